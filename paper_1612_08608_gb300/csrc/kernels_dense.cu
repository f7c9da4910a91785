// Local SGD step of dense softmax regression on bf16 features (the dense
// variant of Eq. A.1, first line), on the 5th-generation tensor cores.
//
//   forward  Z = X_b W^T           X_b [B x d] bf16, W [C x d] (bf16 copy of the fp32 master)
//            R = (softmax(Z) - onehot(y)) / B   -> bf16, stored transposed R^T [C x B]
//   gradient G = R^T X_b           [C x d], fp32 accumulate
//            W_half = (1 - eta l2) W - eta G    (fp32 master, in place), then NOTIFY
//
// Both GEMMs use 128 x 256 output tiles and are persistent and
// warp-specialised: one lane issues TMA loads (128-byte swizzled, K-major
// tiles of 64 bf16) into a ring of stages guarded by full/empty mbarriers;
// another issues tcgen05.mma (M=128, N=256, K=16, bf16 x bf16 -> fp32 in
// TMEM) into one of two accumulators and commits each stage back to its empty
// barrier; epilogue warps (eight in the forward kernel, four in the gradient
// kernel) drain the other accumulator meanwhile (a warp reaches the TMEM
// lanes 32 (w mod 4) .. + 31, i.e. tile rows).
//
// Softmax needs all C logits of a row, more than one CTA's 256 TMEM
// columns: the forward kernel runs as a cluster of ceil(C/256) CTAs along
// the classes, and the CTAs exchange per-row maxima and exp-sums through
// distributed shared memory.
//
// Every wait is time-limited; a wait that runs out records an error in the
// context's device state, and the CTA still passes every barrier and frees
// its TMEM before returning.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "asap_internal.h"

namespace asap {

namespace {

constexpr int kTileM = 128;
constexpr int kTileN = 256;
constexpr int kTileK = 64;                  // one 128-byte swizzle row of bf16
// Operand stages of the TMA -> tcgen05 rings (48 KB each).
constexpr int kFwdStages = 4;
constexpr int kGradStages = 2;
constexpr uint32_t kABytes = kTileM * kTileK * 2;   // 16 KB
constexpr uint32_t kBBytes = kTileN * kTileK * 2;   // 32 KB
constexpr uint32_t kTmemCols = 256;
// Gradient epilogue: the fp32 master tile [128 classes x 256 features] passes
// through shared memory as 8 chunks of 32 columns (128-byte swizzled rows).
constexpr int kWBoxCols = 32;
constexpr uint32_t kWBoxBytes = kTileM * kWBoxCols * 4;          // 16 KB
constexpr unsigned long long kWaitNs = 2000000000ull;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long now_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = now_ns();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (now_ns() - t0 > kWaitNs) return false;
  }
}

__device__ __forceinline__ void tma_2d(void* dst, const CUtensorMap* m, uint64_t* bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(smem_u32(bar)) : "memory");
}

// The same 2-D load, written to the same shared-memory offset of every CTA of
// the cluster in `mask` and completing on the mbarrier at `bar`'s offset in
// each of them (the CTAs read the same tile of this GPU's memory).
__device__ __forceinline__ void tma_2d_multicast(void* dst, const CUtensorMap* m, uint64_t* bar, int x, int y,
                                                 uint16_t mask) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.multicast::cluster"
      " [%0], [%1, {%2, %3}], [%4], %5;"
      :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(smem_u32(bar)), "h"(mask)
      : "memory");
}

__device__ __forceinline__ void tma_3d(void* dst, const CUtensorMap* m, uint64_t* bar, int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];"
      :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tma_store_3d(const CUtensorMap* m, const void* src, int x, int y, int z) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];"
               :: "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(src)) : "memory");
}

// --- tcgen05 -----------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" :: "r"(smem_u32(slot)),
               "r"(ncols) : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" :: "r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, fp32 accumulator).
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
      :: "r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate) : "memory");
}

// Arrive on `bar` once every tcgen05.mma issued so far by this thread is done.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" :: "r"(smem_u32(bar))
               : "memory");
}

// The same arrival on the mbarrier at `bar`'s offset in every CTA of the
// cluster in `mask`.
__device__ __forceinline__ void umma_commit_multicast(uint64_t* bar, uint16_t mask) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;"
               :: "r"(smem_u32(bar)), "h"(mask) : "memory");
}

// 32 consecutive fp32 accumulator columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}

// Shared-memory matrix descriptor: K-major tile, rows of 128 bytes, 128-byte
// swizzle (the layout TMA writes with CU_TENSOR_MAP_SWIZZLE_128B), 8-row
// groups 1024 bytes apart.
__device__ __forceinline__ uint64_t smem_desc_sw128(const void* p) {
  const uint32_t a = smem_u32(p);
  uint64_t d = 0;
  d |= static_cast<uint64_t>((a & 0x3FFFFu) >> 4);     // start address
  d |= static_cast<uint64_t>(1) << 16;                  // leading byte offset (unused for this layout)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;          // stride byte offset: 8 rows x 128 B
  d |= static_cast<uint64_t>(1) << 46;                  // descriptor version for tcgen05
  d |= static_cast<uint64_t>(2) << 61;                  // 128-byte swizzle
  return d;
}

// Instruction descriptor: bf16 A and B (K-major), fp32 D, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

__device__ __forceinline__ void record_error(DevState* st, unsigned code, unsigned worker, unsigned round) {
  if (atomicCAS(&st->err_code, 0u, code) == 0u) {
    st->err_worker = worker;
    st->err_round = round;
  }
}

// --- cluster helpers ----------------------------------------------------
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Store to the shared memory of cluster CTA `rank`, at `local`'s offset.
__device__ __forceinline__ void st_dsmem_f32(float* local, uint32_t rank, float v) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.f32 [%0], %1;" :: "r"(remote), "f"(v) : "memory");
}

// Offset of the first 1024-byte aligned byte of the dynamic shared memory.
// Regions are then formed from the base pointer by pointer arithmetic (no
// integer round trip of the address), so that the compiler keeps them in
// the shared address space and emits plain shared-memory accesses.
__device__ __forceinline__ size_t align1024_off(const unsigned char* raw) {
  return (1024u - (smem_u32(raw) & 1023u)) & 1023u;
}

// Relaxed arrival on the mbarrier at `local`'s offset in the shared memory of
// cluster CTA `rank` (order earlier writes with a release fence first).
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint64_t* local, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" :: "r"(remote) : "memory");
}

// Time-limited wait on a local mbarrier whose arrivals come from other CTAs
// of the cluster (acquire at cluster scope: their prior writes are visible).
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity) {
  const unsigned long long t0 = now_ns();
  for (;;) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
    if (ok) return true;
    if (now_ns() - t0 > kWaitNs) return false;
  }
}

// Barrier among the epilogue warps (barrier 1) that also returns the OR of
// `v` over them, so that they take every decision together.
constexpr int kEpiWarps = 16;                          // forward epilogue warps: four per TMEM lane quarter
constexpr int kEpiParts = kEpiWarps / 4;               // column parts of a row
constexpr int kEpiChunks = kTileN / 32 / kEpiParts;    // 32-column chunks per epilogue thread

__device__ __forceinline__ bool epi_bar_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, %2, p;\n selp.u32 %0, 1, 0, q;\n}"
      : "=r"(r) : "r"(static_cast<uint32_t>(v)), "n"(kEpiWarps * 32) : "memory");
  return r != 0;
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, %0;" :: "n"(kEpiWarps * 32) : "memory"); }

// ----------------------------------------------------------------------------
// Forward: logits, softmax across the cluster, R^T, loss partials.
//
// Persistent clusters of Cq = ceil(C/256) CTAs, one CTA per SM; CTA rank q
// owns classes [256q, 256q+256) of every row tile (i, mt) its cluster walks
// (row tiles cluster, cluster + n_clusters, ...).  Per CTA:
//   warp 0      TMA producer of the operand ring (X and W k-tiles);
//   warp 1      tcgen05.mma issuer into one of two TMEM accumulators, so the
//               next row tile's GEMM runs while this one's epilogue drains;
//   warps 2-9   epilogue, two threads per row (128 columns each): a single
//               pass over their logits gives a running max m and sum of
//               exp(z - m); each thread stores its (m, s) into every cluster
//               CTA's double-buffered slot (remote shared-memory stores, then
//               a release arrival on that CTA's "full" mbarrier; "free"
//               mbarriers guard a slot's reuse), so that the combination
//               reads local shared memory; then R = (softmax - onehot) / B is
//               written to R^T from registers.
constexpr int kFwdThreads = (2 + kEpiWarps) * 32;
// X tiles are loaded in 32-row parts (4 KB each, 1024-byte aligned under the 128-byte swizzle)
constexpr int kXPart = 32;
constexpr uint32_t kXPartBytes = kXPart * kTileK * 2;
constexpr int kMaxCq = 4;                                       // C <= 1024
constexpr int kStatsSlot = kMaxCq * kEpiParts * 2 * kTileM;     // floats per stats slot

struct FwdSmem {
  unsigned char* a;      // kFwdStages x kABytes
  unsigned char* b;      // kFwdStages x kBBytes
  float* stats;          // [2 slots][kMaxCq source CTAs][kEpiParts][2: m, s][128 rows]
  uint64_t* full;        // [kFwdStages]
  uint64_t* empty;       // [kFwdStages]
  uint64_t* acc_full;    // [2]
  uint64_t* acc_empty;   // [2]
  uint64_t* st_full;     // [2]: every cluster CTA's (m, s) of the slot are written
  uint64_t* st_free;     // [2]: every cluster CTA has read the slot
  uint32_t* tmem_slot;
  float* red;            // [kEpiWarps]
};

constexpr size_t fwd_smem_bytes() {
  return 1024 + static_cast<size_t>(kFwdStages) * (kABytes + kBBytes) + 4 * kStatsSlot * 2 + 8 * (2 * kFwdStages + 8) + 16 + 4 * kEpiWarps;
}

__device__ __forceinline__ FwdSmem fwd_carve(unsigned char* raw) {
  size_t p = align1024_off(raw);
  FwdSmem s;
  s.a = raw + p;
  p += kFwdStages * kABytes;
  s.b = raw + p;
  p += kFwdStages * kBBytes;
  s.stats = reinterpret_cast<float*>(raw + p);
  p += 4 * kStatsSlot * 2;
  s.full = reinterpret_cast<uint64_t*>(raw + p);
  s.empty = s.full + kFwdStages;
  s.acc_full = s.empty + kFwdStages;
  s.acc_empty = s.acc_full + 2;
  s.st_full = s.acc_empty + 2;
  s.st_free = s.st_full + 2;
  p += 8 * (2 * kFwdStages + 8);
  s.tmem_slot = reinterpret_cast<uint32_t*>(raw + p);
  p += 16;
  s.red = reinterpret_cast<float*>(raw + p);
  return s;
}

__global__ void __launch_bounds__(kFwdThreads, 1)
    k_dense_fwd(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW, DenseFwdArgs a) {
  extern __shared__ unsigned char smem_raw[];
  const FwdSmem sm = fwd_carve(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Cq = a.Cq, q = static_cast<int>(blockIdx.x) % Cq, cl_id = static_cast<int>(blockIdx.x) / Cq;
  const int n_clusters = static_cast<int>(gridDim.x) / Cq;
  const int MT = a.B / kTileM;
  const int total = a.N * MT;                                   // row tiles
  const int n_my = total > cl_id ? (total - cl_id + n_clusters - 1) / n_clusters : 0;
  const int k_tiles = a.d / kTileK;
  const int c0 = q * kTileN;
  const uint16_t cmask = static_cast<uint16_t>((1u << Cq) - 1u);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kFwdStages; ++s) {
      mbar_init(sm.full + s, 1);
      mbar_init(sm.empty + s, Cq);                         // every cluster CTA's MMA is done with the stage
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(sm.acc_full + s, 1);
      mbar_init(sm.acc_empty + s, kEpiWarps);            // one arrival per epilogue warp
      mbar_init(sm.st_full + s, kEpiWarps * Cq);         // every epilogue warp of every cluster CTA
      mbar_init(sm.st_free + s, kEpiWarps * Cq);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(sm.tmem_slot, 2 * kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  cluster_sync();   // every CTA's barriers exist before any remote arrival
  const uint32_t tmem = *sm.tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      long long g = 0;
      bool ok = true;
      for (int n = 0; n < n_my && ok; ++n) {
        const int rt_i = cl_id + n * n_clusters, i = rt_i / MT, mt = rt_i - i * MT;
        const int row0 = (i * a.nb + a.t) * a.B + mt * kTileM;   // row of X
        for (int kt = 0; kt < k_tiles; ++kt, ++g) {
          const int s = static_cast<int>(g % kFwdStages);
          if (g >= kFwdStages && !mbar_wait(sm.empty + s, static_cast<uint32_t>(((g / kFwdStages) - 1) & 1))) {
            record_error(a.st, ASAP_ERR_CUDA, i, a.round);
            ok = false;
            break;
          }
          mbar_expect_tx(sm.full + s, kABytes + kBBytes);
          // The X tile is the same for the cluster's CTAs: each loads its
          // share of the 32-row parts and multicasts it to all of them.
          for (int j = q; j < kTileM / kXPart; j += Cq)
            tma_2d_multicast(sm.a + s * kABytes + j * kXPartBytes, &tmX, sm.full + s, kt * kTileK, row0 + j * kXPart,
                             cmask);
          tma_3d(sm.b + s * kBBytes, &tmW, sm.full + s, kt * kTileK, c0, i);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(kTileM, kTileN);
      long long g = 0;
      bool ok = true;
      for (int n = 0; n < n_my && ok; ++n) {
        const int ab = n & 1;
        if (n >= 2 && !mbar_wait(sm.acc_empty + ab, static_cast<uint32_t>(((n >> 1) - 1) & 1))) {
          record_error(a.st, ASAP_ERR_CUDA, 0xfffffff9u, a.round);
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + static_cast<uint32_t>(ab) * kTmemCols;
        for (int kt = 0; kt < k_tiles; ++kt, ++g) {
          const int s = static_cast<int>(g % kFwdStages);
          if (!mbar_wait(sm.full + s, static_cast<uint32_t>((g / kFwdStages) & 1))) {
            record_error(a.st, ASAP_ERR_CUDA, 0xfffffff9u, a.round);
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < kTileK / 16; ++kk) {
            const uint64_t ad = smem_desc_sw128(sm.a + s * kABytes + kk * 32);
            const uint64_t bd = smem_desc_sw128(sm.b + s * kBBytes + kk * 32);
            umma_bf16(acc, ad, bd, idesc, (kt | kk) != 0 ? 1u : 0u);
          }
          umma_commit_multicast(sm.empty + s, cmask);   // the stage's X parts came from every CTA
        }
        if (ok) umma_commit(sm.acc_full + ab);
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue (warps 2 .. 2 + kEpiWarps - 1) ----------------
    const int ew = warp - 2;
    const int quarter = warp & 3;                               // TMEM lanes 32*quarter .. +31
    const int part = ew >> 2;                                   // columns [128 part, 128 part + 128)
    const int r = quarter * 32 + lane;                          // row within the tile
    const int ch0 = part * kEpiChunks;
    const bool issuer = ew == 0 && lane == 0;
    float v[32];
    for (int n = 0; n < n_my; ++n) {
      const int ab = n & 1, slot = n & 1;
      const int rt_i = cl_id + n * n_clusters, i = rt_i / MT, mt = rt_i - i * MT;
      bool ok = mbar_wait(sm.acc_full + ab, static_cast<uint32_t>((n >> 1) & 1));
      if (epi_bar_or(!ok)) {
        if (issuer) record_error(a.st, ASAP_ERR_CUDA, 0xfffffff8u, a.round);
        break;
      }
      tc_fence_after();
      const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(ab) * kTmemCols;
      const int yb = a.y[(i * a.nb + a.t) * a.B + mt * kTileM + r];
      // One pass: running max and rescaled exp-sum over this thread's columns.
      float m = -INFINITY, s = 0.f, zy = 0.f;
      for (int ch = ch0; ch < ch0 + kEpiChunks; ++ch) {
        tmem_ld32(trow + ch * 32, v);
        float cm = m;
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (c0 + ch * 32 + j < a.C) cm = fmaxf(cm, v[j]);
        if (cm > -INFINITY) s *= __expf(m - cm);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int c = c0 + ch * 32 + j;
          if (c < a.C) s += __expf(v[j] - cm);
          if (c == yb) zy = v[j];
        }
        m = cm;
      }
      // Exchange (m, s) with the cluster: every peer must have read its slot of
      // tile n-2 before this thread writes into it again.
      ok = n < 2 || mbar_wait_cluster(sm.st_free + slot, static_cast<uint32_t>(((n >> 1) - 1) & 1));
      if (epi_bar_or(!ok)) {
        if (issuer) record_error(a.st, ASAP_ERR_CUDA, 0xfffffff7u, a.round);
        break;
      }
      float* slot_stats = sm.stats + slot * kStatsSlot;
      float* mine = slot_stats + (q * kEpiParts + part) * 2 * kTileM + r;   // this thread's entry, in every CTA
      for (int p = 0; p < Cq; ++p) {
        st_dsmem_f32(mine, static_cast<uint32_t>(p), m);
        st_dsmem_f32(mine + kTileM, static_cast<uint32_t>(p), s);
      }
      __syncwarp();
      if (lane == 0) {
        // One release fence for the warp's stores, then relaxed arrivals.
        asm volatile("fence.acq_rel.cluster;" ::: "memory");
        for (int p = 0; p < Cq; ++p) mbar_arrive_cluster_relaxed(sm.st_full + slot, static_cast<uint32_t>(p));
      }
      ok = mbar_wait_cluster(sm.st_full + slot, static_cast<uint32_t>((n >> 1) & 1));
      if (epi_bar_or(!ok)) {
        if (issuer) record_error(a.st, ASAP_ERR_CUDA, 0xfffffff6u, a.round);
        break;
      }
      float gmax = -INFINITY;
      for (int e = 0; e < Cq * kEpiParts; ++e) gmax = fmaxf(gmax, slot_stats[e * 2 * kTileM + r]);
      float S = 0.f;
      for (int e = 0; e < Cq * kEpiParts; ++e) {
        const float mp = slot_stats[e * 2 * kTileM + r];
        if (mp > -INFINITY) S += slot_stats[(e * 2 + 1) * kTileM + r] * __expf(mp - gmax);
      }
      // Our slot is read: peers may refill it for tile n+2.
      __syncwarp();
      if (lane == 0)
        for (int p = 0; p < Cq; ++p) mbar_arrive_cluster_relaxed(sm.st_free + slot, static_cast<uint32_t>(p));
      const float invS = 1.0f / S;
      // R^T: this thread's row of the tile, class after class (a warp writes 64
      // contiguous bytes per class).
      __nv_bfloat16* rt = reinterpret_cast<__nv_bfloat16*>(a.RT) +
                          (static_cast<int64_t>(i) * Cq * kTileN + c0) * a.B + mt * kTileM + r;
      for (int ch = ch0; ch < ch0 + kEpiChunks; ++ch) {
        tmem_ld32(trow + ch * 32, v);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int cl = ch * 32 + j, c = c0 + cl;
          float rv = 0.f;
          if (c < a.C) rv = (__expf(v[j] - gmax) * invS - (c == yb ? 1.f : 0.f)) * a.inv_B;
          rt[static_cast<int64_t>(cl) * a.B] = __float2bfloat16_rn(rv);
        }
      }
      // The accumulator is free for tile n+2.
      tc_fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(smem_u32(sm.acc_empty + ab))
                                  : "memory");
      // loss of the rows whose label falls in this thread's classes
      const int lo = c0 + ch0 * 32;
      float l = (yb >= lo && yb < lo + kEpiChunks * 32) ? (gmax + __logf(S) - zy) : 0.f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
      if (lane == 0) sm.red[ew] = l;
      epi_bar();
      if (issuer) {
        float lt = 0.f;
        for (int w2 = 0; w2 < kEpiWarps; ++w2) lt += sm.red[w2];
        a.loss_part[(static_cast<int64_t>(i) * MT + mt) * Cq + q] = lt;
      }
      epi_bar();   // sm.red is rewritten by the next tile
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();   // no CTA leaves while peers may still read its slots or arrive on its barriers
  if (warp == 1) tmem_dealloc(tmem, 2 * kTmemCols);
}

// ----------------------------------------------------------------------------
// Gradient and update: G tile [128 classes x 256 features] = R^T X_b, then
// W = (1 - eta l2) W - eta G on the fp32 master.
//
// Persistent and warp-specialised, one CTA per SM walking tiles
// blockIdx.x, blockIdx.x + gridDim.x, ...:
//   warp 0      TMA producer of the operand ring (R^T and X^T k-tiles);
//   warp 1      tcgen05.mma issuer into one of two TMEM accumulators
//               (2 x 256 columns), so tile n+1's GEMM runs while tile n's
//               epilogue drains the other;
//   warps 2-5   epilogue: each thread updates one row of a 16 KB chunk of
//               the master tile (128 rows x 32 columns) in shared memory and
//               the warp arrives on the chunk's "updated" mbarrier;
//   warp 6      master I/O: TMA loads of the chunks (up to kWBufs ahead),
//               TMA stores of the updated ones, NOTIFY.
// The epilogue warps never wait on each other or on a store; the I/O warp
// alone waits for stores to finish reading a buffer before reloading it.
// The 3-D master map clips rows beyond C, so a tile never touches the next
// worker's rows.  A worker's NOTIFY is published by the CTA that completes
// its last tile, once that tile's stores are complete (checked one tile
// later, so that the I/O warp keeps loading meanwhile).
constexpr int kGradThreads = 224;
constexpr int kIoWarp = 6;
// Master chunks in shared memory: the kernel is bound by master bytes in
// flight, so they take what the 2-stage operand ring leaves (GB300, N=32,
// d=2048, C=1000: 3 stages + 5 chunks 135 us, 2 + 8 129 us, 4 + 2 224 us;
// extra L2 prefetches of later chunks were slower still).
constexpr int kWBufs = 8;
constexpr int kChunksPerTile = kTileN / kWBoxCols;        // 8
constexpr uint32_t kGradTmemCols = 2 * kTmemCols;        // two accumulators

struct GradSmem {
  unsigned char* a;      // kGradStages x kABytes
  unsigned char* b;      // kGradStages x kBBytes
  unsigned char* w;      // kWBufs x kWBoxBytes
  uint64_t* full;        // [kGradStages]
  uint64_t* empty;       // [kGradStages]
  uint64_t* acc_full;    // [2]
  uint64_t* acc_empty;   // [2]
  uint64_t* wfull;       // [kWBufs]: chunk loaded
  uint64_t* wupd;        // [kWBufs]: chunk updated by the four epilogue warps
  uint32_t* tmem_slot;
  int* fail;
};

constexpr size_t grad_smem_bytes() {
  return 1024 + static_cast<size_t>(kGradStages) * (kABytes + kBBytes) + static_cast<size_t>(kWBufs) * kWBoxBytes +
         8 * (2 * kGradStages + 4 + 2 * kWBufs) + 16 + 16;
}

__device__ __forceinline__ GradSmem grad_carve(unsigned char* raw) {
  size_t p = align1024_off(raw);
  GradSmem s;
  s.a = raw + p;
  p += kGradStages * kABytes;
  s.b = raw + p;
  p += kGradStages * kBBytes;
  s.w = raw + p;
  p += kWBufs * kWBoxBytes;
  s.full = reinterpret_cast<uint64_t*>(raw + p);
  s.empty = s.full + kGradStages;
  s.acc_full = s.empty + kGradStages;
  s.acc_empty = s.acc_full + 2;
  s.wfull = s.acc_empty + 2;
  s.wupd = s.wfull + kWBufs;
  p += 8 * (2 * kGradStages + 4 + 2 * kWBufs);
  s.tmem_slot = reinterpret_cast<uint32_t*>(raw + p);
  p += 16;
  s.fail = reinterpret_cast<int*>(raw + p);
  return s;
}

struct GradTile {
  int i, mt, nt;
};

__device__ __forceinline__ GradTile grad_tile(long long tau, int MT, int NT) {
  GradTile t;
  const long long per = static_cast<long long>(MT) * NT;
  t.i = static_cast<int>(tau / per);
  const int rem = static_cast<int>(tau - static_cast<long long>(t.i) * per);
  t.mt = rem / NT;
  t.nt = rem - t.mt * NT;
  return t;
}

__global__ void __launch_bounds__(kGradThreads, 1)
    k_dense_grad(const __grid_constant__ CUtensorMap tmR, const __grid_constant__ CUtensorMap tmXT,
                 const __grid_constant__ CUtensorMap tmWf, DenseGradArgs a) {
  extern __shared__ unsigned char smem_raw[];
  const GradSmem sm = grad_carve(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int MT = (a.C + kTileM - 1) / kTileM, NT = a.d / kTileN;
  const long long total = static_cast<long long>(a.N) * MT * NT;
  const int n_tiles = total > blockIdx.x ? static_cast<int>((total - blockIdx.x + gridDim.x - 1) / gridDim.x) : 0;
  const int k_tiles = a.B / kTileK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kGradStages; ++s) {
      mbar_init(sm.full + s, 1);
      mbar_init(sm.empty + s, 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(sm.acc_full + s, 1);
      mbar_init(sm.acc_empty + s, 4);   // one arrival per epilogue warp
    }
    for (int s = 0; s < kWBufs; ++s) {
      mbar_init(sm.wfull + s, 1);
      mbar_init(sm.wupd + s, 4);
    }
    *sm.fail = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(sm.tmem_slot, kGradTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *sm.tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      long long g = 0;   // k-tile counter over all of this CTA's tiles
      bool ok = true;
      for (int n = 0; n < n_tiles && ok; ++n) {
        const GradTile t = grad_tile(blockIdx.x + static_cast<long long>(n) * gridDim.x, MT, NT);
        const int a_row = t.i * a.Cq * kTileN + t.mt * kTileM;          // row of R^T
        const int b_row = (t.i * a.nb + a.t) * a.d + t.nt * kTileN;     // row of X^T
        for (int kt = 0; kt < k_tiles; ++kt, ++g) {
          const int s = static_cast<int>(g % kGradStages);
          if (g >= kGradStages && !mbar_wait(sm.empty + s, static_cast<uint32_t>(((g / kGradStages) - 1) & 1))) {
            record_error(a.st, ASAP_ERR_CUDA, t.i, a.round);
            atomicOr(sm.fail, 1);
            ok = false;
            break;
          }
          mbar_expect_tx(sm.full + s, kABytes + kBBytes);
          tma_2d(sm.a + s * kABytes, &tmR, sm.full + s, kt * kTileK, a_row);
          tma_2d(sm.b + s * kBBytes, &tmXT, sm.full + s, kt * kTileK, b_row);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(kTileM, kTileN);
      long long g = 0;
      bool ok = true;
      for (int n = 0; n < n_tiles && ok; ++n) {
        const int ab = n & 1;
        if (n >= 2 && !mbar_wait(sm.acc_empty + ab, static_cast<uint32_t>(((n >> 1) - 1) & 1))) {
          record_error(a.st, ASAP_ERR_CUDA, 0xfffffffcu, a.round);
          atomicOr(sm.fail, 1);
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + static_cast<uint32_t>(ab) * kTmemCols;
        for (int kt = 0; kt < k_tiles; ++kt, ++g) {
          const int s = static_cast<int>(g % kGradStages);
          if (!mbar_wait(sm.full + s, static_cast<uint32_t>((g / kGradStages) & 1))) {
            record_error(a.st, ASAP_ERR_CUDA, 0xfffffffcu, a.round);
            atomicOr(sm.fail, 1);
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < kTileK / 16; ++kk) {
            const uint64_t ad = smem_desc_sw128(sm.a + s * kABytes + kk * 32);
            const uint64_t bd = smem_desc_sw128(sm.b + s * kBBytes + kk * 32);
            umma_bf16(acc, ad, bd, idesc, (kt | kk) != 0 ? 1u : 0u);
          }
          umma_commit(sm.empty + s);
        }
        if (ok) umma_commit(sm.acc_full + ab);
      }
    }
    __syncwarp();
  } else if (warp == kIoWarp) {
    // ---------------- master I/O ----------------
    if (lane == 0) {
      const long long n_chunks = static_cast<long long>(n_tiles) * kChunksPerTile;
      auto chunk_xyz = [&](long long h, int& x, int& y, int& z) {
        const GradTile t = grad_tile(blockIdx.x + (h / kChunksPerTile) * gridDim.x, MT, NT);
        x = t.nt * kTileN + static_cast<int>(h % kChunksPerTile) * kWBoxCols;
        y = t.mt * kTileM;
        z = t.i;
      };
      auto load_chunk = [&](long long h) {
        const int b = static_cast<int>(h % kWBufs);
        int x, y, z;
        chunk_xyz(h, x, y, z);
        mbar_expect_tx(sm.wfull + b, kWBoxBytes);
        tma_3d(sm.w + b * kWBoxBytes, &tmWf, sm.wfull + b, x, y, z);
      };
      auto notify = [&](int n) {   // tile n's stores are complete
        const GradTile t = grad_tile(blockIdx.x + static_cast<long long>(n) * gridDim.x, MT, NT);
        asm volatile("fence.proxy.async.global;" ::: "memory");
        __threadfence();
        const unsigned per = static_cast<unsigned>(MT * NT);
        const unsigned done = atomicAdd(&a.worker_ticket[t.i], 1u);
        if (done == per - 1) {
          a.worker_ticket[t.i] = 0u;
          __threadfence();
          if (t.i != a.skip_worker)
            asm volatile("st.release.gpu.global.u32 [%0], %1;" :: "l"(a.ready + t.i), "r"(a.round + 1u) : "memory");
        }
      };
      for (long long h = 0; h < n_chunks && h < kWBufs; ++h) load_chunk(h);
      bool ok = true;
      for (long long h = 0; h < n_chunks; ++h) {
        const int b = static_cast<int>(h % kWBufs);
        if (!mbar_wait(sm.wupd + b, static_cast<uint32_t>((h / kWBufs) & 1))) {
          record_error(a.st, ASAP_ERR_CUDA, 0xfffffffau, a.round);
          atomicOr(sm.fail, 1);
          ok = false;
          break;
        }
        int x, y, z;
        chunk_xyz(h, x, y, z);
        tma_store_3d(&tmWf, sm.w + b * kWBoxBytes, x, y, z);
        asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        const long long n = h / kChunksPerTile;
        if (h % kChunksPerTile == kChunksPerTile - 1 && n >= 1) {
          asm volatile("cp.async.bulk.wait_group 8;" ::: "memory");   // tile n-1's stores are complete
          notify(static_cast<int>(n - 1));
        }
        // Reload the previous chunk's buffer once its store has read it.
        if (h >= 1 && h - 1 + kWBufs < n_chunks) {
          asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
          load_chunk(h - 1 + kWBufs);
        }
      }
      asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
      if (ok && n_tiles > 0) notify(n_tiles - 1);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue (warps 2-5) ----------------
    const int quarter = warp & 3;                             // TMEM lanes 32*quarter .. +31
    const int r = quarter * 32 + lane;                        // tile row (class mt*128 + r)
    bool failed = false;
    for (int n = 0; n < n_tiles && !failed; ++n) {
      const int ab = n & 1;
      if (!__all_sync(0xffffffffu, mbar_wait(sm.acc_full + ab, static_cast<uint32_t>((n >> 1) & 1)))) {
        if (lane == 0) record_error(a.st, ASAP_ERR_CUDA, 0xfffffffbu, a.round);
        failed = true;
        break;
      }
      tc_fence_after();
      const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(ab) * kTmemCols;
      for (int c = 0; c < kChunksPerTile; ++c) {
        const long long h = static_cast<long long>(n) * kChunksPerTile + c;
        const int b = static_cast<int>(h % kWBufs);
        if (!__all_sync(0xffffffffu, mbar_wait(sm.wfull + b, static_cast<uint32_t>((h / kWBufs) & 1)))) {
          if (lane == 0) record_error(a.st, ASAP_ERR_CUDA, 0xfffffffbu, a.round);
          failed = true;
          break;
        }
        float gv[32];
        tmem_ld32(trow + c * kWBoxCols, gv);
        unsigned char* row = sm.w + b * kWBoxBytes + r * 128;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          float4* p = reinterpret_cast<float4*>(row + ((j ^ (r & 7)) << 4));   // 128-byte swizzle
          float4 x = *p;
          x.x = fmaf(-a.lr, gv[4 * j + 0], a.decay * x.x);
          x.y = fmaf(-a.lr, gv[4 * j + 1], a.decay * x.y);
          x.z = fmaf(-a.lr, gv[4 * j + 2], a.decay * x.z);
          x.w = fmaf(-a.lr, gv[4 * j + 3], a.decay * x.w);
          *p = x;
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // the updated rows are visible to TMA
        __syncwarp();
        if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(smem_u32(sm.wupd + b))
                                    : "memory");
      }
      if (failed) break;
      // This accumulator may be overwritten by tile n+2.
      tc_fence_before();
      __syncwarp();
      if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(smem_u32(sm.acc_empty + ab))
                                  : "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, kGradTmemCols);
}

}  // namespace

size_t dense_smem_bytes() { return fwd_smem_bytes(); }

size_t dense_grad_smem_bytes() { return grad_smem_bytes(); }

cudaError_t dense_configure() {
  const int smem = static_cast<int>(dense_smem_bytes());
  cudaError_t e = cudaFuncSetAttribute(k_dense_fwd, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_dense_fwd, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_dense_grad, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(dense_grad_smem_bytes()));
}

// Clusters of `cq` forward CTAs that fit on the device at once (cached).
static int fwd_active_clusters(int cq) {
  static int cache[5] = {0, 0, 0, 0, 0};
  if (cq < 1 || cq > 4) return 0;
  if (cache[cq] == 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cq, 1, 1);
    cfg.blockDim = dim3(kFwdThreads, 1, 1);
    cfg.dynamicSmemBytes = dense_smem_bytes();
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cq;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k_dense_fwd, &cfg) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = 1;
    }
    cache[cq] = n;
  }
  return cache[cq];
}

cudaError_t launch_dense_fwd(const CUtensorMap& tmX, const CUtensorMap& tmW, const DenseFwdArgs& f, int N,
                             cudaStream_t s) {
  DenseFwdArgs fa = f;
  fa.N = N;
  const int row_tiles = N * (f.B / kTileM);
  int clusters = fwd_active_clusters(f.Cq);
  if (clusters > row_tiles) clusters = row_tiles;
  if (clusters < 1) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(f.Cq * clusters, 1, 1);
  cfg.blockDim = dim3(kFwdThreads, 1, 1);
  cfg.dynamicSmemBytes = dense_smem_bytes();
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = f.Cq;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_dense_fwd, tmX, tmW, fa);
}

cudaError_t launch_dense_grad(const CUtensorMap& tmR, const CUtensorMap& tmXT, const CUtensorMap& tmWf,
                              const DenseGradArgs& g, int N, int sm_count, cudaStream_t s) {
  DenseGradArgs ga = g;
  ga.N = N;
  const long long tiles = static_cast<long long>(N) * ((g.C + kTileM - 1) / kTileM) * (g.d / kTileN);
  const int grid = static_cast<int>(tiles < sm_count ? tiles : sm_count);
  if (grid < 1) return cudaSuccess;
  k_dense_grad<<<grid, kGradThreads, dense_grad_smem_bytes(), s>>>(tmR, tmXT, tmWf, ga);
  return cudaGetLastError();
}

}  // namespace asap
