// Local minibatch SGD step for sparse linear models (Eq. A.1, first line),
// one fused kernel per step:
//
//   margins        m_b = sum_e val_e * wv[pos_e]
//                  r_b = d loss(y_b, m_b) / d m_b        (hinge or logistic)
//   column sums    g[p] = sum_{e : pos_e = p} r_{row_e} val_e
//                  then NOTIFY ready[i] = t+1
//
// Each step's minibatch has, per worker, a list of the distinct columns it
// touches.  The lists of all workers are laid out slab-major (by column slab
// of the stochastic reduce, then worker, then column) and `pos` indexes that
// list.  `wv[pos]` holds w_i[col] for the step's columns: the previous
// round's reduce writes it while it holds the column slab in shared memory
// (or, after parameters were written from the host, the gather kernel
// below).  The reduce applies w_i[col] -= eta/B * g[pos] to the slab before
// mixing it, so w_{t+1/2} never has to be written to HBM.
//
// One cluster of Q CTAs per worker (grid N x Q, no inter-cluster waits).
// The minibatch's entries are stored once, sorted by (column, row), and
// streamed twice through a ring of shared-memory stages by an issuer warp
// with bulk copies (cp.async.bulk, mbarrier completion) -- a gather warp
// fetches a margin tile's w values as soon as the tile lands -- while four
// consumer warps work on the stage that has landed, each on its own
// 256-entry share of the 1024-entry tile and without CTA-wide barriers:
//   pass 1 (margins): CTA q takes the 256-entry segments s = q nseg/Q ...
//     in tiles of four; a warp's products val * wv[pos] and their rows go to
//     shared memory at the entry's slot (slots of a 256-entry segment
//     ordered by row, then column), a segmented scan over the slots keyed by
//     row sums each row's products in order, and the warp adds them to its
//     own partial margins.  The four warps' partials are added in order; a
//     cluster barrier; every CTA then adds the Q partials of each row in rank
//     order (distributed shared memory), forms r and, in CTA 0, the loss sum.
//   pass 2 (column sums): CTA q takes the entries [bnd[q], bnd[q+1]), cut
//     at column boundaries, in 1024-entry tiles; a warp's segmented scan
//     keyed by list position sums each column's r_row * val; runs that end
//     inside the warp's share are stored by the warp, and the two runs at
//     its edges are fragments that the gather warp, idle by then, adds up
//     in order.
// A last cluster barrier and CTA 0 publishes NOTIFY.  No atomics, no waits
// on other clusters, every sum in a fixed order: the result does not depend
// on the schedule.  The kernel is a programmatic dependent of the previous
// round's reduce (set-up and the first bulk copies of static batch data run
// while that reduce drains); its registers are bounded for five CTAs per SM.
#include <cuda_runtime.h>

#include <cstdint>

#include "asap_internal.h"

namespace asap {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kConsumers = kLocalStepThreads - 64;          // four consumer warps
constexpr int kPerThread = kTileEntries / kConsumers;       // consecutive entries per consumer thread
static_assert(kPerThread == 8, "a consumer thread takes 8 consecutive entries of a tile");
constexpr unsigned long long kCopyWaitNs = 2000000000ull;   // a bulk copy never takes this long

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

__device__ __forceinline__ void st_release_u32(unsigned int* p, unsigned int v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ unsigned long long globaltimer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}

// Time-limited wait on an mbarrier phase; false if the limit ran out.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned n = 1;; ++n) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((n & 255u) == 0 && globaltimer_ns() - t0 > kCopyWaitNs) return false;
  }
}

// 4-byte asynchronous copy global -> shared (a gather), and an arrival on an
// mbarrier once all of this thread's earlier such copies have landed.
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src))
               : "memory");
}

__device__ __forceinline__ void cp_async_arrive(uint64_t* bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" :: "r"(smem_u32(bar)) : "memory");
}

// Untiled bulk copy global -> shared (16-byte aligned, size a multiple of 16).
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_id_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}

// Load of `local`'s offset in the shared memory of cluster CTA `rank`.
__device__ __forceinline__ float ld_dsmem(const float* local, uint32_t rank) {
  uint32_t remote;
  float v;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(remote) : "memory");
  return v;
}

// Barrier among the consumer warps only (the producer warp keeps streaming).
__device__ __forceinline__ void consumer_bar() {
  asm volatile("bar.sync 1, %0;" :: "n"(kConsumers) : "memory");
}

__device__ __forceinline__ void record_error(DevState* st, unsigned code, unsigned worker, unsigned round) {
  if (atomicCAS(&st->err_code, 0u, code) == 0u) {
    st->err_worker = worker;
    st->err_round = round;
  }
}

// loss(y, m) and r = d loss / d m.
template <int LOSS>
__device__ __forceinline__ void loss_and_r(float y, float m, float& l, float& r) {
  const float z = y * m;
  if (LOSS == ASAP_LOSS_HINGE) {
    l = fmaxf(0.f, 1.f - z);
    r = (z < 1.f) ? -y : 0.f;                 // strict: the corner z = 1 takes r = 0
  } else {
    // ln(1 + e^{-z}) = max(-z, 0) + ln(1 + e^{-|z|});  sigmoid(-z) = 1 / (1 + e^{z})
    l = fmaxf(-z, 0.f) + log1pf(expf(-fabsf(z)));
    r = -y / (1.f + expf(z));
  }
}

// Shared-memory layout of the local-step kernel (mirrored by
// local_step_smem_bytes): the ring of stages, each holding one tile's list
// positions, values and two uint16 arrays (pass 1: slots and rows; pass 2:
// rows), a margin tile's positions replaced in place by the gathered w
// values;
// per consumer warp a 256-entry scratch (pass 1: products and rows by slot;
// pass 2: run sums and their list positions); the per-warp partial margins and r
// of the worker's B rows; the column-run fragments at sub-tile edges.
struct StepSmem {
  unsigned char* stage0;
  uint64_t* full;
  uint64_t* empty;
  uint64_t* gath;       // [stages]: the w values of a margin tile are in the stage
  uint64_t* fready;     // [kFragRing]: every warp has left its fragments of a column-sum tile
  uint64_t* ffree;      // [kFragRing]: the merger has read a slot's fragments
  float* prod;          // [kTileEntries]: warp w uses [256 w, 256 w + 256)
  int* okey;            // [kTileEntries]: list position of a run ending at the pair, else -1
  float* mpart;         // [4][B]: per-warp partial margins (warp 0's row holds the CTA's sum after pass 1)
  float* r;             // [B]
  int* fkey;            // [kFragRing][4][2]: first / last column-run fragment of each warp's sub-tile
  float* fval;          // [kFragRing][4][2]
  float* red;           // [kConsumers / 32]
  int* ctl;             // [1]: a copy timed out
};

// pos (in margin tiles overwritten by the gathered w values), val and two
// uint16 arrays
constexpr size_t kStageBytes = static_cast<size_t>(kTileEntries) * 12;
constexpr int kWarps = kConsumers / 32;
constexpr int kIssuerWarp = kWarps, kGatherWarp = kWarps + 1;
// Fragments of a column-sum tile wait in a ring until the merger (the gather
// warp, idle in pass 2) has added them up; a consumer waits for the slot's
// "free" barrier before it reuses it.
constexpr int kFragRing = 8;
constexpr int kNoKey = -2;

// Every region is formed from `raw` by pointer arithmetic (offsets only, no
// integer round trip of the address), so that the compiler keeps the
// pointers in the shared address space and emits plain shared-memory
// accesses.
__device__ __forceinline__ StepSmem carve_step(unsigned char* raw, int B, int stages) {
  StepSmem m;
  size_t off = (128u - (smem_u32(raw) & 127u)) & 127u;   // 128-byte aligned stages
  m.stage0 = raw + off;
  off += kStageBytes * stages;
  m.full = reinterpret_cast<uint64_t*>(raw + off);
  off += 8 * stages;
  m.empty = reinterpret_cast<uint64_t*>(raw + off);
  off += 8 * stages;
  m.gath = reinterpret_cast<uint64_t*>(raw + off);
  off += 8 * stages;
  m.fready = reinterpret_cast<uint64_t*>(raw + off);
  off += 8 * kFragRing;
  m.ffree = reinterpret_cast<uint64_t*>(raw + off);
  off += 8 * kFragRing;
  off = (off + 15) & ~static_cast<size_t>(15);             // prod and okey are accessed as 16-byte vectors
  m.prod = reinterpret_cast<float*>(raw + off);
  off += 4 * kTileEntries;
  m.okey = reinterpret_cast<int*>(raw + off);
  off += 4 * kTileEntries;
  m.mpart = reinterpret_cast<float*>(raw + off);
  off += 4 * static_cast<size_t>(kWarps) * B;
  m.r = reinterpret_cast<float*>(raw + off);
  off += 4 * static_cast<size_t>(B);
  off = (off + 15) & ~static_cast<size_t>(15);             // fragments are read as 16-byte vectors
  m.fkey = reinterpret_cast<int*>(raw + off);
  off += 4 * kFragRing * kWarps * 2;
  m.fval = reinterpret_cast<float*>(raw + off);
  off += 4 * kFragRing * kWarps * 2;
  m.red = reinterpret_cast<float*>(raw + off);
  off += 4 * kWarps;
  m.ctl = reinterpret_cast<int*>(raw + off);
  return m;
}

// Segmented inclusive scan over one warp's sub-tile: lane l holds the eight
// consecutive pairs 8l .. 8l+7 (key, value); a run is a maximal stretch of
// equal keys, and nothing is carried in from before the sub-tile.  On
// return val[u] is the sum of its run's values from the run's first pair in
// the sub-tile up to and including pair u; next_key is the key of the pair
// after this lane's last (kNoKey after the sub-tile's last pair).  Fixed
// order of additions: within a lane left to right, then a fixed shuffle
// tree over the lanes.
__device__ __forceinline__ void seg_scan_warp(const int (&key)[kPerThread], float (&val)[kPerThread], int& next_key) {
  const int lane = threadIdx.x & 31;
  int prev_key = __shfl_up_sync(kFull, key[kPerThread - 1], 1);
  if (lane == 0) prev_key = kNoKey - 1;
  next_key = __shfl_down_sync(kFull, key[0], 1);
  if (lane == 31) next_key = kNoKey;
  bool any_head = false;
  int pk = prev_key;
#pragma unroll
  for (int u = 0; u < kPerThread; ++u) {
    const bool head = key[u] != pk;
    if (u > 0 && !head) val[u] += val[u - 1];
    any_head = any_head || head;
    pk = key[u];
  }
  // inclusive scan over the lanes of (a head seen, running value of the last run)
  float v = val[kPerThread - 1];
  int f = any_head ? 1 : 0;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float vo = __shfl_up_sync(kFull, v, off);
    const int fo = __shfl_up_sync(kFull, f, off);
    if (lane >= off) {
      if (!f) v += vo;
      f |= fo;
    }
  }
  const float ev = __shfl_up_sync(kFull, v, 1);   // the run through the previous lane's last pair
  if (lane > 0) {
    pk = prev_key;
#pragma unroll
    for (int u = 0; u < kPerThread; ++u) {        // pairs before this lane's first head
      if (key[u] != pk) break;
      val[u] += ev;
      pk = key[u];
    }
  }
}

template <int LOSS>
__global__ void __launch_bounds__(kLocalStepThreads, 5) k_local_step(const LocalStepArgs a) {   // five CTAs per SM
  extern __shared__ unsigned char step_smem_raw[];
  const bool big = a.B > kRSmemRows;           // partial margins and r in global memory
  const StepSmem sm = carve_step(step_smem_raw, big ? 0 : a.B, a.stages);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q = static_cast<int>(cluster_rank());
  const int Q = a.Q;
  const int cl = static_cast<int>(cluster_id_x());
  const int i = a.worker_of ? a.worker_of[cl] : cl;
  const BatchDesc dsc = a.desc[i];
  const int nnz = dsc.nnz;
  // Pass 1: CTA q takes the 256-entry slot segments [s0, s1) in tiles of up
  // to four (the CTAs' shares differ by at most one segment).
  const int nseg = (nnz + kSlotSegment - 1) / kSlotSegment;
  const int s0 = static_cast<int>(static_cast<long long>(q) * nseg / Q);
  const int s1 = static_cast<int>(static_cast<long long>(q + 1) * nseg / Q);
  constexpr int kSegsPerTile = kTileEntries / kSlotSegment;
  const int n1 = (s1 - s0 + kSegsPerTile - 1) / kSegsPerTile;
  const int p1_begin = s0 * kSlotSegment, p1_end = min(s1 * kSlotSegment, nnz);
  const int* bnd = reinterpret_cast<const int*>(a.block + dsc.bnd);
  const int lo = bnd[q], hi = bnd[q + 1];
  const int T0 = lo & ~7;                      // 16-byte aligned start of the first column tile
  const int n2 = hi > lo ? (hi - T0 + kTileEntries - 1) / kTileEntries : 0;
  // per-warp partial margins (warp w's row at w B) and r: in shared memory,
  // or for large minibatches in global scratch; the two kinds of pointer
  // are kept apart so that shared accesses stay shared-memory instructions
  float* gpart = a.mpart_big + (static_cast<size_t>(i) * Q + q) * kWarps * a.B;
  float* grr = a.r_big + (static_cast<size_t>(i) * Q + q) * a.B;

  if (tid == 0) {
    for (int st = 0; st < a.stages; ++st) {
      mbar_init(sm.full + st, 1);
      mbar_init(sm.empty + st, kWarps);
      mbar_init(sm.gath + st, 32);
    }
    for (int f = 0; f < kFragRing; ++f) {
      mbar_init(sm.fready + f, kWarps);
      mbar_init(sm.ffree + f, 1);
    }
    sm.ctl[0] = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  for (int b = tid; b < kWarps * a.B; b += kLocalStepThreads) {
    if (big) gpart[b] = 0.f;
    else sm.mpart[b] = 0.f;
  }
  __syncthreads();
  // The stochastic reduce that follows is a programmatic dependent: its CTAs
  // may take SMs as this grid drains; it waits for this grid's results.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  // This grid is itself a programmatic dependent of the previous round's
  // reduce, which may still be running: everything above and the issuer's
  // bulk copies touch only this step's own (static) batch block; the gather
  // and consumer warps wait for the previous grid before they read the
  // exported w values or write anything it reads (column sums, loss).

  bool ok = true;
  if (warp == kIssuerWarp) {
    // ================= issuer warp =================
    // Lane 0 issues every tile of both passes in order as stages come free;
    // the warp arrives on the cluster barrier between the passes once pass 1
    // is issued, so that it never holds up the consumers there.
    auto issue = [&](int it) -> bool {
      const int st = it % a.stages;
      if (it >= a.stages && !mbar_wait_bounded(sm.empty + st, ((it / a.stages) - 1) & 1)) return false;
      unsigned char* base = sm.stage0 + kStageBytes * st;
      const bool pass1 = it < n1;
      const int e0 = pass1 ? p1_begin + it * kTileEntries : T0 + (it - n1) * kTileEntries;
      const int len = min(kTileEntries, (pass1 ? p1_end : hi) - e0);
      const uint32_t n8 = static_cast<uint32_t>((len + 7) & ~7);   // whole 16-byte rows of uint16
      mbar_expect_tx(sm.full + st, n8 * (pass1 ? 12u : 10u));
      bulk_load(base, a.block + dsc.cpos + 4 * static_cast<int64_t>(e0), 4 * n8, sm.full + st);
      bulk_load(base + 4 * kTileEntries, a.block + dsc.cval + 4 * static_cast<int64_t>(e0), 4 * n8, sm.full + st);
      if (pass1) {
        bulk_load(base + 8 * kTileEntries, a.block + dsc.cslot + 2 * static_cast<int64_t>(e0), 2 * n8, sm.full + st);
        bulk_load(base + 10 * kTileEntries, a.block + dsc.crow + 2 * static_cast<int64_t>(e0), 2 * n8, sm.full + st);
      } else {
        bulk_load(base + 8 * kTileEntries, a.block + dsc.crow + 2 * static_cast<int64_t>(e0), 2 * n8, sm.full + st);
      }
      return true;
    };
    bool pok = true;
    if (lane == 0)
      for (int it = 0; it < n1 && pok; ++it) pok = issue(it);
    __syncwarp();
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
    if (lane == 0) {
      for (int it = n1; it < n1 + n2 && pok; ++it) pok = issue(it);
      if (!pok) sm.ctl[0] = 1;
    }
    __syncwarp();
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
  } else if (warp == kGatherWarp) {
    // ================= gather warp =================
    // As soon as margin tile k has landed, every lane gathers 32 of its w
    // values with 4-byte asynchronous copies, each over the list position
    // it was addressed by (read before the copy is issued), and arrives on
    // gath[k] when they are in: the gathers of the next tiles run while the
    // consumers work on this one.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    bool gok = true;
    for (int k = 0; k < n1 && gok; ++k) {
      const int st = k % a.stages;
      gok = __all_sync(kFull, mbar_wait_bounded(sm.full + st, (k / a.stages) & 1));
      if (!gok) break;
      int* spos = reinterpret_cast<int*>(sm.stage0 + kStageBytes * st);
      const int len = min(kTileEntries, p1_end - (p1_begin + k * kTileEntries));
      // four consecutive positions per lane and vector load, two loads ahead
      // of their copies, so that no copy waits on its own position's load
      for (int j0 = lane * 4; j0 < len; j0 += 256) {
        const int j1 = j0 + 128;
        const int4 p0 = *reinterpret_cast<const int4*>(spos + j0);
        const int4 p1 = j1 < len ? *reinterpret_cast<const int4*>(spos + j1) : make_int4(0, 0, 0, 0);
        const int pp[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int j = (u < 4 ? j0 : j1) + (u & 3);
          if (j < len) cp_async4(spos + j, a.wv + pp[u]);
        }
      }
      cp_async_arrive(sm.gath + st);
    }
    if (!gok && lane == 0) sm.ctl[0] = 1;
    __syncwarp();
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
    // ---- pass 2: the column runs at the edges of the consumer warps' shares,
    // added up in share order as every warp leaves a tile's fragments ----
    float* g = a.gsum;
    int open_key = kNoKey;                     // lane 0: the run the fragments continue
    float open_sum = 0.f;
    bool mok = gok;
    for (int k = 0; k < n2 && mok; ++k) {
      const int slot = k % kFragRing;
      mok = __all_sync(kFull, mbar_wait_bounded(sm.fready + slot, (k / kFragRing) & 1));
      if (!mok) break;
      if (lane == 0) {
        static_assert(kWarps * 2 == 8, "a tile leaves eight fragments");
        const int fb = slot * kWarps * 2;
        const int4 k0 = *reinterpret_cast<const int4*>(sm.fkey + fb);
        const int4 k1 = *reinterpret_cast<const int4*>(sm.fkey + fb + 4);
        const float4 v0 = *reinterpret_cast<const float4*>(sm.fval + fb);
        const float4 v1 = *reinterpret_cast<const float4*>(sm.fval + fb + 4);
        const int fks[8] = {k0.x, k0.y, k0.z, k0.w, k1.x, k1.y, k1.z, k1.w};
        const float fvs[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        mbar_arrive(sm.ffree + slot);          // the slot is read
#pragma unroll
        for (int f = 0; f < 8; ++f) {
          const int fk = fks[f];
          if (fk == kNoKey) continue;
          const float fv = fvs[f];
          if (fk == open_key) {
            open_sum += fv;
          } else {
            if (open_key >= 0) g[open_key] = open_sum;
            open_key = fk;
            open_sum = fv;
          }
        }
      }
      __syncwarp();
    }
    if (lane == 0 && mok && open_key >= 0) g[open_key] = open_sum;
    if (!mok && lane == 0) {
      record_error(a.st, ASAP_ERR_CUDA, static_cast<unsigned>(i), a.round);
      sm.ctl[0] = 1;
    }
  } else {
    // ================= consumer warps =================
    // Warp w takes entries [256 w, 256 w + 256) of every tile (its sub-tile)
    // and works through the tiles on its own: it meets the other consumer
    // warps only at the ring's mbarriers and between the passes.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int sub = warp * kSlotSegment;       // the warp's sub-tile within a tile
    const int j0 = sub + lane * kPerThread;    // this lane's eight consecutive pairs
    float* wprod = sm.prod + sub;
    int* wokey = sm.okey + sub;
    uint16_t* wrows = reinterpret_cast<uint16_t*>(wokey);   // pass 1: the row of every slot
    const size_t wrow = static_cast<size_t>(warp) * a.B;   // this warp's partial margins
    // ---- pass 1: products by slot; each row's sum by a scan over the slots ----
    for (int it = 0; it < n1; ++it) {
      const int st = it % a.stages;
      ok = __all_sync(kFull, mbar_wait_bounded(sm.gath + st, (it / a.stages) & 1));
      if (!ok) break;
      const unsigned char* base = sm.stage0 + kStageBytes * st;
      const float* sval = reinterpret_cast<const float*>(base + 4 * kTileEntries);
      const uint16_t* sslot = reinterpret_cast<const uint16_t*>(base + 8 * kTileEntries);
      const uint16_t* scrow = reinterpret_cast<const uint16_t*>(base + 10 * kTileEntries);   // the entries' rows
      const float* wvs = reinterpret_cast<const float*>(base);   // gathered over the positions
      const int len = min(kTileEntries, p1_end - (p1_begin + it * kTileEntries));
      const bool active = sub < len;           // warp-uniform
      int key[kPerThread];
      float val[kPerThread];
      if (active) {
#pragma unroll
        for (int u = 0; u < kPerThread; ++u) {   // consecutive lanes, consecutive entries
          const int j = sub + u * 32 + lane;
          if (j < len) {                         // the product and the row go to the entry's slot
            const int sl = sslot[j];
            wprod[sl] = sval[j] * wvs[j];
            wrows[sl] = scrow[j];
          }
        }
        __syncwarp();
        // slots j0 .. j0+7 of the segment (a row's slots are adjacent): vector loads
        const float4 q0 = *reinterpret_cast<const float4*>(wprod + lane * kPerThread);
        const float4 q1 = *reinterpret_cast<const float4*>(wprod + lane * kPerThread + 4);
        const uint4 rw = *reinterpret_cast<const uint4*>(wrows + lane * kPerThread);
        const float pv[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
        const unsigned rws[4] = {rw.x, rw.y, rw.z, rw.w};
#pragma unroll
        for (int u = 0; u < kPerThread; ++u) {
          const bool in = j0 + u < len;
          key[u] = in ? static_cast<int>((rws[u >> 1] >> (16 * (u & 1))) & 0xffffu) : -1;
          val[u] = in ? pv[u] : 0.f;
        }
      }
      __syncwarp();                            // the stage and wprod are read
      if (lane == 0) mbar_arrive(sm.empty + st);
      if (active) {
        int next_key;
        seg_scan_warp(key, val, next_key);
        // A row's slots form one run per segment: each run end adds the
        // row's partial to the warp's own margins (no other warp writes them).
#pragma unroll
        for (int u = 0; u < kPerThread; ++u) {
          const int nk = u + 1 < kPerThread ? key[u + 1] : next_key;
          if (key[u] >= 0 && nk != key[u]) {
            if (big) gpart[wrow + key[u]] += val[u];
            else sm.mpart[wrow + key[u]] += val[u];
          }
        }
      }
    }
    // ---- the CTA's partial margins: the four warps' rows added in order ----
    consumer_bar();
    for (int b = tid; b < a.B; b += kConsumers) {
      if (big) {
        float m = gpart[b];
        for (int w = 1; w < kWarps; ++w) m += gpart[static_cast<size_t>(w) * a.B + b];
        gpart[b] = m;
      } else {
        float m = sm.mpart[b];
        for (int w = 1; w < kWarps; ++w) m += sm.mpart[static_cast<size_t>(w) * a.B + b];
        sm.mpart[b] = m;
      }
    }
    // ---- the worker's margins: the Q partials of every row in rank order ----
    if (big) __threadfence();
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
    const float* y = reinterpret_cast<const float*>(a.block + dsc.y);
    float lsum = 0.f;
    constexpr int kRowsAtOnce = 2;
    for (int b0 = tid; b0 < a.B; b0 += kRowsAtOnce * kConsumers) {
      // the Q partials of two rows first, then each row's sum in rank order:
      // the remote loads overlap
      float mq[kRowsAtOnce][kMaxStepCluster];
#pragma unroll
      for (int u = 0; u < kRowsAtOnce; ++u) {
        const int b = b0 + u * kConsumers;
#pragma unroll
        for (int qq = 0; qq < kMaxStepCluster; ++qq)
          if (qq < Q && b < a.B)
            mq[u][qq] = big ? __ldcg(a.mpart_big + (static_cast<size_t>(i) * Q + qq) * kWarps * a.B + b)
                            : ld_dsmem(sm.mpart + b, qq);
      }
#pragma unroll
      for (int u = 0; u < kRowsAtOnce; ++u) {
        const int b = b0 + u * kConsumers;
        if (b >= a.B) break;
        float m = 0.f;
#pragma unroll
        for (int qq = 0; qq < kMaxStepCluster; ++qq)
          if (qq < Q) m += mq[u][qq];
        float l, r;
        loss_and_r<LOSS>(y[b], m * a.mscale, l, r);
        if (big) grr[b] = r;
        else sm.r[b] = r;
        lsum += l;
      }
    }
    if (q == 0) {
      lsum = warp_sum(lsum);
      if (lane == 0) sm.red[warp] = lsum;
    }
    consumer_bar();
    if (q == 0 && tid == 0) {
      float tot = 0.f;
      for (int w2 = 0; w2 < kWarps; ++w2) tot += sm.red[w2];
      a.loss_part[i] = tot;
    }
    ok = ok && !sm.ctl[0];
    // ---- pass 2: column sums over [lo, hi) ----
    // Runs that end inside a warp's sub-tile are complete and stored by the
    // warp.  The run through a sub-tile's first pair and the run through its
    // last may continue in the neighbouring sub-tiles: they are left as
    // fragments, which the gather warp adds up in sub-tile order once every
    // warp is through the tile (the CTA's range starts and ends at column
    // bounds).
    float* g = a.gsum;
    for (int k = 0; k < n2 && ok; ++k) {
      const int it = n1 + k;
      const int st = it % a.stages;
      ok = __all_sync(kFull, mbar_wait_bounded(sm.full + st, (it / a.stages) & 1));
      if (!ok) break;
      const unsigned char* base = sm.stage0 + kStageBytes * st;
      const int* spos = reinterpret_cast<const int*>(base);
      const float* sval = reinterpret_cast<const float*>(base + 4 * kTileEntries);
      const uint16_t* srw = reinterpret_cast<const uint16_t*>(base + 8 * kTileEntries);
      const int e_base = T0 + k * kTileEntries;
      int key[kPerThread];
      float val[kPerThread];
      const int4 p0 = *reinterpret_cast<const int4*>(spos + j0);
      const int4 p1 = *reinterpret_cast<const int4*>(spos + j0 + 4);
      const float4 v0 = *reinterpret_cast<const float4*>(sval + j0);
      const float4 v1 = *reinterpret_cast<const float4*>(sval + j0 + 4);
      const uint4 rw = *reinterpret_cast<const uint4*>(srw + j0);
      const int pk[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
      const float pv[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
      const unsigned rws[4] = {rw.x, rw.y, rw.z, rw.w};
#pragma unroll
      for (int u = 0; u < kPerThread; ++u) {
        const int e = e_base + j0 + u;
        const bool valid = e >= lo && e < hi;
        const int row = static_cast<int>((rws[u >> 1] >> (16 * (u & 1))) & 0xffffu);
        key[u] = valid ? pk[u] : -1;
        val[u] = valid ? (big ? __ldcg(grr + row) : sm.r[row]) * pv[u] : 0.f;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(sm.empty + st);   // the stage is read
      int next_key;
      seg_scan_warp(key, val, next_key);
      const int first_key = __shfl_sync(kFull, key[0], 0);
      const int last_key = __shfl_sync(kFull, key[kPerThread - 1], 31);
      const int fr = (k % kFragRing) * kWarps * 2 + warp * 2;
      // the slot's fragments of tile k - kFragRing have been read
      if (k >= kFragRing) {
        ok = __all_sync(kFull, mbar_wait_bounded(sm.ffree + (k % kFragRing), ((k / kFragRing) - 1) & 1));
        if (!ok) break;
      }
      int ok8[kPerThread];
#pragma unroll
      for (int u = 0; u < kPerThread; ++u) {
        const int nk = u + 1 < kPerThread ? key[u + 1] : next_key;
        const bool end = key[u] >= 0 && nk != key[u];
        const bool at_last = lane == 31 && u == kPerThread - 1;
        ok8[u] = -1;
        if (end) {
          if (at_last) {                       // the run through the last pair
            sm.fkey[fr + 1] = key[u];
            sm.fval[fr + 1] = val[u];
          } else if (key[u] == first_key) {    // the run through the first pair
            sm.fkey[fr] = key[u];
            sm.fval[fr] = val[u];
          } else {
            ok8[u] = key[u];
          }
        }
      }
      // sub-tile edges without a fragment
      if (lane == 0 && (first_key < 0 || first_key == last_key)) sm.fkey[fr] = kNoKey;
      if (lane == 31 && last_key < 0) sm.fkey[fr + 1] = kNoKey;
      // complete runs: stored with consecutive lanes on consecutive pairs
      *reinterpret_cast<int4*>(wokey + lane * kPerThread) = make_int4(ok8[0], ok8[1], ok8[2], ok8[3]);
      *reinterpret_cast<int4*>(wokey + lane * kPerThread + 4) = make_int4(ok8[4], ok8[5], ok8[6], ok8[7]);
      *reinterpret_cast<float4*>(wprod + lane * kPerThread) = make_float4(val[0], val[1], val[2], val[3]);
      *reinterpret_cast<float4*>(wprod + lane * kPerThread + 4) = make_float4(val[4], val[5], val[6], val[7]);
      __syncwarp();
      if (lane == 0) mbar_arrive(sm.fready + (k % kFragRing));   // releases the fragments to the merger
#pragma unroll
      for (int u = 0; u < kPerThread; ++u) {
        const int j = u * 32 + lane;
        const int kk = wokey[j];
        if (kk >= 0) g[kk] = wprod[j];
      }
      __syncwarp();                            // wokey / wprod are reused by the next sub-tile
    }
    if (!ok && lane == 0) record_error(a.st, ASAP_ERR_CUDA, static_cast<unsigned>(i), a.round);
  }
  // ---- NOTIFY: every CTA's column sums are visible, then CTA 0 publishes ----
  __threadfence();
  const int all_ok = __syncthreads_or(!ok || sm.ctl[0]) == 0;
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
  if (q == 0 && tid == 0 && a.notify && i != a.skip_worker) {
    __threadfence();
    if (all_ok) st_release_u32(&a.ready[i], a.round + 1u);
  }
}

// wv[e] = W[i][s*S + cl] for every entry e of a step's column list
// (parameters written from the host, or changed by an earlier local step of
// the round, have no exported copy).  One warp per slab, four entries per
// lane in flight.
__global__ void __launch_bounds__(kThreads) k_gather_wv(const float* __restrict__ W, int64_t ld,
                                                       const uint32_t* __restrict__ list,
                                                       const int* __restrict__ slab_off, long long n_slabs, int S,
                                                       float* __restrict__ wv) {
  constexpr int kU = 4;
  const int lane = threadIdx.x & 31;
  const long long nw = static_cast<long long>(gridDim.x) * (kThreads / 32);
  for (long long s = static_cast<long long>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5); s < n_slabs;
       s += nw) {
    const int a0 = slab_off[s], a1 = slab_off[s + 1];
    const float* Ws = W + s * S;
    for (int e0 = a0 + lane; e0 < a1; e0 += kU * 32) {
      uint32_t code[kU];
      float v[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) code[u] = e0 + 32 * u < a1 ? list[e0 + 32 * u] : kListPad;
#pragma unroll
      for (int u = 0; u < kU; ++u)
        v[u] = code[u] != kListPad ? Ws[static_cast<int64_t>(code[u] >> 16) * ld + (code[u] & 0xffffu)] : 0.f;
#pragma unroll
      for (int u = 0; u < kU; ++u)
        if (code[u] != kListPad) wv[e0 + 32 * u] = v[u];
    }
  }
}

// W[i][s*S + cl] -= scale * g[e] for every entry {i << 16 | cl} of a slab-major
// column list: the update of a local step that is not the round's last (the
// last one is applied inside the stochastic reduce).  The entries of a list
// are distinct, so every parameter is written by one thread.  One warp per
// slab, four entries per lane in flight.
__global__ void __launch_bounds__(kThreads) k_apply_update(float* __restrict__ W, int64_t ld,
                                                          const uint32_t* __restrict__ list,
                                                          const int* __restrict__ slab_off, long long n_slabs, int S,
                                                          const float* __restrict__ g, float scale) {
  constexpr int kU = 4;
  const int lane = threadIdx.x & 31;
  const long long nw = static_cast<long long>(gridDim.x) * (kThreads / 32);
  for (long long s = static_cast<long long>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5); s < n_slabs;
       s += nw) {
    const int a0 = slab_off[s], a1 = slab_off[s + 1];
    float* Ws = W + s * S;
    for (int e0 = a0 + lane; e0 < a1; e0 += kU * 32) {
      uint32_t code[kU];
      float gv[kU], wv[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const bool in = e0 + 32 * u < a1;
        code[u] = in ? list[e0 + 32 * u] : kListPad;
        gv[u] = in ? g[e0 + 32 * u] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < kU; ++u)
        wv[u] = code[u] != kListPad ? Ws[static_cast<int64_t>(code[u] >> 16) * ld + (code[u] & 0xffffu)] : 0.f;
#pragma unroll
      for (int u = 0; u < kU; ++u)
        if (code[u] != kListPad)
          Ws[static_cast<int64_t>(code[u] >> 16) * ld + (code[u] & 0xffffu)] = fmaf(-scale, gv[u], wv[u]);
    }
  }
}

}  // namespace

// One warp per slab; at most one wave of 8-warp CTAs.
static int slab_warp_grid(long long n_slabs, int sm_count) {
  const long long ctas = (n_slabs + kThreads / 32 - 1) / (kThreads / 32);
  const long long cap = 8LL * sm_count;
  const long long g = ctas < cap ? ctas : cap;
  return static_cast<int>(g > 0 ? g : 1);
}

cudaError_t launch_apply_update(float* W, int64_t ld, const uint32_t* list, const int* slab_off, long long n_slabs,
                                int S, const float* gsum, float scale, int sm_count, cudaStream_t s) {
  k_apply_update<<<slab_warp_grid(n_slabs, sm_count), kThreads, 0, s>>>(W, ld, list, slab_off, n_slabs, S, gsum,
                                                                        scale);
  return cudaGetLastError();
}

size_t local_step_smem_bytes(int B, int stages) {
  const size_t b_smem = B > kRSmemRows ? 0 : static_cast<size_t>(B);
  return 128 + kStageBytes * stages + 24 * static_cast<size_t>(stages) + 16 * kFragRing + 16 + 8 * kTileEntries +
         4 * (kWarps + 1) * b_smem + 16 + 8 * kFragRing * kWarps * 2 + 4 * kWarps + 4;
}

cudaError_t local_step_configure(size_t smem) {
  cudaError_t e = cudaFuncSetAttribute(k_local_step<ASAP_LOSS_HINGE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_local_step<ASAP_LOSS_LOGISTIC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem));
}

cudaError_t launch_local_step(const LocalStepArgs& a, int loss, size_t smem, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.N * a.Q);
  cfg.blockDim = dim3(kLocalStepThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = a.Q;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // a programmatic dependent of the kernel before it (the previous round's
  // reduce): the kernel waits for that grid itself (griddepcontrol.wait)
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (loss == ASAP_LOSS_HINGE) return cudaLaunchKernelEx(&cfg, k_local_step<ASAP_LOSS_HINGE>, a);
  return cudaLaunchKernelEx(&cfg, k_local_step<ASAP_LOSS_LOGISTIC>, a);
}

cudaError_t launch_gather_wv(const float* W, int64_t ld, const uint32_t* list, const int* slab_off, long long n_slabs,
                             int S, float* wv, int sm_count, cudaStream_t s) {
  k_gather_wv<<<slab_warp_grid(n_slabs, sm_count), kThreads, 0, s>>>(W, ld, list, slab_off, n_slabs, S, wv);
  return cudaGetLastError();
}

}  // namespace asap
