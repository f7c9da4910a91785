// Stochastic reduce (Eq. A.1, second line; Section 3):
//   W_next[i, :] = sum_{m < k+1} wgt[i, m] * W_half[nbr[i, m], :]
// plus, fused, the round's metrics (consensus error ||W_next - 1 wbar^T||_F
// and the mean minibatch loss) and the NOTIFY-ACK bookkeeping of Section 4.
//
// Data movement.  W is [N][ld] fp32 (ld a multiple of 64).  The kernel is
// persistent: CTA b walks column slabs b, b + grid, ...  A slab is S columns
// (8 to 1024, about 32 KB) of *all* N rows.  One producer warp brings slabs into a ring of
// shared-memory stages with TMA 2-D tiled loads (one box per 256 rows), so
// every element of W is read from HBM exactly once however many neighbours
// use it; sixteen compute warps mix and write the outputs straight from
// registers.  A stage goes back to the producer when all the compute warps
// have arrived on its "empty" mbarrier: no CTA-wide barrier in steady state.
//
// Sparse models (FUSED): the local step left, per distinct (worker, column)
// of the minibatch, the column sum g of r_b x_b (kernels_sparse.cu).  The
// producer also copies the slab's part of that list (and of the next
// round's list) into the stage; once a slab has landed two updater warps
// apply the round's last local update to it, w -= eta / (B s) g, and release
// it to the compute warps through a "ready" mbarrier -- so w_{t+1/2} exists
// only in shared memory.  s is the round's L2 shrink, prod_j (1 - eta_j l2)
// over its local steps, which also scales the mixing weights (true w =
// s * stored w).  After mixing the compute warps export w_{t+1} at the next
// round's columns, which is all the next margin kernel reads.
//
// Consensus error per column: with K the column's value in row 0 (a shift
// against cancellation), sum_i (w_i - wbar)^2 = sum_i (w_i - K)^2 -
// (sum_i (w_i - K))^2 / N.  Squares accumulate per thread in fp32 (a few
// dozen slabs per thread; GB300's fp64 pipe is narrow), the per-column sums
// are combined across warps by the producer warp when the stage comes back,
// and the block and launch totals are formed in float-float pairs (fp32 hi +
// lo, a fixed order).  The complete graph (all-reduce, equal weights) writes
// the column mean to every row and adds nothing.
//
// Protocol (Section 4, NOTIFY-ACK): before touching any input each CTA waits,
// with a time limit, until ready[j] == round+1 for every worker j and
// consumed[j] >= round.  The last CTA to finish (ticket) reduces the metric
// partials in a fixed order and ACKs: consumed[j] = round+1,
// stamp_next[j] = round+1.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>

#include "asap_internal.h"

namespace asap {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr unsigned long long kTmaWaitNs = 2000000000ull;   // 2 s: a TMA load never takes this long
constexpr int kCompute = kMixComputeWarps * 32;            // compute threads
constexpr int kProducerWarp = kMixComputeWarps;
constexpr int kUpdater0 = kMixComputeWarps + 1;             // first updater warp

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ unsigned int ld_acquire_u32(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_u32(unsigned int* p, unsigned int v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
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

// Bounded wait on an mbarrier phase; false if the limit ran out.  The timer
// is read every 256 polls only (each try_wait already suspends the thread
// for a while), so waiting warps take few issue slots.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned n = 1;; ++n) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((n & 255u) == 0 && globaltimer_ns() - t0 > kTmaWaitNs) return false;
  }
}

// L2 policy for the parameter stream: each element is read once and written
// once per round, so it should not push the round's small lists out of L2.
__device__ __forceinline__ uint64_t evict_first_policy() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;"
      :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

// The next round's w values (a few MB) should stay in L2 for the margin
// kernel's gathers.
__device__ __forceinline__ uint64_t evict_last_policy() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ void st_f32_hint(float* p, float v, uint64_t policy) {
  asm volatile("st.global.L2::cache_hint.f32 [%0], %1, %2;" :: "l"(p), "f"(v), "l"(policy) : "memory");
}

__device__ __forceinline__ void st_f4_hint(float* p, float4 v, uint64_t policy) {
  asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;"
               :: "l"(p), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "l"(policy) : "memory");
}

// Untiled bulk copy global -> shared (16-byte aligned, size a multiple of 16).
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void record_error(DevState* st, unsigned code, unsigned worker, unsigned round) {
  if (atomicCAS(&st->err_code, 0u, code) == 0u) {
    st->err_worker = worker;
    st->err_round = round;
  }
}

// Wait until *flag >= target (time-limited).  Returns 0 on success,
// ASAP_ERR_TIMEOUT if the limit ran out, ASAP_ERR_STATE if exact and the
// flag went past target.
__device__ unsigned wait_flag(const unsigned int* flag, unsigned target, bool exact, unsigned long long limit_ns) {
  unsigned v = ld_acquire_u32(flag);
  if (v < target) {
    const unsigned long long t0 = globaltimer_ns();
    do {
      __nanosleep(128);
      v = ld_acquire_u32(flag);
      if (v < target && globaltimer_ns() - t0 > limit_ns) return ASAP_ERR_TIMEOUT;
    } while (v < target);
  }
  return (exact && v != target) ? ASAP_ERR_STATE : 0u;
}

__device__ __forceinline__ float4 f4_fma(float w, float4 x, float4 acc) {
  acc.x = fmaf(w, x.x, acc.x);
  acc.y = fmaf(w, x.y, acc.y);
  acc.z = fmaf(w, x.z, acc.z);
  acc.w = fmaf(w, x.w, acc.w);
  return acc;
}

__device__ __forceinline__ float4 f4_add(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}

// A float-float value hi + lo (|lo| at most half an ulp of hi): the block
// sums are carried in fp32 pairs, since this GPU's fp64 pipe is narrow (an
// fp64 tree over the block took ~2 us, in the last CTA's finalisation ~7).
struct F2 {
  float hi, lo;
};

// hi + lo of a + b: the rounding error of hi_a + hi_b is recovered exactly
// by Knuth's two-sum, the low parts are added to it, and the pair is
// renormalised.  The result does not depend on the order of a and b.
__device__ __forceinline__ F2 f2_add(F2 a, F2 b) {
  const float s = a.hi + b.hi;
  const float bv = s - a.hi;
  const float e = ((a.hi - (s - bv)) + (b.hi - bv)) + (a.lo + b.lo);
  const float hi = s + e;
  return F2{hi, e - (hi - s)};
}

__device__ __forceinline__ F2 f2_of(double v) {
  const float h = static_cast<float>(v);
  return F2{h, static_cast<float>(v - static_cast<double>(h))};
}

// Sum over all threads of the block (kMixThreads) in a fixed order; valid in
// thread 0.
__device__ __forceinline__ F2 block_sum_f2(F2 v, F2* scratch) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
    v = f2_add(v, F2{__shfl_xor_sync(kFull, v.hi, o), __shfl_xor_sync(kFull, v.lo, o)});
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  F2 t{0.f, 0.f};
  if (threadIdx.x == 0)
    for (int k = 0; k < kMixThreads / 32; ++k) t = f2_add(t, scratch[k]);
  return t;
}

// Two block sums at once, each in the order block_sum_f2 takes (so each
// result equals that of a separate call); valid in thread 0.  `scratch`
// holds two pairs per warp.
__device__ __forceinline__ void block_sum2_f2(F2& u, F2& v, F2* scratch) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    u = f2_add(u, F2{__shfl_xor_sync(kFull, u.hi, o), __shfl_xor_sync(kFull, u.lo, o)});
    v = f2_add(v, F2{__shfl_xor_sync(kFull, v.hi, o), __shfl_xor_sync(kFull, v.lo, o)});
  }
  constexpr int kW = kMixThreads / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) {
    scratch[warp] = u;
    scratch[kW + warp] = v;
  }
  __syncthreads();
  F2 tu{0.f, 0.f}, tv{0.f, 0.f};
  if (threadIdx.x == 0)
    for (int k = 0; k < kW; ++k) {
      tu = f2_add(tu, scratch[k]);
      tv = f2_add(tv, scratch[kW + k]);
    }
  u = tu;
  v = tv;
}

__device__ __forceinline__ void compute_bar() { asm volatile("bar.sync 1, %0;" :: "n"(kCompute) : "memory"); }

// Barrier among the compute warps that also returns the OR of `v` over them.
__device__ __forceinline__ bool compute_bar_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, %2, p;\n selp.u32 %0, 1, 0, q;\n}"
      : "=r"(r) : "r"(static_cast<uint32_t>(v)), "n"(kCompute) : "memory");
  return r != 0;
}

struct MixSmem {
  unsigned char* stage0;
  size_t stage_bytes;
  uint64_t* full;
  uint64_t* empty;
  uint64_t* ready;   // FUSED: the producer has applied the slab's update
  float4* part;      // [stages][warps][nq]: per-warp column sums (consensus / complete-graph mean)
  int* info;         // [stages][4]: n_upd, n_exp, exp_base
  int* nbr;
  float* wgt;
  double* dscratch;
  int* flags;        // [0]: fail, [1]: last, [2]: failed CTAs of the launch (last CTA)
  unsigned* seen;    // [32]: bitmap of workers whose NOTIFY this CTA has seen (gated reduces)
};

// Shared-memory layout; every region starts 16-byte aligned (the slab
// stages 1024-byte aligned).  mix_smem_bytes() mirrors it.
// Regions are formed from `raw` by pointer arithmetic (offsets only), so that
// the compiler keeps the pointers in the shared address space and emits
// plain shared-memory accesses.
__device__ __forceinline__ MixSmem carve(unsigned char* raw, const MixArgs& a, int kp1) {
  MixSmem m;
  auto a16 = [](size_t v) { return (v + 15) & ~static_cast<size_t>(15); };
  size_t off = (1024u - (smem_u32(raw) & 1023u)) & 1023u;   // 1024-byte aligned stages
  m.stage_bytes = mix_stage_bytes(a.S, a.rows_pad, a.max_region);
  m.stage0 = raw + off;
  off += m.stage_bytes * a.stages;
  m.full = reinterpret_cast<uint64_t*>(raw + off);
  off += 8 * a.stages;
  m.empty = reinterpret_cast<uint64_t*>(raw + off);
  off += 8 * a.stages;
  m.ready = reinterpret_cast<uint64_t*>(raw + off);
  off = a16(off + 8 * a.stages);
  m.dscratch = reinterpret_cast<double*>(raw + off);
  off = a16(off + 16 * (kMixThreads / 32));
  m.flags = reinterpret_cast<int*>(raw + off);
  off = a16(off + 16);
  m.seen = reinterpret_cast<unsigned*>(raw + off);
  off = a16(off + 4 * 32);
  m.info = reinterpret_cast<int*>(raw + off);
  off = a16(off + 16 * a.stages);
  m.part = reinterpret_cast<float4*>(raw + off);
  off = a16(off + 16 * static_cast<size_t>(a.stages) * kCompute);
  m.nbr = reinterpret_cast<int*>(raw + off);
  off = a16(off + 4 * static_cast<size_t>(a.N) * kp1);
  m.wgt = reinterpret_cast<float*>(raw + off);
  return m;
}

// KP1 > 0: sparse graph with KP1 neighbours per row (compile-time);
// KP1 == 0: sparse graph, runtime a.kp1 (<= kMaxKp1Sparse);
// KP1 < 0: complete graph with equal weights.
template <int KP1, bool SHADOW, bool FUSED>
__global__ void __launch_bounds__(kMixThreads, 1) k_mix(const __grid_constant__ CUtensorMap tmap, const MixArgs a) {
  extern __shared__ unsigned char smem_raw[];
  const int kp1 = KP1 > 0 ? KP1 : (KP1 == 0 ? a.kp1 : 0);
  MixSmem sm = carve(smem_raw, a, kp1);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int S = a.S, nq = S >> 2;            // column quads per slab, a power of two <= 256
  const int lq = __ffs(nq) - 1;
  const int QB = nq < 64 ? nq : 64;           // quads per TMA box row (a box spans <= 256 columns)
  const int lqb = __ffs(QB) - 1;
  const int box_col = a.rows_pad << lqb;      // float4s per column box of a slab
  const int G = kCompute >> lq;               // row groups: compute threads that share a column quad
  const size_t slab_floats = static_cast<size_t>(a.rows_pad) * S;
  const size_t list_off = (slab_floats * 4 + 15) & ~static_cast<size_t>(15);
  const size_t list_bytes = (static_cast<size_t>(a.max_region) * 4 + 15) & ~static_cast<size_t>(15);

  if (tid == 0) { sm.flags[0] = 0; sm.flags[1] = 0; }
  if (tid < 32) sm.seen[tid] = 0u;
  __syncthreads();
  // A gated reduce (NOTIFY_ACK or ASYNC, sparse models) runs while the local
  // step may still be running: it reads the column sums of worker j only
  // after j's NOTIFY (or, ASYNC, counts the read as stale).  Otherwise
  // (BSP) it starts once the local step's grid has finished.
  const bool gated = FUSED && a.sync_mode != kSyncBsp;
  if (!gated) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    // The next round's local step (a programmatic dependent) may now be
    // scheduled as this grid drains; it waits for this grid before it reads
    // what this grid writes.  A gated reduce leaves the trigger to its exit,
    // since the local step it overlaps is still running.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  }

  // ---- NOTIFY / ACK checks (time-limited waits) ----
  for (int j = tid; j < a.N; j += kMixThreads) {
    unsigned e = 0;
    const bool own = j >= a.own_lo && j < a.own_lo + a.own_n;
    if (a.expect_notify && !gated && own) e = wait_flag(a.ready + j, a.round + 1u, true, a.wait_ns);
    if (!e) e = wait_flag(a.consumed + j, a.round, false, a.wait_ns);
    if (e) {
      record_error(a.st, e, j, a.round);
      if (e == ASAP_ERR_TIMEOUT) atomicAdd(&a.st->timeouts, 1ull);
      atomicOr(&sm.flags[0], 1);
    }
  }
  __syncthreads();
  bool failed = sm.flags[0] != 0;

  float s2 = 0.f;      // compute threads: sum of (w - K)^2;  producer lanes: -sum of S1^2 / N
  if (!failed) {
    if (KP1 >= 0) {
      for (int idx = tid; idx < a.N * kp1; idx += kMixThreads) {
        sm.nbr[idx] = a.nbr[idx] * QB;       // float4 offset of the neighbour's row within a box column
        sm.wgt[idx] = a.wgt[idx] * a.wscale;
      }
    }
    if (tid == 0) {
      for (int s = 0; s < a.stages; ++s) {
        mbar_init(sm.full + s, 1);
        mbar_init(sm.empty + s, kMixComputeWarps);
        mbar_init(sm.ready + s, kMixUpdaterWarps);
      }
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    const long long stride = gridDim.x;
    const long long n_my = (a.n_slabs - blockIdx.x + stride - 1) / stride;   // slabs of this CTA
    const float inv_n = 1.0f / static_cast<float>(a.N);

    const uint64_t policy = evict_first_policy();
    if (warp == kProducerWarp) {
      // ================= producer warp =================
      float term = 0.f;
      const float inv_n_term = 1.0f / static_cast<float>(a.N);
      unsigned long long n_read = 0, n_current = 0;   // gated: (slab, worker) inputs, and those current
      int n_seen = 0;                                 // gated: workers whose NOTIFY this CTA has seen
      // List offsets of the next 32 slabs, one slab per lane, loaded ahead so
      // that issuing a stage never waits on a global load.
      int4 offs = make_int4(0, 0, 0, 0);
      for (long long it = 0; it < n_my + a.stages; ++it) {
        if (FUSED && (it & 31) == 0 && it < n_my) {
          const long long sl = blockIdx.x + (it + lane) * stride;
          if (it + lane < n_my)
            offs = make_int4(__ldg(a.upd_off + sl), __ldg(a.upd_off + sl + 1), __ldg(a.exp_off + sl),
                             __ldg(a.exp_off + sl + 1));
        }
        int4 o = make_int4(0, 0, 0, 0);
        if (FUSED) {
          const int src = static_cast<int>(it & 31);
          o.x = __shfl_sync(kFull, offs.x, src);
          o.y = __shfl_sync(kFull, offs.y, src);
          o.z = __shfl_sync(kFull, offs.z, src);
          o.w = __shfl_sync(kFull, offs.w, src);
        }
        if (it >= a.stages) {
          const long long done = it - a.stages;
          const int st = static_cast<int>(done % a.stages);
          bool ok = (lane == 0) ? mbar_wait_bounded(sm.empty + st, static_cast<uint32_t>((done / a.stages) & 1))
                                : true;
          ok = __shfl_sync(kFull, ok, 0) != 0;   // warp-uniform outcome
          __syncwarp();
          if (!ok) {
            if (lane == 0) record_error(a.st, ASAP_ERR_CUDA, 0xfffffffeu, a.round);
            failed = true;
            break;
          }
          if (KP1 >= 0) {
            const float4* p = sm.part + static_cast<size_t>(st) * kCompute;
            for (int q = lane; q < nq; q += 32) {
              float4 t = p[q];
              for (int g = 1; g < G; ++g) t = f4_add(t, p[g * nq + q]);
              term = fmaf(fmaf(t.x, t.x, fmaf(t.y, t.y, fmaf(t.z, t.z, t.w * t.w))), inv_n_term, term);
            }
          }
          __syncwarp();
        }
        if (FUSED && gated && it < n_my) {
          // The slab's updates come from workers w0 .. w1 (a region is sorted
          // by worker): their NOTIFY for the round before the slab's column
          // sums are copied (NOTIFY_ACK, time-limited waits), or just noted
          // (ASYNC).  The warp checks 32 workers at a time; a worker seen
          // once stays seen for the rest of the launch.
          const int nu = o.y - o.x;
          if (n_seen == a.N) {
            n_read += static_cast<unsigned long long>(a.N);
            n_current += static_cast<unsigned long long>(a.N);
          } else if (nu > 0) {
            const unsigned w0 = __ldg(a.upd_list + o.x) >> 16;
            unsigned w1 = w0;
            for (int e = nu - 1; e >= 0 && e >= nu - 4; --e) {
              const uint32_t c = __ldg(a.upd_list + o.x + e);
              if (c != kListPad) { w1 = c >> 16; break; }
            }
            bool acquired = false;
            for (unsigned j0 = w0; j0 <= w1 && j0 < static_cast<unsigned>(a.N); j0 += 32) {
              const unsigned j = j0 + lane;
              const bool in = j <= w1 && j < static_cast<unsigned>(a.N);
              const unsigned bit = 1u << (j & 31u);
              bool cur = in && (sm.seen[j >> 5] & bit) != 0;
              bool fresh = false;
              if (in && !cur && !failed) {
                if (a.sync_mode == kSyncNotifyAck) {
                  const unsigned er = wait_flag(a.ready + j, a.round + 1u, true, a.wait_ns);
                  if (er) {
                    record_error(a.st, er, j, a.round);
                    if (er == ASAP_ERR_TIMEOUT) atomicAdd(&a.st->timeouts, 1ull);
                    failed = true;
                  } else {
                    fresh = true;
                  }
                } else {
                  fresh = ld_acquire_u32(a.ready + j) == a.round + 1u;
                }
                if (fresh) atomicOr(sm.seen + (j >> 5), bit);
                cur = fresh;
              }
              n_seen += __popc(__ballot_sync(kFull, fresh));
              acquired = acquired || __any_sync(kFull, fresh);
              n_read += __popc(__ballot_sync(kFull, in));
              n_current += __popc(__ballot_sync(kFull, in && cur));
            }
            failed = __any_sync(kFull, failed);
            __syncwarp();
            // newly acquired column sums, to the bulk copy's async proxy
            if (acquired && lane == 0) asm volatile("fence.proxy.async.global;" ::: "memory");
          }
        }
        if (it < n_my && lane == 0) {
          const long long slab = blockIdx.x + it * stride;
          const int st = static_cast<int>(it % a.stages);
          unsigned char* base = sm.stage0 + st * sm.stage_bytes;
          uint32_t bytes = static_cast<uint32_t>(a.n_boxes) * a.box_rows * S * 4u;
          int n_upd = 0, n_exp = 0, x0 = 0, u0 = 0;
          if (FUSED) {
            u0 = o.x;
            n_upd = o.y - o.x;
            x0 = o.z;
            n_exp = o.w - o.z;
            bytes += 8u * n_upd + 4u * n_exp;
          }
          int* info = sm.info + 4 * st;
          info[0] = n_upd;
          info[1] = n_exp;
          info[2] = x0;
          info[3] = u0;
          mbar_expect_tx(sm.full + st, bytes);
          // Slab layout in shared memory: [column box][row][QB quads].
          for (int xb = 0; xb < nq / QB; ++xb)
            for (int b = 0; b < a.n_boxes; ++b)
              tma_load_2d(base + (static_cast<size_t>(xb) * a.rows_pad + static_cast<size_t>(b) * a.box_rows) * QB * 16,
                          &tmap, sm.full + st, static_cast<int>(slab * S + xb * QB * 4), b * a.box_rows, policy);
          if (FUSED) {
            if (n_upd > 0) {
              bulk_load(base + list_off, a.upd_list + u0, 4u * n_upd, sm.full + st);
              bulk_load(base + list_off + list_bytes, a.gsum + u0, 4u * n_upd, sm.full + st);
            }
            if (n_exp > 0) bulk_load(base + list_off + 2 * list_bytes, a.exp_list + x0, 4u * n_exp, sm.full + st);
          }
        }
        __syncwarp();
      }
      s2 = -term;
      if (gated && lane == 0 && n_read) {
        atomicAdd(&a.st->inputs_read, n_read);
        atomicAdd(&a.st->inputs_current, n_current);
      }
    } else if (warp >= kUpdater0) {
      // ================= updater warps (FUSED) =================
      // Once a slab has landed, apply w -= eta/B (1 - eta l2)^-1 g to it and
      // release it to the compute warps.
      if (FUSED) {
        const int ut = tid - kUpdater0 * 32;
        for (long long it = 0; it < n_my; ++it) {
          const int st = static_cast<int>(it % a.stages);
          const bool ok = __all_sync(kFull, mbar_wait_bounded(sm.full + st, static_cast<uint32_t>((it / a.stages) & 1)));
          if (!ok) {
            if (lane == 0) record_error(a.st, ASAP_ERR_CUDA, 0xfffffffdu, a.round);
            failed = true;
            break;
          }
          unsigned char* bj = sm.stage0 + st * sm.stage_bytes;
          float* xj = reinterpret_cast<float*>(bj);
          const uint32_t* ul = reinterpret_cast<const uint32_t*>(bj + list_off);
          const float* ug = reinterpret_cast<const float*>(bj + list_off + list_bytes);
          const int n_upd = sm.info[4 * st];
          // Four entries per thread in flight: the (worker, column) pairs of
          // one list are distinct, so the four read-modify-writes never alias.
          constexpr int kUpd = kMixUpdaterWarps * 32, kU = 4;
          for (int e0 = ut; e0 < n_upd; e0 += kU * kUpd) {
            uint32_t code[kU];
            float gv[kU], wv[kU] = {};
            int off[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) {
              const int e = e0 + u * kUpd;
              code[u] = e < n_upd ? ul[e] : kListPad;
              gv[u] = e < n_upd ? ug[e] : 0.f;
            }
#pragma unroll
            for (int u = 0; u < kU; ++u) {
              const int i = static_cast<int>(code[u] >> 16), cl = static_cast<int>(code[u] & 0xffffu);
              const int q = cl >> 2;
              off[u] = 4 * ((i << lqb) + (q >> lqb) * box_col + (q & (QB - 1))) + (cl & 3);
              if (code[u] != kListPad) wv[u] = xj[off[u]];
            }
#pragma unroll
            for (int u = 0; u < kU; ++u)
              if (code[u] != kListPad) xj[off[u]] = fmaf(-a.upd_scale, gv[u], wv[u]);
          }
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // before this stage's next TMA
          __syncwarp();
          if (lane == 0) mbar_arrive(sm.ready + st);
        }
      }
    } else {
      // ================= compute warps =================
      // Thread t owns column quad q = t mod nq of every slab for the rows
      // i = g, g + G, ... (g = t / nq): with ~32 KB slabs that is 4 rows.
      const int q_t = tid & (nq - 1), g_t = tid >> lq;
      const uint64_t keep = evict_last_policy();
      const int qoff = (q_t >> lqb) * box_col + (q_t & (QB - 1));   // float4 offset of (row 0, quad q_t)
      const int rows_t = (a.N - g_t + G - 1) / G;
      auto xq = [&](int q) { return (q >> lqb) * box_col + (q & (QB - 1)); };
      // With a compile-time neighbour count and at most kCacheRows rows per
      // thread, the neighbour offsets of the thread's rows (its quad folded
      // in) stay in registers as 16-bit pairs, and an equal weight in one
      // register: the slab loop then reads only the slab from shared memory.
      constexpr int kCacheRows = 4;
      constexpr int kC = KP1 > 0 ? KP1 : 1;
      constexpr int kPk = (kCacheRows * kC + 1) / 2;
      const bool cached = KP1 > 0 && rows_t <= kCacheRows;
      uint32_t pko[kPk];
#pragma unroll
      for (int u = 0; u < kPk; ++u) pko[u] = 0u;
      if (KP1 > 0 && cached) {
#pragma unroll
        for (int rr = 0; rr < kCacheRows; ++rr)
#pragma unroll
          for (int m = 0; m < kC; ++m) {
            const int e = rr * kC + m;
            const uint32_t off = rr < rows_t ? static_cast<uint32_t>(sm.nbr[(g_t + rr * G) * kC + m] + qoff) : 0u;
            pko[e >> 1] |= (off & 0xffffu) << (16 * (e & 1));
          }
      }
      const bool uni = a.uniform_w != 0;
      const float wu = uni && KP1 >= 0 ? sm.wgt[0] : 0.f;
      for (long long it = 0; it < n_my; ++it) {
        const long long slab = blockIdx.x + it * stride;
        const int st = static_cast<int>(it % a.stages);
        bool ok = __all_sync(kFull, mbar_wait_bounded(FUSED ? sm.ready + st : sm.full + st,
                                                      static_cast<uint32_t>((it / a.stages) & 1)));
        unsigned char* base = sm.stage0 + st * sm.stage_bytes;
        float* x = reinterpret_cast<float*>(base);
        const float4* x4 = reinterpret_cast<const float4*>(base);
        const int* info = sm.info + 4 * st;
        float4* part = sm.part + static_cast<size_t>(st) * kCompute;
        const long long c0 = slab * S;
        if (ok && KP1 < 0) {
          // Complete graph: this thread's share of its column's sum.
          float4 cs = make_float4(0.f, 0.f, 0.f, 0.f);
          for (int r = 0; r < rows_t; ++r) cs = f4_add(cs, x4[(g_t + r * G) * QB + qoff]);
          part[tid] = cs;
        }
        if (KP1 < 0) ok = !compute_bar_or(!ok);   // uniform decision; the column sums are visible
        if (!ok) {
          if (lane == 0) record_error(a.st, ASAP_ERR_CUDA, 0xffffffffu, a.round);
          failed = true;
          break;
        }
        if constexpr (KP1 < 0) {
          // Complete graph: column means (threads t < nq), then every row gets them.
          if (tid < nq) {
            float4 t = part[tid];
            for (int g = 1; g < G; ++g) t = f4_add(t, part[g * nq + tid]);
            const float sc = inv_n * a.wscale;
            part[tid] = make_float4(t.x * sc, t.y * sc, t.z * sc, t.w * sc);
          }
          compute_bar();
          const float4 mean = part[q_t];
          for (int r = 0; r < rows_t; ++r) {
            const int i = g_t + r * G;
            const long long c = c0 + 4 * q_t;
            if (c < a.ld) {
              st_f4_hint(a.out + static_cast<int64_t>(i) * a.ld + c, mean, policy);
              if (SHADOW) {
                __nv_bfloat162 lo = __floats2bfloat162_rn(mean.x, mean.y);
                __nv_bfloat162 hi = __floats2bfloat162_rn(mean.z, mean.w);
                uint2 pk;
                pk.x = *reinterpret_cast<uint32_t*>(&lo);
                pk.y = *reinterpret_cast<uint32_t*>(&hi);
                *reinterpret_cast<uint2*>(a.shadow + static_cast<int64_t>(i) * a.ld + c) = pk;
              }
            }
          }
          if (FUSED) {
            const uint32_t* xl = reinterpret_cast<const uint32_t*>(base + list_off + 2 * list_bytes);
            const int n_exp = info[1], xbase = info[2];
            const float* means = reinterpret_cast<const float*>(part);
            for (int e = tid; e < n_exp; e += kCompute) {
              const uint32_t code = xl[e];
              if (code != kListPad) a.wv_out[xbase + e] = means[code & 0xffffu];
            }
          }
          compute_bar();   // the means are read before the next slab's sums overwrite them
        } else {
          const float4 K = x4[qoff];        // shift: row 0 of the (updated) slab
          float4 s1 = make_float4(0.f, 0.f, 0.f, 0.f);
          float sq = 0.f;
          auto mix_one = [&](int i) -> float4 {
            const int* nb = sm.nbr + i * kp1;
            const float* wt = sm.wgt + i * kp1;
            const float4 xa = x4[nb[0] + qoff];
            float4 acc = make_float4(wt[0] * xa.x, wt[0] * xa.y, wt[0] * xa.z, wt[0] * xa.w);
#pragma unroll
            for (int m = 1; m < (KP1 > 0 ? KP1 : kMaxKp1Sparse); ++m) {
              if (KP1 == 0 && m >= kp1) break;
              acc = f4_fma(wt[m], x4[nb[m] + qoff], acc);
            }
            return acc;
          };
          auto emit = [&](int i, float4 acc) {
            const long long c = c0 + 4 * q_t;
            if (c < a.ld) {
              st_f4_hint(a.out + static_cast<int64_t>(i) * a.ld + c, acc, policy);
              if (SHADOW) {
                __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x, acc.y);
                __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z, acc.w);
                uint2 pk;
                pk.x = *reinterpret_cast<uint32_t*>(&lo);
                pk.y = *reinterpret_cast<uint32_t*>(&hi);
                *reinterpret_cast<uint2*>(a.shadow + static_cast<int64_t>(i) * a.ld + c) = pk;
              }
            }
            const float dx = acc.x - K.x, dy = acc.y - K.y, dz = acc.z - K.z, dw = acc.w - K.w;
            s1 = f4_add(s1, make_float4(dx, dy, dz, dw));
            sq = fmaf(dx, dx, fmaf(dy, dy, fmaf(dz, dz, fmaf(dw, dw, sq))));
          };
          if (KP1 > 0 && cached) {
            // the same operations in the same order as mix_one, offsets from registers
            auto mix_c = [&](int rr) -> float4 {
              const float* wt = sm.wgt + (g_t + rr * G) * kC;
              auto xo = [&](int m) {
                const int e = rr * kC + m;
                return static_cast<int>((pko[e >> 1] >> (16 * (e & 1))) & 0xffffu);
              };
              const float w0 = uni ? wu : wt[0];
              const float4 xa = x4[xo(0)];
              float4 acc = make_float4(w0 * xa.x, w0 * xa.y, w0 * xa.z, w0 * xa.w);
#pragma unroll
              for (int m = 1; m < kC; ++m) acc = f4_fma(uni ? wu : wt[m], x4[xo(m)], acc);
              return acc;
            };
#pragma unroll
            for (int rr = 0; rr < kCacheRows; rr += 2) {   // two rows in flight
              if (rr + 1 < rows_t) {
                const float4 a0 = mix_c(rr);
                const float4 a1 = mix_c(rr + 1);
                emit(g_t + rr * G, a0);
                emit(g_t + (rr + 1) * G, a1);
              } else if (rr < rows_t) {
                emit(g_t + rr * G, mix_c(rr));
              }
            }
          } else {
            int r = 0;
            for (; r + 1 < rows_t; r += 2) {      // two rows in flight
              const int i0 = g_t + r * G, i1 = i0 + G;
              const float4 a0 = mix_one(i0);
              const float4 a1 = mix_one(i1);
              emit(i0, a0);
              emit(i1, a1);
            }
            if (r < rows_t) emit(g_t + r * G, mix_one(g_t + r * G));
          }
          s2 += sq;
          part[tid] = s1;
          if (FUSED) {
            // w_{t+1} at the next round's columns, recomputed with the same
            // operations in the same order as the stored outputs.
            const uint32_t* xl = reinterpret_cast<const uint32_t*>(base + list_off + 2 * list_bytes);
            const int n_exp = info[1], xbase = info[2];
            for (int e = tid; e < n_exp; e += kCompute) {
              const uint32_t code = xl[e];
              if (code == kListPad) continue;
              const int i = static_cast<int>(code >> 16), cl = static_cast<int>(code & 0xffffu);
              const int* nb = sm.nbr + i * kp1;
              const float* wt = sm.wgt + i * kp1;
              const int xo = xq(cl >> 2), comp = cl & 3;
              float v = (uni ? wu : wt[0]) * x[4 * (nb[0] + xo) + comp];
#pragma unroll
              for (int m = 1; m < (KP1 > 0 ? KP1 : kMaxKp1Sparse); ++m) {
                if (KP1 == 0 && m >= kp1) break;
                v = fmaf(uni ? wu : wt[m], x[4 * (nb[m] + xo) + comp], v);
              }
              st_f32_hint(a.wv_out + xbase + e, v, keep);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(sm.empty + st);
      }
    }
  }

  // ---- per-CTA partial, ticket, and the last CTA's finalisation ----
  F2* scratch = reinterpret_cast<F2*>(sm.dscratch);
  const F2 csum = block_sum_f2(F2{s2, 0.f}, scratch);
  if (failed) atomicOr(&sm.flags[0], 1);
  __syncthreads();
  if (tid == 0) a.cons_part[blockIdx.x] = static_cast<double>(csum.hi) + static_cast<double>(csum.lo);
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    if (sm.flags[0]) atomicAdd(&a.st->mix_ticket, 0x10000u);   // high half counts failed CTAs
    // Every CTA adds its failure before its ticket, to the same word: the
    // last ticket's old value already holds every CTA's failure count.
    const unsigned t = atomicAdd(&a.st->mix_ticket, 1u);
    sm.flags[1] = ((t & 0xffffu) == gridDim.x - 1) ? 1 : 0;
    sm.flags[2] = static_cast<int>(t >> 16);
  }
  __syncthreads();
  if (!sm.flags[1]) return;
  __threadfence();
  bool any_fail = sm.flags[2] != 0;
  // Consensus partials of every CTA, and the loss partials: read together
  // unless NOTIFY_ACK must first see every worker's NOTIFY (the loss
  // partials of workers without any update in this launch's slabs).
  const bool loss_after_notify = gated && a.sync_mode == kSyncNotifyAck;
  const int n_cons = static_cast<int>(gridDim.x);
  const int n_lp = a.have_loss ? a.n_loss_part : 0;
  F2 ctot{0.f, 0.f}, ltot{0.f, 0.f};
  for (int b = tid; b < (loss_after_notify ? n_cons : max(n_cons, n_lp)); b += kMixThreads) {
    if (b < n_cons) ctot = f2_add(ctot, f2_of(__ldcg(a.cons_part + b)));
    if (!loss_after_notify && b < n_lp) ltot = f2_add(ltot, F2{__ldcg(a.loss_part + b), 0.f});
  }
  if (loss_after_notify) {
    if (!any_fail) {
      for (int j = tid; j < a.N; j += kMixThreads) {
        const unsigned er = wait_flag(a.ready + j, a.round + 1u, true, a.wait_ns);
        if (er) {
          record_error(a.st, er, j, a.round);
          atomicOr(&sm.flags[0], 2);
        }
      }
      __syncthreads();
      any_fail = (sm.flags[0] & 2) != 0;
    }
    for (int b = tid; b < n_lp; b += kMixThreads) ltot = f2_add(ltot, F2{__ldcg(a.loss_part + b), 0.f});
  }
  block_sum2_f2(ctot, ltot, scratch);
  if (tid == 0) {
    const int slot = static_cast<int>(a.round % kMetricsCap);
    a.metrics_cons[slot] = any_fail ? __int_as_float(0x7fc00000) : sqrtf(fmaxf(ctot.hi + ctot.lo, 0.f));
    a.metrics_loss[slot] = (a.have_loss && !any_fail) ? (ltot.hi + ltot.lo) * a.loss_norm
                                                      : __int_as_float(0x7fc00000);
    if (!any_fail) {
      atomicAdd(&a.st->reduces, static_cast<unsigned long long>(a.own_n));
      if (a.expect_notify)
        atomicAdd(&a.st->consistent_inputs, static_cast<unsigned long long>(a.own_n) * (KP1 < 0 ? a.N : kp1));
    }
    a.st->mix_ticket = 0u;
  }
  if (!any_fail) {
    __threadfence();
    for (int j = tid; j < a.N; j += kMixThreads) {
      a.stamp_next[j] = a.round + 1u;
      st_release_u32(a.consumed + j, a.round + 1u);
    }
  }
}

template <int KP1, bool SHADOW, bool FUSED>
struct MixKernel {
  static cudaError_t attr(size_t smem) {
    return cudaFuncSetAttribute(k_mix<KP1, SHADOW, FUSED>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem));
  }
  static cudaError_t occ(size_t smem, int* blocks) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, k_mix<KP1, SHADOW, FUSED>, kMixThreads, smem);
  }
  static cudaError_t launch(const CUtensorMap& tmap, const MixArgs& a, int grid, size_t smem, cudaStream_t s) {
    // A programmatic dependent of the local step's last kernel.
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kMixThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_mix<KP1, SHADOW, FUSED>, tmap, a);
  }
};

// Dispatch over (complete / k+1, shadow, fused); Op is a functor template.
template <template <int, bool, bool> class K, bool SHADOW, bool FUSED>
struct ByKp1 {
  template <typename F>
  static cudaError_t go(bool complete, int kp1, F&& f) {
    if (complete) return f(K<-1, SHADOW, FUSED>());
    switch (kp1) {
      case 1: return f(K<1, SHADOW, FUSED>());
      case 2: return f(K<2, SHADOW, FUSED>());
      case 3: return f(K<3, SHADOW, FUSED>());
      case 5: return f(K<5, SHADOW, FUSED>());
      default: return f(K<0, SHADOW, FUSED>());
    }
  }
};

template <typename F>
cudaError_t dispatch(bool complete, bool fused, int kp1, bool shadow, F&& f) {
  if (shadow) {
    if (fused) return cudaErrorInvalidValue;   // dense models never fuse a sparse update
    return ByKp1<MixKernel, true, false>::go(complete, kp1, f);
  }
  return fused ? ByKp1<MixKernel, false, true>::go(complete, kp1, f)
               : ByKp1<MixKernel, false, false>::go(complete, kp1, f);
}

__global__ void k_cast_bf16(const float* __restrict__ src, uint16_t* __restrict__ dst, int64_t n) {
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    __nv_bfloat16 b = __float2bfloat16_rn(src[i]);
    dst[i] = *reinterpret_cast<uint16_t*>(&b);
  }
}

}  // namespace

ASAP_HD size_t mix_stage_bytes(int S, int rows_pad, int max_region) {
  const size_t slab = (static_cast<size_t>(rows_pad) * S * 4 + 15) & ~static_cast<size_t>(15);
  const size_t list = (static_cast<size_t>(max_region) * 4 + 15) & ~static_cast<size_t>(15);
  return (slab + 3 * list + 1023) & ~static_cast<size_t>(1023);
}

size_t mix_smem_bytes(int N, int kp1, int S, int rows_pad, int stages, int max_region) {
  auto a16 = [](size_t v) { return (v + 15) & ~static_cast<size_t>(15); };
  size_t b = 1024 + mix_stage_bytes(S, rows_pad, max_region) * stages;   // alignment slack + stages
  b = a16(b + 24 * static_cast<size_t>(stages));                         // full / empty / ready
  b = a16(b + 16 * (kMixThreads / 32));                                   // block-sum scratch (two fp32 pairs a warp)
  b = a16(b + 16);                                                        // flags
  b = a16(b + 4 * 32);                                                    // NOTIFY bitmap
  b = a16(b + 16 * static_cast<size_t>(stages));                          // stage info
  b = a16(b + 16 * static_cast<size_t>(stages) * kMixComputeWarps * 32);  // partial sums
  b = a16(b + 4 * static_cast<size_t>(N) * kp1);                          // neighbour offsets
  return b + 4 * static_cast<size_t>(N) * kp1;                            // weights
}

cudaError_t mix_configure(bool complete, bool fused, int kp1, bool shadow, size_t smem) {
  return dispatch(complete, fused, kp1, shadow, [&](auto k) { return decltype(k)::attr(smem); });
}

cudaError_t mix_occupancy(bool complete, bool fused, int kp1, bool shadow, size_t smem, int* blocks) {
  return dispatch(complete, fused, kp1, shadow, [&](auto k) { return decltype(k)::occ(smem, blocks); });
}

cudaError_t launch_mix(const CUtensorMap& tmap, const MixArgs& a, bool complete, bool fused, int grid, size_t smem,
                       cudaStream_t s) {
  return dispatch(complete, fused, a.kp1, a.shadow != nullptr,
                  [&](auto k) { return decltype(k)::launch(tmap, a, grid, smem, s); });
}

cudaError_t launch_cast_bf16(const float* src, uint16_t* dst, int64_t n, cudaStream_t s) {
  const int grid = static_cast<int>(std::min<int64_t>((n + kThreads - 1) / kThreads, 4096));
  k_cast_bf16<<<grid > 0 ? grid : 1, kThreads, 0, s>>>(src, dst, n);
  return cudaGetLastError();
}

}  // namespace asap
