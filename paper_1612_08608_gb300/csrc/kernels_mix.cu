// Stochastic reduce (Eq. A.1, second line; Section 3):
//   W_next[i, :] = sum_{m < k+1} wgt[i, m] * W[nbr[i, m], :]
// plus, fused, the round's metrics (consensus error ||W_next - 1 wbar^T||_F
// and the mean minibatch loss) and the NOTIFY-ACK bookkeeping of Section 4.
//
// Layout and data movement.  W is [N][ld] fp32 (ld a multiple of 64).  The
// kernel is persistent: CTA b walks column slabs b, b + grid, ...  A slab is
// S columns of *all* N rows; it is brought into shared memory by TMA 2-D
// tiled loads (one box per 256 rows) into a ring of `stages` buffers guarded
// by mbarriers, so every element of W is read from HBM exactly once however
// many neighbours use it.  Each output row is then k+1 float4 shared-memory
// reads per float4 written; outputs go straight from registers to HBM.
// The complete graph (all-reduce, k = N-1, equal weights) needs only the
// column mean, which the slab pass computes anyway: every row gets it.
//
// Consensus error: the column mean of W_next equals the column mean of W
// scaled by the weight scale when P is doubly stochastic (Appendix A), so
// the mean comes from the input slab and the squared deviations from the
// output registers.  Partial sums per CTA are fp64; the last CTA to finish
// (ticket) reduces them in a fixed order, so the metric is deterministic.
//
// Protocol (Section 4, NOTIFY-ACK): before touching any input each CTA
// waits, with a time limit, until ready[j] == round+1 for every worker j
// (j's half-step model is complete) and consumed[j] >= round (the buffer
// about to be overwritten was fully read by the previous reduce).  The last
// CTA then ACKs: consumed[j] = round+1, stamp_next[j] = round+1.
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

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}

// Bounded wait on an mbarrier phase; false if the limit ran out.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer_ns() - t0 > kTmaWaitNs) return false;
  }
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      :: "r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
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

__device__ __forceinline__ double block_sum_f64(double v, double* scratch) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  double t = 0.0;
  if (threadIdx.x == 0)
    for (int k = 0; k < kThreads / 32; ++k) t += scratch[k];
  return t;   // valid in thread 0
}

struct MixSmem {
  float* slabs;
  uint64_t* full;
  int* nbr;
  float* wgt;
  float4* mean;
  float4* red;
  double* dscratch;
  int* flags;   // [0]: fail, [1]: last
};

__device__ __forceinline__ MixSmem carve(unsigned char* raw, const MixArgs& a, int kp1) {
  MixSmem m;
  uintptr_t base = (reinterpret_cast<uintptr_t>(raw) + 1023) & ~static_cast<uintptr_t>(1023);
  const size_t slab_bytes = (static_cast<size_t>(a.rows_pad) * a.S * 4 + 1023) & ~static_cast<size_t>(1023);
  m.slabs = reinterpret_cast<float*>(base);
  base += slab_bytes * a.stages;
  m.full = reinterpret_cast<uint64_t*>(base);
  base += 8 * a.stages;
  m.dscratch = reinterpret_cast<double*>(base);
  base += 8 * (kThreads / 32);
  m.flags = reinterpret_cast<int*>(base);
  base += 16;
  m.mean = reinterpret_cast<float4*>(base);
  base += 16 * (a.S / 4);
  m.red = reinterpret_cast<float4*>(base);
  base += 16 * kThreads;
  m.nbr = reinterpret_cast<int*>(base);
  base += 4 * static_cast<size_t>(a.N) * kp1;
  m.wgt = reinterpret_cast<float*>(base);
  return m;
}

// KP1 > 0: sparse graph with KP1 neighbours per row (compile-time);
// KP1 == 0: sparse graph, runtime a.kp1 (<= kMaxKp1Sparse);
// KP1 < 0: complete graph with equal weights.
template <int KP1, bool SHADOW>
__global__ void __launch_bounds__(kThreads, 1) k_mix(const __grid_constant__ CUtensorMap tmap, const MixArgs a) {
  extern __shared__ unsigned char smem_raw[];
  const int kp1 = KP1 > 0 ? KP1 : (KP1 == 0 ? a.kp1 : 0);
  MixSmem sm = carve(smem_raw, a, kp1);
  const int tid = threadIdx.x;
  const int S = a.S, nq = S >> 2;
  const int lq = __ffs(nq) - 1;            // nq is a power of two
  const int G = kThreads >> lq;            // row groups in the mean pass
  const size_t slab_floats = ((static_cast<size_t>(a.rows_pad) * S * 4 + 1023) & ~static_cast<size_t>(1023)) / 4;

  if (tid == 0) { sm.flags[0] = 0; sm.flags[1] = 0; }
  __syncthreads();

  // ---- NOTIFY / ACK checks (time-limited waits) ----
  for (int j = tid; j < a.N; j += kThreads) {
    unsigned e = 0;
    if (a.expect_notify) e = wait_flag(a.ready + j, a.round + 1u, true, a.wait_ns);
    if (!e) e = wait_flag(a.consumed + j, a.round, false, a.wait_ns);
    if (e) {
      record_error(a.st, e, j, a.round);
      if (e == ASAP_ERR_TIMEOUT) atomicAdd(&a.st->timeouts, 1ull);
      atomicOr(&sm.flags[0], 1);
    }
  }
  __syncthreads();
  bool failed = sm.flags[0] != 0;

  double cons = 0.0;
  if (!failed) {
    if (KP1 >= 0) {
      for (int idx = tid; idx < a.N * kp1; idx += kThreads) {
        sm.nbr[idx] = a.nbr[idx];
        sm.wgt[idx] = a.wgt[idx] * a.wscale;
      }
    }
    if (tid == 0) {
      for (int s = 0; s < a.stages; ++s) mbar_init(sm.full + s, 1);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    const long long stride = gridDim.x;
    const uint32_t tx_bytes = static_cast<uint32_t>(a.n_boxes) * a.box_rows * S * 4u;
    auto issue = [&](int stage, long long slab) {
      mbar_expect_tx(sm.full + stage, tx_bytes);
      float* dst = sm.slabs + stage * slab_floats;
      for (int b = 0; b < a.n_boxes; ++b)
        tma_load_2d(dst + static_cast<size_t>(b) * a.box_rows * S, &tmap, sm.full + stage,
                    static_cast<int>(slab * S), b * a.box_rows);
    };
    if (tid == 0) {
      for (int s = 0; s < a.stages; ++s) {
        const long long slab = blockIdx.x + s * stride;
        if (slab < a.n_slabs) issue(s, slab);
      }
    }

    const float inv_n = 1.0f / static_cast<float>(a.N);
    const int q_m = tid & (nq - 1), g_m = tid >> lq;
    int it = 0;
    for (long long slab = blockIdx.x; slab < a.n_slabs; slab += stride, ++it) {
      const int stage = it % a.stages;
      const uint32_t parity = static_cast<uint32_t>((it / a.stages) & 1);
      const bool ok = mbar_wait_bounded(sm.full + stage, parity);
      if (__syncthreads_or(!ok)) {
        if (tid == 0) record_error(a.st, ASAP_ERR_CUDA, 0xffffffffu, a.round);
        failed = true;
        break;
      }
      const float4* x4 = reinterpret_cast<const float4*>(sm.slabs + stage * slab_floats);
      const long long c0 = slab * S;

      // Column sums over all N rows: strided partials, then a fixed tree.
      float4 part = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int j = g_m; j < a.N; j += G) part = f4_add(part, x4[j * nq + q_m]);
      sm.red[tid] = part;
      __syncthreads();
      for (int h = G >> 1; h >= 1; h >>= 1) {
        if (g_m < h) sm.red[tid] = f4_add(sm.red[tid], sm.red[tid + (h << lq)]);
        __syncthreads();
      }
      if (tid < nq) {
        const float4 t = sm.red[tid];
        const float sc = inv_n * a.wscale;
        sm.mean[tid] = make_float4(t.x * sc, t.y * sc, t.z * sc, t.w * sc);
      }
      __syncthreads();

      float cacc = 0.f;
      for (int idx = tid; idx < (a.N << lq); idx += kThreads) {
        const int i = idx >> lq, q = idx & (nq - 1);
        const float4 mean = sm.mean[q];
        float4 acc;
        if (KP1 < 0) {
          acc = mean;
        } else {
          const int* nb = sm.nbr + i * kp1;
          const float* wt = sm.wgt + i * kp1;
          const float4 x0 = x4[nb[0] * nq + q];
          acc = make_float4(wt[0] * x0.x, wt[0] * x0.y, wt[0] * x0.z, wt[0] * x0.w);
#pragma unroll
          for (int m = 1; m < (KP1 > 0 ? KP1 : kMaxKp1Sparse); ++m) {
            if (KP1 == 0 && m >= kp1) break;
            acc = f4_fma(wt[m], x4[nb[m] * nq + q], acc);
          }
          const float dx = acc.x - mean.x, dy = acc.y - mean.y, dz = acc.z - mean.z, dw = acc.w - mean.w;
          cacc = fmaf(dx, dx, fmaf(dy, dy, fmaf(dz, dz, fmaf(dw, dw, cacc))));
        }
        const long long c = c0 + 4 * q;
        if (c < a.ld) {
          *reinterpret_cast<float4*>(a.out + static_cast<int64_t>(i) * a.ld + c) = acc;
          if (SHADOW) {
            __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x, acc.y);
            __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z, acc.w);
            uint2 pk;
            pk.x = *reinterpret_cast<uint32_t*>(&lo);
            pk.y = *reinterpret_cast<uint32_t*>(&hi);
            *reinterpret_cast<uint2*>(a.shadow + static_cast<int64_t>(i) * a.ld + c) = pk;
          }
        }
      }
      cons += static_cast<double>(cacc);
      __syncthreads();   // every thread is done with this stage and with mean/red
      if (tid == 0) {
        const long long nxt = slab + a.stages * stride;
        if (nxt < a.n_slabs) issue(stage, nxt);
      }
    }
  }

  // ---- per-CTA partial, ticket, and the last CTA's finalisation ----
  const double csum = block_sum_f64(cons, sm.dscratch);
  if (tid == 0) {
    a.cons_part[blockIdx.x] = csum;
    if (failed) atomicOr(&sm.flags[0], 1);
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    if (sm.flags[0]) atomicAdd(&a.st->mix_ticket, 0x10000u);   // high half counts failed CTAs
    const unsigned t = atomicAdd(&a.st->mix_ticket, 1u);
    sm.flags[1] = ((t & 0xffffu) == gridDim.x - 1) ? 1 : 0;
  }
  __syncthreads();
  if (!sm.flags[1]) return;
  __threadfence();
  const unsigned ticket = atomicAdd(&a.st->mix_ticket, 0u);
  const bool any_fail = (ticket >> 16) != 0;
  double v = 0.0;
  for (int b = tid; b < static_cast<int>(gridDim.x); b += kThreads) v += __ldcg(a.cons_part + b);
  const double ctot = block_sum_f64(v, sm.dscratch);
  double lv = 0.0;
  if (a.have_loss)
    for (int b = tid; b < a.n_loss_part; b += kThreads) lv += static_cast<double>(__ldcg(a.loss_part + b));
  const double ltot = block_sum_f64(lv, sm.dscratch);
  if (tid == 0) {
    const int slot = static_cast<int>(a.round % kMetricsCap);
    a.metrics_cons[slot] = any_fail ? __int_as_float(0x7fc00000) : static_cast<float>(sqrt(ctot));
    a.metrics_loss[slot] = (a.have_loss && !any_fail) ? static_cast<float>(ltot * a.loss_norm)
                                                      : __int_as_float(0x7fc00000);
    if (!any_fail) {
      a.st->reduces += static_cast<unsigned long long>(a.N);
      if (a.expect_notify)
        a.st->consistent_inputs += static_cast<unsigned long long>(a.N) * (KP1 < 0 ? a.N : kp1);
    }
    a.st->mix_ticket = 0u;
  }
  if (!any_fail) {
    __threadfence();
    for (int j = tid; j < a.N; j += kThreads) {
      a.stamp_next[j] = a.round + 1u;
      st_release_u32(a.consumed + j, a.round + 1u);
    }
  }
}

template <int KP1, bool SHADOW>
cudaError_t set_attr(size_t smem) {
  return cudaFuncSetAttribute(k_mix<KP1, SHADOW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem));
}

template <bool SHADOW>
cudaError_t launch_t(const CUtensorMap& tmap, const MixArgs& a, bool complete, int grid, size_t smem,
                     cudaStream_t s) {
  if (complete) {
    k_mix<-1, SHADOW><<<grid, kThreads, smem, s>>>(tmap, a);
  } else {
    switch (a.kp1) {
      case 1: k_mix<1, SHADOW><<<grid, kThreads, smem, s>>>(tmap, a); break;
      case 2: k_mix<2, SHADOW><<<grid, kThreads, smem, s>>>(tmap, a); break;
      case 3: k_mix<3, SHADOW><<<grid, kThreads, smem, s>>>(tmap, a); break;
      case 5: k_mix<5, SHADOW><<<grid, kThreads, smem, s>>>(tmap, a); break;
      default: k_mix<0, SHADOW><<<grid, kThreads, smem, s>>>(tmap, a); break;
    }
  }
  return cudaGetLastError();
}

template <bool SHADOW>
cudaError_t configure_t(bool complete, int kp1, size_t smem) {
  if (complete) return set_attr<-1, SHADOW>(smem);
  switch (kp1) {
    case 1: return set_attr<1, SHADOW>(smem);
    case 2: return set_attr<2, SHADOW>(smem);
    case 3: return set_attr<3, SHADOW>(smem);
    case 5: return set_attr<5, SHADOW>(smem);
    default: return set_attr<0, SHADOW>(smem);
  }
}

template <int KP1, bool SHADOW>
cudaError_t occ_one(size_t smem, int* blocks) {
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, k_mix<KP1, SHADOW>, kThreads, smem);
}

template <bool SHADOW>
cudaError_t occupancy_t(bool complete, int kp1, size_t smem, int* blocks) {
  if (complete) return occ_one<-1, SHADOW>(smem, blocks);
  switch (kp1) {
    case 1: return occ_one<1, SHADOW>(smem, blocks);
    case 2: return occ_one<2, SHADOW>(smem, blocks);
    case 3: return occ_one<3, SHADOW>(smem, blocks);
    case 5: return occ_one<5, SHADOW>(smem, blocks);
    default: return occ_one<0, SHADOW>(smem, blocks);
  }
}

__global__ void k_cast_bf16(const float* __restrict__ src, uint16_t* __restrict__ dst, int64_t n) {
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    __nv_bfloat16 b = __float2bfloat16_rn(src[i]);
    dst[i] = *reinterpret_cast<uint16_t*>(&b);
  }
}

}  // namespace

size_t mix_smem_bytes(int N, int kp1, int S, int rows_pad, int stages) {
  const size_t slab_bytes = (static_cast<size_t>(rows_pad) * S * 4 + 1023) & ~static_cast<size_t>(1023);
  return 1024 + slab_bytes * stages + 8 * stages + 8 * (kThreads / 32) + 16 + 16 * (S / 4) + 16 * kThreads +
         8 * static_cast<size_t>(N) * kp1;
}

cudaError_t mix_configure(bool complete, int kp1, bool shadow, size_t smem) {
  return shadow ? configure_t<true>(complete, kp1, smem) : configure_t<false>(complete, kp1, smem);
}

cudaError_t mix_occupancy(bool complete, int kp1, bool shadow, size_t smem, int* blocks) {
  return shadow ? occupancy_t<true>(complete, kp1, smem, blocks) : occupancy_t<false>(complete, kp1, smem, blocks);
}

cudaError_t launch_mix(const CUtensorMap& tmap, const MixArgs& a, bool complete, int grid, size_t smem,
                       cudaStream_t s) {
  return a.shadow ? launch_t<true>(tmap, a, complete, grid, smem, s)
                  : launch_t<false>(tmap, a, complete, grid, smem, s);
}

cudaError_t launch_cast_bf16(const float* src, uint16_t* dst, int64_t n, cudaStream_t s) {
  const int grid = static_cast<int>(std::min<int64_t>((n + kThreads - 1) / kThreads, 4096));
  k_cast_bf16<<<grid > 0 ? grid : 1, kThreads, 0, s>>>(src, dst, n);
  return cudaGetLastError();
}

}  // namespace asap
