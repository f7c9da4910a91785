// Local minibatch SGD step for sparse linear models (Eq. A.1, first line).
//
// The step is split so that no kernel touches w at random addresses:
//
//   margin kernel   m_b = sum_e val_e * wv[pos_e]          (8 lanes per row)
//                   r_b = d loss(y_b, m_b) / d m_b        (hinge or logistic)
//   update kernel   g[p] = sum_{e : pos_e = p} r_{row_e} val_e   (column sums)
//                   then NOTIFY ready[i] = t+1
//
// Each round's minibatch has, per worker, a list of the distinct columns it
// touches.  The lists of all workers are laid out slab-major (by column slab
// of the stochastic reduce, then worker, then column) and `pos` indexes that
// list.  `wv[pos]` holds w_i[col] for the round's columns: the previous
// round's reduce writes it while it holds the column slab in shared memory
// (or, after parameters were written from the host, the gather kernel
// below).  The reduce applies w_i[col] -= eta/B * g[pos] to the slab before
// mixing it, so w_{t+1/2} never has to be written to HBM.
//
// Margin kernel: 8 lanes per row (4 rows in flight per warp), 128-bit loads
// of (pos, val), the L2-resident wv gathered, a fixed butterfly sum.
// Update kernel: entries sorted by (column, row) are
// cut into 32-entry chunks, one warp per chunk; a segmented warp scan sums
// each column's run and the warp holding a run's first entry owns it,
// finishing runs that cross into later chunks itself.  No atomics on data,
// every sum in a fixed order: the result does not depend on the schedule.
#include <cuda_runtime.h>

#include <cstdint>

#include "asap_internal.h"

namespace asap {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kMarginRowsPerCta = 32;     // 8 warps x 4 rows
constexpr int kUpdateChunksPerCta = 32;   // 8 warps x 4 chunks of 32 entries

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

__device__ __forceinline__ int4 ld_stream_i4(const int4* p) {
  int4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.s32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__device__ __forceinline__ float4 ld_stream_f4(const float4* p) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "l"(p));
  return v;
}

// Gather of an exported w value, keeping the line in L2 (it is re-read by
// other rows of the minibatch).
__device__ __forceinline__ float ld_keep(const float* p, uint64_t policy) {
  float v;
  asm volatile("ld.global.nc.L2::cache_hint.f32 %0, [%1], %2;" : "=f"(v) : "l"(p), "l"(policy));
  return v;
}

// Programmatic dependent launch: the next kernel in the stream may start its
// CTAs now; this kernel waits here for the previous kernel's results.
__device__ __forceinline__ void allow_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void wait_previous() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void st_release_u32(unsigned int* p, unsigned int v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
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

template <int LOSS>
__global__ void __launch_bounds__(kThreads) k_margin_loss(SparseStepArgs a) {
  // 8 lanes per row, so that each warp keeps the loads of 4 rows in flight.
  constexpr int kLanesPerRow = 8;
  const int i = blockIdx.y;
  const BatchDesc dsc = a.desc[i];
  const int* rp = reinterpret_cast<const int*>(a.block + dsc.rp);
  const float* y = reinterpret_cast<const float*>(a.block + dsc.y);
  const int4* pos4 = reinterpret_cast<const int4*>(a.block + dsc.posw);
  const float4* val4 = reinterpret_cast<const float4*>(a.block + dsc.val);
  allow_dependents();
  const float* wv = a.wv;
  uint64_t keep;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(keep));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sub = lane / kLanesPerRow, sl = lane % kLanesPerRow;
  const int b = blockIdx.x * kMarginRowsPerCta + warp * (32 / kLanesPerRow) + sub;   // 8 warps x 4 rows
  float lsum = 0.f;
  float acc = 0.f;
  if (b < a.B) {
    const int q0 = rp[b] >> 2, q1 = rp[b + 1] >> 2;
    // Four quads per lane per pass, all loads issued before the sums; the
    // summation order is the sequential one (quad after quad).
    constexpr int kU = 4;
    for (int q = q0 + sl; q < q1; q += kU * kLanesPerRow) {
      int4 p[kU];
      float4 v[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int qq = q + u * kLanesPerRow;
        if (qq < q1) {
          p[u] = ld_stream_i4(pos4 + qq);
          v[u] = ld_stream_f4(val4 + qq);
        } else {
          p[u] = make_int4(0, 0, 0, 0);
          v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
      float g[4 * kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        g[4 * u + 0] = ld_keep(wv + p[u].x, keep);
        g[4 * u + 1] = ld_keep(wv + p[u].y, keep);
        g[4 * u + 2] = ld_keep(wv + p[u].z, keep);
        g[4 * u + 3] = ld_keep(wv + p[u].w, keep);
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        if (q + u * kLanesPerRow < q1) {
          acc = fmaf(v[u].x, g[4 * u + 0], acc);
          acc = fmaf(v[u].y, g[4 * u + 1], acc);
          acc = fmaf(v[u].z, g[4 * u + 2], acc);
          acc = fmaf(v[u].w, g[4 * u + 3], acc);
        }
      }
    }
  }
#pragma unroll
  for (int o = kLanesPerRow / 2; o > 0; o >>= 1) acc += __shfl_xor_sync(kFull, acc, o);
  if (b < a.B && sl == 0) {
    float l, r;
    loss_and_r<LOSS>(y[b], acc * a.mscale, l, r);
    a.r[static_cast<int64_t>(i) * a.B + b] = r;
    lsum = l;
  }
  // fixed-order sum of the CTA's 32 row losses
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) lsum += __shfl_xor_sync(kFull, lsum, o);
  __shared__ float part[kThreads / 32];
  if (lane == 0) part[warp] = lsum;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < kThreads / 32; ++k) s += part[k];
    a.loss_part[static_cast<int64_t>(i) * gridDim.x + blockIdx.x] = s;
  }
}

__global__ void __launch_bounds__(kThreads) k_column_sums(SparseStepArgs a) {
  allow_dependents();
  const int i = blockIdx.y;
  const BatchDesc dsc = a.desc[i];
  const int nnz = dsc.nnz;
  const int* cpos = reinterpret_cast<const int*>(a.block + dsc.cpos);
  const float* cval = reinterpret_cast<const float*>(a.block + dsc.cval);
  const uint16_t* crow = reinterpret_cast<const uint16_t*>(a.block + dsc.crow);
  const float* r = a.r + static_cast<int64_t>(i) * a.B;
  float* g = a.gsum;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const unsigned le_mask = (lane == 31) ? kFull : ((2u << lane) - 1u);

  const int n_chunks = (nnz + 31) >> 5;
  constexpr int kPerWarp = kUpdateChunksPerCta / (kThreads / 32);   // 4 chunks per warp per pass
  for (int first = blockIdx.x * kUpdateChunksPerCta; first < n_chunks; first += gridDim.x * kUpdateChunksPerCta) {
    // Load the warp's chunks first (independent), then scan them one by one.
    int cv[kPerWarp], cpv[kPerWarp], cnx[kPerWarp], rw[kPerWarp];
    float pv[kPerWarp];
#pragma unroll
    for (int u = 0; u < kPerWarp; ++u) {
      const int chunk = first + warp + u * (kThreads / 32);
      const int e = chunk * 32 + lane;
      const bool valid = chunk < n_chunks && e < nnz;
      cv[u] = valid ? cpos[e] : -1;
      cpv[u] = (lane == 0 && chunk < n_chunks && e > 0) ? cpos[e - 1] : -2;
      // the entry after the chunk: does lane 31's run continue past it?
      cnx[u] = (lane == 31 && chunk < n_chunks && e + 1 < nnz) ? cpos[e + 1] : -3;
      pv[u] = valid ? cval[e] : 0.f;
      rw[u] = valid ? crow[e] : -1;
    }
    wait_previous();   // r comes from the margin kernel
#pragma unroll
    for (int u = 0; u < kPerWarp; ++u)
      if (rw[u] >= 0) pv[u] *= r[rw[u]];
#pragma unroll
    for (int u = 0; u < kPerWarp; ++u) {
    const int chunk = first + warp + u * (kThreads / 32);
    if (chunk >= n_chunks) break;                  // warp-uniform
    const int e = chunk * 32 + lane;
    const bool valid = e < nnz;
    const int c = cv[u];
    int cprev = __shfl_up_sync(kFull, c, 1);
    if (lane == 0) cprev = cpv[u];
    const bool head = valid && (c != cprev);
    float p = pv[u];
    const unsigned heads = __ballot_sync(kFull, head);
    const unsigned hl = heads & le_mask;
    const int start = hl ? (31 - __clz(hl)) : -1;   // first lane of this lane's run, -1: began earlier
    const int s_eff = start < 0 ? 0 : start;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const float v = __shfl_up_sync(kFull, p, off);
      if (lane - off >= s_eff) p += v;
    }
    const bool next_head = __shfl_down_sync(kFull, head, 1);
    const bool next_valid = __shfl_down_sync(kFull, valid, 1);
    // Runs that end inside the chunk: the tail lane writes if the run began here.
    if (valid && lane < 31 && (next_head || !next_valid) && start >= 0) g[c] = p;
    // The run through lane 31.
    const int c31 = __shfl_sync(kFull, c, 31);
    const int start31 = __shfl_sync(kFull, start, 31);
    const float p31 = __shfl_sync(kFull, p, 31);
    if (c31 >= 0 && start31 >= 0) {
      const int e31 = chunk * 32 + 31;
      bool cont = (e31 + 1 < nnz) && (__shfl_sync(kFull, cnx[u], 31) == c31);
      float acc = p31;
      int base = e31 + 1;
      while (cont) {
        const int e2 = base + lane;
        const bool in_run = (e2 < nnz) && (cpos[e2] == c31);
        const float q = in_run ? r[crow[e2]] * cval[e2] : 0.f;
        acc += warp_sum(q);
        const unsigned run = __ballot_sync(kFull, in_run);
        cont = (run == kFull) && (base + 32 < nnz) && (cpos[base + 32] == c31);
        base += 32;
      }
      if (lane == 0) g[c31] = acc;
    }
    }
  }

  // A CTA without chunks has not waited for the margin kernel yet.  Were no
  // CTA to wait (an all-empty minibatch), this grid could complete before the
  // margin kernel, and the reduce would read its loss partials too early.
  wait_previous();

  // NOTIFY: the last CTA of worker i publishes ready[i] = round + 1 once all
  // of worker i's column sums are visible device-wide.  The CTA barrier
  // orders this CTA's writes before thread 0's fence, which is cumulative.
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned int done = atomicAdd(&a.worker_ticket[i], 1u);
    if (done == gridDim.x - 1) {
      a.worker_ticket[i] = 0u;
      __threadfence();
      if (a.notify && i != a.skip_worker) st_release_u32(&a.ready[i], a.round + 1u);
    }
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

cudaError_t launch_margin(const SparseStepArgs& a, int N, int loss, int margin_ctas, cudaStream_t s) {
  const dim3 g1(margin_ctas, N);
  if (loss == ASAP_LOSS_HINGE)
    k_margin_loss<ASAP_LOSS_HINGE><<<g1, kThreads, 0, s>>>(a);
  else
    k_margin_loss<ASAP_LOSS_LOGISTIC><<<g1, kThreads, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_update(const SparseStepArgs& a, int N, int update_ctas, cudaStream_t s) {
  // Launched as a programmatic dependent of the margin kernel.
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(update_ctas, N);
  cfg.blockDim = dim3(kThreads);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_column_sums, a);
}

cudaError_t launch_gather_wv(const float* W, int64_t ld, const uint32_t* list, const int* slab_off, long long n_slabs,
                             int S, float* wv, int sm_count, cudaStream_t s) {
  k_gather_wv<<<slab_warp_grid(n_slabs, sm_count), kThreads, 0, s>>>(W, ld, list, slab_off, n_slabs, S, wv);
  return cudaGetLastError();
}

int margin_ctas_for(int B) { return (B + kMarginRowsPerCta - 1) / kMarginRowsPerCta; }
int update_ctas_for(int max_nnz) {
  const int chunks = (max_nnz + 31) / 32;
  const int c = (chunks + kUpdateChunksPerCta - 1) / kUpdateChunksPerCta;
  return c < 1 ? 1 : c;
}

}  // namespace asap
