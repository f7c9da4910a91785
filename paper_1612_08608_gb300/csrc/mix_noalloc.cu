// asap_mix_noalloc: the stochastic reduce with its consensus error, for
// callers that must not allocate device memory.
//
// Some callers cannot call cudaMalloc: a host framework that reserves
// (nearly) all of HBM for its own pool and tracks every byte, where an
// untracked cudaMalloc fails or breaks its budget; or a latency-critical
// loop, where cudaMalloc / cudaFree may synchronise the device and take an
// unbounded time.  The context API allocates its scratch at creation, so it
// does not suit them.  This entry point takes only caller-owned inputs and
// outputs.  Its one piece of scratch (a ticket counter and per-slab partial
// sums of the consensus error) is the file-scope array below, which every
// GPU that loads this library holds until the process exits.
//
// Compared with the context's reduce kernel it uses plain vectorised loads
// instead of a TMA pipeline, no NOTIFY-ACK flags and at most 256 workers;
// the arithmetic (weights applied in row order, column means from the
// input, fp64 partial sums) is the same.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <mutex>

#include "asap_internal.h"

namespace asap {
void set_thread_error(const char* msg);
}

namespace {

using namespace asap;

constexpr int kNoAllocMaxN = 256;
constexpr int kNoAllocMaxSlabs = 32768;               // consensus partials: one per column slab
constexpr int kNoAllocTicketBytes = 256;
constexpr size_t kNoAllocScratchBytes = kNoAllocTicketBytes + 8u * kNoAllocMaxSlabs;   // 262,400 bytes
constexpr int kNoAllocMaxDevices = 64;

// [0, 4): ticket counter; [256, 256 + 8 * kNoAllocMaxSlabs): double partials.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

struct NoAllocArgs {
  const float* in;
  float* out;
  int64_t ld;
  int N;
  int kp1;
  const int* nbr;
  const float* wgt;
  int S;           // slab width (columns), a power of two >= 4
  long long n_slabs;
  float* consensus_out;
  unsigned int* ticket;
  double* partial;
};

// Block sums are carried as float-float pairs hi + lo in fp32 arithmetic
// (this GPU's fp64 pipe is narrow): the rounding error of each addition of
// the high parts is recovered exactly (Knuth's two-sum) and kept in lo.
struct Pair {
  float hi, lo;
};

__device__ __forceinline__ Pair pair_add(Pair a, Pair b) {
  const float s = a.hi + b.hi;
  const float bv = s - a.hi;
  const float e = ((a.hi - (s - bv)) + (b.hi - bv)) + (a.lo + b.lo);
  const float hi = s + e;
  return Pair{hi, e - (hi - s)};
}

// Sum over the block in a fixed order; valid in thread 0.
__device__ __forceinline__ Pair block_sum(Pair v, Pair* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
    v = pair_add(v, Pair{__shfl_xor_sync(0xffffffffu, v.hi, o), __shfl_xor_sync(0xffffffffu, v.lo, o)});
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  Pair t{0.f, 0.f};
  if (threadIdx.x == 0)
    for (int w = 0; w < kThreads / 32; ++w) t = pair_add(t, red[w]);
  return t;
}

__global__ void __launch_bounds__(kThreads) k_mix_noalloc(const NoAllocArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int S = a.S, nq = S >> 2;
  const int lq = __ffs(nq) - 1;
  float4* slab = reinterpret_cast<float4*>(smem);                       // [N][nq]
  float4* mean = slab + static_cast<size_t>(a.N) * nq;                  // [nq]
  float4* red4 = mean + nq;                                             // [kThreads]
  Pair* red = reinterpret_cast<Pair*>(red4 + kThreads);                 // [kThreads / 32]
  int* flag = reinterpret_cast<int*>(red + kThreads / 32);
  const int tid = threadIdx.x;
  const int G = kThreads >> lq;
  const int q_m = tid & (nq - 1), g_m = tid >> lq;
  const float inv_n = 1.0f / static_cast<float>(a.N);

  for (long long s = blockIdx.x; s < a.n_slabs; s += gridDim.x) {
    const long long c0 = s * S;
    for (int idx = tid; idx < (a.N << lq); idx += kThreads) {
      const int i = idx >> lq, q = idx & (nq - 1);
      const long long c = c0 + 4 * q;
      slab[idx] = (c < a.ld) ? *reinterpret_cast<const float4*>(a.in + static_cast<int64_t>(i) * a.ld + c)
                             : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    __syncthreads();
    float4 part = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int j = g_m; j < a.N; j += G) {
      const float4 x = slab[j * nq + q_m];
      part.x += x.x; part.y += x.y; part.z += x.z; part.w += x.w;
    }
    red4[tid] = part;
    __syncthreads();
    for (int h = G >> 1; h >= 1; h >>= 1) {
      if (g_m < h) {
        const float4 o = red4[tid + (h << lq)];
        float4 t = red4[tid];
        t.x += o.x; t.y += o.y; t.z += o.z; t.w += o.w;
        red4[tid] = t;
      }
      __syncthreads();
    }
    if (tid < nq) {
      const float4 t = red4[tid];
      mean[tid] = make_float4(t.x * inv_n, t.y * inv_n, t.z * inv_n, t.w * inv_n);
    }
    __syncthreads();
    float cacc = 0.f;
    for (int idx = tid; idx < (a.N << lq); idx += kThreads) {
      const int i = idx >> lq, q = idx & (nq - 1);
      const int* nb = a.nbr + i * a.kp1;
      const float* wt = a.wgt + i * a.kp1;
      // Ids outside [0, N) are clamped so that a bad table cannot read
      // outside the slab; the caller must pass valid ids.
      const float w0 = __ldg(wt);
      const float4 x0 = slab[min(max(__ldg(nb), 0), a.N - 1) * nq + q];
      float4 acc = make_float4(w0 * x0.x, w0 * x0.y, w0 * x0.z, w0 * x0.w);
      for (int m = 1; m < a.kp1; ++m) {
        const float w = __ldg(wt + m);
        const float4 x = slab[min(max(__ldg(nb + m), 0), a.N - 1) * nq + q];
        acc.x = fmaf(w, x.x, acc.x);
        acc.y = fmaf(w, x.y, acc.y);
        acc.z = fmaf(w, x.z, acc.z);
        acc.w = fmaf(w, x.w, acc.w);
      }
      const float4 mu = mean[q];
      const float dx = acc.x - mu.x, dy = acc.y - mu.y, dz = acc.z - mu.z, dw = acc.w - mu.w;
      cacc = fmaf(dx, dx, fmaf(dy, dy, fmaf(dz, dz, fmaf(dw, dw, cacc))));
      const long long c = c0 + 4 * q;
      if (c < a.ld) *reinterpret_cast<float4*>(a.out + static_cast<int64_t>(i) * a.ld + c) = acc;
    }
    const Pair ps = block_sum(Pair{cacc, 0.f}, red);
    if (tid == 0) a.partial[s] = static_cast<double>(ps.hi) + static_cast<double>(ps.lo);
    __syncthreads();   // the slab buffer is reused by the next slab
  }

  // The last CTA sums the per-slab partials in a fixed order (the result does
  // not depend on which CTA finishes last).
  __threadfence();
  __syncthreads();
  if (tid == 0) flag[0] = (atomicAdd(a.ticket, 1u) == gridDim.x - 1) ? 1 : 0;
  __syncthreads();
  if (!flag[0]) return;
  __threadfence();
  Pair v{0.f, 0.f};
  for (long long s = tid; s < a.n_slabs; s += kThreads) {
    const double p = __ldcg(a.partial + s);
    const float h = static_cast<float>(p);
    v = pair_add(v, Pair{h, static_cast<float>(p - static_cast<double>(h))});
  }
  const Pair total = block_sum(v, red);
  if (tid == 0) {
    a.consensus_out[0] = sqrtf(fmaxf(total.hi + total.lo, 0.f));
    *a.ticket = 0u;
  }
}

struct DeviceSlot {
  void* scratch = nullptr;
  int sm_count = 0;
  unsigned long long ctx_id = 0;   // the CUDA context the address belongs to
};

// Unique id of the calling thread's current CUDA context (0: none current).
// A device reset, or a host framework that resets its primary context,
// reloads this library's module at a new address; the id tells the cached
// scratch address apart from a stale one.  The driver entry points are
// looked up through the runtime, so the library needs no link to libcuda.
unsigned long long current_context_id() {
  typedef CUresult (*GetCurrentFn)(CUcontext*);
  typedef CUresult (*GetIdFn)(CUcontext, unsigned long long*);
  static GetCurrentFn get_current = nullptr;
  static GetIdFn get_id = nullptr;
  static bool looked_up = false;
  if (!looked_up) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<GetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<GetIdFn>(p);
    looked_up = true;
  }
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

std::mutex g_noalloc_mu;
DeviceSlot g_noalloc_dev[kNoAllocMaxDevices];

asap_status reject(asap_status s, const char* msg) {
  set_thread_error(msg);
  return s;
}

}  // namespace

extern "C" asap_status asap_mix_noalloc(const float* W_in, float* W_out, int N, int64_t d, int64_t ld,
                                        const int32_t* nbr, const float* wgt, int kp1, float* consensus_out,
                                        void* cuda_stream) {
  if (!W_in || !W_out || !nbr || !wgt || !consensus_out)
    return reject(ASAP_ERR_ARG, "asap_mix_noalloc: NULL pointer");
  if (N < 1 || N > kNoAllocMaxN) return reject(ASAP_ERR_ARG, "asap_mix_noalloc: need 1 <= N <= 256");
  if (kp1 < 1 || kp1 > kMaxKp1Sparse) return reject(ASAP_ERR_ARG, "asap_mix_noalloc: need 1 <= k+1 <= 32");
  if (d < 1 || ld < d || ld % 4 != 0)
    return reject(ASAP_ERR_ARG, "asap_mix_noalloc: need d >= 1, ld >= d and ld a multiple of 4");
  if ((reinterpret_cast<uintptr_t>(W_in) | reinterpret_cast<uintptr_t>(W_out)) & 15u)
    return reject(ASAP_ERR_ARG, "asap_mix_noalloc: W_in and W_out must be 16-byte aligned");
  int S = 256;
  while (S > 4 && static_cast<size_t>(N) * S * 4 > 16384) S >>= 1;
  const long long n_slabs = (ld + S - 1) / S;
  if (n_slabs > kNoAllocMaxSlabs)
    return reject(ASAP_ERR_ARG, "asap_mix_noalloc: ld too large for the built-in scratch "
                                "(at most 32768 slabs of 256 columns for N <= 16, 16 columns for N = 256)");
  {
    // Every CTA reads rows of W_in that other CTAs may already have written
    // to W_out: the two ranges must not overlap at all.
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(W_in), b0 = reinterpret_cast<uintptr_t>(W_out);
    const uintptr_t bytes = static_cast<uintptr_t>(N) * static_cast<uintptr_t>(ld) * sizeof(float);
    if (a0 < b0 + bytes && b0 < a0 + bytes)
      return reject(ASAP_ERR_ARG, "asap_mix_noalloc: W_in and W_out must not overlap");
  }

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kNoAllocMaxDevices)
    return reject(ASAP_ERR_CUDA, "asap_mix_noalloc: no usable current device");
  DeviceSlot slot;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    DeviceSlot& ds = g_noalloc_dev[dev];
    const unsigned long long cur = current_context_id();
    if (!ds.scratch || cur == 0 || cur != ds.ctx_id) {
      // First call on this device (or in a new context of it): resolve the
      // device address of the file-scope scratch (the host-side name is only
      // a stand-in).  This also makes the device's primary context current.
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p)
        return reject(ASAP_ERR_CUDA, "asap_mix_noalloc: cudaGetSymbolAddress failed for the scratch array");
      int sms = 0;
      if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return reject(ASAP_ERR_CUDA, "asap_mix_noalloc: cannot query the SM count");
      ds.scratch = p;
      ds.sm_count = sms;
      ds.ctx_id = current_context_id();
    }
    slot = ds;
  }
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  unsigned char* base = static_cast<unsigned char*>(slot.scratch);
  NoAllocArgs a;
  a.in = W_in;
  a.out = W_out;
  a.ld = ld;
  a.N = N;
  a.kp1 = kp1;
  a.nbr = nbr;
  a.wgt = wgt;
  a.S = S;
  a.n_slabs = n_slabs;
  a.consensus_out = consensus_out;
  a.ticket = reinterpret_cast<unsigned int*>(base);
  a.partial = reinterpret_cast<double*>(base + kNoAllocTicketBytes);
  // The ticket must start at zero; the array keeps whatever the last call left.
  if (cudaMemsetAsync(a.ticket, 0, sizeof(unsigned int), s) != cudaSuccess)
    return reject(ASAP_ERR_CUDA, "asap_mix_noalloc: clearing the ticket failed");
  const int nq = S / 4;
  const size_t smem = 16 * (static_cast<size_t>(N) * nq + nq + kThreads) + 8 * (kThreads / 32) + 16;
  const int grid = static_cast<int>(std::min<long long>(n_slabs, 4LL * slot.sm_count));
  k_mix_noalloc<<<grid, kThreads, smem, s>>>(a);
  if (cudaGetLastError() != cudaSuccess) return reject(ASAP_ERR_CUDA, "asap_mix_noalloc: launch failed");
  return ASAP_OK;
}
