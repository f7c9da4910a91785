// Host runtime behind include/asap.h: context and device memory, graph
// schedule, shard layout (index builder), launch sequencing of one ASAP
// round (Eq. A.1), NOTIFY-ACK state and error reporting.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <memory>
#include <string>
#include <thread>
#include <limits>
#include <vector>

#include "asap_internal.h"


using namespace asap;

namespace {

thread_local std::string g_last_error;

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

}  // namespace

namespace asap {
// Records a failure message for asap_last_error(NULL) on this thread.
void set_thread_error(const char* msg) { g_last_error = msg; }
}  // namespace asap

struct asap_ctx {
  int dev = 0, sm_count = 0;
  int N = 0;
  int64_t d = 0;
  uint64_t seed = 0;
  int k = 0;
  asap_graph_kind kind = ASAP_GRAPH_IDENTITY;
  bool regen = false;
  bool have_explicit = false;
  std::vector<int32_t> ex_nbr;
  std::vector<float> ex_wgt;
  int tab_kp1 = 1;          // neighbours per row in the device tables (0 for COMPLETE)
  int64_t graph_round_in_slot0 = -2;

  asap_loss loss = ASAP_LOSS_NONE;
  int C = 1, B = 0;
  float lr = 0.f, l2 = 0.f;
  // schedule: local steps per round, eta_k = lr (constant) or lr / (1 + gamma k)
  int tau = 1;
  int lr_kind = ASAP_LR_CONSTANT;
  float lr_gamma = 0.f;
  // left by the last local step for the fused reduce
  float pend_wscale = 1.f;          // true w = pend_wscale * stored values
  float pend_upd = 0.f;             // eta / (B pend_wscale)
  int64_t pend_k = 0;               // global step of the last local step
  int64_t P = 0, ld = 0;

  float* W[2] = {nullptr, nullptr};
  uint16_t* Wbf[2] = {nullptr, nullptr};
  unsigned* ready = nullptr;
  unsigned* consumed = nullptr;
  unsigned* stamp = nullptr;     // [2][N]
  unsigned* ticket = nullptr;    // [N]
  DevState* st = nullptr;
  float* m_loss = nullptr;
  float* m_cons = nullptr;
  float* r_scr = nullptr;
  float* loss_part = nullptr;
  float* mpart_big = nullptr;        // sparse, B > kRSmemRows: per-warp partial margins [N][Q][4][B]
  float* r_big = nullptr;            // sparse, B > kRSmemRows: r [N][Q][B]
  int* d_worker_of = nullptr;        // sparse: worker of each local-step cluster (a permutation)
  bool permuted = false;             // d_worker_of differs from the identity
  // worker-sharded mode (asap_set_worker_range): this context steps workers
  // [own_lo, own_lo + own_n); the rows of the others are delivered by the caller
  bool sharded = false;
  int own_lo = 0, own_n = 0;
  std::vector<unsigned char> delivered;   // [N] row j written this round (asap_write_rows)
  double* cons_part = nullptr;
  int cons_cap = 0;
  int32_t* d_nbr = nullptr;
  float* d_wgt = nullptr;
  int32_t* h_nbr = nullptr;
  float* h_wgt = nullptr;
  // Regenerated graphs: the ring's two halves hold batches of kGraphBatch
  // rounds (batch b = round / kGraphBatch in half b & 1), uploaded on the
  // copy stream one batch at a time.
  int64_t graph_half_batch[2] = {-1, -1};
  cudaEvent_t graph_half_ev[2] = {};   // the half's last upload
  bool graph_half_used[2] = {false, false};
  cudaEvent_t graph_order_ev = nullptr; // the stream's work before an upload

  // sparse shards
  asap_residency residency = ASAP_SHARDS_DEVICE;
  unsigned char* pool = nullptr;  // device or pinned host
  bool pool_pinned = false;
  size_t pool_bytes = 0;
  std::vector<size_t> block_off, block_bytes;
  int nb = 0;
  BatchDesc* d_desc = nullptr;
  // per batch block: the slab-major column list and its slab offsets
  std::vector<size_t> list_off, soff_off;
  std::vector<int64_t> list_len;
  int max_region = 0;               // entries of the largest slab region of any list
  int64_t max_list = 0;
  float* wv[2] = {nullptr, nullptr};  // w at the list positions of round t's steps: wv[t & 1] (the
                                    // reduce of round t writes wv[(t+1) & 1] while round t's step may run)
  float* gsum = nullptr;            // column sums at the current round's list positions
  int64_t wv_step = -1;             // global local step whose column list wv holds (-1: none)
  // host residency: a round reads its own block and the next one
  static constexpr int kStaging = 3;
  unsigned char* staging[kStaging] = {nullptr, nullptr, nullptr};
  size_t staging_bytes = 0;
  int64_t staged_round[kStaging] = {-1, -1, -1};
  bool free_recorded[kStaging] = {false, false, false};
  cudaEvent_t staged_ev[kStaging] = {}, free_ev[kStaging] = {};
  int step_q = 1;                   // CTAs per worker (cluster size) of the local step
  int step_stages = 3;              // ring stages of the local step
  size_t step_smem = 0;
  int max_nnz = 0;

  // dense softmax shards and scratch
  uint16_t* X = nullptr;     // [N][nb*B][d] bf16
  uint16_t* XT = nullptr;    // [N][nb][d][B] bf16
  int32_t* Yd = nullptr;     // [N][nb*B]
  uint16_t* RT = nullptr;    // [N][Cq*256][B] bf16
  int Cq = 0;
  int n_loss_part = 0;
  CUtensorMap tmX, tmXT, tmR, tmWbf[2], tmWf[2];
  bool dense_configured = false;

  cudaStream_t stream = nullptr, own_stream = nullptr, copy_stream = nullptr;
  // An event recorded after every round's reduce (a ring), so that a metrics
  // read waits for its own rounds only while later rounds keep the GPU busy.
  static constexpr int kRoundEvents = 64;
  cudaEvent_t round_ev[kRoundEvents] = {};
  int64_t round_ev_round[kRoundEvents] = {};   // round recorded in each slot, -1: none
  cudaStream_t read_stream = nullptr;

  CUtensorMap tmap[2];
  int S = 0, rows_pad = 0, box_rows = 0, n_boxes = 0, stages = 0;
  int s_cap = 1024;                 // upper bound on the slab width (lowered for skewed column lists)
  bool fused_cfg = false;
  long long n_slabs = 0;
  int mix_grid = 0;
  size_t mix_smem = 0;
  long long configured_key = -1;

  // per-kernel timing (asap_set_kernel_timing)
  bool timing = false;
  std::vector<cudaEvent_t> tev;   // 2 per timed launch
  std::vector<int> tkind;
  size_t tused = 0;

  int64_t round = 0;
  int64_t graph_ready_round = -1;   // round whose tables are staged in graph_nbr/graph_wgt
  const int* graph_nbr = nullptr;
  const float* graph_wgt = nullptr;
  bool graph_uniform = false;       // every weight of the staged table is equal
  bool step_pending = false;
  int skip_notify = -1;
  int sync_mode = kSyncBsp;         // how a sparse reduce meets its local step (asap_set_sync_mode)
  unsigned long long wait_ns = 200000000ull;
  uint64_t launches = 0;
  std::string err;
};

namespace {

asap_status fail(asap_ctx* c, asap_status s, const std::string& msg) {
  if (c) c->err = msg;
  g_last_error = msg;
  return s;
}

asap_status cuda_fail(asap_ctx* c, cudaError_t e, const char* what) {
  std::string m = std::string(what) + ": " + cudaGetErrorString(e);
  return fail(c, e == cudaErrorMemoryAllocation ? ASAP_ERR_OOM : ASAP_ERR_CUDA, m);
}

#define CU(call, what)                                   \
  do {                                                   \
    cudaError_t e_ = (call);                             \
    if (e_ != cudaSuccess) return cuda_fail(c, e_, what); \
  } while (0)

template <typename T>
void dfree(T*& p) {
  if (p) cudaFree(p);
  p = nullptr;
}

void free_shards(asap_ctx* c) {
  if (c->pool) {
    if (c->pool_pinned)
      cudaFreeHost(c->pool);
    else
      cudaFree(c->pool);
  }
  c->pool = nullptr;
  c->pool_bytes = 0;
  dfree(c->d_desc);
  dfree(c->X);
  dfree(c->XT);
  dfree(c->Yd);
  dfree(c->wv[0]);
  dfree(c->wv[1]);
  dfree(c->gsum);
  dfree(c->mpart_big);
  dfree(c->r_big);
  for (int b = 0; b < asap_ctx::kStaging; ++b) {
    dfree(c->staging[b]);
    c->staged_round[b] = -1;
    c->free_recorded[b] = false;
  }
  c->block_off.clear();
  c->block_bytes.clear();
  c->list_off.clear();
  c->soff_off.clear();
  c->list_len.clear();
  c->max_region = 0;
  c->max_list = 0;
  c->wv_step = -1;
  c->nb = 0;
}

// Host copy of the graph of round `rnd`: nbr/wgt with c->k + 1 entries per row.
asap_status graph_host(asap_ctx* c, int64_t rnd, int32_t* nbr, float* wgt) {
  const int kp1 = c->k + 1;
  if (c->kind == ASAP_GRAPH_EXPLICIT) {
    std::copy(c->ex_nbr.begin(), c->ex_nbr.end(), nbr);
    if (wgt) std::copy(c->ex_wgt.begin(), c->ex_wgt.end(), wgt);
    return ASAP_OK;
  }
  const char* why = "";
  asap_status s = build_graph_host(c->kind, c->N, c->k, c->seed, c->regen ? rnd : 0, nbr, &why);
  if (s != ASAP_OK) return fail(c, s, why);
  if (wgt) std::fill(wgt, wgt + static_cast<size_t>(c->N) * kp1, 1.0f / static_cast<float>(kp1));
  return ASAP_OK;
}

bool is_complete_kernel(const asap_ctx* c) { return c->kind == ASAP_GRAPH_COMPLETE; }

asap_status setup_mix(asap_ctx* c) {
  const int N = c->N;
  c->n_boxes = (N + 255) / 256;
  // Rows per TMA box, a multiple of 4 so that every box starts 128-byte
  // aligned in shared memory (S >= 8 floats per row).
  c->box_rows = ((N + c->n_boxes - 1) / c->n_boxes + 3) / 4 * 4;
  c->rows_pad = c->n_boxes * c->box_rows;
  // Slab: S columns of all rows, about 32 KB (8 <= S <= 1024, a power of 2).
  int S = 1024;
  while (S > 8 && static_cast<size_t>(c->rows_pad) * S * 4 > 32768) S >>= 1;
  int maxS = 8;
  while (static_cast<int64_t>(maxS) * 2 <= c->ld && maxS < 1024) maxS <<= 1;
  c->S = std::min(std::min(S, maxS), c->s_cap);
  c->n_slabs = (c->ld + c->S - 1) / c->S;
  c->tab_kp1 = is_complete_kernel(c) ? 0 : c->k + 1;
  c->configured_key = -1;
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return fail(c, ASAP_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  for (int b = 0; b < 2; ++b) {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(c->ld), static_cast<cuuint64_t>(N)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(c->ld) * 4};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(std::min(c->S, 256)), static_cast<cuuint32_t>(c->box_rows)};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&c->tmap[b], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, c->W[b], dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(c, ASAP_ERR_CUDA, "cuTensorMapEncodeTiled failed for the parameter buffer");
  }
  return ASAP_OK;
}

// bf16 tiled map with 128-byte swizzle (64-element inner box), for the
// tensor-core operands.
asap_status bf16_map(asap_ctx* c, CUtensorMap* m, void* base, int rank, const cuuint64_t* dims,
                     const cuuint64_t* strides_bytes, const cuuint32_t* box) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return fail(c, ASAP_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, base, dims, strides_bytes, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(c, ASAP_ERR_CUDA, "cuTensorMapEncodeTiled failed for a bf16 operand");
  return ASAP_OK;
}

// Maps of the two bf16 parameter copies: [N][C][d], box 64 x 256 x 1.
asap_status setup_dense_param_maps(asap_ctx* c) {
  for (int b = 0; b < 2; ++b) {
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(c->d), static_cast<cuuint64_t>(c->C),
                          static_cast<cuuint64_t>(c->N)};
    cuuint64_t str[2] = {static_cast<cuuint64_t>(c->d) * 2, static_cast<cuuint64_t>(c->ld) * 2};
    cuuint32_t box[3] = {64, 256, 1};
    asap_status s = bf16_map(c, &c->tmWbf[b], c->Wbf[b], 3, dims, str, box);
    if (s != ASAP_OK) return s;
    // fp32 master [N][C][d] for the gradient epilogue: boxes of 32 x 128 x 1, 128-byte swizzle.
    EncodeTiledFn enc = get_encode_fn();
    cuuint64_t strf[2] = {static_cast<cuuint64_t>(c->d) * 4, static_cast<cuuint64_t>(c->ld) * 4};
    cuuint32_t boxf[3] = {32, 128, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult rr = enc(&c->tmWf[b], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, c->W[b], dims, strf, boxf, estr,
                      CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (rr != CUDA_SUCCESS) return fail(c, ASAP_ERR_CUDA, "cuTensorMapEncodeTiled failed for the fp32 master");
  }
  return ASAP_OK;
}

asap_status configure_mix_launch(asap_ctx* c, bool fused) {
  const bool complete = is_complete_kernel(c);
  const bool shadow = c->Wbf[0] != nullptr;
  const int region = fused ? c->max_region : 0;
  const long long key = (complete ? 1 : 0) | (shadow ? 2 : 0) | (fused ? 4 : 0) |
                        (static_cast<long long>(c->tab_kp1) << 3) | (static_cast<long long>(region) << 12);
  if (key == c->configured_key) return ASAP_OK;
  // Stages of ~32 KB slabs: three keep enough bytes in flight per SM to
  // stream at full rate; more only queue in the memory system (on GB300 the
  // reduce alone and the dense reduce run 3-10 % faster with 3 than with 5).
  // The fused reduce holds each slab longer (the update precedes the mix)
  // and wants one more.  Fewer when the footprint does not fit.
  const int want = fused ? 4 : 3;
  c->stages = 2;
  for (int st = want; st > 2; --st)
    if (mix_smem_bytes(c->N, c->tab_kp1, c->S, c->rows_pad, st, region) <= (220u << 10)) {
      c->stages = st;
      break;
    }
  c->mix_smem = mix_smem_bytes(c->N, c->tab_kp1, c->S, c->rows_pad, c->stages, region);
  if (c->mix_smem > (227u << 10)) return fail(c, ASAP_ERR_ARG, "reduce stages do not fit in shared memory");
  CU(mix_configure(complete, fused, c->tab_kp1, shadow, c->mix_smem), "configuring the reduce kernel");
  int blocks = 0;
  CU(mix_occupancy(complete, fused, c->tab_kp1, shadow, c->mix_smem, &blocks), "occupancy of the reduce kernel");
  if (blocks < 1) return fail(c, ASAP_ERR_ARG, "reduce kernel does not fit on an SM for this N");
  c->mix_grid = static_cast<int>(std::min<long long>(c->n_slabs, static_cast<long long>(c->sm_count) * blocks));
  if (c->mix_grid > c->cons_cap) return fail(c, ASAP_ERR_ARG, "internal: reduce grid exceeds its scratch");
  c->fused_cfg = fused;
  c->configured_key = key;
  return ASAP_OK;
}

asap_status reset_protocol(asap_ctx* c, int64_t rnd) {
  std::vector<unsigned> v(c->N, static_cast<unsigned>(rnd));
  CU(cudaMemcpy(c->ready, v.data(), 4 * c->N, cudaMemcpyHostToDevice), "resetting NOTIFY flags");
  CU(cudaMemcpy(c->consumed, v.data(), 4 * c->N, cudaMemcpyHostToDevice), "resetting ACK flags");
  CU(cudaMemcpy(c->stamp + (rnd & 1) * c->N, v.data(), 4 * c->N, cudaMemcpyHostToDevice), "resetting stamps");
  CU(cudaMemset(c->ticket, 0, 4 * c->N), "resetting tickets");
  c->round = rnd;
  c->step_pending = false;
  c->graph_ready_round = -1;
  for (int i = 0; i < asap_ctx::kRoundEvents; ++i) c->round_ev_round[i] = -1;
  return ASAP_OK;
}

asap_status alloc_params(asap_ctx* c) {
  CU(cudaStreamSynchronize(c->stream), "synchronising before re-allocation");
  for (int b = 0; b < 2; ++b) {
    dfree(c->W[b]);
    dfree(c->Wbf[b]);
  }
  c->ld = static_cast<int64_t>(align_up(static_cast<size_t>(c->P), 64));
  const size_t bytes = static_cast<size_t>(c->N) * c->ld * 4;
  for (int b = 0; b < 2; ++b) {
    CU(cudaMalloc(&c->W[b], bytes), "allocating the parameter buffers");
    CU(cudaMemset(c->W[b], 0, bytes), "zeroing the parameter buffers");
    if (c->loss == ASAP_LOSS_SOFTMAX) {
      CU(cudaMalloc(&c->Wbf[b], bytes / 2), "allocating the bf16 parameter copy");
      CU(cudaMemset(c->Wbf[b], 0, bytes / 2), "zeroing the bf16 parameter copy");
    }
  }
  asap_status s = setup_mix(c);
  if (s != ASAP_OK) return s;
  if (c->loss == ASAP_LOSS_SOFTMAX) {
    s = setup_dense_param_maps(c);
    if (s != ASAP_OK) return s;
  }
  return reset_protocol(c, 0);
}

asap_status upload_fixed_graph(asap_ctx* c) {
  c->graph_round_in_slot0 = -2;
  c->graph_ready_round = -1;
  c->graph_half_batch[0] = c->graph_half_batch[1] = -1;
  if (c->tab_kp1 == 0 || c->regen) return ASAP_OK;
  const size_t n = static_cast<size_t>(c->N) * c->tab_kp1;
  std::vector<int32_t> nbr(n);
  std::vector<float> wgt(n);
  asap_status s = graph_host(c, 0, nbr.data(), wgt.data());
  if (s != ASAP_OK) return s;
  CU(cudaStreamSynchronize(c->stream), "synchronising before a graph upload");
  CU(cudaMemcpy(c->d_nbr, nbr.data(), n * 4, cudaMemcpyHostToDevice), "uploading the graph");
  CU(cudaMemcpy(c->d_wgt, wgt.data(), n * 4, cudaMemcpyHostToDevice), "uploading the graph weights");
  c->graph_round_in_slot0 = 0;
  return ASAP_OK;
}

// Device tables for round `rnd`.  Regenerated graphs are built on the host
// kGraphBatch rounds at a time into one half of a pinned ring and uploaded
// with one copy per table on the copy stream, so that the context stream
// meets an upload once per batch instead of carrying two small copies
// between the kernels of every round.  The upload into a half waits for the
// stream's earlier work (every reduce that read the half's previous batch),
// and the stream waits for the upload.
asap_status graph_tables(asap_ctx* c, int64_t rnd, const int** nbr, const float** wgt) {
  *nbr = nullptr;
  *wgt = nullptr;
  if (c->tab_kp1 == 0) return ASAP_OK;
  const size_t n = static_cast<size_t>(c->N) * c->tab_kp1;
  if (!c->regen) {
    *nbr = c->d_nbr;
    *wgt = c->d_wgt;
    return ASAP_OK;
  }
  const int64_t b = rnd / kGraphBatch;
  const int half = static_cast<int>(b & 1);
  const size_t h0 = static_cast<size_t>(half) * kGraphBatch * n;   // first entry of the half
  if (c->graph_half_batch[half] != b) {
    if (c->graph_half_used[half]) CU(cudaEventSynchronize(c->graph_half_ev[half]), "waiting for a graph upload");
    for (int j = 0; j < kGraphBatch; ++j) {
      asap_status s = graph_host(c, b * kGraphBatch + j, c->h_nbr + h0 + j * n, c->h_wgt + h0 + j * n);
      if (s != ASAP_OK) return s;
    }
    CU(cudaEventRecord(c->graph_order_ev, c->stream), "graph upload order");
    CU(cudaStreamWaitEvent(c->copy_stream, c->graph_order_ev, 0), "graph upload order");
    CU(cudaMemcpyAsync(c->d_nbr + h0, c->h_nbr + h0, kGraphBatch * n * 4, cudaMemcpyHostToDevice, c->copy_stream),
       "graph upload");
    CU(cudaMemcpyAsync(c->d_wgt + h0, c->h_wgt + h0, kGraphBatch * n * 4, cudaMemcpyHostToDevice, c->copy_stream),
       "graph upload");
    CU(cudaEventRecord(c->graph_half_ev[half], c->copy_stream), "graph upload event");
    CU(cudaStreamWaitEvent(c->stream, c->graph_half_ev[half], 0), "graph upload");
    c->graph_half_used[half] = true;
    c->graph_half_batch[half] = b;
  }
  const size_t at = h0 + static_cast<size_t>(rnd % kGraphBatch) * n;
  *nbr = c->d_nbr + at;
  *wgt = c->d_wgt + at;
  return ASAP_OK;
}

// Stage the graph of round r (no-op when it is already staged).
asap_status prepare_graph(asap_ctx* c, int64_t r) {
  if (c->graph_ready_round == r) return ASAP_OK;
  asap_status s = graph_tables(c, r, &c->graph_nbr, &c->graph_wgt);
  if (s != ASAP_OK) return s;
  c->graph_uniform = true;
  if (c->kind == ASAP_GRAPH_EXPLICIT)
    for (float w : c->ex_wgt)
      if (w != c->ex_wgt[0]) c->graph_uniform = false;
  c->graph_ready_round = r;
  return ASAP_OK;
}

constexpr size_t kTimedLaunches = 8192;

// Bracket one launch with timing events (no-op unless timing is on).
void time_begin(asap_ctx* c, int kind) {
  if (!c->timing || c->tused >= kTimedLaunches) return;
  cudaEventRecord(c->tev[2 * c->tused], c->stream);
  c->tkind[c->tused] = kind;
}

void time_end(asap_ctx* c) {
  if (!c->timing || c->tused >= kTimedLaunches) return;
  cudaEventRecord(c->tev[2 * c->tused + 1], c->stream);
  ++c->tused;
}

asap_status check_device_error(asap_ctx* c) {
  DevState h;
  CU(cudaMemcpy(&h, c->st, sizeof(DevState), cudaMemcpyDeviceToHost), "reading device state");
  if (h.err_code == 0) return ASAP_OK;
  const unsigned zero = 0;
  CU(cudaMemcpy(&c->st->err_code, &zero, 4, cudaMemcpyHostToDevice), "clearing device error");
  char buf[200];
  if (h.err_code == ASAP_ERR_TIMEOUT)
    snprintf(buf, sizeof buf, "device: NOTIFY/ACK wait ran out (worker %u, round %u); parameters are undefined "
             "until asap_write_params", h.err_worker, h.err_round);
  else if (h.err_code == ASAP_ERR_STATE)
    snprintf(buf, sizeof buf, "device: round stamp mismatch (worker %u, round %u)", h.err_worker, h.err_round);
  else
    snprintf(buf, sizeof buf, "device: error %u (worker %u, round %u)", h.err_code, h.err_worker, h.err_round);
  return fail(c, static_cast<asap_status>(h.err_code), buf);
}

asap_status sync_all(asap_ctx* c) {
  CU(cudaStreamSynchronize(c->stream), "synchronising the context stream");
  if (c->copy_stream) CU(cudaStreamSynchronize(c->copy_stream), "synchronising the copy stream");
  return check_device_error(c);
}

// The device image of minibatch t (host only): per worker the labels, the
// entries sorted by (column, row) -- list position, value, row and the
// entry's slot inside its margin segment -- and the Q column-sum ranges cut
// at column boundaries; then the batch's
// slab-major list of distinct (worker, column) pairs and its slab offsets.
// Used by asap_load_shards and, for tests, asap_debug_batch_image.
struct BatchImage {
  std::vector<unsigned char> img;
  std::vector<BatchDesc> desc;
  size_t list_off = 0, soff_off = 0;
  int64_t list_len = 0;
  int max_region = 0, max_nnz = 0;
  const char* err = nullptr;
};

void build_batch_image(int N, int B, int64_t d, int S, long long n_slabs, int Q, int t,
                       const int64_t* const* rowptr, const int32_t* const* col, const float* const* val,
                       const float* const* y, BatchImage& bt) {
  std::vector<std::vector<uint64_t>> keys(N);
  std::vector<std::vector<int32_t>> ucol(N), run_of(N), upos(N);
  std::vector<int64_t> nnz(N, 0);
  for (int i = 0; i < N; ++i) {
    const int64_t* rp = rowptr[i];
    if (!rp) continue;   // a worker this context does not step (worker-sharded): no entries
    const int64_t r0 = static_cast<int64_t>(t) * B;
    const int64_t a0 = rp[r0], a1 = rp[r0 + B];
    nnz[i] = a1 - a0;
    if (nnz[i] > (1ll << 30)) { bt.err = "a minibatch holds more than 2^30 entries"; return; }
    std::vector<uint64_t>& k = keys[i];
    k.resize(nnz[i]);
    for (int64_t e = 0; e < nnz[i]; ++e) {
      const int32_t cc = col[i][a0 + e];
      if (cc < 0 || cc >= d) { bt.err = "column id out of range [0, d)"; return; }
      k[e] = (static_cast<uint64_t>(static_cast<uint32_t>(cc)) << 32) | static_cast<uint64_t>(e);
    }
    std::sort(k.begin(), k.end());   // by column, then by entry (= by row)
    run_of[i].resize(nnz[i]);
    for (int64_t e = 0; e < nnz[i]; ++e) {
      const int32_t cc = static_cast<int32_t>(k[e] >> 32);
      if (e == 0 || cc != static_cast<int32_t>(k[e - 1] >> 32)) ucol[i].push_back(cc);
      run_of[i][e] = static_cast<int32_t>(ucol[i].size()) - 1;
    }
    bt.max_nnz = std::max<int>(bt.max_nnz, static_cast<int>(nnz[i]));
  }
  // Slab-major positions.
  std::vector<int32_t> cnt(static_cast<size_t>(n_slabs) * N, 0);
  for (int i = 0; i < N; ++i)
    for (int32_t cc : ucol[i]) cnt[static_cast<size_t>(cc / S) * N + i]++;
  std::vector<int32_t> soff(n_slabs + 1), start(static_cast<size_t>(n_slabs) * N);
  int64_t tot = 0;
  for (long long sl = 0; sl < n_slabs; ++sl) {
    soff[sl] = static_cast<int32_t>(tot);
    int64_t acc = tot;
    for (int i = 0; i < N; ++i) {
      start[static_cast<size_t>(sl) * N + i] = static_cast<int32_t>(acc);
      acc += cnt[static_cast<size_t>(sl) * N + i];
    }
    const int64_t n = acc - tot, np = (n + 3) / 4 * 4;
    bt.max_region = std::max<int>(bt.max_region, static_cast<int>(np));
    tot += np;
    if (tot >= (1ll << 31)) { bt.err = "column list of a minibatch too long"; return; }
  }
  soff[n_slabs] = static_cast<int32_t>(tot);
  std::vector<uint32_t> list(tot, kListPad);
  for (int i = 0; i < N; ++i) {
    upos[i].resize(ucol[i].size());
    for (size_t u = 0; u < ucol[i].size(); ++u) {
      const int32_t cc = ucol[i][u];
      const int sl = cc / S;
      const int32_t pos = start[static_cast<size_t>(sl) * N + i]++;
      list[pos] = (static_cast<uint32_t>(i) << 16) | static_cast<uint32_t>(cc - sl * S);
      upos[i][u] = pos;
    }
  }
  // Layout of the block image.
  bt.desc.resize(N);
  size_t off = 0;
  for (int i = 0; i < N; ++i) {
    BatchDesc& dd = bt.desc[i];
    dd.y = static_cast<int64_t>(off);
    off = align_up(off + 4 * static_cast<size_t>(B), 16);
    dd.cpos = static_cast<int64_t>(off);
    off = align_up(off + 4 * static_cast<size_t>(nnz[i]), 16);
    dd.cval = static_cast<int64_t>(off);
    off = align_up(off + 4 * static_cast<size_t>(nnz[i]), 16);
    dd.crow = static_cast<int64_t>(off);
    off = align_up(off + 2 * static_cast<size_t>(nnz[i]), 16);
    dd.cslot = static_cast<int64_t>(off);
    off = align_up(off + 2 * static_cast<size_t>(nnz[i]), 16);
    dd.bnd = static_cast<int64_t>(off);
    off = align_up(off + 4 * static_cast<size_t>(Q + 1), 16);
    dd.nnz = static_cast<int32_t>(nnz[i]);
    dd.pad_ = 0;
  }
  bt.list_off = off;
  off = align_up(off + 4 * static_cast<size_t>(tot), 16);
  bt.soff_off = off;
  off = align_up(off + 4 * static_cast<size_t>(n_slabs + 1), 256);
  bt.list_len = tot;
  bt.img.assign(off, 0);
  unsigned char* base = bt.img.data();
  std::memcpy(base + bt.list_off, list.data(), 4 * list.size());
  std::memcpy(base + bt.soff_off, soff.data(), 4 * soff.size());
  std::vector<int32_t> fill(B);
  for (int i = 0; i < N; ++i) {
    const BatchDesc& dd = bt.desc[i];
    float* y_o = reinterpret_cast<float*>(base + dd.y);
    int32_t* cp_o = reinterpret_cast<int32_t*>(base + dd.cpos);
    float* cv_o = reinterpret_cast<float*>(base + dd.cval);
    uint16_t* cr_o = reinterpret_cast<uint16_t*>(base + dd.crow);
    uint16_t* cs_o = reinterpret_cast<uint16_t*>(base + dd.cslot);
    int32_t* bd_o = reinterpret_cast<int32_t*>(base + dd.bnd);
    const int64_t* rp = rowptr[i];
    if (!rp) continue;   // labels and ranges stay zero
    const int64_t r0 = static_cast<int64_t>(t) * B, a0 = rp[r0];
    for (int b = 0; b < B; ++b) y_o[b] = y[i][r0 + b];
    std::vector<uint16_t> erow(nnz[i]);
    for (int b = 0; b < B; ++b)
      for (int64_t e = rp[r0 + b] - a0; e < rp[r0 + b + 1] - a0; ++e) erow[e] = static_cast<uint16_t>(b);
    for (int64_t e = 0; e < nnz[i]; ++e) {
      const int64_t k = static_cast<int64_t>(keys[i][e] & 0xffffffffu);
      cp_o[e] = upos[i][run_of[i][e]];
      cv_o[e] = val[i][a0 + k];
      cr_o[e] = erow[k];
    }
    // Margin segments of kSlotSegment sorted entries: slots row by row, a
    // row's entries in sorted (column) order.
    for (int64_t e0 = 0; e0 < nnz[i]; e0 += kSlotSegment) {
      const int64_t e1 = std::min<int64_t>(e0 + kSlotSegment, nnz[i]);
      std::fill(fill.begin(), fill.end(), 0);
      for (int64_t e = e0; e < e1; ++e) fill[cr_o[e]]++;
      int32_t acc = 0;
      for (int b = 0; b < B; ++b) {
        const int32_t n = fill[b];
        fill[b] = acc;
        acc += n;
      }
      for (int64_t e = e0; e < e1; ++e) {
        const int32_t sl = fill[cr_o[e]]++;
        cs_o[e] = static_cast<uint16_t>(sl);
      }
    }
    // Column-sum ranges of the Q CTAs: cut at the first column boundary at
    // or after q nnz / Q.
    bd_o[0] = 0;
    for (int q = 1; q < Q; ++q) {
      int64_t e = std::max<int64_t>(q * nnz[i] / Q, bd_o[q - 1]);
      while (e > 0 && e < nnz[i] && cp_o[e] == cp_o[e - 1]) ++e;
      bd_o[q] = static_cast<int32_t>(e);
    }
    bd_o[Q] = static_cast<int32_t>(nnz[i]);
  }
}

// eta_k of global local step k.
float lr_at(const asap_ctx* c, int64_t k) {
  if (c->lr_kind == ASAP_LR_INVERSE) return static_cast<float>(c->lr / (1.0 + c->lr_gamma * static_cast<double>(k)));
  return c->lr;
}

// Make the block of global local step r available on the device (host residency).
// Slot r % 3; a slot is rewritten only after the last kernel that reads its
// previous block (the step's update, or the reduce of its round) has finished.
asap_status stage_block(asap_ctx* c, int64_t r) {
  const int slot = static_cast<int>(r % asap_ctx::kStaging);
  if (c->staged_round[slot] == r) return ASAP_OK;
  const int t = static_cast<int>(r % c->nb);
  if (c->free_recorded[slot]) CU(cudaStreamWaitEvent(c->copy_stream, c->free_ev[slot], 0), "staging wait");
  CU(cudaMemcpyAsync(c->staging[slot], c->pool + c->block_off[t], c->block_bytes[t], cudaMemcpyHostToDevice,
                     c->copy_stream),
     "copying a minibatch block to the device");
  CU(cudaEventRecord(c->staged_ev[slot], c->copy_stream), "staging event");
  c->staged_round[slot] = r;
  return ASAP_OK;
}

// Device address of round r's batch block (staging it first when the
// shards live on the host; the context stream then waits for the copy).
asap_status block_of(asap_ctx* c, int64_t r, const unsigned char** out) {
  const int t = static_cast<int>(r % c->nb);
  if (c->residency != ASAP_SHARDS_HOST) {
    *out = c->pool + c->block_off[t];
    return ASAP_OK;
  }
  asap_status s = stage_block(c, r);
  if (s != ASAP_OK) return s;
  const int slot = static_cast<int>(r % asap_ctx::kStaging);
  CU(cudaStreamWaitEvent(c->stream, c->staged_ev[slot], 0), "waiting for a staged block");
  *out = c->staging[slot];
  return ASAP_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
extern "C" {

const char* asap_version(void) { return "asap-gb300 0.1 (sm_103a)"; }

const char* asap_last_error(const asap_ctx* c) { return c ? c->err.c_str() : g_last_error.c_str(); }

asap_status asap_debug_batch_image(int N, int64_t d, int batch, int slab_cols, int ctas_per_worker, int t,
                                   const int64_t* const* rowptr, const int32_t* const* col, const float* const* val,
                                   const float* const* y, unsigned char* image, int64_t cap, int64_t* image_bytes,
                                   int64_t* desc_out, int64_t* list_out) {
  if (N < 1 || N > kMaxWorkers || d < 1 || batch < 1 || batch > 65535 || t < 0 || ctas_per_worker < 1 ||
      ctas_per_worker > kMaxStepCluster || !rowptr || !col || !val || !y || !image_bytes || !desc_out || !list_out)
    return fail(nullptr, ASAP_ERR_ARG, "bad arguments to asap_debug_batch_image");
  if (slab_cols < 8 || slab_cols > 1024 || (slab_cols & (slab_cols - 1)))
    return fail(nullptr, ASAP_ERR_ARG, "slab_cols must be a power of two in [8, 1024]");
  const int64_t ld = (d + 63) / 64 * 64;
  const long long n_slabs = (ld + slab_cols - 1) / slab_cols;
  BatchImage bt;
  build_batch_image(N, batch, d, slab_cols, n_slabs, ctas_per_worker, t, rowptr, col, val, y, bt);
  if (bt.err) return fail(nullptr, ASAP_ERR_ARG, bt.err);
  *image_bytes = static_cast<int64_t>(bt.img.size());
  if (!image || cap < static_cast<int64_t>(bt.img.size())) return fail(nullptr, ASAP_ERR_ARG, "image buffer too small");
  std::memcpy(image, bt.img.data(), bt.img.size());
  for (int i = 0; i < N; ++i) {
    const BatchDesc& q = bt.desc[i];
    const int64_t v[8] = {q.y, q.cpos, q.cval, q.crow, q.cslot, q.bnd, q.nnz, 0};
    std::memcpy(desc_out + 8 * static_cast<size_t>(i), v, sizeof v);
  }
  list_out[0] = static_cast<int64_t>(bt.list_off);
  list_out[1] = static_cast<int64_t>(bt.soff_off);
  list_out[2] = bt.list_len;
  return ASAP_OK;
}

asap_status asap_build_graph(asap_graph_kind kind, int N, int k, uint64_t graph_seed, int64_t round,
                             int32_t* nbr_out) {
  if (!nbr_out || N < 1 || N > kMaxWorkers) return fail(nullptr, ASAP_ERR_ARG, "bad arguments to asap_build_graph");
  const char* why = "";
  asap_status s = build_graph_host(kind, N, k, graph_seed, round, nbr_out, &why);
  if (s != ASAP_OK) return fail(nullptr, s, why);
  return ASAP_OK;
}

// Streams, events, flags, metrics and the parameter buffers of a new
// context.  On failure asap_create hands the partly built context to
// asap_destroy, which frees whatever exists.
static asap_status init_ctx(asap_ctx* c) {
  const int N = c->N, k = c->k;
  c->P = c->d;
  CU(cudaGetDevice(&c->dev), "cudaGetDevice");
  CU(cudaDeviceGetAttribute(&c->sm_count, cudaDevAttrMultiProcessorCount, c->dev), "querying SM count");
  CU(cudaStreamCreateWithFlags(&c->own_stream, cudaStreamNonBlocking), "creating a stream");
  CU(cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking), "creating a copy stream");
  CU(cudaStreamCreateWithFlags(&c->read_stream, cudaStreamNonBlocking), "creating a read stream");
  c->stream = c->own_stream;
  for (int i = 0; i < asap_ctx::kRoundEvents; ++i) {
    CU(cudaEventCreateWithFlags(&c->round_ev[i], cudaEventDisableTiming), "creating events");
    c->round_ev_round[i] = -1;
  }
  for (int h = 0; h < 2; ++h) {
    CU(cudaEventCreateWithFlags(&c->graph_half_ev[h], cudaEventDisableTiming), "creating events");
    c->graph_half_used[h] = false;
  }
  CU(cudaEventCreateWithFlags(&c->graph_order_ev, cudaEventDisableTiming), "creating events");
  for (int b = 0; b < asap_ctx::kStaging; ++b) {
    CU(cudaEventCreateWithFlags(&c->staged_ev[b], cudaEventDisableTiming), "creating events");
    CU(cudaEventCreateWithFlags(&c->free_ev[b], cudaEventDisableTiming), "creating events");
  }
  CU(cudaMalloc(&c->ready, 4 * N), "allocating flags");
  CU(cudaMalloc(&c->consumed, 4 * N), "allocating flags");
  CU(cudaMalloc(&c->stamp, 8 * N), "allocating stamps");
  CU(cudaMemset(c->stamp, 0, 8 * N), "zeroing stamps");
  CU(cudaMalloc(&c->ticket, 4 * N), "allocating tickets");
  CU(cudaMalloc(&c->d_worker_of, 4 * static_cast<size_t>(N)), "allocating the local-step map");
  CU(cudaMalloc(&c->st, sizeof(DevState)), "allocating device state");
  CU(cudaMemset(c->st, 0, sizeof(DevState)), "zeroing device state");
  CU(cudaMalloc(&c->m_loss, 4 * kMetricsCap), "allocating metrics");
  CU(cudaMalloc(&c->m_cons, 4 * kMetricsCap), "allocating metrics");
  CU(cudaMemset(c->m_loss, 0xff, 4 * kMetricsCap), "clearing metrics");
  CU(cudaMemset(c->m_cons, 0xff, 4 * kMetricsCap), "clearing metrics");
  c->cons_cap = c->sm_count * 32;
  CU(cudaMalloc(&c->cons_part, 8 * static_cast<size_t>(c->cons_cap)), "allocating reduce scratch");
  const int kp1_tab = std::min(k + 1, kMaxKp1Sparse);
  const size_t ring = static_cast<size_t>(kGraphRing) * N * kp1_tab;
  CU(cudaMalloc(&c->d_nbr, ring * 4), "allocating graph slots");
  CU(cudaMalloc(&c->d_wgt, ring * 4), "allocating graph slots");
  CU(cudaHostAlloc(&c->h_nbr, ring * 4, cudaHostAllocDefault), "allocating pinned graph slots");
  CU(cudaHostAlloc(&c->h_wgt, ring * 4, cudaHostAllocDefault), "allocating pinned graph slots");
  asap_status s = alloc_params(c);
  if (s != ASAP_OK) return s;
  return upload_fixed_graph(c);
}

asap_status asap_create(int N, int64_t d, uint64_t graph_seed, int k, asap_ctx** out) {
  if (!out) return fail(nullptr, ASAP_ERR_ARG, "out is NULL");
  *out = nullptr;
  if (N < 1 || N > kMaxWorkers || d < 1 || k < 0 || k > N - 1)
    return fail(nullptr, ASAP_ERR_ARG, "need 1 <= N <= 1024, d >= 1, 0 <= k <= N-1");
  std::unique_ptr<asap_ctx> holder(new asap_ctx());
  asap_ctx* c = holder.get();
  c->N = N;
  c->d = d;
  c->seed = graph_seed;
  c->k = k;
  c->kind = (k == 0) ? ASAP_GRAPH_IDENTITY
            : (k == N - 1) ? ASAP_GRAPH_COMPLETE
            : (k == 1) ? ASAP_GRAPH_RING
                       : ASAP_GRAPH_RANDOM_REGULAR;
  if (c->kind == ASAP_GRAPH_RANDOM_REGULAR && k + 1 > kMaxKp1Sparse)
    return fail(nullptr, ASAP_ERR_ARG, "k+1 > 32 is supported only for the complete graph");
  asap_status s = init_ctx(c);
  if (s != ASAP_OK) {
    g_last_error = c->err;
    asap_destroy(holder.release());
    return s;
  }
  *out = holder.release();
  return ASAP_OK;
}

void asap_destroy(asap_ctx* c) {
  if (!c) return;
  if (c->stream) cudaStreamSynchronize(c->stream);
  if (c->copy_stream) cudaStreamSynchronize(c->copy_stream);
  free_shards(c);
  for (int b = 0; b < 2; ++b) {
    dfree(c->W[b]);
    dfree(c->Wbf[b]);
  }
  dfree(c->ready);
  dfree(c->consumed);
  dfree(c->stamp);
  dfree(c->ticket);
  dfree(c->d_worker_of);
  dfree(c->st);
  dfree(c->m_loss);
  dfree(c->m_cons);
  dfree(c->r_scr);
  dfree(c->loss_part);
  dfree(c->RT);
  dfree(c->cons_part);
  dfree(c->d_nbr);
  dfree(c->d_wgt);
  if (c->h_nbr) cudaFreeHost(c->h_nbr);
  if (c->h_wgt) cudaFreeHost(c->h_wgt);
  for (int h = 0; h < 2; ++h)
    if (c->graph_half_ev[h]) cudaEventDestroy(c->graph_half_ev[h]);
  if (c->graph_order_ev) cudaEventDestroy(c->graph_order_ev);
  for (auto& e : c->tev)
    if (e) cudaEventDestroy(e);
  for (int b = 0; b < asap_ctx::kStaging; ++b) {
    if (c->staged_ev[b]) cudaEventDestroy(c->staged_ev[b]);
    if (c->free_ev[b]) cudaEventDestroy(c->free_ev[b]);
  }
  for (int i = 0; i < asap_ctx::kRoundEvents; ++i)
    if (c->round_ev[i]) cudaEventDestroy(c->round_ev[i]);
  if (c->read_stream) {
    cudaStreamSynchronize(c->read_stream);
    cudaStreamDestroy(c->read_stream);
  }
  if (c->own_stream) cudaStreamDestroy(c->own_stream);
  if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
  delete c;
}

asap_status asap_set_graph(asap_ctx* c, asap_graph_kind kind, int regenerate_every_round) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (kind == ASAP_GRAPH_EXPLICIT && !c->have_explicit)
    return fail(c, ASAP_ERR_ARG, "EXPLICIT needs asap_set_mixing");
  if (kind == ASAP_GRAPH_EXPLICIT && regenerate_every_round)
    return fail(c, ASAP_ERR_ARG, "an explicit graph cannot be regenerated");
  if (kind != ASAP_GRAPH_EXPLICIT) {
    std::vector<int32_t> probe(static_cast<size_t>(c->N) * (c->k + 1));
    const char* why = "";
    asap_status s = build_graph_host(kind, c->N, c->k, c->seed, 0, probe.data(), &why);
    if (s != ASAP_OK) return fail(c, s, why);
    if (kind != ASAP_GRAPH_COMPLETE && c->k + 1 > kMaxKp1Sparse)
      return fail(c, ASAP_ERR_ARG, "k+1 > 32 is supported only for the complete graph");
  }
  asap_status s0 = asap_sync(c);
  if (s0 != ASAP_OK) return s0;
  c->kind = kind;
  c->regen = regenerate_every_round != 0 && kind == ASAP_GRAPH_RANDOM_REGULAR;
  asap_status s = setup_mix(c);
  if (s != ASAP_OK) return s;
  return upload_fixed_graph(c);
}

asap_status asap_set_mixing(asap_ctx* c, const int32_t* nbr, const float* wgt) {
  if (!c || !nbr || !wgt) return fail(c, ASAP_ERR_ARG, "NULL argument");
  const int N = c->N, kp1 = c->k + 1;
  if (kp1 > kMaxKp1Sparse) return fail(c, ASAP_ERR_ARG, "explicit mixing supports k+1 <= 32");
  std::vector<double> colsum(N, 0.0);
  for (int i = 0; i < N; ++i) {
    double rs = 0.0;
    for (int m = 0; m < kp1; ++m) {
      const int j = nbr[i * kp1 + m];
      const float w = wgt[i * kp1 + m];
      if (j < 0 || j >= N) return fail(c, ASAP_ERR_GRAPH, "neighbour id out of range");
      if (m > 0 && j <= nbr[i * kp1 + m - 1]) return fail(c, ASAP_ERR_GRAPH, "rows must be strictly ascending");
      if (!(w >= 0.f) || !std::isfinite(w)) return fail(c, ASAP_ERR_GRAPH, "weights must be finite and >= 0");
      rs += w;
      colsum[j] += w;
    }
    if (std::fabs(rs - 1.0) > 1e-6) return fail(c, ASAP_ERR_GRAPH, "a row of P does not sum to 1");
  }
  for (int j = 0; j < N; ++j)
    if (std::fabs(colsum[j] - 1.0) > 1e-6)
      return fail(c, ASAP_ERR_GRAPH, "a column of P does not sum to 1 (P must be doubly stochastic)");
  asap_status s0 = asap_sync(c);
  if (s0 != ASAP_OK) return s0;
  c->ex_nbr.assign(nbr, nbr + static_cast<size_t>(N) * kp1);
  c->ex_wgt.assign(wgt, wgt + static_cast<size_t>(N) * kp1);
  c->have_explicit = true;
  c->kind = ASAP_GRAPH_EXPLICIT;
  c->regen = false;
  asap_status s = setup_mix(c);
  if (s != ASAP_OK) return s;
  return upload_fixed_graph(c);
}

asap_status asap_set_model(asap_ctx* c, asap_loss loss, int num_classes, int batch, float lr, float l2) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (loss != ASAP_LOSS_NONE && loss != ASAP_LOSS_HINGE && loss != ASAP_LOSS_LOGISTIC && loss != ASAP_LOSS_SOFTMAX)
    return fail(c, ASAP_ERR_ARG, "unknown loss");
  if (loss != ASAP_LOSS_NONE && (batch < 1 || batch > 65535 || !(lr > 0.f) || !(l2 >= 0.f) || !(lr * l2 < 1.f)))
    return fail(c, ASAP_ERR_ARG, "need 1 <= batch <= 65535, lr > 0, l2 >= 0, lr*l2 < 1");
  if (loss == ASAP_LOSS_SOFTMAX &&
      (num_classes < 2 || num_classes > 1024 || c->d % 256 != 0 || batch % 128 != 0 ||
       static_cast<int64_t>(c->N) * ((num_classes + 255) / 256) * 256 > (1ll << 31) / batch))
    return fail(c, ASAP_ERR_ARG, "softmax needs 2 <= C <= 1024, d % 256 == 0 and B % 128 == 0");
  if (loss != ASAP_LOSS_SOFTMAX && num_classes != 1) return fail(c, ASAP_ERR_ARG, "num_classes must be 1");
  if (c->sharded && loss == ASAP_LOSS_SOFTMAX)
    return fail(c, ASAP_ERR_ARG, "worker-sharded contexts take hinge or logistic models");
  asap_status s0 = asap_sync(c);
  if (s0 != ASAP_OK) return s0;
  free_shards(c);
  c->loss = loss;
  c->C = num_classes;
  c->B = batch;
  c->lr = lr;
  c->l2 = l2;
  c->P = (loss == ASAP_LOSS_SOFTMAX) ? c->d * num_classes : c->d;
  asap_status s = alloc_params(c);
  if (s != ASAP_OK) return s;
  s = upload_fixed_graph(c);
  if (s != ASAP_OK) return s;
  dfree(c->r_scr);
  dfree(c->loss_part);
  dfree(c->RT);
  c->n_loss_part = 0;
  if (loss == ASAP_LOSS_HINGE || loss == ASAP_LOSS_LOGISTIC) {
    c->n_loss_part = c->N;
    // The local step: one cluster of Q CTAs per worker, Q as large as keeps
    // all clusters resident (at most 8, the portable size).  Two ring stages
    // keep a CTA small enough for five per SM at the usual minibatch sizes
    // (the kernel's registers are bounded for five).
    c->step_stages = 2;
    c->step_smem = local_step_smem_bytes(batch, c->step_stages);
    int smem_sm = 0;
    CU(cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, c->dev),
       "querying shared memory per SM");
    const int64_t per_sm = std::max<int64_t>(1, std::min<int64_t>(5, smem_sm / static_cast<int64_t>(c->step_smem + 1024)));
    c->step_q = kMaxStepCluster;
    while (c->step_q > 1 && static_cast<int64_t>(c->N) * c->step_q > per_sm * c->sm_count) c->step_q >>= 1;
    CU(local_step_configure(c->step_smem), "configuring the local-step kernel");
    c->permuted = false;
  } else if (loss == ASAP_LOSS_SOFTMAX) {
    c->Cq = (num_classes + 255) / 256;
    c->n_loss_part = c->N * (batch / 128) * c->Cq;
    const size_t rt = static_cast<size_t>(c->N) * c->Cq * 256 * batch;
    CU(cudaMalloc(&c->RT, 2 * rt), "allocating the softmax residual scratch");
    CU(cudaMemset(c->RT, 0, 2 * rt), "zeroing the softmax residual scratch");
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(batch), static_cast<cuuint64_t>(c->N) * c->Cq * 256};
    cuuint64_t str[1] = {static_cast<cuuint64_t>(batch) * 2};
    cuuint32_t box[2] = {64, 128};
    s = bf16_map(c, &c->tmR, c->RT, 2, dims, str, box);
    if (s != ASAP_OK) return s;
    if (!c->dense_configured) {
      CU(dense_configure(), "configuring the tensor-core kernels");
      c->dense_configured = true;
    }
  }
  if (c->n_loss_part > 0) {
    CU(cudaMalloc(&c->loss_part, 4 * static_cast<size_t>(c->n_loss_part)), "allocating step scratch");
    // Workers that a worker-sharded context does not step contribute 0.
    CU(cudaMemset(c->loss_part, 0, 4 * static_cast<size_t>(c->n_loss_part)), "zeroing step scratch");
  }
  return ASAP_OK;
}

asap_status asap_set_schedule(asap_ctx* c, int local_steps, asap_lr_schedule kind, float gamma) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (local_steps < 1 || local_steps > 4096) return fail(c, ASAP_ERR_ARG, "local_steps must be in [1, 4096]");
  if (kind != ASAP_LR_CONSTANT && kind != ASAP_LR_INVERSE) return fail(c, ASAP_ERR_ARG, "unknown schedule");
  if (!(gamma >= 0.f) || !std::isfinite(gamma)) return fail(c, ASAP_ERR_ARG, "gamma must be finite and >= 0");
  if (c->step_pending) return fail(c, ASAP_ERR_ARG, "a local step is pending: reduce first");
  if (c->loss == ASAP_LOSS_SOFTMAX && local_steps != 1)
    return fail(c, ASAP_ERR_ARG, "softmax models take one local step per round");
  c->tau = local_steps;
  c->lr_kind = kind;
  c->lr_gamma = gamma;
  c->wv_step = -1;   // the step numbering may change: gather at the next step
  return ASAP_OK;
}

asap_status asap_set_stream(asap_ctx* c, void* s) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  cudaStream_t ns = s ? static_cast<cudaStream_t>(s) : c->own_stream;
  if (ns != c->stream) {
    CU(cudaStreamSynchronize(c->stream), "synchronising the old stream");
    c->stream = ns;
  }
  return ASAP_OK;
}

asap_status asap_set_shard_residency(asap_ctx* c, asap_residency r) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (r != ASAP_SHARDS_DEVICE && r != ASAP_SHARDS_HOST) return fail(c, ASAP_ERR_ARG, "unknown residency");
  if (r == c->residency) return ASAP_OK;
  if (c->nb) {
    // Move the loaded shards; the layout is the same in both places.
    asap_status s0 = sync_all(c);
    if (s0 != ASAP_OK) return s0;
    unsigned char* np = nullptr;
    if (r == ASAP_SHARDS_DEVICE) {
      CU(cudaMalloc(&np, c->pool_bytes), "allocating device shard memory");
      CU(cudaMemcpy(np, c->pool, c->pool_bytes, cudaMemcpyHostToDevice), "moving shards to the device");
      cudaFreeHost(c->pool);
      for (int b = 0; b < asap_ctx::kStaging; ++b) dfree(c->staging[b]);
    } else {
      CU(cudaHostAlloc(&np, c->pool_bytes, cudaHostAllocDefault), "allocating pinned shard memory");
      CU(cudaMemcpy(np, c->pool, c->pool_bytes, cudaMemcpyDeviceToHost), "moving shards to the host");
      cudaFree(c->pool);
      size_t mb = 0;
      for (size_t b : c->block_bytes) mb = std::max(mb, b);
      c->staging_bytes = mb;
      for (int b = 0; b < asap_ctx::kStaging; ++b) CU(cudaMalloc(&c->staging[b], mb), "allocating staging buffers");
    }
    c->pool = np;
    c->pool_pinned = (r == ASAP_SHARDS_HOST);
    for (int b = 0; b < asap_ctx::kStaging; ++b) {
      c->staged_round[b] = -1;
      c->free_recorded[b] = false;
    }
  }
  c->residency = r;
  return ASAP_OK;
}

asap_status asap_shard_block_bytes(asap_ctx* c, int64_t round, uint64_t* bytes) {
  if (!c || !bytes || round < 0) return fail(c, ASAP_ERR_ARG, "bad argument");
  if (!c->nb) return fail(c, ASAP_ERR_ARG, "no shards loaded");
  *bytes = c->block_bytes[static_cast<size_t>(round % c->nb)];
  return ASAP_OK;
}

asap_status asap_load_shards(asap_ctx* c, const int64_t* const* rowptr, const int32_t* const* col,
                             const float* const* val, const float* const* y, const int64_t* n_rows) {
  if (!c || !rowptr || !col || !val || !y || !n_rows) return fail(c, ASAP_ERR_ARG, "NULL argument");
  if (c->loss != ASAP_LOSS_HINGE && c->loss != ASAP_LOSS_LOGISTIC)
    return fail(c, ASAP_ERR_ARG, "set a hinge or logistic model before loading CSR shards");
  const int N = c->N, B = c->B;
  int nb = -1;
  // Worker-sharded: the shards of workers outside the owned range are not
  // read (their pointers may be NULL) and get empty minibatches.
  std::vector<const int64_t*> rp_use(rowptr, rowptr + N);
  for (int i = 0; i < N; ++i) {
    if (c->sharded && (i < c->own_lo || i >= c->own_lo + c->own_n)) {
      rp_use[i] = nullptr;
      continue;
    }
    if (!rowptr[i] || !col[i] || !val[i] || !y[i]) return fail(c, ASAP_ERR_ARG, "NULL shard pointer");
    if (n_rows[i] < B) return fail(c, ASAP_ERR_ARG, "a shard has fewer rows than one minibatch");
    const int64_t nbi = n_rows[i] / B;
    if (nb >= 0 && nbi != nb) return fail(c, ASAP_ERR_ARG, "all shards must hold the same number of minibatches");
    nb = static_cast<int>(std::min<int64_t>(nbi, 1 << 30));
    if (rowptr[i][0] != 0) return fail(c, ASAP_ERR_ARG, "rowptr must start at 0");
    for (int64_t r = 0; r < nbi * B; ++r)
      if (rowptr[i][r + 1] < rowptr[i][r]) return fail(c, ASAP_ERR_ARG, "rowptr must be non-decreasing");
  }
  asap_status s0 = asap_sync(c);
  if (s0 != ASAP_OK) return s0;
  free_shards(c);
  c->s_cap = 1024;
  s0 = setup_mix(c);
  if (s0 != ASAP_OK) return s0;
  const int Q = c->step_q;
  // Build every minibatch's image; narrow the slabs and rebuild while a
  // slab's column list is too long for the fused reduce's shared memory.
  for (;;) {
    const int S = c->S;
    const long long n_slabs = c->n_slabs;

    std::vector<BatchImage> built(nb);
    auto build_batch = [&](int t) {
      build_batch_image(N, B, c->d, S, n_slabs, Q, t, rp_use.data(), col, val, y, built[t]);
    };
    {
      const unsigned nthr = std::max(1u, std::min(32u, std::thread::hardware_concurrency()));
      std::vector<std::thread> pool;
      for (unsigned w = 0; w < nthr; ++w)
        pool.emplace_back([&, w]() {
          for (int t = static_cast<int>(w); t < nb; t += static_cast<int>(nthr)) build_batch(t);
        });
      for (auto& th : pool) th.join();
    }
    size_t total = 0;
    int max_nnz = 0, max_region = 0;
    int64_t max_list = 0;
    for (int t = 0; t < nb; ++t)
      if (built[t].err) return fail(c, ASAP_ERR_ARG, built[t].err);
    for (int t = 0; t < nb; ++t) max_region = std::max(max_region, built[t].max_region);
    // Two stages of the fused reduce (slab + three list regions each) must fit
    // in shared memory; skewed column popularity calls for narrower slabs.
    if (mix_smem_bytes(N, std::min(c->k + 1, kMaxKp1Sparse), S, c->rows_pad, 2, max_region) > (220u << 10)) {
      if (S <= 8) return fail(c, ASAP_ERR_ARG, "a column slab's list does not fit in shared memory");
      c->s_cap = S / 2;
      asap_status sm = setup_mix(c);
      if (sm != ASAP_OK) return sm;
      continue;
    }
    max_region = 0;
    c->block_off.assign(nb, 0);
    c->block_bytes.assign(nb, 0);
    c->list_off.assign(nb, 0);
    c->soff_off.assign(nb, 0);
    c->list_len.assign(nb, 0);
    std::vector<BatchDesc> desc(static_cast<size_t>(nb) * N);
    for (int t = 0; t < nb; ++t) {
      if (built[t].err) return fail(c, ASAP_ERR_ARG, built[t].err);
      c->block_off[t] = total;
      c->block_bytes[t] = built[t].img.size();
      c->list_off[t] = built[t].list_off;
      c->soff_off[t] = built[t].soff_off;
      c->list_len[t] = built[t].list_len;
      total += built[t].img.size();
      max_nnz = std::max(max_nnz, built[t].max_nnz);
      max_region = std::max(max_region, built[t].max_region);
      max_list = std::max(max_list, built[t].list_len);
      std::copy(built[t].desc.begin(), built[t].desc.end(), desc.begin() + static_cast<size_t>(t) * N);
    }
    if (c->residency == ASAP_SHARDS_HOST) {
      CU(cudaHostAlloc(&c->pool, total, cudaHostAllocDefault), "allocating pinned shard memory");
      c->pool_pinned = true;
      size_t mb = 0;
      for (int t = 0; t < nb; ++t) {
        std::memcpy(c->pool + c->block_off[t], built[t].img.data(), built[t].img.size());
        mb = std::max(mb, built[t].img.size());
        std::vector<unsigned char>().swap(built[t].img);
      }
      c->staging_bytes = mb;
      for (int b = 0; b < asap_ctx::kStaging; ++b) CU(cudaMalloc(&c->staging[b], mb), "allocating staging buffers");
    } else {
      CU(cudaMalloc(&c->pool, total), "allocating device shard memory");
      c->pool_pinned = false;
      for (int t = 0; t < nb; ++t) {
        CU(cudaMemcpy(c->pool + c->block_off[t], built[t].img.data(), built[t].img.size(), cudaMemcpyHostToDevice),
           "copying shards to the device");
        std::vector<unsigned char>().swap(built[t].img);
      }
    }
    c->pool_bytes = total;
    CU(cudaMalloc(&c->d_desc, desc.size() * sizeof(BatchDesc)), "allocating batch descriptors");
    CU(cudaMemcpy(c->d_desc, desc.data(), desc.size() * sizeof(BatchDesc), cudaMemcpyHostToDevice),
       "copying batch descriptors");
    const size_t lb = 4 * static_cast<size_t>(std::max<int64_t>(max_list, 4));
    CU(cudaMalloc(&c->wv[0], lb), "allocating the list value buffer");
    CU(cudaMalloc(&c->wv[1], lb), "allocating the list value buffer");
    CU(cudaMalloc(&c->gsum, lb), "allocating the column-sum buffer");
    CU(cudaMemset(c->wv[0], 0, lb), "zeroing the list value buffer");
    CU(cudaMemset(c->wv[1], 0, lb), "zeroing the list value buffer");
    CU(cudaMemset(c->gsum, 0, lb), "zeroing the column-sum buffer");
    if (B > kRSmemRows) {
      CU(cudaMalloc(&c->mpart_big, 16 * static_cast<size_t>(N) * Q * B), "allocating the partial margins");
      CU(cudaMalloc(&c->r_big, 4 * static_cast<size_t>(N) * Q * B), "allocating the step scratch");
    }
    c->nb = nb;
    c->max_nnz = max_nnz;
    c->max_region = max_region;
    c->max_list = max_list;
    c->wv_step = -1;
    c->configured_key = -1;
    return ASAP_OK;
  }
}

asap_status asap_load_dense_shards(asap_ctx* c, const uint16_t* const* X, const int32_t* const* y,
                                   const int64_t* n_rows) {
  if (!c || !X || !y || !n_rows) return fail(c, ASAP_ERR_ARG, "NULL argument");
  if (c->loss != ASAP_LOSS_SOFTMAX) return fail(c, ASAP_ERR_ARG, "set a softmax model before loading dense shards");
  if (c->residency != ASAP_SHARDS_DEVICE) return fail(c, ASAP_ERR_ARG, "dense shards are device-resident only");
  const int N = c->N, B = c->B;
  const int64_t d = c->d;
  int64_t nb = -1;
  for (int i = 0; i < N; ++i) {
    if (!X[i] || !y[i]) return fail(c, ASAP_ERR_ARG, "NULL shard pointer");
    if (n_rows[i] < B) return fail(c, ASAP_ERR_ARG, "a shard has fewer rows than one minibatch");
    if (nb >= 0 && n_rows[i] / B != nb)
      return fail(c, ASAP_ERR_ARG, "all shards must hold the same number of minibatches");
    nb = n_rows[i] / B;
    for (int64_t r = 0; r < nb * B; ++r)
      if (y[i][r] < 0 || y[i][r] >= c->C) return fail(c, ASAP_ERR_ARG, "class id out of range [0, C)");
  }
  if (static_cast<int64_t>(N) * nb * B > (1ll << 31) || static_cast<int64_t>(N) * nb * d > (1ll << 31))
    return fail(c, ASAP_ERR_ARG, "dense shards too large for 32-bit tile coordinates");
  asap_status s0 = asap_sync(c);
  if (s0 != ASAP_OK) return s0;
  free_shards(c);
  const size_t rows = static_cast<size_t>(nb) * B;
  const size_t xe = static_cast<size_t>(N) * rows * d;
  CU(cudaMalloc(&c->X, 2 * xe), "allocating dense features");
  CU(cudaMalloc(&c->XT, 2 * xe), "allocating transposed dense features");
  CU(cudaMalloc(&c->Yd, 4 * static_cast<size_t>(N) * rows), "allocating labels");
  std::vector<uint16_t> tr(rows * d);
  for (int i = 0; i < N; ++i) {
    CU(cudaMemcpy(c->X + static_cast<size_t>(i) * rows * d, X[i], 2 * rows * d, cudaMemcpyHostToDevice),
       "copying dense features");
    CU(cudaMemcpy(c->Yd + static_cast<size_t>(i) * rows, y[i], 4 * rows, cudaMemcpyHostToDevice), "copying labels");
    // Per minibatch, the features transposed to [d][B] (the K-major operand
    // of the gradient GEMM, whose reduction runs over the batch).
    const unsigned nthr = std::max(1u, std::min(16u, std::thread::hardware_concurrency()));
    std::vector<std::thread> pool;
    for (unsigned w = 0; w < nthr; ++w)
      pool.emplace_back([&, w]() {
        for (int64_t t = w; t < nb; t += nthr) {
          const uint16_t* src = X[i] + static_cast<size_t>(t) * B * d;
          uint16_t* dst = tr.data() + static_cast<size_t>(t) * d * B;
          for (int b = 0; b < B; ++b)
            for (int64_t k = 0; k < d; ++k) dst[k * B + b] = src[static_cast<size_t>(b) * d + k];
        }
      });
    for (auto& th : pool) th.join();
    CU(cudaMemcpy(c->XT + static_cast<size_t>(i) * rows * d, tr.data(), 2 * rows * d, cudaMemcpyHostToDevice),
       "copying transposed features");
  }
  {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(N) * rows};
    cuuint64_t str[1] = {static_cast<cuuint64_t>(d) * 2};
    cuuint32_t box[2] = {64, 32};   // 32-row parts, multicast across the forward kernel's cluster
    asap_status s = bf16_map(c, &c->tmX, c->X, 2, dims, str, box);
    if (s != ASAP_OK) return s;
  }
  {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(B), static_cast<cuuint64_t>(N) * nb * d};
    cuuint64_t str[1] = {static_cast<cuuint64_t>(B) * 2};
    cuuint32_t box[2] = {64, 256};
    asap_status s = bf16_map(c, &c->tmXT, c->XT, 2, dims, str, box);
    if (s != ASAP_OK) return s;
  }
  c->nb = static_cast<int>(nb);
  return ASAP_OK;
}

asap_status asap_local_step(asap_ctx* c) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (c->loss == ASAP_LOSS_NONE) return fail(c, ASAP_ERR_ARG, "no model set (asap_set_model)");
  if (!c->nb) return fail(c, ASAP_ERR_ARG, "no shards loaded");
  if (c->step_pending) return fail(c, ASAP_ERR_ARG, "local step already taken this round; reduce first");
  const int64_t r = c->round;
  const int t = static_cast<int>(r % c->nb);
  if (c->loss == ASAP_LOSS_SOFTMAX) {
    if (c->tau != 1) return fail(c, ASAP_ERR_ARG, "softmax models take one local step per round");
    asap_status sg = prepare_graph(c, r);
    if (sg != ASAP_OK) return sg;
    DenseFwdArgs f;
    f.C = c->C;
    f.Cq = c->Cq;
    f.d = static_cast<int>(c->d);
    f.B = c->B;
    f.nb = c->nb;
    f.t = t;
    f.y = c->Yd;
    f.RT = c->RT;
    f.loss_part = c->loss_part;
    f.inv_B = 1.0f / static_cast<float>(c->B);
    f.st = c->st;
    f.round = static_cast<unsigned>(r);
    DenseGradArgs g;
    g.C = c->C;
    g.Cq = c->Cq;
    g.d = static_cast<int>(c->d);
    g.B = c->B;
    g.nb = c->nb;
    g.t = t;
    g.W = c->W[r & 1];
    g.ld = c->ld;
    const float eta = lr_at(c, r);
    g.lr = eta;
    g.decay = 1.0f - eta * c->l2;
    g.ready = c->ready;
    g.worker_ticket = c->ticket;
    g.skip_worker = c->skip_notify;
    g.st = c->st;
    g.round = static_cast<unsigned>(r);
    c->skip_notify = -1;
    time_begin(c, ASAP_KERNEL_DENSE_FWD);
    CU(launch_dense_fwd(c->tmX, c->tmWbf[r & 1], f, c->N, c->stream), "launching the dense forward kernel");
    time_end(c);
    time_begin(c, ASAP_KERNEL_DENSE_GRAD);
    CU(launch_dense_grad(c->tmR, c->tmXT, c->tmWf[r & 1], g, c->N, c->sm_count, c->stream),
       "launching the dense gradient kernel");
    time_end(c);
    c->launches += 2;
    c->step_pending = true;
    return ASAP_OK;
  }
  // tau local steps: step j is global step k = r tau + j on minibatch k mod nb.
  // L2 shrinks every worker's w by the same (1 - eta_k l2) per step, kept as
  // one scale s (true w = s * stored values) until the reduce applies it.
  float s_scale = 1.0f;
  for (int j = 0; j < c->tau; ++j) {
    const int64_t k = r * c->tau + j;
    const int tk = static_cast<int>(k % c->nb);
    const bool last = j == c->tau - 1;
    const unsigned char* block = nullptr;
    asap_status sb = block_of(c, k, &block);
    if (sb != ASAP_OK) return sb;
    if (c->wv_step != k) {
      // No exported w values for this step's columns (parameters came from
      // the host, or an earlier local step of the round changed them): gather.
      time_begin(c, ASAP_KERNEL_GATHER);
      CU(launch_gather_wv(c->W[r & 1], c->ld, reinterpret_cast<const uint32_t*>(block + c->list_off[tk]),
                          reinterpret_cast<const int*>(block + c->soff_off[tk]), c->n_slabs, c->S, c->wv[r & 1],
                          c->sm_count, c->stream),
         "launching the gather kernel");
      time_end(c);
      c->launches += 1;
      c->wv_step = k;
    }
    LocalStepArgs a;
    a.block = block;
    a.desc = c->d_desc + static_cast<size_t>(tk) * c->N;
    a.wv = c->wv[r & 1];
    a.gsum = c->gsum;
    a.mpart_big = c->mpart_big;
    a.r_big = c->r_big;
    a.loss_part = c->loss_part;
    a.ready = c->ready;
    a.st = c->st;
    a.worker_of = (c->permuted || c->sharded) ? c->d_worker_of : nullptr;
    a.N = c->sharded ? c->own_n : c->N;
    a.B = c->B;
    a.Q = c->step_q;
    a.stages = c->step_stages;
    a.round = static_cast<unsigned>(r);
    a.mscale = s_scale;
    a.notify = last ? 1 : 0;
    a.skip_worker = last ? c->skip_notify : -1;
    if (last) {
      c->skip_notify = -1;
      asap_status sg = prepare_graph(c, r);   // upload a regenerated graph ahead of the reduce
      if (sg != ASAP_OK) return sg;
    }
    time_begin(c, ASAP_KERNEL_LOCAL_STEP);
    CU(launch_local_step(a, c->loss, c->step_smem, c->stream), "launching the local-step kernel");
    time_end(c);
    c->launches += 1;
    const float eta = lr_at(c, k);
    const float s_next = s_scale * (1.0f - eta * c->l2);
    const float upd = eta / (static_cast<float>(c->B) * s_next);
    if (!last || c->sharded) {
      // w_stored -= eta / (B s') g at the step's columns; the reduce applies
      // the round's last update itself, except in a worker-sharded context,
      // whose owned rows must hold x - eta g before they are sent.
      time_begin(c, ASAP_KERNEL_APPLY);
      CU(launch_apply_update(c->W[r & 1], c->ld, reinterpret_cast<const uint32_t*>(block + c->list_off[tk]),
                             reinterpret_cast<const int*>(block + c->soff_off[tk]), c->n_slabs, c->S, c->gsum, upd,
                             c->sm_count, c->stream),
         "launching the local update kernel");
      time_end(c);
      c->launches += 1;
      if (c->residency == ASAP_SHARDS_HOST) {
        const int slot = static_cast<int>(k % asap_ctx::kStaging);
        CU(cudaEventRecord(c->free_ev[slot], c->stream), "staging event");   // block k is no longer read
        c->free_recorded[slot] = true;
        asap_status ss = stage_block(c, k + 2);                                 // prefetch
        if (ss != ASAP_OK) return ss;
      }
    }
    if (last) {
      c->pend_wscale = s_next;
      c->pend_upd = upd;
      c->pend_k = k;
    }
    s_scale = s_next;
  }
  if (c->sharded) std::fill(c->delivered.begin(), c->delivered.end(), 0);
  c->step_pending = true;
  return ASAP_OK;
}

asap_status asap_stochastic_reduce(asap_ctx* c) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  const int64_t r = c->round;
  const bool sparse = c->loss == ASAP_LOSS_HINGE || c->loss == ASAP_LOSS_LOGISTIC;
  const bool fused = c->step_pending && sparse && !c->sharded;
  if (c->sharded && c->step_pending) {
    // The NOTIFY of a worker stepped elsewhere is the delivery of its row:
    // every in-neighbour of an owned worker must have arrived this round.
    const size_t kp1 = static_cast<size_t>(c->k) + 1;
    std::vector<int32_t> nbr(static_cast<size_t>(c->N) * kp1);
    std::vector<float> wgt(nbr.size());
    asap_status sg = graph_host(c, r, nbr.data(), wgt.data());
    if (sg != ASAP_OK) return sg;
    for (int i = c->own_lo; i < c->own_lo + c->own_n; ++i)
      for (size_t q = 0; q < kp1; ++q) {
        const int j = nbr[i * kp1 + q];
        if ((j < c->own_lo || j >= c->own_lo + c->own_n) && !c->delivered[j])
          return fail(c, ASAP_ERR_ARG, "an in-neighbour's row was not delivered this round (asap_write_rows)");
      }
  }
  asap_status s = configure_mix_launch(c, fused);
  if (s != ASAP_OK) return s;
  s = prepare_graph(c, r);
  if (s != ASAP_OK) return s;
  const int* nbr = c->graph_nbr;
  const float* wgt = c->graph_wgt;
  const int uniform = c->graph_uniform ? 1 : 0;
  c->graph_ready_round = -1;
  MixArgs a = {};
  a.out = c->W[(r + 1) & 1];
  a.shadow = c->Wbf[(r + 1) & 1];
  a.ld = c->ld;
  a.N = c->N;
  a.kp1 = c->tab_kp1;
  a.nbr = nbr;
  a.wgt = wgt;
  a.wscale = (c->step_pending && sparse) ? c->pend_wscale : 1.0f;
  a.uniform_w = uniform;
  a.S = c->S;
  a.rows_pad = c->rows_pad;
  a.box_rows = c->box_rows;
  a.n_boxes = c->n_boxes;
  a.stages = c->stages;
  a.n_slabs = c->n_slabs;
  if (fused) {
    const unsigned char* bt = nullptr;
    const unsigned char* bn = nullptr;
    const int64_t kl = c->pend_k;            // the round's last local step; the next round starts at kl + 1
    s = block_of(c, kl, &bt);
    if (s != ASAP_OK) return s;
    s = block_of(c, kl + 1, &bn);
    if (s != ASAP_OK) return s;
    const int t = static_cast<int>(kl % c->nb), tn = static_cast<int>((kl + 1) % c->nb);
    a.upd_list = reinterpret_cast<const uint32_t*>(bt + c->list_off[t]);
    a.upd_off = reinterpret_cast<const int*>(bt + c->soff_off[t]);
    a.gsum = c->gsum;
    a.upd_scale = c->pend_upd;
    a.exp_list = reinterpret_cast<const uint32_t*>(bn + c->list_off[tn]);
    a.exp_off = reinterpret_cast<const int*>(bn + c->soff_off[tn]);
    a.wv_out = c->wv[(r + 1) & 1];
    a.max_region = c->max_region;
  }
  a.cons_part = c->cons_part;
  a.loss_part = c->loss_part;
  a.n_loss_part = c->step_pending ? c->n_loss_part : 0;
  a.loss_norm = c->B > 0 ? 1.0f / (static_cast<float>(c->N) * static_cast<float>(c->B)) : 0.f;
  a.have_loss = c->step_pending ? 1 : 0;
  a.metrics_loss = c->m_loss;
  a.metrics_cons = c->m_cons;
  a.ready = c->ready;
  a.consumed = c->consumed;
  a.stamp_next = c->stamp + ((r + 1) & 1) * c->N;
  a.st = c->st;
  a.round = static_cast<unsigned>(r);
  a.expect_notify = c->step_pending ? 1 : 0;
  a.wait_ns = c->wait_ns;
  a.sync_mode = fused ? c->sync_mode : kSyncBsp;
  a.own_lo = c->sharded ? c->own_lo : 0;
  a.own_n = c->sharded ? c->own_n : c->N;
  time_begin(c, ASAP_KERNEL_REDUCE);
  CU(launch_mix(c->tmap[r & 1], a, is_complete_kernel(c), fused, c->mix_grid, c->mix_smem, c->stream),
     "launching the stochastic reduce");
  time_end(c);
  c->launches += 1;
  const int ev = static_cast<int>(r % asap_ctx::kRoundEvents);
  CU(cudaEventRecord(c->round_ev[ev], c->stream), "round event");
  c->round_ev_round[ev] = r;
  c->wv_step = fused ? c->pend_k + 1 : -1;
  if (fused && c->residency == ASAP_SHARDS_HOST) {
    const int slot = static_cast<int>(c->pend_k % asap_ctx::kStaging);
    CU(cudaEventRecord(c->free_ev[slot], c->stream), "staging event");   // block pend_k is no longer read
    c->free_recorded[slot] = true;
    s = stage_block(c, c->pend_k + 2);                                    // prefetch
    if (s != ASAP_OK) return s;
  }
  c->round = r + 1;
  c->step_pending = false;
  return ASAP_OK;
}

asap_status asap_round(asap_ctx* c, int T) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (T < 0) return fail(c, ASAP_ERR_ARG, "T must be >= 0");
  for (int t = 0; t < T; ++t) {
    if (c->loss != ASAP_LOSS_NONE) {
      asap_status s = asap_local_step(c);
      if (s != ASAP_OK) return s;
    }
    asap_status s = asap_stochastic_reduce(c);
    if (s != ASAP_OK) return s;
  }
  return ASAP_OK;
}

asap_status asap_sync(asap_ctx* c) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  return sync_all(c);
}

asap_status asap_read_params(asap_ctx* c, float* host_out, int64_t* round_out) {
  if (!c || !host_out) return fail(c, ASAP_ERR_ARG, "NULL argument");
  asap_status s = sync_all(c);
  if (s != ASAP_OK) return s;
  CU(cudaMemcpy2D(host_out, c->P * 4, c->W[c->round & 1], c->ld * 4, c->P * 4, c->N, cudaMemcpyDeviceToHost),
     "reading parameters");
  if (round_out) *round_out = c->round;
  return ASAP_OK;
}

asap_status asap_write_params(asap_ctx* c, const float* host_in, int64_t round) {
  if (!c || !host_in || round < 0) return fail(c, ASAP_ERR_ARG, "bad argument");
  asap_status s = sync_all(c);
  if (s != ASAP_OK) return s;
  float* dst = c->W[round & 1];
  CU(cudaMemcpy2D(dst, c->ld * 4, host_in, c->P * 4, c->P * 4, c->N, cudaMemcpyHostToDevice), "writing parameters");
  if (c->Wbf[round & 1]) {
    CU(launch_cast_bf16(dst, c->Wbf[round & 1], static_cast<int64_t>(c->N) * c->ld, c->stream), "bf16 copy");
    c->launches += 1;
    CU(cudaStreamSynchronize(c->stream), "bf16 copy");
  }
  c->wv_step = -1;
  return reset_protocol(c, round);
}

asap_status asap_write_params_device(asap_ctx* c, const float* dev_in, int64_t ld_in, int64_t round) {
  if (!c || !dev_in || round < 0 || ld_in < c->P) return fail(c, ASAP_ERR_ARG, "bad argument");
  asap_status s = sync_all(c);
  if (s != ASAP_OK) return s;
  float* dst = c->W[round & 1];
  CU(cudaMemcpy2DAsync(dst, c->ld * 4, dev_in, ld_in * 4, c->P * 4, c->N, cudaMemcpyDeviceToDevice, c->stream),
     "writing parameters");
  if (c->Wbf[round & 1]) {
    CU(launch_cast_bf16(dst, c->Wbf[round & 1], static_cast<int64_t>(c->N) * c->ld, c->stream), "bf16 copy");
    c->launches += 1;
  }
  CU(cudaStreamSynchronize(c->stream), "writing parameters");
  c->wv_step = -1;
  return reset_protocol(c, round);
}

asap_status asap_read_param_columns(asap_ctx* c, int64_t first, int64_t count, float* host_out) {
  if (!c || !host_out || first < 0 || count < 1 || first + count > c->P) return fail(c, ASAP_ERR_ARG, "bad argument");
  asap_status s = sync_all(c);
  if (s != ASAP_OK) return s;
  CU(cudaMemcpy2D(host_out, count * 4, c->W[c->round & 1] + first, c->ld * 4, count * 4, c->N,
                  cudaMemcpyDeviceToHost),
     "reading parameter columns");
  return ASAP_OK;
}

asap_status asap_read_metrics(asap_ctx* c, int64_t first, int64_t count, float* loss_out, float* cons_out) {
  if (!c || first < 0 || count < 0) return fail(c, ASAP_ERR_ARG, "bad argument");
  if (first + count > c->round || first < c->round - kMetricsCap)
    return fail(c, ASAP_ERR_ARG, "rounds outside the kept metrics window");
  const int64_t last = first + count - 1;
  const int ev = static_cast<int>((count > 0 ? last : 0) % asap_ctx::kRoundEvents);
  if (count == 0 || c->round_ev_round[ev] != last) {
    // No event for the last requested round: drain everything.
    asap_status s = sync_all(c);
    if (s != ASAP_OK) return s;
  } else {
    // Wait for round `last` only; rounds queued after it keep running.  A
    // device error recorded by then is reported after a full drain.
    CU(cudaStreamWaitEvent(c->read_stream, c->round_ev[ev], 0), "waiting for the round");
    unsigned code = 0;
    CU(cudaMemcpyAsync(&code, &c->st->err_code, 4, cudaMemcpyDeviceToHost, c->read_stream), "reading device state");
    CU(cudaStreamSynchronize(c->read_stream), "waiting for the round");
    if (code != 0) {
      asap_status s = sync_all(c);
      if (s != ASAP_OK) return s;
    }
  }
  // Pageable destinations: each copy returns once it is done.
  for (int64_t r = first; r < first + count;) {
    const int64_t slot = r % kMetricsCap;
    const int64_t n = std::min<int64_t>(first + count - r, kMetricsCap - slot);
    if (loss_out)
      CU(cudaMemcpyAsync(loss_out + (r - first), c->m_loss + slot, 4 * n, cudaMemcpyDeviceToHost, c->read_stream),
         "metrics");
    if (cons_out)
      CU(cudaMemcpyAsync(cons_out + (r - first), c->m_cons + slot, 4 * n, cudaMemcpyDeviceToHost, c->read_stream),
         "metrics");
    r += n;
  }
  CU(cudaStreamSynchronize(c->read_stream), "metrics");
  // A worker-sharded context holds the other workers' rows only where they
  // were delivered: its consensus error over all rows is not defined.
  if (c->sharded && cons_out) std::fill(cons_out, cons_out + count, std::numeric_limits<float>::quiet_NaN());
  return ASAP_OK;
}

asap_status asap_read_counters(asap_ctx* c, uint64_t* reduces, uint64_t* consistent, uint64_t* timeouts) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  CU(cudaStreamSynchronize(c->stream), "synchronising");
  DevState h;
  CU(cudaMemcpy(&h, c->st, sizeof h, cudaMemcpyDeviceToHost), "reading counters");
  if (reduces) *reduces = h.reduces;
  if (consistent) *consistent = h.consistent_inputs;
  if (timeouts) *timeouts = h.timeouts;
  return ASAP_OK;
}

asap_status asap_get_graph(asap_ctx* c, int64_t round, int32_t* nbr_out, float* wgt_out) {
  if (!c || round < 0) return fail(c, ASAP_ERR_ARG, "bad argument");
  const size_t n = static_cast<size_t>(c->N) * (c->k + 1);
  std::vector<int32_t> nbr(n);
  std::vector<float> wgt(n);
  asap_status s = graph_host(c, round, nbr.data(), wgt.data());
  if (s != ASAP_OK) return s;
  if (nbr_out) std::copy(nbr.begin(), nbr.end(), nbr_out);
  if (wgt_out) std::copy(wgt.begin(), wgt.end(), wgt_out);
  return ASAP_OK;
}

asap_status asap_set_sync_mode(asap_ctx* c, asap_sync_mode mode) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (mode != ASAP_SYNC_BSP && mode != ASAP_SYNC_NOTIFY_ACK && mode != ASAP_SYNC_ASYNC)
    return fail(c, ASAP_ERR_ARG, "unknown synchronisation mode");
  if (c->step_pending) return fail(c, ASAP_ERR_ARG, "a local step is pending: reduce first");
  if (c->sharded && mode != ASAP_SYNC_BSP)
    return fail(c, ASAP_ERR_ARG, "a worker-sharded context reduces after the delivery of its rows (BSP)");
  c->sync_mode = mode == ASAP_SYNC_NOTIFY_ACK ? kSyncNotifyAck : mode == ASAP_SYNC_ASYNC ? kSyncAsync : kSyncBsp;
  return ASAP_OK;
}

asap_status asap_set_worker_order(asap_ctx* c, const int32_t* order) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (c->step_pending) return fail(c, ASAP_ERR_ARG, "a local step is pending: reduce first");
  if (c->sharded) return fail(c, ASAP_ERR_ARG, "the worker order of a worker-sharded context is its range");
  if (!order) {
    c->permuted = false;
    return ASAP_OK;
  }
  std::vector<int> seen(c->N, 0);
  bool identity = true;
  for (int q = 0; q < c->N; ++q) {
    if (order[q] < 0 || order[q] >= c->N || seen[order[q]]++) return fail(c, ASAP_ERR_ARG, "not a permutation of [0, N)");
    identity = identity && order[q] == q;
  }
  asap_status s0 = asap_sync(c);
  if (s0 != ASAP_OK) return s0;
  CU(cudaMemcpy(c->d_worker_of, order, 4 * static_cast<size_t>(c->N), cudaMemcpyHostToDevice), "uploading the worker order");
  c->permuted = !identity;
  return ASAP_OK;
}

asap_status asap_set_worker_range(asap_ctx* c, int first, int count) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  if (c->loss != ASAP_LOSS_HINGE && c->loss != ASAP_LOSS_LOGISTIC)
    return fail(c, ASAP_ERR_ARG, "set a hinge or logistic model first");
  if (first < 0 || count < 1 || first > c->N - count) return fail(c, ASAP_ERR_ARG, "range outside [0, N)");
  if (c->step_pending) return fail(c, ASAP_ERR_ARG, "a local step is pending: reduce first");
  asap_status s0 = asap_sync(c);
  if (s0 != ASAP_OK) return s0;
  free_shards(c);   // the minibatch images depend on the range
  const bool whole = first == 0 && count == c->N;
  c->sharded = !whole;
  c->own_lo = whole ? 0 : first;
  c->own_n = whole ? c->N : count;
  c->delivered.assign(c->N, 0);
  c->permuted = false;
  c->sync_mode = kSyncBsp;
  std::vector<int32_t> own(c->N);
  for (int q = 0; q < c->N; ++q) own[q] = q < c->own_n ? c->own_lo + q : q;
  CU(cudaMemcpy(c->d_worker_of, own.data(), 4 * static_cast<size_t>(c->N), cudaMemcpyHostToDevice),
     "uploading the owned workers");
  return ASAP_OK;
}

asap_status asap_read_rows(asap_ctx* c, const int32_t* rows, int count, float* host_out, float* scale_out) {
  if (!c || (count > 0 && (!rows || !host_out)) || count < 0) return fail(c, ASAP_ERR_ARG, "bad argument");
  for (int q = 0; q < count; ++q)
    if (rows[q] < 0 || rows[q] >= c->N) return fail(c, ASAP_ERR_ARG, "row outside [0, N)");
  asap_status s = sync_all(c);
  if (s != ASAP_OK) return s;
  const float* src = c->W[c->round & 1];
  for (int q = 0; q < count; ++q)
    CU(cudaMemcpyAsync(host_out + static_cast<size_t>(q) * c->P, src + static_cast<size_t>(rows[q]) * c->ld,
                       4 * static_cast<size_t>(c->P), cudaMemcpyDeviceToHost, c->stream),
       "reading rows");
  CU(cudaStreamSynchronize(c->stream), "reading rows");
  if (scale_out) *scale_out = (c->sharded && c->step_pending) ? c->pend_wscale : 1.0f;
  return ASAP_OK;
}

asap_status asap_write_rows(asap_ctx* c, const int32_t* rows, int count, const float* host_in) {
  if (!c || (count > 0 && (!rows || !host_in)) || count < 0) return fail(c, ASAP_ERR_ARG, "bad argument");
  if (!c->sharded) return fail(c, ASAP_ERR_ARG, "rows are delivered to worker-sharded contexts only");
  if (!c->step_pending) return fail(c, ASAP_ERR_ARG, "deliver rows between the local step and the reduce");
  for (int q = 0; q < count; ++q) {
    if (rows[q] < 0 || rows[q] >= c->N) return fail(c, ASAP_ERR_ARG, "row outside [0, N)");
    if (rows[q] >= c->own_lo && rows[q] < c->own_lo + c->own_n)
      return fail(c, ASAP_ERR_ARG, "an owned worker's row is this context's own");
  }
  float* dst = c->W[c->round & 1];
  for (int q = 0; q < count; ++q) {
    CU(cudaMemcpyAsync(dst + static_cast<size_t>(rows[q]) * c->ld, host_in + static_cast<size_t>(q) * c->P,
                       4 * static_cast<size_t>(c->P), cudaMemcpyHostToDevice, c->stream),
       "writing rows");
    c->delivered[rows[q]] = 1;
  }
  CU(cudaStreamSynchronize(c->stream), "writing rows");
  return ASAP_OK;
}

asap_status asap_read_consistency(asap_ctx* c, uint64_t* inputs_read, uint64_t* inputs_current) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  CU(cudaStreamSynchronize(c->stream), "synchronising");
  DevState h;
  CU(cudaMemcpy(&h, c->st, sizeof h, cudaMemcpyDeviceToHost), "reading counters");
  if (inputs_read) *inputs_read = h.inputs_read;
  if (inputs_current) *inputs_current = h.inputs_current;
  return ASAP_OK;
}

asap_status asap_set_wait_limit_ns(asap_ctx* c, uint64_t ns) {
  if (!c || ns == 0) return fail(c, ASAP_ERR_ARG, "bad argument");
  c->wait_ns = ns;
  return ASAP_OK;
}

asap_status asap_debug_skip_notify(asap_ctx* c, int worker) {
  if (!c || worker < -1 || worker >= c->N) return fail(c, ASAP_ERR_ARG, "bad worker");
  c->skip_notify = worker;
  return ASAP_OK;
}

asap_status asap_set_kernel_timing(asap_ctx* c, int enable) {
  if (!c) return fail(nullptr, ASAP_ERR_ARG, "ctx is NULL");
  CU(cudaStreamSynchronize(c->stream), "synchronising");
  if (enable && c->tev.empty()) {
    c->tev.resize(2 * kTimedLaunches);
    c->tkind.resize(kTimedLaunches);
    for (auto& e : c->tev) CU(cudaEventCreate(&e), "creating timing events");
  }
  c->timing = enable != 0;
  c->tused = 0;
  return ASAP_OK;
}

asap_status asap_read_kernel_times(asap_ctx* c, uint64_t* launches, double* total_ms) {
  if (!c || !launches || !total_ms) return fail(c, ASAP_ERR_ARG, "NULL argument");
  CU(cudaStreamSynchronize(c->stream), "synchronising");
  for (int k = 0; k < ASAP_KERNEL_KINDS; ++k) {
    launches[k] = 0;
    total_ms[k] = 0.0;
  }
  for (size_t u = 0; u < c->tused; ++u) {
    float ms = 0.f;
    CU(cudaEventElapsedTime(&ms, c->tev[2 * u], c->tev[2 * u + 1]), "reading timing events");
    launches[c->tkind[u]] += 1;
    total_ms[c->tkind[u]] += ms;
  }
  c->tused = 0;
  return ASAP_OK;
}

asap_status asap_kernel_launches(asap_ctx* c, uint64_t* launches) {
  if (!c || !launches) return fail(c, ASAP_ERR_ARG, "NULL argument");
  *launches = c->launches;
  return ASAP_OK;
}

}  // extern "C"
