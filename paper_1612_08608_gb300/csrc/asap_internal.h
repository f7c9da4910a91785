// Internal declarations shared by the host runtime and the kernels of the
// ASAP library.  Nothing here is part of the public ABI (include/asap.h).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <string>
#include <vector>

#include "asap.h"

#ifdef __CUDACC__
#define ASAP_HD __host__ __device__
#else
#define ASAP_HD
#endif

namespace asap {

constexpr int kMaxWorkers = 1024;
constexpr int kMaxKp1Sparse = 32;     // neighbours per row for the sparse reduce
constexpr int kMetricsCap = 65536;    // rounds of metrics kept on the device
constexpr int kGraphRing = 64;        // device slots for per-round graphs: two halves of
constexpr int kGraphBatch = kGraphRing / 2;   // rounds uploaded together
constexpr int kThreads = 256;         // block size of every kernel here

// Device-side protocol and error state (one per context).
struct DevState {
  unsigned int err_code;     // first asap_status raised on the device (0 = none)
  unsigned int err_worker;
  unsigned int err_round;
  unsigned int mix_ticket;   // CTAs of the current reduce that have finished
  unsigned long long reduces;
  unsigned long long consistent_inputs;
  unsigned long long timeouts;
  unsigned long long inputs_read;        // (slab, worker) update blocks read by gated reduces
  unsigned long long inputs_current;     // ... whose worker had published NOTIFY for the round
};

// How the stochastic reduce of a sparse model meets its local step.
//   BSP        the reduce starts when the whole local-step grid has finished
//              (the kernel boundary is the barrier)
//   NOTIFY_ACK the reduce is launched while the local step runs; it streams
//              W at once and copies a slab's column sums only after the
//              NOTIFY of every worker with updates in the slab (time-limited)
//   ASYNC      measurement only: as NOTIFY_ACK but without the waits; a
//              block of updates copied before its worker's NOTIFY is stale
constexpr int kSyncBsp = 0;
constexpr int kSyncNotifyAck = 1;
constexpr int kSyncAsync = 2;

constexpr uint32_t kListPad = 0xffffffffu;   // padding entry of a column list

// Where one worker's minibatch lives inside a batch block (byte offsets from
// the block start).  The minibatch's entries are kept in one order only,
// sorted by (column, row); `cpos` indexes the batch's slab-major column list
// (one entry per distinct (worker, column) of the minibatch).  For the
// margins the sorted entries are cut into segments of kSlotSegment (one
// consumer warp's share of a tile); inside a segment every entry has a slot,
// the slots of one row contiguous (rows in order, a row's entries by
// column); the local step puts each entry's product and row at its slot.
// For the column sums the entries are split among the worker's Q CTAs at
// column boundaries (`bnd`).
struct BatchDesc {
  int64_t y;      // float [B]
  int64_t cpos;   // int32 [nnz]: list position of the entry's column
  int64_t cval;   // float [nnz]
  int64_t crow;   // uint16 [nnz]: row within the batch
  int64_t cslot;  // uint16 [nnz]: slot within its segment
  int64_t bnd;    // int32 [Q+1]: column-sum ranges of the worker's CTAs
  int32_t nnz;
  int32_t pad_;
};

// Entries per ring stage of the local step (a tile), and per margin slot
// segment (a consumer warp's 256-entry share of a tile).
constexpr int kTileEntries = 1024;
constexpr int kSlotSegment = 256;
// Per-warp partial margins and r stay in shared memory for minibatches of
// at most this many rows (else in global scratch).
constexpr int kRSmemRows = 2048;
constexpr int kLocalStepThreads = 192;   // four consumer warps, a bulk-copy issuer warp, a gather warp
constexpr int kMaxStepCluster = 8;       // CTAs per worker (portable cluster size)

// Arguments of the fused sparse local step (kernels_sparse.cu): one cluster
// of Q CTAs per worker.
struct LocalStepArgs {
  const unsigned char* block;  // batch block of this step
  const BatchDesc* desc;       // [N] descriptors of this step's batch
  const float* wv;             // w values at the step's list positions
  float* gsum;                 // column sums at the step's list positions
  float* mpart_big;            // [N][Q][4][B] per-warp partial margins (B > kRSmemRows only)
  float* r_big;                // [N][Q][B] r (B > kRSmemRows only)
  float* loss_part;            // [N]: minibatch loss sum per worker
  unsigned int* ready;         // NOTIFY flags [N]
  DevState* st;
  const int* worker_of;        // worker of each cluster (a permutation or, worker-sharded, the owned
                               // workers), or nullptr
  int N, B, Q, stages;         // N: clusters launched (workers stepped)
  unsigned int round;
  int skip_worker;             // fault injection: do not NOTIFY this worker
  float mscale;                // true w = mscale * (stored values): margins are scaled by it
  int notify;                  // publish NOTIFY (last local step of the round)
};

// Arguments of the stochastic reduce.
struct MixArgs {
  float* out;                  // next parameter buffer
  uint16_t* shadow;            // bf16 copy of `out` (softmax) or nullptr
  int64_t ld;                  // row stride of W (floats), multiple of 64
  int N;
  int kp1;                     // neighbours per row (sparse kind)
  const int* nbr;              // [N][kp1]
  const float* wgt;            // [N][kp1]
  float wscale;                // the round's L2 shrink prod_j (1 - eta_j l2) after local steps, else 1
  int uniform_w;               // every weight of the table equals wgt[0]
  int S;                       // slab width (columns)
  int rows_pad;                // smem rows per slab (box_rows * n_boxes)
  int box_rows;
  int n_boxes;
  int stages;
  long long n_slabs;
  // fused sparse update / export (FUSED kernels only)
  const uint32_t* upd_list;    // this round's column list (slab-major)
  const int* upd_off;          // [n_slabs + 1] slab regions of upd_list
  const float* gsum;           // column sums at upd_list positions
  float upd_scale;             // eta / (B wscale) of the round's last local step
  const uint32_t* exp_list;    // next round's column list
  const int* exp_off;          // [n_slabs + 1]
  float* wv_out;               // w_{t+1} at exp_list positions
  int max_region;              // entries: the largest slab region of any list
  // metrics and protocol
  double* cons_part;           // scratch [gridDim.x]
  const float* loss_part;      // [n_loss_part] from the local step
  int n_loss_part;
  float loss_norm;             // 1 / (N B)
  int have_loss;
  float* metrics_loss;         // ring of kMetricsCap
  float* metrics_cons;
  unsigned int* ready;
  unsigned int* consumed;
  unsigned int* stamp_next;    // [N] stamp of the buffer being written
  DevState* st;
  unsigned int round;
  int expect_notify;
  unsigned long long wait_ns;
  int sync_mode;               // kSync* (FUSED reduces; others are BSP)
  int own_lo, own_n;           // workers stepped in this context: the NOTIFY waits and the counters cover
                               // [own_lo, own_lo + own_n); a worker-sharded context learns of the others'
                               // NOTIFY on the host, when their rows are delivered
};

// Arguments of the dense softmax-regression step (kernels_dense.cu).
struct DenseFwdArgs {
  int C, Cq, d, B, nb, t;      // Cq = ceil(C / 256) CTAs per cluster
  int N;                       // workers (set by the launcher)
  const int* y;                // [N][nb*B] class ids
  uint16_t* RT;                // [N][Cq*256][B] bf16: R^T
  float* loss_part;            // [N][B/128][Cq]
  float inv_B;
  DevState* st;
  unsigned int round;
};

struct DenseGradArgs {
  int C, Cq, d, B, nb, t;
  int N;                       // workers (set by the launcher)
  float* W;                    // fp32 master [N][ld], worker row = C x d class-major
  int64_t ld;
  float lr;
  float decay;                 // 1 - lr * l2
  unsigned int* ready;
  unsigned int* worker_ticket;
  int skip_worker;
  DevState* st;
  unsigned int round;
};

asap_status build_graph_host(asap_graph_kind kind, int N, int k, uint64_t seed, int64_t round,
                             int32_t* nbr, const char** why);

// Launchers (kernels_*.cu).  Each returns the cudaError_t of the launch.
cudaError_t launch_local_step(const LocalStepArgs& a, int loss, size_t smem, cudaStream_t s);
size_t local_step_smem_bytes(int B, int stages);
cudaError_t local_step_configure(size_t smem);
cudaError_t launch_apply_update(float* W, int64_t ld, const uint32_t* list, const int* slab_off, long long n_slabs,
                                int S, const float* gsum, float scale, int sm_count, cudaStream_t s);
cudaError_t launch_gather_wv(const float* W, int64_t ld, const uint32_t* list, const int* slab_off, long long n_slabs,
                             int S, float* wv, int sm_count, cudaStream_t s);
constexpr int kMixComputeWarps = 16;
constexpr int kMixUpdaterWarps = 2;
// compute warps + one TMA producer warp + the warps that apply the fused update
constexpr int kMixThreads = (kMixComputeWarps + 1 + kMixUpdaterWarps) * 32;
cudaError_t launch_mix(const CUtensorMap& tmap, const MixArgs& a, bool complete, bool fused, int grid, size_t smem,
                       cudaStream_t s);
ASAP_HD size_t mix_stage_bytes(int S, int rows_pad, int max_region);
size_t mix_smem_bytes(int N, int kp1, int S, int rows_pad, int stages, int max_region);
cudaError_t mix_configure(bool complete, bool fused, int kp1, bool shadow, size_t smem);
cudaError_t mix_occupancy(bool complete, bool fused, int kp1, bool shadow, size_t smem, int* blocks);
size_t dense_smem_bytes();
cudaError_t dense_configure();
cudaError_t launch_dense_fwd(const CUtensorMap& tmX, const CUtensorMap& tmW, const DenseFwdArgs& f, int N,
                             cudaStream_t s);
cudaError_t launch_dense_grad(const CUtensorMap& tmR, const CUtensorMap& tmXT, const CUtensorMap& tmWf,
                              const DenseGradArgs& g, int N, int sm_count, cudaStream_t s);
cudaError_t launch_cast_bf16(const float* src, uint16_t* dst, int64_t n, cudaStream_t s);

}  // namespace asap
