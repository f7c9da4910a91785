/*
 * asap.h -- C ABI of the GB300 implementation of ASAP's data-parallel hot
 * path (Kadav & Kruus, "ASAP: Asynchronous Approximate Data-Parallel
 * Computation", arXiv 1612.08608).
 *
 * One context holds N simulated workers on one GPU.  Worker i owns a
 * parameter vector w_i (fp32) and a private data shard.  One round is the
 * paper's Eq. A.1:
 *
 *     w_{t+1/2}^i = w_t^i - eta * grad f_i(w_t^i)          (local SGD step)
 *     w_{t+1}^i   = sum_j P_t[i, j] * w_{t+1/2}^j          (stochastic reduce)
 *
 * where P_t is a doubly-stochastic mixing matrix with k+1 non-zeros per row
 * (k in-neighbours plus the worker itself) from a sparse communication
 * graph (Section 3, "stochastic reduce"; Appendix A, "Network requirement").
 * NOTIFY-ACK (Section 4, "Fine-grained synchronization") is kept as
 * per-worker round counters in device memory: worker i publishes
 * ready[i] = t+1 after its step, a reduce reads worker j's half-step model
 * only when ready[j] == t+1, and consumed[i] = t+1 acknowledges that every
 * input of worker i's reduce has been read.  Parameters are double-buffered
 * (W[t & 1] holds round t), so no reduce ever sees a torn or mixed-version
 * input, whatever the schedule.
 *
 * Conventions for every entry point:
 *  - The return value is an asap_status; no C++ exception crosses the ABI.
 *  - Host pointers passed in are read during the call and never retained;
 *    the caller keeps ownership.  Device memory is allocated and owned by the
 *    context and released by asap_destroy.
 *  - Calls marked "async" enqueue work on the context's stream and return;
 *    they report launch errors at once.  Errors found on the device (a wait
 *    that ran out, a stamp that did not match) are reported by the next
 *    "syncing" call (asap_read_params, asap_read_metrics, asap_sync).
 *  - asap_last_error(ctx) gives a one-line description of the last failure;
 *    asap_last_error(NULL) gives the last failure of asap_create or of a
 *    context-free helper on this thread.
 *  - A context is not thread-safe; use one host thread per context.
 */
#ifndef ASAP_H
#define ASAP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct asap_ctx asap_ctx;

typedef enum {
  ASAP_OK = 0,
  ASAP_ERR_ARG = 1,     /* invalid argument, size or call order             */
  ASAP_ERR_CUDA = 2,    /* a CUDA runtime call or kernel launch failed       */
  ASAP_ERR_OOM = 3,     /* device or pinned host allocation failed           */
  ASAP_ERR_TIMEOUT = 4, /* a device-side NOTIFY/ACK wait ran out            */
  ASAP_ERR_STATE = 5,   /* a round stamp did not match (protocol violation)  */
  ASAP_ERR_GRAPH = 6    /* the requested graph cannot be built / is invalid  */
} asap_status;

/* Communication graphs (Section 3.1 and Fig. 2).  Row i of P lists i and its
 * in-neighbours in ascending order; the default weights are 1/(k+1). */
typedef enum {
  ASAP_GRAPH_RING = 1,           /* chain closed into a ring: i <- i-1 (k = 1)        */
  ASAP_GRAPH_ROOT = 2,           /* root expander: i <- i-1, i-isqrt(N) (k = 2, N>=4) */
  ASAP_GRAPH_RANDOM_REGULAR = 3, /* seeded random k-regular digraph (see below)       */
  ASAP_GRAPH_COMPLETE = 4,       /* all-reduce: every worker (k = N-1)                */
  ASAP_GRAPH_EXPLICIT = 5,       /* user weights, see asap_set_mixing                 */
  ASAP_GRAPH_IDENTITY = 6        /* no communication (k = 0)                          */
} asap_graph_kind;

typedef enum {
  ASAP_LOSS_NONE = 0,     /* no local step: the context only mixes              */
  ASAP_LOSS_HINGE = 1,    /* linear SVM, l = max(0, 1 - y m) (Section 6)         */
  ASAP_LOSS_LOGISTIC = 2, /* l = ln(1 + exp(-y m))                              */
  ASAP_LOSS_SOFTMAX = 3   /* dense softmax regression on bf16 features          */
} asap_loss;

typedef enum {
  ASAP_SHARDS_DEVICE = 0, /* shards copied to HBM once at load time             */
  ASAP_SHARDS_HOST = 1    /* shards kept in pinned host memory; each round's
                             minibatch block is copied to the GPU as the round
                             runs (overlapped with the previous round)         */
} asap_residency;

/* Create a context for N workers with d parameters each (d features; for
 * softmax regression the model is C x d, see asap_set_model).  k is the
 * number of in-neighbours besides the worker itself.  The default graph is
 * IDENTITY for k = 0, RING for k = 1, COMPLETE for k = N-1 and
 * RANDOM_REGULAR otherwise, built from graph_seed and fixed for all rounds.
 * W_0 = 0 (Appendix A takes w_0 = 0).  Uses the current CUDA device.
 * Limits: 1 <= N <= 1024, 1 <= d, 0 <= k <= N-1.  On failure *out = NULL. */
asap_status asap_create(int N, int64_t d, uint64_t graph_seed, int k, asap_ctx** out);

/* Choose the graph kind, and whether a new graph is drawn from
 * (graph_seed, round) every round (Section 3.1 wants graphs that are cheap
 * to build, so that they can be rebuilt, e.g. around a failure).  The kind must match k (RING: 1,
 * ROOT: 2, COMPLETE: N-1, IDENTITY: 0).  RANDOM_REGULAR construction:
 * SplitMix64 seeded with graph_seed ^ (0x9E3779B97F4A7C15 * (round+1));
 * a uniform random Hamiltonian cycle (Fisher-Yates), then k-1 permutation
 * layers drawn by Fisher-Yates with rejection (a node may not receive from
 * itself or twice from the same node); at most 100,000 draws per layer,
 * else ASAP_ERR_GRAPH.  Call before the first round that should use it. */
asap_status asap_set_graph(asap_ctx* ctx, asap_graph_kind kind, int regenerate_every_round);

/* Explicit mixing weights (kind EXPLICIT), fixed for all rounds.
 * nbr: N*(k+1) int32, row-major, each row strictly ascending, ids in [0,N);
 * wgt: N*(k+1) float, >= 0.  P must be doubly stochastic: every row sum and
 * every column sum within 1e-6 of 1 (Appendix A), else ASAP_ERR_GRAPH.
 * Rows may omit the worker itself.  Requires k+1 <= 32. */
asap_status asap_set_mixing(asap_ctx* ctx, const int32_t* nbr, const float* wgt);

/* The local objective f_i of Eq. A.1.  loss: ASAP_LOSS_*; num_classes: C for
 * SOFTMAX (then each worker's model is C x d, class-major), 1 otherwise;
 * batch: minibatch rows B per worker per round (round t uses rows
 * [(t mod nb) B, (t mod nb) B + B), nb = floor(rows / B)); lr: eta (> 0);
 * l2: coefficient of (l2/2) ||w||^2 in f_i (0 <= lr*l2 < 1).
 * SOFTMAX requires d % 256 == 0, B % 128 == 0, 2 <= C <= 1024.  Re-setting the
 * model clears the shards and resets W to 0. */
asap_status asap_set_model(asap_ctx* ctx, asap_loss loss, int num_classes, int batch, float lr, float l2);

/* Learning-rate schedules for asap_set_schedule. */
typedef enum {
  ASAP_LR_CONSTANT = 0, /* eta_k = lr                                   */
  ASAP_LR_INVERSE = 1   /* eta_k = lr / (1 + gamma k)  (Bottou's SVM-SGD) */
} asap_lr_schedule;

/* Local steps per round and the learning-rate schedule.  Eq. A.1 writes the
 * rate as eta_t; in Section 5 each replica trains on a handful of local
 * examples between two exchanges.  Each round runs local_steps (>= 1)
 * minibatch steps per worker before the reduce: step j of round t is global
 * step k = t * local_steps + j, on minibatch k mod nb, at rate eta_k;
 * asap_local_step runs all of them and the round's loss metric is its last
 * step's.  The L2 shrink of the intermediate steps is kept as one scale per
 * round (all workers take the same steps) and applied in the reduce.
 * SOFTMAX models take the schedule with local_steps = 1 only.  Defaults:
 * 1, ASAP_LR_CONSTANT.  Keeps W, shards and the round counter; the
 * minibatch of a round follows the new local_steps from the next call on. */
asap_status asap_set_schedule(asap_ctx* ctx, int local_steps, asap_lr_schedule kind, float gamma);

/* Stream for all device work of this context (a cudaStream_t, e.g.
 * torch.cuda.current_stream().cuda_stream).  NULL selects the context's own
 * non-blocking stream (the default). */
asap_status asap_set_stream(asap_ctx* ctx, void* cuda_stream);

/* Where the shards live.  Default DEVICE.  Called after loading, it moves
 * the loaded shards (synchronous). */
asap_status asap_set_shard_residency(asap_ctx* ctx, asap_residency residency);

/* Bytes of the minibatch block that round `round` reads (all workers: the
 * padded CSR rows, labels and the column-sorted copy).  With HOST residency
 * this is what one round copies to the GPU.  Host only. */
asap_status asap_shard_block_bytes(asap_ctx* ctx, int64_t round, uint64_t* bytes);

/* Load one CSR shard per worker (hinge / logistic).  All pointers are host
 * pointers, one per worker: rowptr[i] has n_rows[i]+1 int64 entries starting
 * at 0; col[i] / val[i] have rowptr[i][n_rows[i]] entries; col ids in
 * [0, d), distinct within a row; y[i] has n_rows[i] labels in {-1, +1}.
 * Every worker needs n_rows[i] >= B.  The library builds, once, the batch
 * layout the kernels read (rows padded to 4 entries; per batch a copy
 * sorted by (column, row)).  Synchronous. */
asap_status asap_load_shards(asap_ctx* ctx, const int64_t* const* rowptr, const int32_t* const* col,
                             const float* const* val, const float* const* y, const int64_t* n_rows);

/* Load one dense shard per worker (softmax): X[i] is n_rows[i] x d bf16
 * (raw uint16 bits, row-major), y[i] n_rows[i] class ids in [0, C).
 * Synchronous. */
asap_status asap_load_dense_shards(asap_ctx* ctx, const uint16_t* const* X_bf16, const int32_t* const* y,
                                   const int64_t* n_rows);

/* Eq. A.1 first line for every worker, then NOTIFY (ready[i] = t+1).
 * Async.  Between this call and asap_stochastic_reduce, for SOFTMAX models
 * the current buffer holds w_{t+1/2}.  For hinge / logistic models it holds
 * w_t with every local step but the round's last applied (values scaled by
 * the inverse L2 shrink of those steps); the last step's update is applied
 * by the reduce to each column slab it loads, so w_{t+1/2} is never stored. */
asap_status asap_local_step(asap_ctx* ctx);

/* Eq. A.1 second line for every worker: wait for the in-neighbours' NOTIFY,
 * W[(t+1)&1] = P_t W[t&1], ACK (consumed[i] = t+1), record the round's
 * metrics, advance t.  Without a preceding asap_local_step it mixes the
 * current parameters (the reduce alone).  Async. */
asap_status asap_stochastic_reduce(asap_ctx* ctx);

/* T rounds of (asap_local_step; asap_stochastic_reduce).  Async. */
asap_status asap_round(asap_ctx* ctx, int T);

/* Wait for all queued work; report device-side errors.  Syncing. */
asap_status asap_sync(asap_ctx* ctx);

/* Copy the current parameters W_t (N rows of P = d or C*d floats, row-major,
 * packed) to host_out; *round_out = t (may be NULL).  Syncing. */
asap_status asap_read_params(asap_ctx* ctx, float* host_out, int64_t* round_out);

/* Set W_t = host_in (N rows of P floats) and the round counter to `round`
 * (resume from a checkpoint, or a custom W_0).  Synchronous. */
asap_status asap_write_params(asap_ctx* ctx, const float* host_in, int64_t round);

/* Set W_t from device memory: dev_in holds N rows of P floats with row
 * stride ld_in (>= P), on the context's device; the round counter becomes
 * `round`.  For parameters that already live in HBM (a resume, or inputs
 * drawn on the device), without a host round trip.  Synchronous. */
asap_status asap_write_params_device(asap_ctx* ctx, const float* dev_in, int64_t ld_in, int64_t round);

/* Copy columns [first, first + count) of every worker's current
 * parameters W_t to host_out (N rows of count floats, row-major): a sample
 * of the model without reading all N x P values.  Syncing. */
asap_status asap_read_param_columns(asap_ctx* ctx, int64_t first, int64_t count, float* host_out);

/* Per-round metrics of rounds [first_round, first_round + count): the mean
 * over workers of the minibatch loss at the pre-step parameters (NaN for a
 * reduce-only round) and the consensus error ||W_{t+1} - 1 wbar^T||_F.
 * The last 65536 rounds are kept.  Either output pointer may be NULL.
 * Waits only until round first_round + count - 1 is complete when that is
 * one of the last 64 rounds launched since the last asap_write_params
 * (rounds queued after it keep running, so a caller may read round t's
 * metrics while round t+1 runs); otherwise, and for count = 0, it
 * synchronises fully.  A device error recorded by then is reported after a
 * full drain, as by asap_sync. */
asap_status asap_read_metrics(asap_ctx* ctx, int64_t first_round, int64_t count, float* loss_out,
                              float* consensus_out);

/* Counters of the NOTIFY-ACK protocol since creation: reduces performed,
 * in-neighbour inputs whose round stamp matched (Section 6.2 reports the
 * share of such consistent reduces), and waits that ran out.  Syncing. */
asap_status asap_read_counters(asap_ctx* ctx, uint64_t* reduces, uint64_t* consistent_inputs,
                               uint64_t* timeouts);

/* The graph used by round `round`: nbr_out N*(k+1) int32 and wgt_out
 * N*(k+1) float (either may be NULL).  Host only. */
asap_status asap_get_graph(asap_ctx* ctx, int64_t round, int32_t* nbr_out, float* wgt_out);

/* How a sparse model's stochastic reduce meets its local step (Section 4
 * contrasts the three; Section 6.2 measures them).
 *   BSP        (default) the reduce starts when the whole local step has
 *              finished: the kernel boundary is the barrier.
 *   NOTIFY_ACK the reduce is launched while the local step runs; it streams
 *              W at once and copies a column slab's updates only after the
 *              NOTIFY for the round of every worker with updates in the slab
 *              (time-limited waits), so a slab waits only for those workers.
 *              Results are identical to BSP.
 *   ASYNC      for measurement only: as NOTIFY_ACK without the waits; an
 *              update read before its worker's NOTIFY is stale, so results
 *              depend on the schedule (asap_read_consistency counts how
 *              many inputs were current).
 * Dense (softmax) models always use BSP.  Not while a local step is
 * pending. */
typedef enum {
  ASAP_SYNC_BSP = 0,
  ASAP_SYNC_NOTIFY_ACK = 1,
  ASAP_SYNC_ASYNC = 2
} asap_sync_mode;
asap_status asap_set_sync_mode(asap_ctx* ctx, asap_sync_mode mode);

/* The order in which the local step's CTA clusters take the workers:
 * cluster q runs worker order[q] (a permutation of [0, N); NULL restores
 * the identity).  The schedule changes, the arithmetic does not: results
 * are bit-identical, which the tests check.  Not while a local step is
 * pending. */
asap_status asap_set_worker_order(asap_ctx* ctx, const int32_t* order);

/* Worker-sharded mode (Section 5, Implementation: each process holds the
 * replicas of some workers, and a worker's model reaches the processes of
 * its out-neighbours as a point-to-point message).  This context steps only
 * workers [first, first + count) of its N-worker system; W keeps all N rows,
 * but the rows of the other workers hold what the caller delivered.  Per
 * round:
 *   asap_local_step       the owned workers' minibatch step; their rows of W_t
 *                         then hold the half step x_j - eta g_j;
 *   asap_read_rows        the owned rows that other processes need;
 *   asap_write_rows       the rows received from other processes (every
 *                         in-neighbour of an owned worker under the round's
 *                         graph, asap_get_graph);
 *   asap_stochastic_reduce  the owned rows of W_{t+1}.  It fails with
 *                         ASAP_ERR_ARG, launching nothing, if an in-neighbour's
 *                         row was not delivered this round: for a worker
 *                         stepped elsewhere the delivery is its NOTIFY.
 * Hinge and logistic models, BSP only, any graph; every process must use the
 * same N, d, graph seed, graph kind and model settings.  Call after
 * asap_set_model and before asap_load_shards (it drops loaded shards);
 * asap_load_shards then reads only the owned workers' shards (the others'
 * pointers may be NULL).  first = 0, count = N restores the whole system.
 * asap_read_metrics then returns this context's share of the mean loss (the
 * sum over owned workers / (N B): the shares of all processes add up to the
 * mean loss) and NaN for the consensus error.  Syncing. */
asap_status asap_set_worker_range(asap_ctx* ctx, int first, int count);

/* Copies rows `rows[0..count)` of the current parameters W_t (row-major,
 * count x P floats, P = d C) to host memory.  Between asap_local_step and
 * asap_stochastic_reduce of a worker-sharded context the owned rows hold
 * the half step in stored form: true values = stored values x *scale_out
 * (the product of the round's L2 shrink factors; 1 without L2).  Processes
 * with the same model settings share the factor, so rows are sent as
 * stored.  Otherwise *scale_out = 1.  scale_out may be NULL.  Syncing. */
asap_status asap_read_rows(asap_ctx* ctx, const int32_t* rows, int count, float* host_out, float* scale_out);

/* Writes rows received from other processes into the current parameters
 * W_t of a worker-sharded context, after its local step and before its
 * reduce: rows[q] (not an owned worker) gets host_in[q * P .. (q+1) * P),
 * in the sender's stored form.  Each row counts as delivered for this round.
 * ASAP_ERR_ARG for an owned or out-of-range row, or outside that window.
 * Syncing. */
asap_status asap_write_rows(asap_ctx* ctx, const int32_t* rows, int count, const float* host_in);

/* Consistency of the gated (NOTIFY_ACK, ASYNC) reduces since creation: the
 * inputs they read -- one per (column slab, worker) block of updates -- and
 * how many of those were current, i.e. read after the worker's NOTIFY for
 * the round (the analogue of Section 6.2's consistent reduces, Fig. 8).
 * NOTIFY_ACK makes every input current.  Syncing. */
asap_status asap_read_consistency(asap_ctx* ctx, uint64_t* inputs_read, uint64_t* inputs_current);

/* Limit for every device-side NOTIFY/ACK wait, in nanoseconds (default
 * 200 ms).  A wait that runs out sets ASAP_ERR_TIMEOUT and the kernel
 * returns without writing the round's output. */
asap_status asap_set_wait_limit_ns(asap_ctx* ctx, uint64_t ns);

/* Fault injection for tests: the next asap_local_step does not publish
 * NOTIFY for `worker` (a stalled worker), so every reduce that depends on it
 * runs into its wait limit.  worker = -1 clears the injection. */
asap_status asap_debug_skip_notify(asap_ctx* ctx, int worker);

/* Host only, for tests (no device needed): the image asap_load_shards builds
 * for minibatch t -- the index structure of Section 5's per-worker updates
 * laid out for the stochastic reduce's column slabs (no counterpart in the
 * paper beyond that).  Shards as in asap_load_shards, each with at least
 * (t + 1) * batch rows (not checked: there is no row count here); batch: B rows;
 * slab_cols: the slab width S (a power of two, 8 to 1024); the column list
 * covers ceil(round_up(d, 64) / S) slabs; ctas_per_worker: Q, the CTAs of
 * one worker's local step (1 to 8).  The image is written to `image` (cap
 * bytes; *image_bytes receives its size; ASAP_ERR_ARG when it does not fit).
 * desc_out (N*8 int64), per worker: byte offsets of the labels (float [B]),
 * of the (column, row)-sorted entries' list positions, values, rows and
 * segment slots (int32 / float / uint16 / uint16 [nnz]) and of the Q+1
 * column-sum range bounds (int32), then nnz, then 0.  Segment g holds sorted entries [256 g,
 * 256 (g+1)); its slots are numbered row by row, a row's entries in sorted
 * order.  The range bounds start at 0, end at nnz and cut the sorted entries
 * at the first column boundary at or after q nnz / Q.  list_out (3 int64):
 * byte offsets of the slab-major list of distinct (worker << 16 | column in
 * slab) codes and of its slab offsets (int32 [n_slabs + 1]), and the list
 * length in entries. */
asap_status asap_debug_batch_image(int N, int64_t d, int batch, int slab_cols, int ctas_per_worker, int t,
                                   const int64_t* const* rowptr, const int32_t* const* col, const float* const* val,
                                   const float* const* y, unsigned char* image, int64_t cap, int64_t* image_bytes,
                                   int64_t* desc_out, int64_t* list_out);

/* Kernel kinds for per-kernel timing. */
typedef enum {
  ASAP_KERNEL_LOCAL_STEP = 0, /* sparse margins, loss derivative, column sums,
                                 NOTIFY (a2-a4), one fused kernel               */
  ASAP_KERNEL_REDUCE = 1,     /* stochastic reduce + ACK + metrics (a5-a7, a9)  */
  ASAP_KERNEL_DENSE_FWD = 2,  /* dense logits, softmax, R^T (a3')               */
  ASAP_KERNEL_DENSE_GRAD = 3, /* dense gradient GEMM + update + NOTIFY (a3')    */
  ASAP_KERNEL_APPLY = 4,      /* update of a local step before the round's last */
  ASAP_KERNEL_GATHER = 5,     /* w at a step's columns from the stored W        */
  ASAP_KERNEL_KINDS = 6
} asap_kernel_kind;

/* Per-kernel timing: while enabled, every kernel launch of the context is
 * bracketed by CUDA events on the context stream (the first 8192 launches
 * after enabling or after the last read). */
asap_status asap_set_kernel_timing(asap_ctx* ctx, int enable);

/* Per kernel kind: timed launches and their total milliseconds, since
 * enabling or since the last read (which resets them).  launches and
 * total_ms have ASAP_KERNEL_KINDS entries.  Syncing. */
asap_status asap_read_kernel_times(asap_ctx* ctx, uint64_t* launches, double* total_ms);

/* Number of this library's kernel launches since creation (host counter). */
asap_status asap_kernel_launches(asap_ctx* ctx, uint64_t* launches);

/* Context-free helper: build graph `kind` for (N, k, graph_seed, round) on
 * the host, exactly as a context would.  nbr_out: N*(k+1) int32.  Needs no
 * GPU. */
asap_status asap_build_graph(asap_graph_kind kind, int N, int k, uint64_t graph_seed, int64_t round,
                             int32_t* nbr_out);

/* Stochastic reduce W_out = P W_in with its consensus error, for callers
 * that cannot allocate device memory (a host framework that owns all of
 * HBM through its own pool, or a latency-critical loop where cudaMalloc /
 * cudaFree may synchronise the device).  The paper has no counterpart: it
 * is the reduce of asap_stochastic_reduce without a context.
 * All pointers are device pointers owned by the caller: W_in, W_out
 * N rows of `ld` floats (row stride ld, ld >= d, ld % 4 == 0, 16-byte
 * aligned, the two ranges of N*ld floats not overlapping; columns [d, ld)
 * are mixed too); nbr / wgt N*kp1
 * int32 / float (row i = the ids in [0, N) and weights of worker i's
 * inputs, summed in the given order; ids outside [0, N) are clamped into
 * range, never read out of bounds); consensus_out one float, set to
 * ||W_out - 1 wbar^T||_F with wbar the column mean of W_in.  Limits:
 * 1 <= N <= 256, 1 <= kp1 <= 32, and ld within the built-in scratch (32768
 * column slabs: ld <= 8,388,608 for N <= 16, ld <= 524,288 for N = 256);
 * larger sizes return ASAP_ERR_ARG without touching the GPU.
 * It calls no cudaMalloc, cudaFree or other allocating routine: its scratch
 * (about 256 KB) is a file-scope device array that every GPU loading this
 * library holds until the process exits.  The first call on each device
 * looks up that array's device address (cudaGetSymbolAddress) with the
 * device current, so make that first call before any stream capture.  The
 * address is kept per device together with the id of the CUDA context it
 * was found in; a call from a different context (after cudaDeviceReset, or
 * a host framework that reset its primary context) looks it up again.  Every
 * call shares the array and clears what must start at zero; calls that
 * overlap on the GPU (other streams, other threads) race on it and must be
 * serialised by the caller.  Async on cuda_stream (NULL: legacy default
 * stream); no device-side error is reported. */
asap_status asap_mix_noalloc(const float* W_in, float* W_out, int N, int64_t d, int64_t ld, const int32_t* nbr,
                             const float* wgt, int kp1, float* consensus_out, void* cuda_stream);

const char* asap_last_error(const asap_ctx* ctx);
const char* asap_version(void);
void asap_destroy(asap_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* ASAP_H */
