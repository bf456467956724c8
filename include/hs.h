/*
 * hs.h - C ABI of libhs: one synchronous data-parallel SGD step over M logical
 * workers whose partitions follow their compute power (arXiv 2110.08941).
 *
 * The paper's method in the terms used here:
 *   - Section 1: M workers each compute a stochastic gradient g^m_t of their
 *     local objective f_m (Eq. 1, the mean loss over the worker's data); the
 *     gradients are averaged, g_t = (1/M) sum_m g^m_t, and the model is updated
 *     theta_{t+1} = theta_t - eta_t g_t.
 *   - Section 4, Eq. 2: compute power CP_m = |D_m| / X_m (samples per second).
 *   - Section 4.1, Algorithm 1 (Dynamic Partitioning): normalise the CPs and
 *     size worker m's partition as CP_m * |D|; the first partition is even.
 *   - Section 4.2 (Enhanced Dynamic Partitioning): weight each g^m by the
 *     normalised compute power before the gradient exchange.
 *
 * On one GPU the M workers are contiguous segments of one global minibatch:
 * worker m owns samples [off_m, off_m + n_m).  Each segment gets its own
 * forward and backward pass and its own gradient G_m, and the update applies
 * sum_m w_m G_m.  On the bf16 MLP step each tile of a layer's weight gradient
 * G_m is formed in tensor memory and folded into the weighted sum there, in
 * worker order, by the kernel that also applies the update; bias gradients (and
 * every range on the slab path: debug read-back, more than 32 workers, layers
 * with fewer 256 x 256 weight tiles than SM pairs, the slab-free variant, the
 * fp32 check path, the CNN) go through per-worker fp32 slabs in
 * device memory and one reduce-and-update pass.  Both forms give the same bits.
 *
 * Conventions for every entry point:
 *   - Pointers marked "device" are CUDA device pointers on the device that was
 *     current at hs_init; "host" pointers are ordinary CPU memory.  The library
 *     never takes ownership of caller memory.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Work is
 *     enqueued on it; calls return before the GPU finishes unless stated.
 *   - Every call returns an hs_status and never throws or aborts.  Invalid
 *     arguments are rejected on the host before any GPU work is enqueued; the
 *     message is available from hs_last_error(ctx).
 *   - A context is not thread-safe and is meant for one stream at a time.
 */
#ifndef HS_H_
#define HS_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct hs_ctx hs_ctx;

typedef enum {
  HS_OK = 0,
  HS_ERR_INVALID_ARG = 1,   /* bad pointer, size, enum or numeric value; nothing was enqueued */
  HS_ERR_CUDA = 2,          /* a CUDA runtime call failed (message has the CUDA error string) */
  HS_ERR_OOM = 3,           /* device workspace allocation failed */
  HS_ERR_UNSUPPORTED = 4,   /* valid request outside what the library implements */
  HS_ERR_DEVICE_CHECK = 5   /* a kernel's own check failed (bounded wait timed out); results invalid */
} hs_status;

typedef enum { HS_MLP = 0, HS_CNN = 1 } hs_arch;

/* HS_BF16: bf16 tensor-core operands (tcgen05), fp32 accumulation, fp32 master
 * parameters and fp32 gradient slabs.  HS_FP32_CHECK: the same step with every
 * contraction in fp32 on the CUDA cores (a check path for tight parity). */
typedef enum { HS_BF16 = 0, HS_FP32_CHECK = 1 } hs_precision;

/* Gradient synchronisation weights w_m in g = sum_m w_m g^m:
 *   HS_SYNC_MEAN        w_m = 1/M                  (Section 1, Sync-SGD / DP-SGD)
 *   HS_SYNC_CP_WEIGHTED w_m = n_m / N              (Section 4.2, EDP-SGD: the normalised
 *                                                   compute power as realised by the integer
 *                                                   partition; weights sum to 1)
 *   HS_SYNC_CP_LITERAL  w_m = (CP_m / sum CP) / M  (Section 4.2 read literally: weight, then
 *                                                   the averaging exchange of Section 1) */
typedef enum { HS_SYNC_MEAN = 0, HS_SYNC_CP_WEIGHTED = 1, HS_SYNC_CP_LITERAL = 2 } hs_sync;

/* Model description (all fields 32-bit for a stable ABI).
 *   MLP: dims[0..n_layers] = d0 (input features), hidden widths, d_L = classes.
 *        Layer l: A_l = H_{l-1} W_l^T + b_l, ReLU on every layer but the last.
 *        HS_BF16 needs d0..d_{L-1} to be multiples of 8 (16-byte rows for TMA).
 *   CNN: dims[0..6] = Cin, H, W, c1, c2, c3, classes: three 3x3 convs with
 *        padding 1 and strides 1, 2, 2 (ReLU after each), global average pool,
 *        one fully connected layer.  n_layers is ignored.
 * Parameter layout (flat fp32): [W1, b1, W2, b2, ...]; linear W row-major
 * [out, in]; conv W [Cout, Cin, 3, 3]; fc W [classes, c3]. */
typedef struct {
  int32_t arch;        /* hs_arch */
  int32_t n_layers;
  const int32_t* dims; /* host; copied by hs_init */
  int32_t precision;   /* hs_precision */
  int32_t sync;        /* hs_sync */
} hs_model_desc;

/* A partition as produced by hs_partition (Algorithm 1).  All pointers are
 * owned by the context and stay valid until the next hs_partition call on it
 * or hs_destroy. */
typedef struct {
  int32_t M, N;
  const int32_t* counts_host;   /* host [M]: n_m, sum = N, each >= 1 */
  const int32_t* offsets_host;  /* host [M+1]: exclusive prefix sum, offsets[M] = N */
  const int32_t* index_map_dev; /* device [N]: index_map[i] = m for offsets[m] <= i < offsets[m+1] */
  const double* weights_host;   /* host [M]: synchronisation weights w_m of the context's hs_sync */
  const double* cp_host;        /* host [M]: normalised compute power the sizes were drawn from */
  uint64_t version;             /* increments on every hs_partition call that changes the sizes */
} hs_partition_t;

/* Algorithm 1's sizing rule on the host, no GPU involved (Section 4.1,
 * Algorithm 1; Eq. 2 gives the CPs).  counts_out[m] = n_m from compute powers
 * cp[0..M-1] (any positive scale) over a batch of N samples:
 *   S = sum cp (fp64, left to right); q_m = (cp_m / S) * N; n_m = floor(q_m),
 *   then N - sum floor(q) extra samples to the largest remainders q_m - floor(q_m)
 *   (ties: lower m); finally every worker with 0 samples takes one from the
 *   largest worker (ties: lower m).
 * Errors: HS_ERR_INVALID_ARG if M < 1, N < M, a null pointer, or any cp not
 * finite and > 0.  counts_out is host [M], caller-owned. */
hs_status hs_partition_sizes(int32_t M, int32_t N, const double* cp, int32_t* counts_out);

/* Number of fp32 parameters P of a model (layout above).  Host only. */
hs_status hs_param_count(const hs_model_desc* model, int64_t* P);

/* Create a context on the current CUDA device for global batch N = global_batch
 * split over M workers.  compute_weights: host [M] initial compute powers, or
 * NULL for the even split of Algorithm 1's first epoch (t = 0).  Allocates all
 * device workspace (per-worker gradient slabs M x P fp32, activations for N
 * rows, the bf16 parameter shadow) and computes the initial partition
 * synchronously.  Errors: HS_ERR_INVALID_ARG (bad model/M/N/weights),
 * HS_ERR_UNSUPPORTED (shape constraint of the precision), HS_ERR_OOM,
 * HS_ERR_CUDA.  On error *out is NULL.
 * Read here from the environment (all give the same results; they select how):
 *   HS_TILE_AVERAGE=0    bf16 MLP: every layer's weight gradients through the
 *                        per-worker slabs (default: averaged in tensor memory
 *                        where a layer has a 256 x 256 weight tile per SM
 *                        pair); =all: averaged in tensor memory on every layer
 *   HS_OVERLAP_UPDATE=0  slab-path updates on the step's stream, not beside the
 *                        remaining products
 *   HS_RELU_BITS=0       bf16: the input-gradient products (MLP; the CNN's
 *                        sub-pixel ones) read ReLU' from the stored activations
 *                        instead of packed bits
 *   HS_CONV_IMPLICIT=0|fwd  bf16 CNN: materialised patch rows everywhere, or
 *                        for the input gradients only
 *   HS_TC_FORM=single    one-SM tensor-core tiles instead of SM pairs (read
 *                        when the library loads)
 *   HS_NARROW_EW=4       256 x 128 SM-pair tiles with four epilogue warps instead
 *                        of two groups of four on alternate tiles
 *   HS_CONV_FIRST=0      bf16 CNN: the first convolution as patch rows plus the
 *                        tiled product instead of its one kernel
 *   HS_SUBPIXEL=classes  bf16 CNN: the stride-2 input gradients as one grouped
 *                        product per sub-pixel class instead of one product
 *                        over the four classes
 *   HS_SUBPIXEL_EW=4|8   bf16 CNN: four or eight epilogue warps on every
 *                        one-product sub-pixel input gradient (default: eight
 *                        where the input has <= 64 channels, else four)
 *   HS_CONV_ABOX=64      bf16 CNN: 64-pixel A boxes instead of 128-pixel ones
 *   HS_KSTAGE=1|2        one k-block per pipeline stage everywhere, or two
 *                        everywhere (read per launch; default: two for the
 *                        forward products, 256 x 128 tiles and convolutions)
 *   HS_CNN_FUSED_UPDATE=0  bf16 CNN: per-worker split-K reductions into the slabs,
 *                        the slab update and the weight permutations as separate
 *                        launches instead of one update kernel (debug read-back
 *                        always takes the separate launches)
 *   HS_CNN_FC_POOL=0     bf16 CNN: the fc layer's logits and input gradient as
 *                        two tensor-core products instead of inside the pooling
 *                        kernels (at most 32 classes)
 *   HS_STEP_GRAPH=0      every hs_step enqueues its kernels one by one (no
 *                        replay of a captured step, see hs_step); =1 replays
 *                        captured steps also above 1e11 parameter-samples */
hs_status hs_init(const hs_model_desc* model, int32_t M, const double* compute_weights,
                  int32_t global_batch, hs_ctx** out);

/* Dynamic Partitioning (Section 4.1, Algorithm 1; Eq. 2).  measured_throughputs:
 * host [M], CP_m = |D_m| / X_m in samples per second measured by the caller over
 * the last epoch (or window); NULL keeps the current partition.  The new sizes
 * follow hs_partition_sizes; the sample->worker map is rebuilt on the device
 * (contiguous segments in worker order) on `stream`.
 * Outputs (each may be NULL): counts_out host [M]; index_map_out device [N]
 * int32 (written on `stream`); out receives the partition view.
 * Errors: HS_ERR_INVALID_ARG (non-finite or <= 0 throughput); nothing changes. */
hs_status hs_partition(hs_ctx* ctx, const double* measured_throughputs, int32_t* counts_out,
                       int32_t* index_map_out, void* stream, hs_partition_t* out);

/* Slab-free formulation of the same step (MLP only; opt-in, off by default).  Every later
 * backward signal is linear in the loss gradient, so scaling sample i's loss gradient by
 * w_{m(i)} / n_{m(i)} instead of 1 / n_{m(i)} makes one weight-gradient product over all N rows
 * equal to sum_m w_m G_m (Eq. 1 with Section 1's / Section 4.2's weights).  No per-worker slabs
 * are written and the update reads one gradient instead of M: same parameters up to rounding
 * order, fewer bytes.  hs_debug_grads then offers g but no slabs (HS_ERR_INVALID_ARG).
 * Errors: HS_ERR_UNSUPPORTED for the CNN. */
hs_status hs_set_fused_sync(hs_ctx* ctx, int32_t enable);

/* Where the compute power handed to Algorithm 1 comes from (Section 4.1: "just the previous
 * epoch or ... a history of epochs").  Each hs_partition call with measured_throughputs c adds c
 * to the history, and the partition is sized from the estimate e:
 *   HS_CP_LAST   e = c (default; param ignored)
 *   HS_CP_EMA    e = param * c + (1 - param) * e_prev, param in (0, 1]; the first c initialises e
 *   HS_CP_WINDOW e = mean of the last `param` measurements (integer in [1, 1024]), summed oldest first
 * fp64 per worker in these operation orders.  Changing the mode clears the history.
 * Errors: HS_ERR_INVALID_ARG for an unknown mode or a parameter out of range. */
typedef enum { HS_CP_LAST = 0, HS_CP_EMA = 1, HS_CP_WINDOW = 2 } hs_cp_history;
hs_status hs_set_cp_history(hs_ctx* ctx, int32_t mode, double param);

/* One synchronous SGD step (Section 1; Eq. 1; Section 4.2 for the weights).
 *   params: device fp32 [P], updated in place: theta <- theta - lr * sum_m w_m G_m,
 *           where G_m is the gradient of worker m's mean cross-entropy over its segment.
 *   x:      fp32 [N, features] (MLP) or [N, Cin, H, W] (CNN, NCHW), row-major.
 *   y:      int32 [N], class labels in [0, classes).
 *           x and y may be device pointers or host pointers (pinned or pageable);
 *           host inputs are copied to a context-owned device buffer on `stream`.
 *   part:   the context's current partition (from hs_init/hs_partition), or NULL
 *           for the same; a stale version is rejected.
 *   loss_out: host float, or NULL.  When non-NULL the call waits for the step and
 *           returns loss = sum_m w_m L_m at the parameters before the update; it
 *           also reports HS_ERR_DEVICE_CHECK if a kernel's bounded wait expired.
 *           When NULL the call is fully asynchronous.
 * Labels outside [0, classes) are clamped by the loss kernel and counted as an
 * error reported through HS_ERR_DEVICE_CHECK at the next synchronising call.
 * CUDA graphs: with device x and y, loss_out NULL and the bf16 shadow current (a previous step
 * or hs_sync_params on the same params), the call only enqueues work on `stream` and may be
 * captured into a graph.  The graph holds this call's pointers, lr and partition plans by value:
 * it stays valid until the next hs_partition, hs_set_* or hs_init/hs_destroy on the context.
 * The library's own graph of the step (contexts of at most 1e11 parameter-samples, P * N, whose
 * step is short enough for its launches to show): once a context has run a step, hs_step captures the step's
 * kernels into a CUDA graph per combination of params, the device x and y it reads (caller's,
 * staging slot or its own copy), momentum state and profiling, keeps the four last used, and
 * replays them, writing lr to device memory with one small kernel first; the kernels and their
 * order are the eager step's, so results are identical.  A call on a stream the caller is
 * capturing is enqueued kernel by kernel.  hs_partition with new sizes, hs_set_debug,
 * hs_set_fused_sync and hs_set_optimizer drop the captured steps; HS_STEP_GRAPH=0 (read by
 * hs_init) keeps every step eager. */
hs_status hs_step(hs_ctx* ctx, float* params, const void* x, const int32_t* y,
                  const hs_partition_t* part, float lr, void* stream, float* loss_out);

/* Double-buffered input staging for a pipelined training loop (an input pipeline; the paper's
 * workers each read their own data shard, Section 1).  Copies one step's x and y (layouts as in
 * hs_step) from host memory into the next of two context-owned device slots, enqueued on
 * `stream` (typically a copy stream other than the step's), after the step that last read that
 * slot has finished with it; returns the slot's device pointers in *x_dev, *y_dev.  hs_step given
 * exactly these pointers makes its own stream wait for the copy, so the copy of step t + 1's
 * inputs overlaps step t.  Pinned host memory makes the copy asynchronous; the host buffers
 * must stay unchanged until the copy has run.
 * Errors: HS_ERR_INVALID_ARG for NULL arguments, or when both slots hold inputs that no hs_step
 * has read yet (at most two staged steps in flight); HS_ERR_OOM on the first use of a slot. */
hs_status hs_stage_inputs(hs_ctx* ctx, const float* x_host, const int32_t* y_host, void* stream,
                          const float** x_dev, const int32_t** y_dev);

/* The training recipe of the paper's experiments (Section 5: SGD with momentum and weight decay)
 * in the fused update.  With d = g + weight_decay * theta (g the synchronised gradient):
 *   b = d on the first step after this call, b = momentum * b + d afterwards, theta <- theta - lr * b.
 * momentum in [0, 1), weight_decay >= 0; both 0 restores plain SGD.  Allocates the momentum buffer
 * (device fp32 [P], one more read and write per parameter per step) on first use and restarts it.
 * Errors: HS_ERR_INVALID_ARG, HS_ERR_OOM. */
hs_status hs_set_optimizer(hs_ctx* ctx, float momentum, float weight_decay);

/* Checkpointing of the momentum buffer: save != 0 copies it to buf_dev (device fp32 [P]); save == 0
 * restores it from buf_dev and the next step continues it (no restart).  Enqueued on `stream`.
 * Errors: HS_ERR_INVALID_ARG without hs_set_optimizer, or when saving a buffer no step started. */
hs_status hs_optimizer_state(hs_ctx* ctx, float* buf_dev, int32_t save, void* stream);

/* Cosine annealing of the learning rate over T steps (Section 5):
 * eta_min + (eta0 - eta_min) * (1 + cos(pi * t / T)) / 2, t clamped to [0, T]; T <= 0 gives eta0.
 * Host only. */
double hs_cosine_lr(double eta0, double eta_min, int64_t t, int64_t T);

/* The bf16 parameter shadow is refreshed by every hs_step for the params
 * pointer it updated.  A caller that writes params in place between steps
 * (checkpoint restore, manual edits) calls this to re-derive the shadow. */
hs_status hs_sync_params(hs_ctx* ctx, const float* params, void* stream);

/* Keep a copy of the synchronised gradient g from each hs_step (costs one
 * extra P x 4 byte write per step).  Off by default. */
hs_status hs_set_debug(hs_ctx* ctx, int32_t enable);

/* Copy the last step's synchronised gradient g (device fp32 [P]; needs
 * hs_set_debug(ctx, 1) before that step, else HS_ERR_INVALID_ARG) and/or the
 * per-worker gradient slabs G_m (device fp32 [M, P], row m = worker m; a bf16
 * MLP step without debug keeps the weight ranges in tensor memory only, so
 * slabs_out then also needs hs_set_debug(ctx, 1) before the step, else
 * HS_ERR_INVALID_ARG).  Either pointer may be NULL.  Copies are enqueued on
 * `stream`. */
hs_status hs_debug_grads(hs_ctx* ctx, float* g_out, float* slabs_out, void* stream);

/* Per-worker losses L_m of the last step (host float [M]); synchronises. */
hs_status hs_worker_losses(hs_ctx* ctx, float* losses_out);

/* Phases of hs_step for device-side timing (CUDA events recorded on the step's stream). */
typedef enum {
  HS_PHASE_CAST = 0,      /* fp32 -> bf16 casts of the inputs (and of params after an external change) */
  HS_PHASE_FORWARD = 1,   /* per-worker forward products, bias + ReLU fused (Eq. 1 f_m) */
  HS_PHASE_LOSS = 2,      /* softmax cross-entropy, loss gradient, per-worker mean losses L_m */
  HS_PHASE_WGRAD = 3,     /* per-worker weight gradients G_m (grouped over the worker segments) */
  HS_PHASE_BIASGRAD = 4,  /* per-worker bias gradients */
  HS_PHASE_DGRAD = 5,     /* input gradients with the ReLU derivative fused */
  HS_PHASE_UPDATE = 6,    /* g = sum_m w_m G_m fused with theta <- theta - lr g (Section 1) */
  HS_PHASE_COUNT = 7
} hs_phase;

/* Record CUDA events around every phase of each hs_step while enabled (adds two event
 * records per phase on the step's stream; off by default). */
hs_status hs_set_profiling(hs_ctx* ctx, int32_t enable);

/* Sum of device time (ms) and kernel launches per phase over the steps since the last read,
 * then reset.  ms_out and launches_out are host [HS_PHASE_COUNT] (either may be NULL).
 * Waits for the recorded events.  Launch counts are kept whether or not profiling is on. */
hs_status hs_read_profile(hs_ctx* ctx, double* ms_out, int64_t* launches_out);

/* The partition of hs_partition and its sample->worker map without a context and without
 * allocating any device memory.  The paper has no counterpart: this is a service for callers
 * that cannot call cudaMalloc - a data-loading process that shares the GPU under a fixed memory
 * budget, or code running under an allocator that forbids new device allocations after start-up -
 * and so cannot create a context (hs_init allocates the whole training workspace).
 *   cp:            host [M] compute powers (as for hs_partition_sizes); M <= 1024, N >= M.
 *   counts_out:    host [M] n_m, or NULL.
 *   index_map_out: device int32 [N], caller-owned: index_map[i] = m for samples of worker m's
 *                  contiguous segment (identical to hs_partition's index_map_out).
 * Device scratch: a static offsets table of 1025 int32 in the library's device image, held by
 * every GPU that loads the library until the process exits.  The first call on a device looks up
 * that table's device address (cudaGetSymbolAddress, with that device current); make that first
 * call before any stream capture.  All calls share the table and it keeps the last call's
 * offsets; calls whose kernels overlap on the GPU (different streams) race on it.
 * `stream` must belong to the current device (the table's address is looked up per device).
 * Each call copies the M + 1 offsets from a host stack array (pageable memory) with
 * cudaMemcpyAsync on `stream`; the runtime stages that copy before the call returns.
 * Errors: HS_ERR_INVALID_ARG for M > 1024, any hs_partition_sizes error, or a stream of another
 * device; HS_ERR_CUDA; the message is returned by hs_last_init_error().  Asynchronous on `stream`. */
hs_status hs_partition_noalloc(int32_t M, int32_t N, const double* cp, int32_t* counts_out,
                               int32_t* index_map_out, void* stream);

/* Free the context and all its device memory (synchronises the device first).
 * NULL is a no-op. */
void hs_destroy(hs_ctx* ctx);

const char* hs_status_string(hs_status s);
/* Last error message of the context ("" if none).  For hs_init failures use
 * hs_last_init_error().  The string is owned by the library. */
const char* hs_last_error(const hs_ctx* ctx);
const char* hs_last_init_error(void);

#ifdef __cplusplus
}
#endif

#endif /* HS_H_ */
