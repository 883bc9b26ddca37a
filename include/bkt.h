/*
 * bkt.h -- C ABI of the GB300-native bucketed LSTM-CTC training step.
 *
 * Method: "Accelerating Recurrent Neural Network Training using Sequence
 * Bucketing and Multi-GPU Data Parallelization" (arXiv 1708.05604).
 *   - bkt_plan_buckets: Section III.A (eq. 1-2, the length histogram f and
 *     procedure DYNAMICBUCKETING), Section III.B step 3 (reshuffle every
 *     epoch) and Section IV.A (shorter buckets are fed first).
 *   - bkt_lstm_ctc_step: the training step of Section IV (an LSTM, ref. [1],
 *     trained with the CTC cost, ref. [15]) over one length-bucketed
 *     mini-batch, forward + back-propagation through time, on one GPU.
 *   - bkt_adadelta_update: the paper's parameter update rule, ADADELTA
 *     (Section III.B step 4, ref. [21]); bkt_sgd_update: plain SGD.
 *   - bkt_average_models: the per-epoch model averaging of the paper's
 *     data-parallel training (Section III.B step 5, eq. 3).
 *
 * Conventions
 *   - Every entry point returns an int status (BKT_OK = 0).  On failure
 *     bkt_last_error() returns a message for the calling thread.
 *   - "host" pointers are ordinary CPU memory; "device" pointers are CUDA
 *     global memory of the device current when the ctx was created.  The
 *     caller owns every buffer it passes; the library owns what it creates
 *     (plans, contexts) and frees it in the matching *_free / *_destroy.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy stream).
 *     Device work is enqueued asynchronously on it; device-side errors are
 *     reported by bkt_ctx_sync_status().
 *   - No entry point falls back to the CPU.  Without a usable GPU the calls
 *     that need one return BKT_ECUDA.
 */
#ifndef BKT_H
#define BKT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BKT_OK 0
#define BKT_EINVAL 1   /* bad argument: sizes, NULL pointers, Q > max length */
#define BKT_ENOMEM 2   /* host or device allocation failed */
#define BKT_ECUDA 3    /* a CUDA runtime call failed (message has the name) */
#define BKT_EDEVICE 4  /* a device-side input check failed (label >= classes or == blank) */
#define BKT_ETIMEOUT 5 /* a bounded device-side wait (tensor-core pipeline or recurrent
                          cluster exchange) reached its iteration cap; the kernel left
                          its loop, its results are invalid, the context stays usable */

#define BKT_GEMM_FP32 0 /* fp32 contractions (tensor cores with split-precision 3xTF32 operands) */
#define BKT_GEMM_BF16 1 /* projection, dX and token-axis contractions: bf16 operands, fp32 accumulation */

/* Emission order of an epoch's mini-batches (bkt_plan_buckets_ordered). */
#define BKT_ORDER_ASCENDING 0       /* shortest bucket first (Section IV.A) */
#define BKT_ORDER_DESCENDING 1      /* longest bucket first */
#define BKT_ORDER_SHUFFLE_BUCKETS 2 /* buckets in a seeded random order, each kept together */
#define BKT_ORDER_SHUFFLE_BATCHES 3 /* all mini-batches in a seeded random order */

/* ------------------------------------------------------------------ */
/* Bucketing planner (host only; no GPU needed).                       */

typedef struct bkt_plan bkt_plan; /* opaque, library-owned */

typedef struct bkt_plan_view {
  int32_t n_buckets;            /* Q */
  const int32_t *bounds;        /* [Q] inclusive upper length of each bucket, ascending; bounds[Q-1] = max length */
  int64_t dp_cost;              /* optimal value of eq. 2: sum over sequences of their bucket's bound */
  int64_t n_seqs;               /* n */
  const int32_t *order;         /* [n] sequence ids (0..n-1) in emission order */
  int32_t n_batches;
  const int32_t *batch_off;     /* [n_batches+1] batch k is order[batch_off[k] .. batch_off[k+1]) */
  const int32_t *batch_bucket;  /* [n_batches] bucket index of each batch (non-decreasing for BKT_ORDER_ASCENDING) */
  int64_t padded_timesteps;     /* sum over batches of |batch| * max length in the batch */
  int64_t unpadded_timesteps;   /* sum of all lengths */
} bkt_plan_view;

/* Plans one epoch (Section III.A, procedure DYNAMICBUCKETING, plus Section
 * III.B step 3 and Section IV.A).
 *   lengths  host int32 [n], every entry >= 1.
 *   n_buckets Q >= 1 and Q <= max(lengths); batch >= 1.
 * Steps: histogram f[l] of the lengths (l = 0..max); the dynamic program
 * dp[q][i] = min_j dp[q-1][j] + i * (f[j+1] + ... + f[i]) with the j loop
 * descending and a strict "<" (ties keep the largest j); walk back from
 * i = max length.  Sequence s goes to the first bucket q with
 * lengths[s] <= bounds[q]; each bucket lists its sequences in ascending id,
 * then one SplitMix64 stream with state seed + (epoch+1)*0x9E3779B97F4A7C15
 * shuffles the buckets in ascending order (Fisher-Yates, k = m-1 down to 1,
 * j = next() mod (k+1)).  Buckets are cut into consecutive batches of
 * `batch` (the last one of a bucket may be smaller) and emitted shortest
 * bucket first.  Empty buckets emit no batch.
 * On success *out receives a plan to be released with bkt_plan_free.     */
int bkt_plan_buckets(const int32_t *lengths, int64_t n, int32_t n_buckets,
                     int32_t batch, uint64_t seed, uint64_t epoch,
                     bkt_plan **out);

/* As bkt_plan_buckets, with the batches emitted in `batch_order` (one of
 * BKT_ORDER_*; Section V names bucket-ordering strategies as future work).
 * Bounds, bucket contents, the in-bucket shuffles and the cut into batches
 * are those of bkt_plan_buckets; only the order in which the batches are
 * emitted changes (order[] is rewritten so every batch stays contiguous):
 *   ASCENDING       buckets 0, 1, ..., Q-1 (identical to bkt_plan_buckets);
 *   DESCENDING      buckets Q-1, ..., 0, batches of a bucket in cut order;
 *   SHUFFLE_BUCKETS the bucket sequence permuted by Fisher-Yates over the Q
 *                   bucket indices (k = Q-1 down to 1, j = next() mod (k+1)),
 *                   drawing from the same SplitMix64 stream after the
 *                   in-bucket shuffles; batches of a bucket in cut order;
 *   SHUFFLE_BATCHES the sequence of all batches (in ascending cut order)
 *                   permuted the same way, k = n_batches-1 down to 1.
 * padded_timesteps and dp_cost do not depend on the order.  An unknown
 * batch_order is BKT_EINVAL.                                            */
int bkt_plan_buckets_ordered(const int32_t *lengths, int64_t n, int32_t n_buckets,
                             int32_t batch, uint64_t seed, uint64_t epoch,
                             int32_t batch_order, bkt_plan **out);

/* Fills *view with pointers into the plan (valid until bkt_plan_free). */
int bkt_plan_get(const bkt_plan *plan, bkt_plan_view *view);

void bkt_plan_free(bkt_plan *plan);

/* ------------------------------------------------------------------ */
/* Model and parameters.                                               */

typedef struct bkt_model_cfg {
  int32_t n_layers;       /* >= 1 stacked LSTM layers */
  int32_t bidirectional;  /* 0 or 1; layer l+1 reads [h_forward, h_reverse] */
  int32_t in_dim;         /* features per time step (4 for pen samples) */
  int32_t hidden;         /* H, units per direction */
  int32_t n_classes;      /* C, output classes including the blank */
  int32_t blank;          /* blank class index, 0 <= blank < C */
  int32_t gemm_precision; /* BKT_GEMM_FP32 or BKT_GEMM_BF16 */
} bkt_model_cfg;

/* Number of fp32 parameters.  Flat layout, every block row-major:
 *   for layer l, for direction d (0 forward, 1 reverse):
 *     W_ih [4H x D_l], W_hh [4H x H], b [4H]   (gate row blocks i, f, g, o)
 *   then W_out [C x dirs*H], b_out [C];   D_0 = in_dim, D_l = dirs*H.
 * Returns 0 for an invalid cfg.                                          */
int64_t bkt_param_count(const bkt_model_cfg *cfg);

/* ------------------------------------------------------------------ */
/* Step context: device workspace for batches up to the given sizes.   */

typedef struct bkt_ctx bkt_ctx; /* opaque, library-owned */

/* Allocates the workspace on the current device.
 *   max_tokens     upper bound on the sum of lengths in one batch
 *   max_batch      upper bound on sequences per batch
 *   max_label_len  upper bound on one sequence's label length U          */
int bkt_ctx_create(const bkt_model_cfg *cfg, int64_t max_tokens,
                   int32_t max_batch, int32_t max_label_len, bkt_ctx **out);

void bkt_ctx_destroy(bkt_ctx *ctx);

/* One mini-batch.  Sequence i has lengths[i] >= 1 feature rows starting at
 * row x_offsets[i] of x, and label_lengths[i] >= 0 labels starting at
 * labels[label_offsets[i]].  The batch may be any subset of a resident
 * dataset, in any order.                                                 */
typedef struct bkt_batch {
  int32_t n_seq;
  const int32_t *lengths;       /* host [n_seq] */
  const int64_t *x_offsets;     /* host [n_seq], in rows of in_dim floats */
  const int32_t *label_lengths; /* host [n_seq] */
  const int64_t *label_offsets; /* host [n_seq] */
  const float *x;               /* device, fp32 rows [*, in_dim] */
  const int32_t *labels;        /* device, int32 in 1..C-1 (never the blank) */
} bkt_batch;

/* The training step on one mini-batch (Section IV): packs the batch
 * time-major sorted by length (the active batch shrinks as sequences end;
 * no padded time step is computed), runs the stacked LSTM forward, the
 * output layer + log-softmax, CTC (log-space forward/backward variables),
 * the softmax gradient, and back-propagation through time.
 *   params  device fp32 [bkt_param_count]
 *   grads   device fp32 [bkt_param_count], overwritten with
 *           d(sum_i loss_i)/d(params)
 *   loss    device fp32 [n_seq]: loss[i] = -ln p(labels_i | x_i) of batch
 *           entry i; +inf when the sequence admits no alignment
 *           (lengths[i] < label_lengths[i] + repeated neighbours), which
 *           then adds nothing to grads.
 * Host-side argument checks return BKT_EINVAL before anything is enqueued.
 * Enqueued on `stream`; the call returns before the GPU finishes.        */
int bkt_lstm_ctc_step(bkt_ctx *ctx, const bkt_batch *batch,
                      const float *params, float *grads, float *loss,
                      void *stream);

/* The same training step without a ctx and without allocating anything.
 * The paper has no counterpart: this entry point exists for callers that
 * cannot allocate device memory, such as a plugin running inside a host
 * framework that owns every byte of GPU memory through its own pool, or a
 * process whose memory budget is fixed at start-up and may not grow.
 * Instead of a ctx workspace it uses one device array of
 * BKT_STATIC_SCRATCH_BYTES that is part of the library image; every GPU
 * that loads the library holds that array until the process exits.
 *   - Arguments and results are exactly those of bkt_lstm_ctc_step; the
 *     limits are n_seq <= 512, label_lengths <= 1023, and a workspace that
 *     fits the array (about (26 H + C + 2 S + 8) * 4 bytes per token for one
 *     bidirectional layer, S = 2U + 1: some 4,500 tokens at H = 128).  A batch beyond them returns
 *     BKT_EINVAL with the needed and available bytes in bkt_last_error().
 *   - It cannot be captured into a CUDA graph: on a stream that is being
 *     captured it returns BKT_EINVAL before anything is enqueued (the
 *     index block goes up from one shared pageable buffer, which a replay
 *     would read as it is then).
 *   - The array used is the current device's; a stream of another device
 *     returns BKT_EINVAL before anything is enqueued.
 *   - All calls share the one array, and it keeps the previous call's
 *     contents (the device error flags are cleared at the start of each
 *     call).  Calls whose GPU work overlaps, on different streams or from
 *     different threads, race on it: order them on one stream.
 *   - The host waits for earlier work on `stream` before uploading the
 *     batch's index arrays (they go through pageable host memory).
 *   - There is no status query: a label outside 1..C-1 shows up as a NaN
 *     loss for that sequence, which then adds nothing to grads.          */
#define BKT_STATIC_SCRATCH_BYTES (64u * 1024u * 1024u)
int bkt_lstm_ctc_step_static(const bkt_model_cfg *cfg, const bkt_batch *batch,
                             const float *params, float *grads, float *loss,
                             void *stream);

/* params[i] -= lr * grads[i] for i < n (device fp32 pointers; 16-byte
 * vectors when both are 16-byte aligned), enqueued on `stream`.          */
int bkt_sgd_update(float *params, const float *grads, int64_t n, float lr,
                   void *stream);

/* ADADELTA (Zeiler 2012, the paper's ref. [21], Algorithm 1; the update
 * rule of Section III.B step 4), for i < n:
 *   eg2[i]  = rho * eg2[i] + (1 - rho) * grads[i]^2
 *   dx      = sqrt(edx2[i] + eps) / sqrt(eg2[i] + eps) * grads[i]
 *   edx2[i] = rho * edx2[i] + (1 - rho) * dx^2
 *   params[i] -= lr * dx
 * (Zeiler's rule is lr = 1; the paper names no constants, the usual ones
 * are rho = 0.95, eps = 1e-6.)  All arrays are device fp32 of n entries;
 * eg2 and edx2 are the caller's running averages, zero before the first
 * update, and are updated in place.  IEEE square roots and division; one
 * element per thread, 16-byte vectors when all four arrays are 16-byte
 * aligned.  BKT_EINVAL: n < 0, a NULL array with n > 0, rho outside
 * [0, 1), eps <= 0 or lr < 0.  Enqueued on `stream`.                    */
int bkt_adadelta_update(float *params, const float *grads, float *eg2,
                        float *edx2, int64_t n, float rho, float eps,
                        float lr, void *stream);

/* Model averaging of the data-parallel training loop (Section III.B step
 * 5, eq. 3 with alpha = 1): V(t) = V_alpha(t) - beta V(t-1), V_alpha the
 * mean over the K parallel models of their parameters after the epoch,
 * V(t-1) the parameters the epoch started from (the paper uses
 * beta = 1e-6, a decay proportional to the weights).  Given
 *   v     device fp32 [n]: the element-wise sum of the K models'
 *         parameters, as an all-reduce with the sum operation leaves it on
 *         every replica; overwritten with V(t);
 *   prev  device fp32 [n]: V(t-1);
 * computes v[i] <- v[i] / K - beta prev[i] (IEEE division, then one fused
 * multiply-add), enqueued on `stream`.  BKT_EINVAL: n < 0, n_models < 1,
 * beta < 0 or NaN, or a NULL array with n > 0.                           */
int bkt_average_models(float *v, const float *prev, int64_t n, int32_t n_models,
                       float beta, void *stream);

/* Waits for the work this ctx enqueued, then returns BKT_OK or the
 * device-side errors raised since the previous call, and clears them:
 * BKT_ETIMEOUT when a bounded wait ran out (it takes precedence),
 * otherwise BKT_EDEVICE for a label outside 1..C-1.  The message lists
 * every flag that was set.                                               */
int bkt_ctx_sync_status(bkt_ctx *ctx);

/* Sequences without any CTC alignment (lengths[i] < label_lengths[i] +
 * repeated neighbours; ref. [15]): their loss is +inf and they add nothing
 * to grads, which is not an error.  Waits for the ctx's work, stores in
 * *count how many such sequences the steps of this ctx met since it was
 * created or since the previous call, and resets the counter.           */
int bkt_ctx_infeasible_count(bkt_ctx *ctx, int64_t *count);

/* Failure-detection hooks (off by default; for tests of the bounded waits).
 *   poll_cap  > 0: every bounded device-side wait of this ctx's kernels
 *             gives up after poll_cap polls instead of the built-in cap
 *             (about 4 M polls); values below 256 are raised to 256;
 *             0 restores the built-in caps.
 *   withhold  bit 0 (BKT_WITHHOLD_EXCHANGE): CTA 0 of every recurrent
 *             cluster (H = 256, 512) sends none of its exchange data, so
 *             its peers' waits run out; bit 1 (BKT_WITHHOLD_TMA): the TMA
 *             producer of every tensor-core GEMM skips the loads of its
 *             first k slab, so the MMA issuer's wait runs out.
 * A step run with a withhold bit set ends with BKT_ETIMEOUT from
 * bkt_ctx_sync_status and invalid results; every wait is bounded, so it
 * finishes, and the next step with the hooks off is normal.  BKT_EINVAL
 * for a negative poll_cap or unknown withhold bits.                      */
#define BKT_WITHHOLD_EXCHANGE 1
#define BKT_WITHHOLD_TMA 2
int bkt_ctx_set_wait_faults(bkt_ctx *ctx, int32_t poll_cap, int32_t withhold);

/* ------------------------------------------------------------------ */
/* Per-kernel timing with CUDA events on the launching stream.         */

typedef struct bkt_kernel_time {
  const char *name;  /* static string */
  int64_t launches;
  double total_ms;
  /* Algorithmic work of all those launches, from their shapes:
   *   flops         floating-point operations of the contraction or
   *                 recurrence (2 per multiply-add; a split-precision
   *                 product counts once);
   *   bytes         the minimum DRAM bytes the kernel must move (each
   *                 input read once, each output written once);
   *   serial_steps  sum over launches of the time steps a launch runs one
   *                 after another (recurrent and CTC kernels), else 0.   */
  double flops;
  double bytes;
  int64_t serial_steps;
} bkt_kernel_time;

/* enable != 0: record an event pair around every kernel this ctx launches
 * from now on; 0: stop.  Counters start from zero on enable.             */
int bkt_ctx_set_timing(bkt_ctx *ctx, int32_t enable);

/* Synchronises, folds the recorded events into per-kernel totals and
 * copies up to `cap` entries to out; *n_out = number of kernels seen.    */
int bkt_ctx_kernel_times(bkt_ctx *ctx, bkt_kernel_time *out, int32_t cap,
                         int32_t *n_out);

/* Message for the last failed call on this thread ("" if none). */
const char *bkt_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* BKT_H */
