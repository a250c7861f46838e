/*
 * fedoptima.h — C ABI of the GB300 server-side hot path of FedOptima
 * (arxiv 2504.13850).
 *
 * The server holds ONE copy of the server-side network M_s (theta_s, its
 * momentum and a bf16 shadow used as tensor-core operand), a slab of
 * `omega` activation batch slots in HBM, one FIFO of slot indices per device
 * (Q^act_k), the consumption counters c_k and the global device-model
 * version t.  Devices are not processes here: an upload is a call to
 * fo_enqueue_activations, a model upload is a call to fo_aggregate.
 *
 * Conventions shared by every entry point
 *   - Return value: FO_OK (0) or a positive outcome code (FO_EMPTY,
 *     FO_FULL, FO_STALE) that leaves the server consistent, or a negative
 *     error.  After FO_ERR_CUDA the handle may only be destroyed.
 *   - Pointers named *_host are host memory; pointers documented as
 *     "host or device" may be either (unified addressing decides the copy
 *     direction).  The caller owns every buffer it passes; the library never
 *     keeps a caller pointer beyond the call.
 *   - All GPU work is enqueued on streams the library owns; only
 *     fo_read_losses, fo_server_get_*, fo_server_synchronize and
 *     fo_server_destroy wait for it.
 *   - A handle is not thread safe: one thread drives one server.
 *   - fo_last_error() returns a message for the last failing call on the
 *     calling thread (empty when there is none).
 */
#ifndef FEDOPTIMA_H
#define FEDOPTIMA_H

#include <stdint.h>

#if defined(__GNUC__)
#define FO_API __attribute__((visibility("default")))
#else
#define FO_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ---------------------------------------------------------------- status */
#define FO_OK 0
#define FO_EMPTY 1           /* no queued activation batch: nothing ran          */
#define FO_FULL 2            /* upload refused: cap omega or ring depth reached   */
#define FO_STALE 3           /* local model older than t - D: not aggregated      */
#define FO_ERR_ARG (-1)      /* bad argument; nothing changed                      */
#define FO_ERR_CUDA (-2)     /* CUDA error; the handle is no longer usable         */
#define FO_ERR_OOM (-3)      /* device or host allocation failed                   */
#define FO_ERR_TIMEOUT (-4)  /* a bounded device-side wait gave up                 */
#define FO_ERR_UNSUPPORTED (-5) /* a layer shape this build has no kernel for      */

/* Size limits of the Task Scheduler (both fo_server_create and
 * fo_sched_create return FO_ERR_ARG beyond them). */
#define FO_MAX_DEVICES (1 << 20)  /* K     */
#define FO_MAX_OMEGA (1 << 24)    /* omega */

/* ------------------------------------------------------------ layer spec */
/* Op kinds of the server-side network M_s (Sec. 3.2: M is split at a layer,
 * M_s holds the remaining layers).  Tensor 0 is the uploaded activation
 * batch xi; op i produces tensor i + 1.  Activations are NHWC; a sequence
 * batch [B, L, d] is carried as H = L, W = 1, C = d.  The last op's output
 * is the logits [B, num_classes]; the server loss f_s is softmax
 * cross-entropy averaged over the batch. */
enum {
  FO_OP_CONV = 1,      /* k x k (k = 1 or 3), stride 1|2, pad k/2.  params W[cout][k][k][cin], b[cout] if bias */
  FO_OP_AFFINE = 2,    /* y = x * scale[c] + shift[c] (batch-norm folded).  params scale[c], shift[c]          */
  FO_OP_RELU = 3,
  FO_OP_MAXPOOL2 = 4,  /* 2x2 window, stride 2                                                                  */
  FO_OP_ADD = 5,       /* y = in0 + in1                                                                         */
  FO_OP_AVGPOOL = 6,   /* global mean over H, W -> [B, C]                                                        */
  FO_OP_FLATTEN = 7,   /* [B, H, W, C] -> [B, H*W*C] in (h, w, c) order                                         */
  FO_OP_LINEAR = 8,    /* y = x W^T + b over the last dim.  params W[cout][cin], b[cout] if bias                 */
  FO_OP_LAYERNORM = 9, /* over the last dim, eps 1e-5, biased variance.  params gamma[c], beta[c]               */
  FO_OP_GELU = 10,     /* exact GELU x * Phi(x)                                                                 */
  FO_OP_ATTENTION = 11,/* in0 = [B, L, 3c] packed q|k|v; `heads` heads of c/heads; keys >= length masked          */
  FO_OP_MEANPOOL = 12, /* mean over the first length[b] tokens: [B, L, c] -> [B, c]                              */
  /* MobileNetV3 bottleneck ops (the MobileNetV3-Large split of Table 4):                                       */
  FO_OP_DWCONV = 13,   /* depthwise k x k (k odd, <= 7), stride 1|2, pad k/2, channels cin.  params W[cin][k][k],
                          b[cin] if bias                                                                        */
  FO_OP_HSWISH = 14,   /* hard swish x * relu6(x + 3) / 6; derivative 0 below -3, (2x + 3) / 6 on [-3, 3], 1 above */
  FO_OP_HSIGMOID = 15, /* hard sigmoid relu6(x + 3) / 6; derivative 1/6 strictly inside (-3, 3), else 0          */
  FO_OP_CHMUL = 16     /* squeeze-and-excite scaling y[b,h,w,c] = in0[b,h,w,c] * in1[b,c] (in1 is [B, 1, 1, C])    */
};

typedef struct fo_op {
  int32_t kind;    /* FO_OP_*                                                   */
  int32_t in0;     /* tensor id of the (first) input, 0 <= in0 <= op index     */
  int32_t in1;     /* second input of FO_OP_ADD / FO_OP_CHMUL, else ignored    */
  int32_t cin;     /* conv/linear input channels; channels c of affine,
                      layernorm, attention and the depthwise convolution      */
  int32_t cout;    /* conv/linear output channels                             */
  int32_t k;       /* conv / depthwise conv kernel size                        */
  int32_t stride;  /* conv / depthwise conv stride                             */
  int32_t bias;    /* conv/linear/depthwise conv: 1 if the op has a bias       */
  int32_t heads;   /* attention heads                                           */
} fo_op;

/* Server optimizer: SGD with momentum, v <- mu v + g, theta <- theta - lr v
 * (Algorithm 4 training branch; v starts at 0). */
typedef struct fo_optimizer {
  float lr;
  float momentum;
} fo_optimizer;

enum { FO_DTYPE_F32 = 0, FO_DTYPE_BF16 = 1 };
enum { FO_SCHED_COUNTER = 0, FO_SCHED_FIFO = 1 };

typedef struct fo_server_cfg {
  int32_t num_devices;  /* K                                                                  */
  int32_t omega;        /* global cap on buffered batches, sum_k |Q_k| <= omega (Sec. 3.4.1) */
  int32_t depth;        /* per-device ring depth, |Q_k| <= depth                             */
  int32_t batch;        /* B                                                                  */
  int32_t in_h, in_w, in_c; /* per-sample activation shape (NHWC)                              */
  int32_t num_classes;
  int32_t dtype;        /* FO_DTYPE_*: uploaded activation type and compute path              */
  int32_t seq;          /* 1: each batch carries int32 lengths[B] (attention mask, mean-pool) */
  int32_t max_delay;    /* D of Algorithm 4                                                   */
  int32_t sched_policy; /* FO_SCHED_COUNTER (Algorithm 3) or FO_SCHED_FIFO (arrival order)    */
} fo_server_cfg;

typedef struct fo_server fo_server;

/* Create a server (initialisation stage, Sec. 3.2).  Allocates theta_s,
 * momentum, gradient, bf16 shadow, the omega-slot activation slab (Eq. 3:
 * memory is mu_model + omega * mu_act, independent of K) and all
 * intermediate tensors for one batch.  Parameters start at zero: load them
 * with fo_server_set_params.  Returns FO_ERR_UNSUPPORTED for layer shapes
 * without a kernel (e.g. bf16 conv channels not a multiple of 64), FO_ERR_ARG
 * for K or omega above FO_MAX_DEVICES / FO_MAX_OMEGA, for an op list whose
 * shapes do not chain, or for any tensor of more than 2^31 - 1 elements per
 * sample (all checked on the host before any CUDA call), FO_ERR_OOM when a
 * device or host allocation fails. */
FO_API int fo_server_create(const fo_op* ops, int n_ops, const fo_optimizer* opt,
                     const fo_server_cfg* cfg, fo_server** out);
FO_API int fo_server_destroy(fo_server* s);

/* Number of parameters of M_s, the server-side model of Sec. 3.2 (length of
 * the flat vector below); -1 for a NULL handle. */
FO_API int64_t fo_server_num_params(const fo_server* s);

/* theta_s, the single server model that every training iteration of
 * Algorithm 4 updates whichever device's activations it takes (Sec. 3.3.2),
 * and its SGD momentum.
 * Flat fp32 vectors in op order: conv W[cout][k][k][cin] then b; linear
 * W[cout][cin] then b; affine scale then shift; layernorm gamma then beta.
 * `host` is host memory of n floats owned by the caller; n must equal
 * fo_server_num_params, else FO_ERR_ARG.  set_* also refreshes the bf16
 * shadow; every call waits for pending steps first. */
FO_API int fo_server_set_params(fo_server* s, const float* host, int64_t n);
FO_API int fo_server_get_params(fo_server* s, float* host, int64_t n);
FO_API int fo_server_set_momentum(fo_server* s, const float* host, int64_t n);
FO_API int fo_server_get_momentum(fo_server* s, float* host, int64_t n);

/* Device-resident access, for running a device's network (M_dk and its
 * auxiliary network, Alg. 1) as a second fo_server on the same GPU and
 * feeding its split-point activations and models to the server.
 * fo_server_tensor: device pointer, NHWC dims (dims4[0..3]) and dtype of
 *   tensor `index` -- 1..n_ops is the output of op index-1 -- as written by
 *   the last fo_server_step.  The pointer stays valid for the server's
 *   lifetime; the contents change with each step, which runs on
 *   fo_server_stream.  A flatten of the uploaded batch is a view of it: its
 *   pointer is the batch slot the last step read.  FO_ERR_ARG for an index
 *   outside 1..n_ops.
 * fo_server_params_device: the fp32 master parameters on the device in the
 *   server's padded layout (*n floats; identical for servers built from the
 *   same op list), for device-to-device aggregation.  Read it only when the
 *   server's stream is idle.
 * fo_server_load_params_device: copies n (padded layout) floats from device
 *   memory `src` into the parameters and refreshes the bf16 shadow, ordered
 *   on the server's stream; returns after the copy is issued.
 *   FO_ERR_ARG when n differs from the padded length. */
FO_API int fo_server_tensor(const fo_server* s, int index, const void** data, int64_t* dims4, int* dtype);
FO_API int fo_server_params_device(fo_server* s, float** theta, int64_t* n);
FO_API int fo_server_load_params_device(fo_server* s, const float* src, int64_t n);
/* The reverse copy (Alg. 1: a device pulls the global model): the
 * parameters (padded layout, n floats) into caller-owned device memory
 * `dst`, ordered on the server's stream.  FO_ERR_ARG when n differs from
 * the padded length. */
FO_API int fo_server_store_params_device(fo_server* s, float* dst, int64_t n);

/* Task Scheduler put() for an activation message (Algorithm 2) plus the
 * server-side flow control of Sec. 3.4.1.  `acts` (host or device) holds
 * B*H*W*C elements of the configured dtype, NHWC; `labels` (host or device)
 * int32[B]; `lengths` (host or device) int32[B] when cfg.seq, else NULL.
 * The caller's buffers are copied to the device before the call returns,
 * so it may reuse them: straight into the slot when the slot is idle, else
 * into one of three device staging buffers that move into the slot once
 * the queued step still reading it has finished (the call does not wait for
 * that step).  The server holds omega slots plus these three staging
 * buffers, whatever the number of devices.  *sender_on (may be NULL) receives the
 * device's Sender Status after the call: 1 = "turn-on" was sent.
 * FO_FULL: the cap omega or the ring depth is reached; the device is turned
 * off and, if its queue is empty, waits in a FIFO of blocked devices.
 * FO_ERR_ARG: bad device id or the device has left. */
FO_API int fo_enqueue_activations(fo_server* s, int device_id, const void* acts,
                           const int32_t* labels, const int32_t* lengths,
                           int* sender_on);

/* Task Scheduler get() (Algorithm 3, counter-based: serve argmin_k c_k over
 * non-empty queues, ties to the lowest k, then c_k += 1) followed by one
 * training iteration of Algorithm 4: forward of M_s, loss f_s, backward
 * (no gradient for the uploaded activations), SGD-momentum update of
 * theta_s.  Asynchronous: returns once the kernels are enqueued.
 * *device_used / *slot_used (may be NULL) receive k and the slot index.
 * FO_EMPTY when every queue is empty (nothing changes). */
FO_API int fo_server_step(fo_server* s, int* device_used, int32_t* slot_used);

/* The server loss f_s of training iterations [first_step, first_step + n)
 * of Algorithm 4 (softmax cross-entropy, batch mean), copied to caller-owned
 * host memory of n floats.  Waits for those steps only (work enqueued after
 * them keeps running), so a caller can read step i's loss while step i + 1
 * executes.  Only the most recent 2^20 steps are kept: FO_ERR_ARG for a
 * range not yet run or older than that. */
FO_API int fo_read_losses(fo_server* s, float* host_out, int64_t first_step, int64_t n);

/* FedAsync aggregation (Algorithm 4, aggregation branch).  `global`
 * (device, n floats) is theta_d || theta~_d and is updated in place:
 * global <- alpha * local + (1 - alpha) * global with
 * alpha = 1 / (t - version + 1), computed as fmaf(alpha, local - global,
 * global) in fp32; then t <- t + 1 and *new_version = t.  `local` (device,
 * n floats, read only) is theta_dk || theta~_dk trained from version t_k =
 * `version`.  FO_STALE when t - version > D (global and t unchanged).
 * FO_ERR_ARG when version < 0 or version > t.  Runs on the server's
 * aggregation stream (fo_server_agg_stream), ordered after earlier
 * aggregations but not after the training steps: the two touch disjoint data
 * and overlap on the GPU (fo_server_synchronize waits for both;
 * fo_server_join_aggregations orders the compute stream after the
 * aggregations enqueued so far).  `local` may also be host memory
 * (page-locked for an asynchronous copy): it is then copied into one of two
 * server-owned device buffers on the upload stream, overlapping the steps
 * already queued, and the call returns once that copy has landed, so the
 * caller may reuse its buffer at once; the buffers grow to the largest n
 * seen (FO_ERR_OOM if that fails). */
FO_API int fo_aggregate(fo_server* s, float* global, const float* local, int64_t n,
                 int device_id, int32_t version, int32_t* new_version);

/* Scheduler state, copied to caller-owned host arrays of K entries: the
 * consumption counters c_k of Algorithm 3, and the Sender Status of each
 * device (1 = on, Sec. 3.4.1).  fo_get_version: the global device-model
 * version t of Algorithm 4 and the completed rounds t / K (either pointer
 * may be NULL).  FO_ERR_ARG for a NULL handle or array. */
FO_API int fo_get_counters(const fo_server* s, uint64_t* c_host);
FO_API int fo_get_sender_status(const fo_server* s, uint8_t* on_host);
FO_API int fo_get_version(const fo_server* s, int32_t* t, int32_t* round);
/* Device leaving (active = 0: further uploads are refused, its queued
 * batches are still consumed) or (re)joining (active = 1: c_k becomes
 * max(c_k, min over the other active devices), Sender on) — Sec. 3.4.2. */
FO_API int fo_set_device_active(fo_server* s, int device_id, int active);

/* Bytes of the activation slab, omega slots of acts + labels + lengths: the
 * omega * mu_act term of Eq. 3, independent of K.  -1 for a NULL handle.
 * The helpers from here to fo_server_kernel_times have no counterpart in
 * the paper: they expose memory, streams and timing to the caller. */
FO_API int64_t fo_server_activation_bytes(const fo_server* s);
/* Wait for all work the server has enqueued (uploads, steps,
 * aggregations); no counterpart in the paper.  FO_ERR_CUDA if any of it
 * failed. */
FO_API int fo_server_synchronize(fo_server* s);
/* The compute stream (a cudaStream_t) the step and aggregation kernels run
 * on, for callers that time them with CUDA events; no counterpart in the
 * paper.  NULL for a NULL handle. */
FO_API void* fo_server_stream(const fo_server* s);
/* The aggregation stream (a cudaStream_t) fo_aggregate runs on, for callers
 * that order their work after aggregations; no counterpart in the paper.
 * NULL for a NULL handle. */
FO_API void* fo_server_agg_stream(const fo_server* s);
/* Makes the compute stream wait for every aggregation enqueued so far
 * (asynchronous; an event on the aggregation stream), e.g. before the caller
 * records a timing event on fo_server_stream; no counterpart in the paper.
 * FO_ERR_ARG for a NULL handle. */
FO_API int fo_server_join_aggregations(fo_server* s);
/* Kernel launches the last fo_server_step enqueued, and all kernels the
 * server has launched since creation (steps and aggregations); no
 * counterpart in the paper.  -1 for a NULL handle. */
FO_API int fo_server_last_step_launches(const fo_server* s);
FO_API int64_t fo_server_kernels_launched(const fo_server* s);
/* Device bytes the server allocated (parameters, momentum, gradient, bf16
 * shadow, activation slab, intermediate tensors, scratch): the whole of Eq.
 * 3's mu_model + omega * mu_act plus this implementation's buffers.  -1 for
 * a NULL handle. */
FO_API int64_t fo_server_device_bytes(const fo_server* s);
/* Waits for the compute stream and reports FO_ERR_TIMEOUT if a tensor-core
 * kernel gave up a bounded wait since creation (FO_OK otherwise); no
 * counterpart in the paper. */
FO_API int fo_server_error(fo_server* s);

/* Optional per-kernel timing of fo_server_step and fo_aggregate (no
 * counterpart in the paper): when enabled, each launch is bracketed by CUDA
 * events on the compute stream.
 * fo_server_kernel_times fills up to `cap` entries (any output array may be
 * NULL) with the name (static string), kernel launches, summed milliseconds
 * and summed algorithmic FLOPs and HBM bytes of every kernel class seen since
 * profiling was enabled or reset (waits for the stream); *n_out receives the
 * number of classes. */
FO_API int fo_server_profile(fo_server* s, int enable);
FO_API int fo_server_profile_reset(fo_server* s);
FO_API int fo_server_kernel_times(fo_server* s, const char** names, int64_t* launches,
                           double* ms, double* flops, double* bytes, int cap, int* n_out);

/* The message of the last error returned on the calling thread (empty
 * when there is none; no counterpart in the paper); a buffer valid until the
 * thread's next call into the library. */
FO_API const char* fo_last_error(void);

/* ------------------------------------------------------------------------
 * Host-only Task Scheduler (Algorithms 2-3 and the flow control of Sec.
 * 3.4.1) without any GPU state: the same logic fo_server uses, for trace
 * replay and tests.  put returns the slot the batch would occupy.
 * 1 <= K <= FO_MAX_DEVICES, 1 <= omega <= FO_MAX_OMEGA, depth >= 1 (a depth
 * above omega acts as omega: the cap is reached first).  Create returns
 * FO_ERR_OOM when the host allocation fails.
 * ---------------------------------------------------------------------- */
typedef struct fo_sched fo_sched;
FO_API int fo_sched_create(int K, int omega, int depth, int policy, fo_sched** out);
FO_API int fo_sched_destroy(fo_sched* s);
FO_API int fo_sched_put(fo_sched* s, int k, int32_t* slot, int* sender_on);
FO_API int fo_sched_get(fo_sched* s, int* k, int32_t* slot);
FO_API int fo_sched_set_active(fo_sched* s, int k, int active);
FO_API int fo_sched_counters(const fo_sched* s, uint64_t* c_host);
FO_API int fo_sched_sender_status(const fo_sched* s, uint8_t* on_host);
FO_API int fo_sched_queued(const fo_sched* s, int k); /* |Q_k|, or the total when k < 0 */

/* ------------------------------------------------------------------------
 * Standalone FedAsync update on caller buffers (the arithmetic of Algorithm
 * 4's aggregation branch without its version bookkeeping), for bandwidth
 * sweeps: global <- fmaf(alpha, local - global, global) over n fp32 elements
 * on `stream` (a cudaStream_t, NULL = default).  global (updated in place)
 * and local (read only) are caller-owned device pointers; alpha in (0, 1].
 * FO_ERR_ARG for a NULL pointer, n < 0 or alpha outside (0, 1].
 * ---------------------------------------------------------------------- */
FO_API int fo_axpby_async(float* global, const float* local, int64_t n, float alpha,
                   void* stream);

/* ------------------------------------------------------------------------
 * Deterministic column sums out[c] = sum_r x[r][c] of a row-major
 * [rows][cols] matrix: the reduction the server uses for bias gradients in
 * the backward pass of Algorithm 4 (the sum over all positions of a layer's
 * output gradient).  x is a device
 * pointer to fp32 (dtype FO_DTYPE_F32) or bf16 (FO_DTYPE_BF16) values, out a
 * device pointer to `cols` floats; partial sums over 128-row chunks are added
 * in a fixed order, so results are bitwise reproducible.  The partial sums
 * live in scratch this call allocates and frees stream-ordered on `stream`
 * (a cudaStream_t, NULL = default stream).  FO_ERR_ARG for rows < 1,
 * cols < 1, an unknown dtype, or more than 65,535 chunks of 128 rows
 * (rows > 8,388,480: the chunks are one grid dimension).
 * ---------------------------------------------------------------------- */
FO_API int fo_column_sums(const void* x, int dtype, int64_t rows, int cols, float* out, void* stream);

/* ------------------------------------------------------------------------
 * Pre-processor split selection (Sec. 3.2, "Splitting the DNN", Eqs. 4-6).
 * Host-only; runs once at initialisation.  The model M has L layers; layer
 * l (1-based) costs O[l-1] floating-point operations per training pass on a
 * device and its output is S[l-1] bytes.  Device k has bandwidth b[k]
 * (bytes/s) and compute o[k] (FLOP/s).  Splitting after layer l costs
 * device k t_train = sum_{i<=l} O_i / o_k and t_transfer = S_l / b_k; the
 * chosen split is
 *     l = argmin_l  max_k  max(t_train_k(l), t_transfer_k(l))
 * over the candidate split points: every l in 1..L when `allowed` is NULL,
 * else the l with allowed[l-1] != 0 (split points between sequential layers,
 * never inside a branch).  Ties go to the smallest l.  Writes l to *split and
 * the minimised time (seconds) to *cost.
 * Errors: FO_ERR_ARG for L < 1, K < 1, a null pointer, a negative O or S, a
 * non-positive b or o, or no allowed candidate (the outputs are untouched).
 * ---------------------------------------------------------------------- */
FO_API int fo_select_split(const double* O, const double* S, int L, const double* b, const double* o, int K,
                           const unsigned char* allowed, int* split, double* cost);

/* ------------------------------------------------------------------------
 * fo_column_sums without any allocation.  The paper has no counterpart: it
 * is an interface for callers that cannot allocate device memory when they
 * need the reduction -- code running while its stream is captured into a
 * CUDA graph, processes whose device memory belongs to an outside allocator
 * (a framework's caching allocator or a fixed arena), and loops that must
 * not allocate after start-up.
 *
 * Same arguments, result and determinism as fo_column_sums; the partial
 * sums go to one fixed device array of 262,144 floats (1 MiB) that the
 * library holds on every GPU it is loaded on until the process exits.
 * Limits: ceil(rows / 128) * cols <= 262,144 (e.g. 65,536 rows x 512
 * columns) and ceil(rows / 128) <= 65,535 (as for fo_column_sums); larger
 * inputs return FO_ERR_ARG with the reason in fo_last_error().
 * The first call on a device looks up the array's device address (once per
 * device, with that device current); make that first call before any stream
 * capture.  All calls share the array, and it keeps the last call's
 * contents: calls that can overlap on the GPU (different streams, no
 * ordering between them) race on it, so order them on one stream or with
 * events.  Nothing in the array needs to start at zero.
 * ---------------------------------------------------------------------- */
FO_API int fo_column_sums_noalloc(const void* x, int dtype, int64_t rows, int cols, float* out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* FEDOPTIMA_H */
