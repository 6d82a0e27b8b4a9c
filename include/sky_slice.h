/*
 * sky_slice.h -- C ABI of the GB300 encoder-slice library.
 *
 * The paper (Sky Computing, Sec. III and Sec. IV-D) partitions a deep BERT
 * encoder by layer index: device i owns the contiguous layers
 * pi[i] .. pi[i+1]-1, runs their forward pass on the activations it receives
 * from device i-1, and, after the last device has finished, runs the backward
 * pass in reverse order, computing the gradients of its own layers locally.
 * This library is that per-device unit of work on one GPU: a "slice" is the
 * post-LN BERT encoder layers [layer_begin, layer_end), and the calls below
 * create it, run its forward and backward pass, and measure what each of its
 * layers costs (the per-layer time and memory the paper's allocator consumes,
 * Sec. IV-B).
 *
 * One encoder layer (Sec. II-C, Eq. 1), rows of X[T,H] with T = B*S tokens:
 *   QKV = X Wqkv^T + bqkv                         (Wqkv[3H,H]: rows Q | K | V)
 *   ctx = softmax(Q K^T / sqrt(D)) V per sequence b and head a, keys j < len[b]
 *   X1  = LayerNorm(ctx Wo^T + bo + X) * gamma1 + beta1
 *   Y   = LayerNorm(GELU(X1 W1^T + b1) W2^T + b2 + X1) * gamma2 + beta2
 * GELU(z) = z * Phi(z) (exact erf form); LayerNorm uses the biased variance.
 *
 * Conventions for every call:
 *   - Every function returns a sky_status and never aborts or throws across
 *     the ABI.  After a failure, sky_last_error() holds a message (per thread).
 *   - Activations are row-major [B, S, H] in the slice's dtype (bf16 bits or
 *     fp32).  Lengths are int32[B] in device memory.  Padded positions
 *     (s >= len[b]) are computed and returned; as keys they get probability 0.
 *   - Device pointers passed in stay owned by the caller and must stay valid
 *     until the work enqueued on the given stream has finished.
 *   - All GPU work goes on the caller's stream (a cudaStream_t passed as
 *     void*; NULL is the legacy default stream).  No call synchronises except
 *     where stated.
 *   - The library is not thread-safe per handle: calls on one handle must not
 *     overlap.  Distinct handles are independent.
 */
#ifndef SKY_SLICE_H
#define SKY_SLICE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SKY_OK = 0,
  SKY_ERR_INVALID_ARG = 1,  /* bad size, null pointer, length outside [1,S] */
  SKY_ERR_OOM = 2,          /* device memory for the slice does not fit     */
  SKY_ERR_CUDA = 3,         /* a CUDA runtime/driver call failed            */
  SKY_ERR_STATE = 4,        /* e.g. backward without a matching forward     */
  SKY_ERR_TIMEOUT = 5,      /* a bounded device-side wait gave up           */
  SKY_ERR_UNSUPPORTED = 6,  /* valid but not implemented (e.g. D != 64 bf16)*/
  SKY_ERR_INFEASIBLE = 7    /* allocator: no partition fits the memory limits */
} sky_status;

typedef enum { SKY_DTYPE_BF16 = 0, SKY_DTYPE_FP32 = 1 } sky_dtype;

/* Slice description.  layer_begin/layer_end are the partition indices
 * [pi[i], pi[i+1]) of Sec. IV-D; they name global layer indices and only
 * matter for reporting (parameters are set per layer by the caller).
 * max_batch * max_seq sizes the activation stash and workspace, which are
 * allocated once, at create.  bf16 slices need head dim D = width/heads = 64. */
typedef struct {
  int32_t width;        /* H */
  int32_t heads;        /* A, width % heads == 0 */
  int32_t ffn;          /* F */
  int32_t layer_begin;  /* l0 */
  int32_t layer_end;    /* l1 > l0 */
  int32_t max_batch;    /* largest B a forward may use */
  int32_t max_seq;      /* largest S a forward may use */
  sky_dtype dtype;      /* storage type of activations and parameters */
  float ln_eps;         /* LayerNorm epsilon (BERT uses 1e-12) */
  int32_t io_fp32;      /* 1: x, y, dy, dx are fp32 even in a bf16 slice.  Inside a
                           slice the residual and gradient streams are fp32, so with
                           fp32 boundaries a chain of slices [a,b), [b,c) reproduces
                           slice [a,c) bit for bit; with slice-dtype boundaries
                           they agree up to one rounding of the boundary tensor. */
  int32_t stash_slots;  /* activation stashes kept (0 or 1: one).  With M > 1, up to M
                           forwards (sky_slice_forward_slot, slots 0..M-1) may precede
                           their backwards, as the micro-batches of a pipelined step do
                           (Sec. III); the stash memory grows M-fold. */
} sky_slice_config;

/* Per-layer cost record (Sec. IV-B: the model benchmark's per-layer FLOPs
 * lf_j and memory lm_j, and the device's measured time for them). */
typedef struct {
  int32_t layer;              /* global layer index */
  int32_t _pad;
  double fwd_ms, bwd_ms;      /* median measured time of this layer */
  double fwd_flops, bwd_flops;/* algorithmic matmul FLOPs of this layer */
  uint64_t param_bytes;       /* 12 parameter tensors, slice dtype */
  uint64_t grad_bytes;        /* 12 gradient tensors, fp32 */
  uint64_t stash_bytes;       /* activations kept from forward for backward */
  uint64_t workspace_bytes;   /* this layer's share of the shared workspace */
} sky_layer_cost;

/* Per-kernel timing record (profiling, see sky_slice_set_profiling). */
typedef struct {
  char name[32];        /* kernel family, e.g. "gemm", "attn_fwd", "ln_fwd" */
  int64_t launches;     /* launches timed since profiling was enabled */
  double total_ms;      /* sum of CUDA-event durations of those launches */
  double flops;         /* algorithmic FLOPs of those launches (0 if n/a) */
  double bytes;         /* algorithmic HBM bytes of those launches */
} sky_kernel_stat;

typedef struct sky_slice sky_slice;  /* opaque, owned by the library */

/* Order of the 12 per-layer tensors in set/get calls (layouts [out, in]):
 *  0 Wqkv[3H,H] 1 bqkv[3H] 2 Wo[H,H] 3 bo[H] 4 gamma1[H] 5 beta1[H]
 *  6 W1[F,H]    7 b1[F]    8 W2[H,F] 9 b2[H] 10 gamma2[H] 11 beta2[H]   */
#define SKY_NUM_PARAMS 12

/* Creates a slice and allocates its parameters, gradients, stash and
 * workspace on the current CUDA device.  Parameters start at zero.
 * Errors: INVALID_ARG (non-positive sizes, width % heads, l0 >= l1, an
 * unknown dtype, ln_eps < 0, io_fp32 not 0 or 1, stash_slots outside
 * [0, 64], max_batch * max_seq above 2^30), UNSUPPORTED (bf16: head dim != 64, width or ffn not a multiple of
 * 8, width above 2048; fp32: head dim above 128, width above 1024 or not a
 * multiple of 4), OOM (the arena does not fit, or exceeds the cap of
 * sky_debug_set_alloc_cap), CUDA. */
sky_status sky_slice_create(const sky_slice_config* cfg, sky_slice** out);

/* Frees everything the slice owns.  NULL is accepted.  Synchronises the device. */
sky_status sky_slice_destroy(sky_slice* s);

/* Copies the 12 parameter tensors of global layer `layer` into the slice.
 * tensors[k] points to tensor k in the slice dtype (host memory if
 * on_device == 0, device memory otherwise).  Synchronous. */
sky_status sky_slice_set_params(sky_slice* s, int32_t layer, const void* const* tensors,
                                int on_device);

/* Copies the 12 parameter tensors of `layer` out (slice dtype).  Synchronous. */
sky_status sky_slice_get_params(sky_slice* s, int32_t layer, void* const* tensors, int on_device);

/* Copies the 12 fp32 gradient tensors of `layer` (from the last backward)
 * out.  Synchronous; also reports a pending device status (see sky_slice_sync). */
sky_status sky_slice_get_grads(sky_slice* s, int32_t layer, void* const* tensors, int on_device);

/* Forward pass of all layers of the slice: y = layer_{l1-1}(...layer_{l0}(x)).
 * x, y: device [B,S,H] in the boundary dtype (the slice dtype, or fp32 with
 * io_fp32; may not alias); d_len: device
 * int32[B], each in [1,S] (checked on the device: a bad length is clamped,
 * and reported as INVALID_ARG by the next synchronising call).  The stash
 * keeps everything the backward needs, so x may be reused once the forward's
 * work on `stream` is done (a bf16 slice with fp32 boundary tensors reads a
 * 16-byte aligned x in place as the first layer's residual until then).
 * Enqueues work on `stream`; no host synchronisation.
 * Errors: INVALID_ARG (B > max_batch, S > max_seq, B or S < 1, null),
 * UNSUPPORTED (y not 16-byte aligned). */
sky_status sky_slice_forward(sky_slice* s, const void* x, const int32_t* d_len, int32_t B,
                             int32_t S, void* y, void* stream);

/* Backward pass of the slice for the most recent forward: given dy = dL/dy
 * (device [B,S,H], boundary dtype) writes dx = dL/dx and overwrites the fp32
 * gradients of every layer.  Must follow a forward on the same handle (the
 * forward's d_len must still be valid).  Enqueues on `stream`.
 * Errors: STATE (no forward since create), INVALID_ARG (null), UNSUPPORTED
 * (dy not 16-byte aligned). */
sky_status sky_slice_backward(sky_slice* s, const void* dy, void* dx, void* stream);

/* Micro-batched use (Sec. III: a device runs the forward passes of several
 * micro-batches before their backward passes, and its layers' gradients are
 * the sum over the micro-batches).  sky_slice_forward_slot is
 * sky_slice_forward keeping the activations in stash `slot`
 * (0 <= slot < stash_slots); sky_slice_backward_slot is sky_slice_backward
 * for the most recent forward into that slot (its x, d_len, B, S).  With
 * accumulate == 0 the backward overwrites the gradients; with accumulate == 1
 * it adds this micro-batch's gradients to them (each layer's gradients are
 * formed in a scratch set and added on the device, in call order, so a
 * fixed order of calls gives the same bits).  sky_slice_forward /
 * sky_slice_backward are slot 0 without accumulation.  Slots are
 * independent: a forward into slot m leaves the other slots' stashes as
 * they were.  Errors: as the calls they extend; INVALID_ARG (slot out of
 * range, accumulate not 0 or 1), STATE (no forward into the slot),
 * UNSUPPORTED (accumulate == 1 on a slice with stash_slots < 2). */
sky_status sky_slice_forward_slot(sky_slice* s, const void* x, const int32_t* d_len, int32_t B,
                                  int32_t S, void* y, int32_t slot, void* stream);
sky_status sky_slice_backward_slot(sky_slice* s, const void* dy, void* dx, int32_t slot,
                                   int32_t accumulate, void* stream);

/* Emulates a slower device (the slow_down factor of Sec. V-B): enqueues on
 * `stream` one single-thread kernel that returns after `ns` nanoseconds of
 * wall time, so work enqueued behind it on that stream starts that much
 * later while other streams keep the GPU's SMs.  ns <= 10^10, else
 * INVALID_ARG; 0 enqueues nothing. */
sky_status sky_device_delay(uint64_t ns, void* stream);

/* A device's training step over its slice (Sec. III: forward through its
 * layers, then backward in reverse order) as one CUDA graph.
 * sky_slice_step_graph_create runs sky_slice_forward(x, d_len, B, S, y) and
 * sky_slice_backward(dy, dx) once on `stream` (checking every argument as
 * those calls do, and synchronising `stream`), then captures the same two
 * calls on a private stream into an executable graph that the slice owns,
 * replacing any earlier one.  sky_slice_step_graph_launch enqueues that graph
 * on `stream`: the same kernels, in the same order, on the same buffers, so
 * its results equal the two calls' bit for bit.  The graph keeps the pointers
 * and B, S it was created with: the caller refills x, d_len and dy in place
 * between launches and keeps all five buffers alive while the graph exists.
 * Replays on one slice must not overlap each other or direct calls on that
 * slice (they share its stash and workspace).  Launches are counted in
 * sky_launch_count at every replay.  With per-kernel timing on at create
 * (sky_slice_set_profiling), every kernel runs in line on one stream with a
 * pair of CUDA events around it captured into the graph; each launch of such
 * a graph then synchronises `stream` and adds the replay's per-kernel times
 * to the records of sky_slice_kernel_stats (kernel times without host launch
 * gaps).  The graph is freed by the next create and by sky_slice_destroy.
 * Errors: those of sky_slice_forward / sky_slice_backward; STATE if no graph
 * exists (launch); CUDA if the capture or instantiation fails. */
sky_status sky_slice_step_graph_create(sky_slice* s, const void* x, const int32_t* d_len,
                                       int32_t B, int32_t S, void* y, const void* dy, void* dx,
                                       void* stream);
sky_status sky_slice_step_graph_launch(sky_slice* s, void* stream);

/* Measures every layer of the slice (the per-layer benchmark of Sec. IV-B):
 * on a fixed input pattern written on the device (parameters as set), runs
 * 2 forward+backward passes at [B,S] directly, then captures one pass with a
 * CUDA event around each layer into a CUDA graph on a stream of its own and
 * replays it 1 + `iters` times (as a step is replayed), and writes the
 * median per-layer times of the last `iters` replays with the analytic FLOPs
 * and the byte counts.
 * lens: host int32[B], the valid length of every sequence (each in [1,S]),
 * so that a workload's own padding mask is measured; NULL measures
 * full-length sequences.  fwd_flops / bwd_flops count attention over those
 * lengths.  The layers are timed inside whole forward + backward passes, as a
 * step runs them: a layer's weight gradients, which run on a second stream,
 * overlap the next layer's interval, and the slice's first layer takes the
 * final join, so the per-layer times add up to the passes' time.  Before it
 * starts, the call waits for all work already enqueued on
 * this slice (its last stream and its weight-gradient stream), because the
 * measurement reuses the slice's stash and workspace.  It allocates its
 * input, output and length buffers (cudaMalloc) and a stream, and frees them
 * and its graph on every return path.  n_out must equal layer_end - layer_begin.
 * Synchronous; overwrites grads, and a following sky_slice_backward needs a
 * new forward (STATE).  Errors: INVALID_ARG (null out, n_out, B or S outside
 * [1, max], iters < 1, a length outside [1,S]), OOM / CUDA (buffers). */
sky_status sky_slice_layer_cost(sky_slice* s, int32_t B, int32_t S, const int32_t* lens,
                                int32_t iters, sky_layer_cost* out, int32_t n_out);

/* Waits for the slice's enqueued work and reports device-side status:
 * INVALID_ARG if a length was outside [1,S], TIMEOUT if a bounded wait gave
 * up, CUDA on an asynchronous CUDA error.  Clears the status word. */
sky_status sky_slice_sync(sky_slice* s);

/* Enables (1) or disables (0) per-kernel CUDA-event timing of the slice's
 * launches; enabling resets the counters. */
sky_status sky_slice_set_profiling(sky_slice* s, int enable);

/* Reads the per-kernel records accumulated while profiling was on
 * (synchronises).  Writes at most n_out records and the count to *n_written. */
sky_status sky_slice_kernel_stats(sky_slice* s, sky_kernel_stat* out, int32_t n_out,
                                  int32_t* n_written);

/* Bytes the slice allocated at create (parameters, grads, stash, workspace). */
sky_status sky_slice_memory(const sky_slice* s, uint64_t* param_bytes, uint64_t* grad_bytes,
                            uint64_t* stash_bytes, uint64_t* workspace_bytes);

/* ---- Local parameter update (Sec. III) ------------------------------------
 * After its backward pass a device updates the weights of its own layers with
 * the gradients it computed (Sec. III); nothing is sent anywhere.  The paper
 * names no optimizer; two rules are provided:
 *   ADAMW: Adam with bias-corrected moments and decoupled weight decay
 *          (w <- w - lr wd w; w <- w - lr m_hat / (sqrt(v_hat) + eps)),
 *   SGD:   heavy-ball momentum with the decay added to the gradient
 *          (b <- momentum b + g + wd w; w <- w - lr b).
 * Weight decay applies to Wqkv, Wo, W1 and W2 only (BERT's choice), not to
 * biases or LayerNorm parameters.  Updates run on fp32 master weights; a bf16
 * slice's parameters are the master weights rounded to nearest bf16 after
 * every step. */
typedef enum { SKY_OPT_SGD = 0, SKY_OPT_ADAMW = 1 } sky_optimizer_kind;
typedef struct {
  int32_t kind;        /* sky_optimizer_kind                         */
  float lr;            /* learning rate (sky_slice_optimizer_step may override) */
  float beta1, beta2;  /* ADAMW moment decay rates, in [0, 1)        */
  float eps;           /* ADAMW denominator term, > 0                */
  float weight_decay;  /* >= 0                                       */
  float momentum;      /* SGD, in [0, 1)                             */
} sky_optimizer_config;

/* Allocates the fp32 master weights (copied from the current parameters) and
 * zeroed optimizer state (AdamW: 2, SGD: 1 fp32 copy of every parameter; a
 * bf16 slice also keeps the master copy) and resets the step count.  Calling
 * it again re-initialises.  Synchronises the device; the memory is freed by
 * sky_slice_destroy.  Errors: INVALID_ARG for a bad config, OOM, UNSUPPORTED
 * when a parameter tensor's size is not a multiple of 4. */
sky_status sky_slice_optimizer_init(sky_slice* s, const sky_optimizer_config* cfg);

/* One update of every parameter from the gradients of the most recent
 * sky_slice_backward, with learning rate `lr` (a schedule is the caller's),
 * enqueued on `stream`.  The slice's parameters are rewritten.  STATE if the
 * optimizer is not initialised. */
sky_status sky_slice_optimizer_step(sky_slice* s, float lr, void* stream);

/* Host copies of one layer's fp32 optimizer tensors, 12 in parameter order:
 * which = 0 master weights, 1 first state (AdamW m, SGD momentum),
 * 2 second state (AdamW v).  Synchronises. */
sky_status sky_slice_get_optimizer_state(sky_slice* s, int32_t layer, int32_t which,
                                         void* const* dst);

/* Host-side cap (bytes) on what sky_slice_create may allocate; 0 = no cap.
 * Lets the out-of-memory path be tested without exhausting a device. */
void sky_debug_set_alloc_cap(uint64_t bytes);

/* Total number of kernels the library has launched in this process (all
 * handles and threads), for accounting of GPU work. */
int64_t sky_launch_count(void);

/* Name of a status code ("SKY_OK", "SKY_ERR_INVALID_ARG", ...), a static
 * string owned by the library; an unknown code gives "SKY_ERR_UNKNOWN". */
const char* sky_status_string(sky_status st);

/* Message of the calling thread's most recent failed call (empty before the
 * first failure; a successful call leaves it unchanged).  The string belongs
 * to the library and stays valid until that thread's next failing call. */
const char* sky_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* SKY_SLICE_H */
