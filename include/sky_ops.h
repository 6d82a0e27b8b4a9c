/*
 * sky_ops.h -- kernel-level C ABI of the encoder-slice library.
 *
 * These are the individual steps of one encoder layer's forward and backward
 * pass (Sec. II-C, Eq. 1; backward in reverse order, Sec. III) exposed one by
 * one, on caller-owned device buffers, so each kernel can be checked and
 * timed on its own.  sky_slice_forward/backward (sky_slice.h) run the same
 * kernels in sequence.
 *
 * Common rules:
 *   - All pointers are device pointers owned by the caller; nothing here
 *     allocates or frees device memory.  Scratch ("workspace") buffers are
 *     passed in, sized by the matching *_workspace_bytes query; their
 *     contents on entry do not matter.
 *   - Matrices are row-major.  "bf16" means bfloat16 bit patterns, "fp32"
 *     IEEE single; the dtype argument selects the storage type of the
 *     activation operands (the tensor-core path is bf16 only; fp32 runs the
 *     exact-fp32 SIMT path used for the tight-tolerance configuration).
 *   - All work is enqueued on `stream`; nothing synchronises.
 *   - Errors: INVALID_ARG for null pointers or non-positive sizes,
 *     UNSUPPORTED for shapes a kernel does not handle (listed per call),
 *     CUDA if a launch fails.  Device-side conditions (bad lengths, timed-out
 *     waits) are written to the int32 status word `d_status` if non-null:
 *     bit 0 = a length outside [1,S] was clamped, bit 1 = a wait timed out.
 */
#ifndef SKY_OPS_H
#define SKY_OPS_H

#include <stddef.h>
#include <stdint.h>

#include "sky_slice.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Contraction forms of the layer's linear maps and their gradients.
 *   XWT: C[M,N] = A[M,K] * B[N,K]^T   forward  (x W^T: activations x weights)
 *   XW : C[M,N] = A[M,K] * B[K,N]     dgrad    (dy W)
 *   XTW: C[M,N] = A[K,M]^T * B[K,N]   wgrad    (dy^T x), K = tokens        */
typedef enum { SKY_GEMM_XWT = 0, SKY_GEMM_XW = 1, SKY_GEMM_XTW = 2 } sky_gemm_form;

/* Epilogues applied to the fp32 accumulator before the store.
 *   STORE     : C = acc (+ bias[n] if bias != NULL)
 *   BIAS_GELU : z = acc + bias[n]; C = GELU(z), aux_out = GELU'(z) -- the
 *               derivative the backward pass needs, stored as IEEE fp16 for
 *               bf16 inputs (finer than bf16 on its range [-0.17, 1.13]) and
 *               as fp32 for fp32 inputs
 *   GELU_BWD  : C = acc * aux[m,n], aux = GELU'(z) as stored by BIAS_GELU
 * sky_gemm takes no residual operand: with the ops of this header the
 * residual is added by sky_layernorm_fwd (its r operand).  The slice
 * (sky_slice.h) adds its residuals inside its own GEMM epilogues. */
typedef enum { SKY_EPI_STORE = 0, SKY_EPI_BIAS_GELU = 1, SKY_EPI_GELU_BWD = 2 } sky_epilogue;

/* Scratch bytes sky_gemm needs for (form, M, N, K) with an fp32 output
 * (deterministic split-K partials); 0 otherwise. */
size_t sky_gemm_workspace_bytes(sky_gemm_form form, int32_t M, int32_t N, int32_t K,
                                sky_dtype in_dtype, sky_dtype out_dtype);

/* C = epilogue(op(A) * op(B)) with fp32 accumulation (Sec. II-C linear
 * layers).  in_dtype: BF16 runs the tcgen05/TMEM tensor-core kernel (the
 * contiguous dimensions -- K for XWT/XW, M for XTW, and N -- multiples of 8,
 * A, B, C 16-byte aligned, else UNSUPPORTED); FP32 runs the SIMT kernel.
 * out_dtype: the storage type of C (BF16 only with BF16 input); an FP32
 * output takes the STORE epilogue (with or without bias).  bias uses
 * in_dtype.  An FP32 output with no bias may split the K range over CTAs; the
 * partial sums go to `workspace` and are added in a fixed order
 * (deterministic). */
sky_status sky_gemm(sky_gemm_form form, int32_t M, int32_t N, int32_t K, sky_dtype in_dtype,
                    const void* A, const void* B, void* C, sky_dtype out_dtype,
                    sky_epilogue epilogue, const void* bias, const void* aux, void* aux_out,
                    void* workspace, size_t workspace_bytes, int32_t* d_status, void* stream);

/* Masked scaled dot-product attention, forward (Eq. 1).
 * qkv: [B*S, 3H] (Q | K | V blocks, head a at columns a*D..a*D+D-1 in each);
 * d_len: int32[B] valid lengths; ctx: [B*S, H] out; lse: fp32 [B, A, S] out,
 * the softmax normaliser of each query row in base-2 units,
 * log2 sum_{j < len} exp2(log2(e) q.k_j / sqrt(D)) (kept for the backward,
 * which takes it in the same units).
 * bf16 needs D = H/A = 64. */
sky_status sky_attention_fwd(const void* qkv, const int32_t* d_len, int32_t B, int32_t S,
                             int32_t H, int32_t A, sky_dtype dtype, void* ctx, float* lse,
                             int32_t* d_status, void* stream);

/* Scratch bytes of sky_attention_bwd: the per-row terms dot(dctx, ctx) and,
 * for bf16, 32 bytes per (row, head) of per-query MMA operand rows.  The
 * workspace must be 16-byte aligned. */
size_t sky_attention_bwd_workspace_bytes(int32_t B, int32_t S, int32_t H, int32_t A);

/* Attention backward: from dctx [B*S, H] and the forward's qkv, ctx and lse,
 * writes dqkv [B*S, 3H] (dQ | dK | dV; rows of padded keys get zero dK, dV). */
sky_status sky_attention_bwd(const void* qkv, const void* ctx, const void* dctx,
                             const float* lse, const int32_t* d_len, int32_t B, int32_t S,
                             int32_t H, int32_t A, sky_dtype dtype, void* dqkv,
                             void* workspace, size_t workspace_bytes, int32_t* d_status,
                             void* stream);

/* Residual + LayerNorm forward (post-LN placement): u = a + r with a the
 * linear layer's fp32 output and r the fp32 residual stream (r may be NULL);
 * y = gamma * (u - mean) * rstd + beta, rstd = 1/sqrt(var + eps), biased
 * variance.  Writes u to u_out (may alias a, or NULL), y to y32 (fp32) and/or
 * y (dtype) -- either may be NULL but not both; gamma, beta: [H] (dtype);
 * mean, rstd: fp32 [T].  H % 8 == 0, H <= 2048 (bf16) or 1024 (fp32).  The
 * [T, H] tensors and gamma, beta must be 16-byte aligned (else UNSUPPORTED). */
sky_status sky_layernorm_fwd(const float* a, const float* r, const void* gamma,
                             const void* beta, int32_t T, int32_t H, float eps, sky_dtype dtype,
                             float* u_out, float* y32, void* y, float* mean, float* rstd,
                             void* stream);

/* Scratch bytes of sky_layernorm_bwd (per-block column partial sums). */
size_t sky_layernorm_bwd_workspace_bytes(int32_t T, int32_t H);

/* LayerNorm backward.  The upstream gradient is dy + dy2 with dy: [T, H] in
 * dy_dtype (FP32 or the slice dtype) and dy2: fp32 [T, H] or NULL (the two
 * contributions meeting at a residual branch point); u, mean, rstd as saved
 * by the forward.  With xhat = (u - mean) * rstd and g = (dy + dy2) * gamma
 * writes du = rstd * (g - mean(g) - xhat * mean(g * xhat)) to du32 (fp32)
 * and/or du (dtype), and the fp32 column sums dgamma = sum dy*xhat,
 * dbeta = sum dy, dbias = sum du (each [H]; any may be NULL), which are
 * deterministic (fixed-order partials in `workspace`).  The [T, H] tensors
 * and gamma must be 16-byte aligned (else UNSUPPORTED). */
sky_status sky_layernorm_bwd(const void* dy, sky_dtype dy_dtype, const float* dy2,
                             const float* u, const void* gamma, const float* mean,
                             const float* rstd, int32_t T, int32_t H, sky_dtype dtype,
                             float* du32, void* du, float* dgamma, float* dbeta, float* dbias,
                             void* workspace, size_t workspace_bytes, void* stream);

/* out = a + b for fp32 a, b [n]; out in out_dtype (the slice's input
 * gradient is the sum of its two branch terms). */
sky_status sky_add_f32(const float* a, const float* b, int64_t n, sky_dtype out_dtype, void* out,
                       void* stream);

/* Widens x [n] (dtype) to fp32: the slice's residual stream is fp32. */
sky_status sky_to_f32(const void* x, int64_t n, sky_dtype dtype, float* out, void* stream);

/* Bias + GELU forward: hpre = z + bias[n], g = hpre * Phi(hpre).  [T, N]. */
sky_status sky_bias_gelu_fwd(const void* z, const void* bias, int32_t T, int32_t N,
                             sky_dtype dtype, void* hpre, void* g, void* stream);

/* GELU backward: dh = dg * (Phi(h) + h * phi(h)), h = hpre.  [T, N]. */
sky_status sky_gelu_bwd(const void* dg, const void* hpre, int32_t T, int32_t N,
                        sky_dtype dtype, void* dh, void* stream);

/* Scratch bytes of sky_column_sum. */
size_t sky_column_sum_workspace_bytes(int32_t T, int32_t N);

/* out[n] = sum over rows t of x[t, n] (fp32, fixed summation order):
 * the bias gradients.  x: [T, N] dtype. */
sky_status sky_column_sum(const void* x, int32_t T, int32_t N, sky_dtype dtype, float* out,
                          void* workspace, size_t workspace_bytes, void* stream);

/* sky_column_sum without any device allocation, for callers that cannot
 * allocate: code that takes all device memory from a fixed pool it does not
 * own (a framework's caching allocator, a pre-sized arena) must not call
 * cudaMalloc around it, and code that must not allocate inside its step loop
 * cannot supply a fresh workspace per call.  (The paper has no counterpart;
 * this is a library-usability variant of the bias-gradient reduction.)
 * Same arguments and result as sky_column_sum minus the workspace: the
 * partial sums live in a 1 MiB device array inside the library, which every
 * device that loads the library holds until the process exits.
 *   - Every call looks up that array's device address on the current
 *     device (cudaGetSymbolAddress, which enqueues no work); the first call
 *     on a device also loads the library's module there, so make that first
 *     call before capturing the stream into a CUDA graph.  A device reset
 *     discards the array's contents with the module; the next call finds
 *     the new address.
 *   - All calls share the array and it keeps the previous call's contents;
 *     nothing in it needs to start at zero, but calls that may overlap on
 *     the GPU (different streams, or different host threads, same device)
 *     race on it and must be serialised by the caller.
 *   - Sizes whose partials exceed 1 MiB are rejected with INVALID_ARG (on a
 *     152-SM GB300 that is N > 262144, for any T); use sky_column_sum then. */
sky_status sky_column_sum_noalloc(const void* x, int32_t T, int32_t N, sky_dtype dtype,
                                  float* out, void* stream);

/* Test hook of the tensor-core GEMM's failure path (not for production use).
 * limit_ns caps every mbarrier wait of GEMM launches made after the call
 * (0 restores the default, 2 s).  skip_loads != 0 makes the TMA producer
 * arrive on its barriers without issuing the copies, so the consumers' waits
 * run out: the kernel then sets the timeout bit (2) of the status word it was
 * given, frees its tensor memory and exits, and the context stays usable.
 * Process-wide setting; pass (0, 0) to restore normal operation. */
void sky_debug_gemm_fault(uint64_t limit_ns, int32_t skip_loads);

/* Number of streaming multiprocessors of the current device (0 on error). */
int32_t sky_device_sm_count(void);

#ifdef __cplusplus
}
#endif
#endif /* SKY_OPS_H */
