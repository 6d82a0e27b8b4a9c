// Internal launchers of the attention and row-wise kernels.
#pragma once
#include <cuda_runtime.h>

#include "../../include/sky_ops.h"

namespace sky {

sky_status attention_fwd(const void* qkv, const int32_t* lens, int B, int S, int H, int A,
                         sky_dtype dt, void* ctx, float* lse, int32_t* status, cudaStream_t st);
// Scratch of attention_bwd (`delta` below), 16-byte aligned: the per-query
// delta terms and, for bf16, the dK/dV kernel's per-query MMA operand rows.
size_t attention_bwd_ws(int B, int S, int A);
// colpart (bf16 only, optional): column sums of the stored dqkv, one row per
// 128-row tile of each sequence: colpart[b * ceil(S/128) + tile][3H].
sky_status attention_bwd(const void* qkv, const void* ctx, const void* dctx, const float* lse,
                         const int32_t* lens, int B, int S, int H, int A, sky_dtype dt, void* dqkv,
                         float* delta, int32_t* status, cudaStream_t st, float* colpart = nullptr);

// LayerNorm launchers: [rows, H] tensors and gamma, beta 16-byte aligned;
// `status` (optional) receives the timeout bit of the streamed backward's
// bounded waits.
sky_status layernorm_fwd(const float* a, const float* r, const void* gamma, const void* beta,
                         int rows, int H, float eps, sky_dtype dt, float* u_out, float* y32,
                         void* y, float* mean, float* rstd, cudaStream_t st);
size_t layernorm_bwd_ws(int rows, int H);
sky_status layernorm_bwd(const void* dy, sky_dtype dy_dt, const float* dy2, const float* u,
                         const void* gamma, const float* mean, const float* rstd, int rows, int H,
                         sky_dtype dt, float* du32, void* du, float* dgamma, float* dbeta,
                         float* dbias, void* ws, size_t ws_bytes, cudaStream_t st,
                         int* deferred_parts = nullptr, int32_t* status = nullptr);
// With `deferred_parts`, layernorm_bwd leaves dgamma / dbeta / dbias as
// per-CTA partials in `ws` (*deferred_parts rows each) and this call, possibly
// on another stream ordered after it, adds them in a fixed order.
sky_status layernorm_bwd_reduce(const void* ws, int parts, int H, float* dgamma, float* dbeta,
                                float* dbias, cudaStream_t st);
// Fixed-order column sums of several partial matrices in one launch:
// seg[i].out[n] = sum over b < seg[i].rows of seg[i].part[b * cols + n].
// The same partials give the same bits as layernorm_bwd_reduce and
// gemm::reduce_rows_f32.
struct ColSegment {
  const float* part;
  float* out;
  int rows, cols;
};
constexpr int kMaxColSegments = 8;
struct ColSegments {
  ColSegment seg[kMaxColSegments];
  int n;
};
sky_status reduce_column_segments(const ColSegments& segs, cudaStream_t st);
sky_status add_f32(const float* a, const float* b, int64_t n, sky_dtype out_dt, void* out,
                   cudaStream_t st);
sky_status f32_to_bf16(const float* x, int64_t n, void* out, cudaStream_t st);
sky_status to_f32(const void* x, int64_t n, sky_dtype dt, float* out, cudaStream_t st);
size_t column_sum_ws(int rows, int N);
sky_status column_sum(const void* x, int rows, int N, sky_dtype dt, float* out, void* ws,
                      size_t ws_bytes, cudaStream_t st);
sky_status bias_gelu_fwd(const void* z, const void* bias, int rows, int N, sky_dtype dt,
                         void* hpre, void* g, cudaStream_t st);
sky_status gelu_bwd(const void* dg, const void* hpre, int rows, int N, sky_dtype dt, void* dh,
                    cudaStream_t st);

}  // namespace sky
