// Internal GEMM launchers (bf16 tensor-core and fp32 SIMT).
#pragma once
#include <cuda_runtime.h>

#include "../../include/sky_ops.h"

namespace sky {
namespace gemm {

// bf16 inputs on tcgen05; C is bf16 unless out_f32.
// colsum (optional, bf16 output, no split): also writes out[n] = sum_m C[m, n]
// (before rounding), with fixed-order partials (one row per 32 rows of C) in
// `ws`.  With `deferred_rows`, the partials go to `colpart` instead, no sum is
// launched and *deferred_rows reports their row count (for reduce_rows_f32,
// possibly on another stream ordered after this launch).
// resid (optional, fp32 output of the STORE epilogue, no split): C = acc +
// bias + resid[m, n], added in that order (the residual branch of Sec. II-C).
// With `ln`, resid holds the pre-LayerNorm sum u of the previous sub-layer and
// the residual added is its LayerNorm output, recomputed in the epilogue from
// the row statistics: gamma[n] * ((u[m, n] - mean[m]) * rstd[m]) + beta[n]
// (Eq. 3; the same expression the LayerNorm forward evaluates, so the sum is
// the one an fp32 copy of the LayerNorm output would give).
struct LnResid {
  const float* mean;  // [M]
  const float* rstd;  // [M]
  const void* gamma;  // [N] bf16
  const void* beta;   // [N] bf16
};
sky_status launch_bf16(sky_gemm_form form, int M, int N, int K, const void* A, const void* B,
                       void* C, bool out_f32, int epi, const void* bias, const void* aux,
                       void* aux_out, void* ws, size_t ws_bytes, int32_t* status,
                       cudaStream_t stream, float* colsum = nullptr, float* colpart = nullptr,
                       size_t colpart_bytes = 0, int* deferred_rows = nullptr,
                       const float* resid = nullptr, const LnResid* ln = nullptr);
// Rows of column partials a bf16 GEMM with M rows writes (upper bound).
int colpart_rows_max(int M);
// out[n] = sum over r of part[r][n] in order r = 0, 1, ... (rowwise.cu).
cudaError_t reduce_rows_f32(const float* part, int rows, int N, float* out, cudaStream_t stream);
size_t workspace_bytes(sky_gemm_form form, int M, int N, int K, bool out_f32);
int choose_splits(int tiles, int k_blocks, int sms);
// Debug controls: per-wait timeout (0 = default 2 s) and the fault-injection
// switch that makes the TMA producer skip its loads (waits then time out).
void set_debug(uint64_t timeout_ns, int skip_loads);

// fp32 SIMT path (exact fp32 FMA accumulation); same forms and epilogues.
sky_status launch_f32(sky_gemm_form form, int M, int N, int K, const float* A, const float* B,
                      float* C, int epi, const float* bias, const float* aux, float* aux_out,
                      cudaStream_t stream);

}  // namespace gemm
}  // namespace sky
