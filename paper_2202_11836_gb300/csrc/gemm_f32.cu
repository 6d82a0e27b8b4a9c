// fp32 SIMT GEMM: exact fp32 FMA accumulation for the tight-tolerance fp32
// slice (tensor-core TF32 would not reach a 1e-4 relative error).  Same
// three contraction forms and epilogues as the bf16 tensor-core kernel.
#include "common.cuh"
#include "gemm.h"

namespace sky {
namespace gemm {

namespace {
constexpr int TM = 64, TN = 64, TK = 16;

// A(m,k) = A[m*am + k*ak], B(k,n) = B[k*bk + n*bn]
__global__ void __launch_bounds__(256) gemm_f32_kernel(int M, int N, int K, const float* A,
                                                       int64_t am, int64_t ak, const float* B,
                                                       int64_t bk, int64_t bn, float* C, int epi,
                                                       const float* bias, const float* aux,
                                                       float* aux_out) {
  __shared__ float sA[TK][TM + 1];
  __shared__ float sB[TK][TN + 1];
  const int m0 = blockIdx.y * TM, n0 = blockIdx.x * TN;
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int i = threadIdx.x; i < TK * TM; i += 256) {
      const int kk = i / TM, mm = i % TM;
      const int m = m0 + mm, k = k0 + kk;
      sA[kk][mm] = (m < M && k < K) ? A[m * am + k * ak] : 0.f;
    }
    for (int i = threadIdx.x; i < TK * TN; i += 256) {
      const int kk = i / TN, nn = i % TN;
      const int n = n0 + nn, k = k0 + kk;
      sB[kk][nn] = (n < N && k < K) ? B[k * bk + n * bn] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = sA[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = sB[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty + 16 * i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx + 16 * j;
      if (n >= N) continue;
      const int64_t off = static_cast<int64_t>(m) * N + n;
      float v = acc[i][j];
      if (bias) v += bias[n];
      if (epi == SKY_EPI_GELU_BWD) v *= aux[off];
      if (epi == SKY_EPI_BIAS_GELU) {
        aux_out[off] = gelu_grad_f(v);
        v = gelu_f(v);
      }
      C[off] = v;
    }
  }
}
}  // namespace

sky_status launch_f32(sky_gemm_form form, int M, int N, int K, const float* A, const float* B,
                      float* C, int epi, const float* bias, const float* aux, float* aux_out,
                      cudaStream_t stream) {
  SKY_CHECK(epi != SKY_EPI_BIAS_GELU || (bias && aux_out), SKY_ERR_INVALID_ARG,
            "BIAS_GELU epilogue needs bias and aux_out");
  SKY_CHECK(epi == SKY_EPI_STORE || epi == SKY_EPI_BIAS_GELU || epi == SKY_EPI_GELU_BWD,
            SKY_ERR_INVALID_ARG, "unknown epilogue %d", epi);
  SKY_CHECK(epi != SKY_EPI_GELU_BWD || aux, SKY_ERR_INVALID_ARG, "GELU' epilogue needs aux");
  int64_t am, ak, bk, bn;
  switch (form) {
    case SKY_GEMM_XWT: am = K; ak = 1; bk = 1; bn = K; break;   // A[M,K], B[N,K]
    case SKY_GEMM_XW: am = K; ak = 1; bk = N; bn = 1; break;    // A[M,K], B[K,N]
    default: am = 1; ak = M; bk = N; bn = 1; break;             // A[K,M], B[K,N]
  }
  dim3 grid(ceil_div(N, TN), ceil_div(M, TM));
  gemm_f32_kernel<<<grid, 256, 0, stream>>>(M, N, K, A, am, ak, B, bk, bn, C, epi, bias, aux,
                                            aux_out);
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "gemm_f32_kernel launch");
}

}  // namespace gemm
}  // namespace sky
