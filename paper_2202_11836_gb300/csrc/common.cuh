// Shared host/device helpers of the encoder-slice library.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <cstdio>
#include <string>

#include "../../include/sky_ops.h"
#include "../../include/sky_slice.h"

namespace sky {

// Device status word bits (sky_ops.h: d_status).
constexpr int32_t kStatusBadLength = 1;
constexpr int32_t kStatusTimeout = 2;

// Records the thread-local error message returned by sky_last_error().
void set_error(const char* fmt, ...);
sky_status cuda_fail(cudaError_t e, const char* what);

#define SKY_CUDA(call)                                        \
  do {                                                        \
    cudaError_t e_ = (call);                                  \
    if (e_ != cudaSuccess) return ::sky::cuda_fail(e_, #call); \
  } while (0)

#define SKY_CHECK(cond, status, ...)   \
  do {                                 \
    if (!(cond)) {                     \
      ::sky::set_error(__VA_ARGS__);   \
      return (status);                 \
    }                                  \
  } while (0)

// bf16 <-> fp32 conversions usable for both storage types.
template <typename T> __device__ __forceinline__ float to_f32(T v);
template <> __device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) {
  return __bfloat162float(v);
}
template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

// GELU(h) = h * Phi(h) and its derivative Phi(h) + h * phi(h), with
// Phi(h) = (1 + erf(h / sqrt 2)) / 2 from CUDA's erff and phi from expf
// (exact-erf form, no tanh approximation).
__device__ __forceinline__ float std_normal_cdf(float h) {
  return 0.5f * (1.f + erff(h * 0.70710678118654752f));
}
__device__ __forceinline__ float gelu_f(float h) { return h * std_normal_cdf(h); }
__device__ __forceinline__ float gelu_grad_f(float h) {
  const float inv_sqrt_2pi = 0.3989422804014327f;
  return std_normal_cdf(h) + h * inv_sqrt_2pi * expf(-0.5f * h * h);
}

// GELU(h) and GELU'(h) together, for the tensor-core epilogues: Phi from the
// erf approximation of Abramowitz & Stegun, Handbook of Mathematical
// Functions, formula 7.1.25 (|erf error| <= 2.5e-5 for all x: well below the
// bf16 rounding of GELU and the fp16 rounding of GELU'), written for
// x = |h| / sqrt 2 so that Phi and phi share one exponential exp(-h^2 / 2):
//   t = 1 / (1 + p x),  Phi(-|h|) = (1/2)(a1 t + a2 t^2 + a3 t^3) exp(-h^2/2).
// The 1/2 is folded into the coefficients and 1/sqrt 2 into p; the
// reciprocal and the exponential use the hardware approximations (relative
// error of a few ulp).  The epilogue is bound by this arithmetic, so the
// three-term formula (two FMAs fewer than the five-term 7.1.26) pays.
__device__ __forceinline__ void gelu_and_grad_as(float h, float& g, float& gp) {
  float t, E;
  const float den = fmaf(fabsf(h), 0.47047f * 0.70710678118654752f, 1.f);
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(t) : "f"(den));
  const float q_poly = t * (0.5f * 0.3480242f + t * (0.5f * -0.0958798f + t * (0.5f * 0.7478556f)));
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(E) : "f"((h * -0.72134752044448170f) * h));  // exp(-h^2/2)
  const float q = q_poly * E;  // Phi(-|h|)
  const float Phi = h >= 0.f ? 1.f - q : q;
  g = h * Phi;
  gp = fmaf(h * 0.3989422804014327f, E, Phi);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

inline int ceil_div(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }

int sm_count();  // cached per device

// Number of kernels this library has launched (all threads, all devices).
void count_launches(int n);

// ---- Programmatic dependent launch ------------------------------------------
// Hot-path kernels launch with programmatic stream serialization: the next
// kernel on the stream may be scheduled once every CTA of the current one
// has started (each calls pdl_trigger() first), and it runs pdl_wait() --
// which returns when the previous grid has completed and its memory is
// visible -- before it reads anything that grid wrote or writes anything it
// reads.  Its launch and set-up then overlap the previous kernel's tail
// instead of following its completion.  SKY_PDL=0 in the environment turns
// the attribute off (plain stream order).
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

bool pdl_enabled();

// cudaLaunchKernelEx with the programmatic-serialization attribute (when
// enabled) and optionally a cluster of `cluster_x` CTAs.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, int cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[2];
  int n = 0;
  if (pdl_enabled()) {
    at[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (cluster_x > 1) {
    at[n].id = cudaLaunchAttributeClusterDimension;
    at[n].val.clusterDim.x = cluster_x;
    at[n].val.clusterDim.y = 1;
    at[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = at;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

}  // namespace sky
