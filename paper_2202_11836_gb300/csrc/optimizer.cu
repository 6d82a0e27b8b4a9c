// Local parameter update of a slice (Sec. III: after its backward pass each
// device updates its own layers' weights with the gradients it computed).
//
// One launch updates every parameter tensor of the slice.  The host cuts the
// tensors into chunks of at most kChunk float4 groups; a chunk table
// (tensor, first group, group count) lets every CTA walk its chunks with no
// per-element search.  Per element the kernel reads the fp32 gradient, the
// fp32 master weight and the optimizer state and writes the master weight,
// the state and (bf16 slices) the parameter rounded to bf16: 30 bytes per
// parameter for AdamW, 22 for SGD -- an HBM-bound stream.
//
// AdamW (Kingma & Ba, Algorithm 1, with decoupled weight decay as in BERT):
//   m <- b1 m + (1 - b1) g,  v <- b2 v + (1 - b2) g^2,
//   w <- w - lr wd w (weight matrices only),
//   w <- w - lr (m / bc1) / (sqrt(v / bc2) + eps),  bc = 1 - b^t.
// SGD with momentum (weight decay added to the gradient):
//   b <- mu b + (g + wd w)  (b <- g + wd w on the first step),  w <- w - lr b.
#include "common.cuh"
#include "optimizer.h"

namespace sky {
namespace opt {

constexpr int kThreads = 256;

__device__ __forceinline__ void store_param(void* p, int64_t i4, const float4& w) {
  __nv_bfloat162 a = __floats2bfloat162_rn(w.x, w.y), b = __floats2bfloat162_rn(w.z, w.w);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&a);
  u.y = *reinterpret_cast<uint32_t*>(&b);
  reinterpret_cast<uint2*>(p)[i4] = u;
}

__global__ void __launch_bounds__(kThreads) adamw_kernel(const Tensor* __restrict__ ts,
                                                         const Chunk* __restrict__ chunks,
                                                         int n_chunks, AdamArgs a) {
  pdl_trigger();
  pdl_wait();
  for (int c = blockIdx.x; c < n_chunks; c += gridDim.x) {
    const Chunk ch = chunks[c];
    const Tensor t = ts[ch.tensor];
    const float wd = t.decay ? a.lr * a.wd : 0.f;
    for (int64_t k = threadIdx.x; k < ch.count; k += kThreads) {
      const int64_t i = ch.first + k;
      const float4 g = reinterpret_cast<const float4*>(t.g)[i];
      float4 w = reinterpret_cast<float4*>(t.w)[i];
      float4 m = reinterpret_cast<float4*>(t.s0)[i];
      float4 v = reinterpret_cast<float4*>(t.s1)[i];
      auto upd = [&](float gg, float& ww, float& mm, float& vv) {
        mm = a.b1 * mm + (1.f - a.b1) * gg;
        vv = a.b2 * vv + (1.f - a.b2) * gg * gg;
        ww = ww - wd * ww;
        ww = ww - a.lr * (mm / a.bc1) / (sqrtf(vv / a.bc2) + a.eps);
      };
      upd(g.x, w.x, m.x, v.x);
      upd(g.y, w.y, m.y, v.y);
      upd(g.z, w.z, m.z, v.z);
      upd(g.w, w.w, m.w, v.w);
      reinterpret_cast<float4*>(t.w)[i] = w;
      reinterpret_cast<float4*>(t.s0)[i] = m;
      reinterpret_cast<float4*>(t.s1)[i] = v;
      if (t.p) store_param(t.p, i, w);
    }
  }
}

__global__ void __launch_bounds__(kThreads) sgd_kernel(const Tensor* __restrict__ ts,
                                                       const Chunk* __restrict__ chunks,
                                                       int n_chunks, SgdArgs a) {
  pdl_trigger();
  pdl_wait();
  for (int c = blockIdx.x; c < n_chunks; c += gridDim.x) {
    const Chunk ch = chunks[c];
    const Tensor t = ts[ch.tensor];
    const float wd = t.decay ? a.wd : 0.f;
    for (int64_t k = threadIdx.x; k < ch.count; k += kThreads) {
      const int64_t i = ch.first + k;
      const float4 g = reinterpret_cast<const float4*>(t.g)[i];
      float4 w = reinterpret_cast<float4*>(t.w)[i];
      float4 b = reinterpret_cast<float4*>(t.s0)[i];
      auto upd = [&](float gg, float& ww, float& bb) {
        const float d = gg + wd * ww;
        bb = a.first ? d : a.mu * bb + d;
        ww = ww - a.lr * bb;
      };
      upd(g.x, w.x, b.x);
      upd(g.y, w.y, b.y);
      upd(g.z, w.z, b.z);
      upd(g.w, w.w, b.w);
      reinterpret_cast<float4*>(t.w)[i] = w;
      reinterpret_cast<float4*>(t.s0)[i] = b;
      if (t.p) store_param(t.p, i, w);
    }
  }
}

void make_chunks(const std::vector<Tensor>& ts, std::vector<Chunk>* out) {
  out->clear();
  for (int t = 0; t < (int)ts.size(); ++t) {
    const int64_t groups = ts[t].n / 4;
    for (int64_t f = 0; f < groups; f += kChunk)
      out->push_back(Chunk{t, f, std::min<int64_t>(kChunk, groups - f)});
  }
}

sky_status launch_adamw(const Tensor* d_ts, const Chunk* d_chunks, int n_chunks, const AdamArgs& a,
                        cudaStream_t st) {
  const int blocks = std::min(n_chunks, 8 * (sm_count() > 0 ? sm_count() : 148));
  if (blocks <= 0) return SKY_OK;
  launch_pdl(adamw_kernel, dim3(blocks), dim3(kThreads), 0, st, 1, d_ts, d_chunks, n_chunks, a);
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "AdamW update launch");
}

sky_status launch_sgd(const Tensor* d_ts, const Chunk* d_chunks, int n_chunks, const SgdArgs& a,
                      cudaStream_t st) {
  const int blocks = std::min(n_chunks, 8 * (sm_count() > 0 ? sm_count() : 148));
  if (blocks <= 0) return SKY_OK;
  launch_pdl(sgd_kernel, dim3(blocks), dim3(kThreads), 0, st, 1, d_ts, d_chunks, n_chunks, a);
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "SGD update launch");
}

}  // namespace opt
}  // namespace sky
