// Parameter-update kernels of a slice (optimizer.cu).
#pragma once
#include <algorithm>
#include <vector>

#include <cuda_runtime.h>

#include "../../include/sky_slice.h"

namespace sky {
namespace opt {

// One parameter tensor: n fp32 elements (n % 4 == 0, all pointers 16-byte
// aligned).  w: fp32 master weights; g: gradient; s0 / s1: optimizer state
// (AdamW m / v, SGD momentum / unused); p: the slice's bf16 copy or null.
struct Tensor {
  float* w;
  const float* g;
  float* s0;
  float* s1;
  void* p;
  int64_t n;
  int decay;  // weight decay applies (weight matrices)
};

// Float4 groups [first, first + count) of tensor `tensor`.
struct Chunk {
  int tensor;
  int64_t first;
  int64_t count;
};
constexpr int64_t kChunk = 2048;  // float4 groups per chunk (8192 elements)

struct AdamArgs {
  float lr, b1, b2, eps, wd, bc1, bc2;
};
struct SgdArgs {
  float lr, mu, wd;
  int first;
};

void make_chunks(const std::vector<Tensor>& ts, std::vector<Chunk>* out);
sky_status launch_adamw(const Tensor* d_ts, const Chunk* d_chunks, int n_chunks, const AdamArgs& a,
                        cudaStream_t st);
sky_status launch_sgd(const Tensor* d_ts, const Chunk* d_chunks, int n_chunks, const SgdArgs& a,
                      cudaStream_t st);

}  // namespace opt
}  // namespace sky
