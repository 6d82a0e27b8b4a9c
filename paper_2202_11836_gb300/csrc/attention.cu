// Masked scaled dot-product attention, Eq. 1: per sequence b and head a,
//   P = softmax_j(Q K^T / sqrt(D)) over the valid keys j < len[b],
//   ctx = P V,
// and its backward (dQ, dK, dV).  All S query rows are computed; padded keys
// get probability exactly 0.
//
// bf16 (D = 64): the tensor-core kernels of attention_tc.cu, plus the
// vectorised delta = rowsum(dO * O) pre-pass here.
// fp32: one warp per query (or key) row with exact fp32 arithmetic, for the
// small fp32 configuration.
#include "common.cuh"
#include "ptx.cuh"

namespace sky {
namespace attn {

constexpr int HD = 64;

using bf16 = __nv_bfloat16;

// delta[b,a,s] = sum_d dctx[b,s,a,d] * ctx[b,s,a,d]  (equals sum_j P_sj dP_sj)
// One warp per token row; each lane takes 8 consecutive elements (16 bytes
// of bf16) per 256-column group, and the 8 lanes covering one 64-wide head
// reduce with shuffles.  NV > 0: the row has exactly NV groups, and every
// load of the row is issued before the first product (more bytes in flight
// per warp); NV == 0: any H that is a multiple of 64, one group at a time.
// Requires D == 64.
// Beside delta it writes the per-query terms the tensor-core dK/dV kernel
// adds inside its score products: xtab[(b*A + a)*2 + 0][s] = lse2 / c and
// xtab[(b*A + a)*2 + 1][s] = delta (c = log2(e)/sqrt(D)), each negated and
// split into a bf16 high and low part, as 16-byte rows [hi, lo, 0 x 6].
template <int NV>
__global__ void attn_delta_bf16(const bf16* __restrict__ ctx, const bf16* __restrict__ dctx, int S,
                                int H, int A, int64_t rows, float* __restrict__ delta,
                                const float* __restrict__ lse, uint4* __restrict__ xtab) {
  pdl_trigger();
  pdl_wait();
  const int64_t row = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int l = threadIdx.x & 31;
  if (row >= rows) return;
  const int64_t b = row / S, s = row % S;
  auto dot8 = [](const uint4& x, const uint4& y) {
    const __nv_bfloat162* xs = reinterpret_cast<const __nv_bfloat162*>(&x);
    const __nv_bfloat162* ys = reinterpret_cast<const __nv_bfloat162*>(&y);
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 p = __bfloat1622float2(xs[i]), q = __bfloat1622float2(ys[i]);
      acc += p.x * q.x + p.y * q.y;
    }
    return acc;
  };
  // lz: the row's lse of this lane's head, loaded beside ctx / dctx (NV > 0)
  auto finish = [&](float acc, int col, float lz) {
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);
    acc += __shfl_xor_sync(0xffffffffu, acc, 2);
    acc += __shfl_xor_sync(0xffffffffu, acc, 4);
    if ((l & 7) == 0 && col < H) {
      const int64_t bh = b * A + col / HD;
      delta[bh * S + s] = acc;
      auto row16 = [](float x) {  // -x as [hi, lo, 0, ...] in bf16
        const bf16 hi = __float2bfloat16_rn(-x);
        const bf16 lo = __float2bfloat16_rn(-x - __bfloat162float(hi));
        return make_uint4(static_cast<uint32_t>(__bfloat16_as_ushort(hi)) |
                              (static_cast<uint32_t>(__bfloat16_as_ushort(lo)) << 16),
                          0u, 0u, 0u);
      };
      constexpr float kC = 1.4426950408889634f * 0.125f;  // log2(e) / sqrt(64)
      xtab[(bh * 2) * S + s] = row16(__fdiv_rn(lz, kC));
      xtab[(bh * 2 + 1) * S + s] = row16(acc);
    }
  };
  if constexpr (NV > 0) {
    uint4 x[NV], y[NV];
    float lz[NV];
#pragma unroll
    for (int v = 0; v < NV; ++v) {
      x[v] = *reinterpret_cast<const uint4*>(ctx + row * H + v * 256 + l * 8);
      y[v] = *reinterpret_cast<const uint4*>(dctx + row * H + v * 256 + l * 8);
      lz[v] = (l & 7) == 0 ? lse[(b * A + (v * 256 + l * 8) / HD) * S + s] : 0.f;
    }
#pragma unroll
    for (int v = 0; v < NV; ++v) finish(dot8(x[v], y[v]), v * 256 + l * 8, lz[v]);
  } else {
    for (int c0 = 0; c0 < H; c0 += 256) {
      const int col = c0 + l * 8;
      float acc = 0.f, lz = 0.f;
      if (col < H) {
        acc = dot8(*reinterpret_cast<const uint4*>(ctx + row * H + col),
                   *reinterpret_cast<const uint4*>(dctx + row * H + col));
        if ((l & 7) == 0) lz = lse[(b * A + col / HD) * S + s];
      }
      finish(acc, col, lz);
    }
  }
}

// Generic form (fp32 path): one warp per (row, head).
template <typename T>
__global__ void attn_delta(const T* __restrict__ ctx, const T* __restrict__ dctx, int S, int H,
                           int A, int D, int64_t rows, float* __restrict__ delta) {
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int l = threadIdx.x & 31;
  if (w >= rows * A) return;
  const int64_t row = w / A;
  const int a = (int)(w % A);
  const T* c = ctx + row * H + a * D;
  const T* dc = dctx + row * H + a * D;
  float acc = 0.f;
  for (int d = l; d < D; d += 32) acc += to_f32(c[d]) * to_f32(dc[d]);
  acc = warp_sum(acc);
  if (l == 0) {
    const int64_t b = row / S, s = row % S;
    delta[(b * A + a) * S + s] = acc;
  }
}

// ----------------------------------------------------------------- fp32 path
// One warp per (query row, head, sequence); p[] staged in shared memory.
__global__ void attn_fwd_f32(const float* __restrict__ qkv, const int32_t* __restrict__ lens,
                             int S, int H, int A, int D, float* __restrict__ ctx,
                             float* __restrict__ lse, int32_t* status) {
  extern __shared__ float sp[];
  const int wpb = blockDim.x >> 5, warp = threadIdx.x >> 5, l = threadIdx.x & 31;
  const int64_t w = (int64_t)blockIdx.x * wpb + warp;
  if (w >= (int64_t)S * A) return;
  const int b = blockIdx.y;
  const int i = (int)(w % S), a = (int)(w / S);
  float* p = sp + warp * S;
  int len = lens[b];
  if (len < 1 || len > S) {
    if (status && l == 0) atomicOr(status, kStatusBadLength);
    len = len < 1 ? 1 : S;
  }
  const int64_t rs = 3 * (int64_t)H;
  const float* q = qkv + ((int64_t)b * S + i) * rs + a * D;
  const float sc = 1.f / sqrtf((float)D);
  float mx = -INFINITY;
  for (int j = l; j < len; j += 32) {
    const float* k = qkv + ((int64_t)b * S + j) * rs + H + a * D;
    float s = 0.f;
    for (int d = 0; d < D; ++d) s = fmaf(q[d], k[d], s);
    s *= sc;
    p[j] = s;
    mx = fmaxf(mx, s);
  }
  mx = warp_max(mx);
  float sum = 0.f;
  for (int j = l; j < len; j += 32) {
    const float e = expf(p[j] - mx);
    p[j] = e;
    sum += e;
  }
  sum = warp_sum(sum);
  __syncwarp();
  const float inv = 1.f / sum;
  for (int d = l; d < D; d += 32) {
    float acc = 0.f;
    for (int j = 0; j < len; ++j)
      acc = fmaf(p[j], qkv[((int64_t)b * S + j) * rs + 2 * H + a * D + d], acc);
    ctx[((int64_t)b * S + i) * H + a * D + d] = acc * inv;
  }
  if (l == 0) lse[((int64_t)b * A + a) * S + i] = (mx + logf(sum)) * 1.4426950408889634f;  // base 2
}

// dQ rows (mode 0) or dK/dV rows (mode 1), one warp per row.
__global__ void attn_bwd_f32(const float* __restrict__ qkv, const float* __restrict__ dctx,
                             const float* __restrict__ lse, const float* __restrict__ delta,
                             const int32_t* __restrict__ lens, int S, int H, int A, int D,
                             float* __restrict__ dqkv, int mode) {
  const int wpb = blockDim.x >> 5, warp = threadIdx.x >> 5, l = threadIdx.x & 31;
  const int64_t w = (int64_t)blockIdx.x * wpb + warp;
  if (w >= (int64_t)S * A) return;
  const int b = blockIdx.y;
  const int r = (int)(w % S), a = (int)(w / S);
  int len = lens[b];
  len = len < 1 ? 1 : (len > S ? S : len);
  const int64_t rs = 3 * (int64_t)H;
  const float sc = 1.f / sqrtf((float)D);
  auto Q = [&](int i, int d) { return qkv[((int64_t)b * S + i) * rs + a * D + d]; };
  auto K = [&](int j, int d) { return qkv[((int64_t)b * S + j) * rs + H + a * D + d]; };
  auto V = [&](int j, int d) { return qkv[((int64_t)b * S + j) * rs + 2 * H + a * D + d]; };
  auto dO = [&](int i, int d) { return dctx[((int64_t)b * S + i) * H + a * D + d]; };
  const float* lse_b = lse + ((int64_t)b * A + a) * S;
  const float* del_b = delta + ((int64_t)b * A + a) * S;
  constexpr int MAXD = 4;  // D <= 128
  float acc0[MAXD] = {}, acc1[MAXD] = {};
  if (mode == 0) {
    const int i = r;
    for (int j = 0; j < len; ++j) {
      float s = 0.f, dp = 0.f;
      for (int d = l; d < D; d += 32) {
        s = fmaf(Q(i, d), K(j, d), s);
        dp = fmaf(dO(i, d), V(j, d), dp);
      }
      s = warp_sum(s);
      dp = warp_sum(dp);
      const float p = exp2f(fmaf(s, sc * 1.4426950408889634f, -lse_b[i]));
      const float ds = p * (dp - del_b[i]);
      for (int d = l, c = 0; d < D; d += 32, ++c) acc0[c] = fmaf(ds, K(j, d), acc0[c]);
    }
    for (int d = l, c = 0; d < D; d += 32, ++c)
      dqkv[((int64_t)b * S + i) * rs + a * D + d] = acc0[c] * sc;
  } else {
    const int j = r;
    if (j < len) {
      for (int i = 0; i < S; ++i) {
        float s = 0.f, dp = 0.f;
        for (int d = l; d < D; d += 32) {
          s = fmaf(Q(i, d), K(j, d), s);
          dp = fmaf(dO(i, d), V(j, d), dp);
        }
        s = warp_sum(s);
        dp = warp_sum(dp);
        const float p = exp2f(fmaf(s, sc * 1.4426950408889634f, -lse_b[i]));
        const float ds = p * (dp - del_b[i]);
        for (int d = l, c = 0; d < D; d += 32, ++c) {
          acc0[c] = fmaf(ds, Q(i, d), acc0[c]);   // dK
          acc1[c] = fmaf(p, dO(i, d), acc1[c]);    // dV
        }
      }
    }
    for (int d = l, c = 0; d < D; d += 32, ++c) {
      dqkv[((int64_t)b * S + j) * rs + H + a * D + d] = acc0[c] * sc;
      dqkv[((int64_t)b * S + j) * rs + 2 * H + a * D + d] = acc1[c];
    }
  }
}

}  // namespace attn

// ------------------------------------------------------------------- host
sky_status attention_fwd_tc(const void* qkv, const int32_t* lens, int B, int S, int H, int A,
                            void* ctx, float* lse, int32_t* status, uint64_t timeout_ns,
                            cudaStream_t stream);

sky_status attention_bwd_tc(const void* qkv, const void* dctx, const float* lse, const float* delta,
                            const uint4* xtab, const int32_t* lens, int B, int S, int H, int A, void* dqkv,
                            int32_t* status, uint64_t timeout_ns, cudaStream_t stream,
                            float* colpart);

sky_status attention_fwd(const void* qkv, const int32_t* lens, int B, int S, int H, int A,
                         sky_dtype dt, void* ctx, float* lse, int32_t* status,
                         cudaStream_t stream) {
  const int D = H / A;
  if (dt == SKY_DTYPE_BF16) {
    SKY_CHECK(D == attn::HD, SKY_ERR_UNSUPPORTED, "bf16 attention needs head dim 64 (got %d)", D);
    return attention_fwd_tc(qkv, lens, B, S, H, A, ctx, lse, status, 2000000000ull, stream);
  } else {
    SKY_CHECK(D <= 128, SKY_ERR_UNSUPPORTED, "fp32 attention needs head dim <= 128");
    const int wpb = 4;
    dim3 grid(ceil_div((int64_t)S * A, wpb), B);
    const size_t smem = (size_t)wpb * S * sizeof(float);
    SKY_CHECK(smem <= 48 * 1024, SKY_ERR_UNSUPPORTED, "fp32 attention: sequence too long");
    attn::attn_fwd_f32<<<grid, wpb * 32, smem, stream>>>(static_cast<const float*>(qkv), lens, S,
                                                         H, A, D, static_cast<float*>(ctx), lse,
                                                         status);
  }
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "attention forward launch");
}

// delta [B][A][S] floats, then (bf16 path) the dK/dV kernel's per-query rows
// [B][A][2][S] x 16 bytes, 16-byte aligned.
static size_t delta_bytes(int B, int S, int A) { return ((size_t)B * A * S * sizeof(float) + 15) & ~(size_t)15; }
size_t attention_bwd_ws(int B, int S, int A) { return delta_bytes(B, S, A) + (size_t)B * A * 2 * S * 16; }

sky_status attention_bwd(const void* qkv, const void* ctx, const void* dctx, const float* lse,
                         const int32_t* lens, int B, int S, int H, int A, sky_dtype dt, void* dqkv,
                         float* delta, int32_t* status, cudaStream_t stream, float* colpart) {
  const int D = H / A;
  const int64_t rows = (int64_t)B * S;
  const int dblocks = ceil_div(rows * A * 32, 256);
  if (dt == SKY_DTYPE_BF16) {
    SKY_CHECK(D == attn::HD, SKY_ERR_UNSUPPORTED, "bf16 attention needs head dim 64 (got %d)", D);
    // every kernel below moves 16-byte vectors of these buffers (checked
    // before the first launch)
    const auto a16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15) == 0; };
    SKY_CHECK(a16(qkv) && a16(ctx) && a16(dctx) && a16(dqkv) && a16(delta), SKY_ERR_INVALID_ARG,
              "bf16 attention backward buffers and workspace must be 16-byte aligned");
    const auto* c = static_cast<const __nv_bfloat16*>(ctx);
    const auto* dc = static_cast<const __nv_bfloat16*>(dctx);
    const dim3 g(ceil_div(rows * 32, 256)), blk(256);
    uint4* xtab = reinterpret_cast<uint4*>(reinterpret_cast<char*>(delta) + delta_bytes(B, S, A));
    cudaError_t le;
    switch (H % 256 == 0 ? H / 256 : 0) {
      case 3: le = launch_pdl(attn::attn_delta_bf16<3>, g, blk, 0, stream, 1, c, dc, S, H, A, rows, delta, lse, xtab); break;
      case 4: le = launch_pdl(attn::attn_delta_bf16<4>, g, blk, 0, stream, 1, c, dc, S, H, A, rows, delta, lse, xtab); break;
      case 8: le = launch_pdl(attn::attn_delta_bf16<8>, g, blk, 0, stream, 1, c, dc, S, H, A, rows, delta, lse, xtab); break;
      default: le = launch_pdl(attn::attn_delta_bf16<0>, g, blk, 0, stream, 1, c, dc, S, H, A, rows, delta, lse, xtab); break;
    }
    count_launches(1);
    if (le != cudaSuccess) return cuda_fail(le, "attention delta launch");
    return attention_bwd_tc(qkv, dctx, lse, delta, xtab, lens, B, S, H, A, dqkv, status, 2000000000ull,
                            stream, colpart);
  } else {
    SKY_CHECK(D <= 128, SKY_ERR_UNSUPPORTED, "fp32 attention needs head dim <= 128");
    attn::attn_delta<float><<<dblocks, 256, 0, stream>>>(static_cast<const float*>(ctx),
                                                         static_cast<const float*>(dctx), S, H, A,
                                                         D, rows, delta);
    const int wpb = 4;
    dim3 grid(ceil_div((int64_t)S * A, wpb), B);
    for (int mode = 0; mode < 2; ++mode)
      attn::attn_bwd_f32<<<grid, wpb * 32, 0, stream>>>(
          static_cast<const float*>(qkv), static_cast<const float*>(dctx), lse, delta, lens, S, H,
          A, D, static_cast<float*>(dqkv), mode);
  }
  count_launches(3);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "attention backward launch");
}

}  // namespace sky
