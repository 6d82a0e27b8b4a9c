// Masked scaled dot-product attention, Eq. 1: per sequence b and head a,
//   P = softmax_j(Q K^T / sqrt(D)) over the valid keys j < len[b],
//   ctx = P V,
// and its backward (dQ, dK, dV).  All S query rows are computed; padded keys
// get probability exactly 0.
//
// bf16 path (D = 64): flash-style tiles of 64 queries x 64 keys.  Q/K/V tiles
// are staged in XOR-swizzled shared memory with cp.async, fragments are read
// with ldmatrix and multiplied with mma.sync m16n8k16 (bf16 in, fp32 accum);
// the row max / row sum of the online softmax are fp32 and reduced with warp
// shuffles within each quad.  Key tiles at or beyond len[b] are skipped.  The
// forward keeps the per-row log-sum-exp; the backward recomputes P from it:
//   kernel dkdv: per key tile, loop over all query tiles, accumulate dV, dK;
//   kernel dq:   per query tile, loop over the valid key tiles, accumulate dQ;
// so no floating-point atomics are used and results are deterministic.
//
// fp32 path: one warp per query (or key) row with exact fp32 arithmetic, for
// the small fp32 configuration.
#include "common.cuh"
#include "ptx.cuh"

namespace sky {
namespace attn {

constexpr int TQ = 64, TKV = 64, HD = 64, NTHR = 128;
constexpr float LOG2E = 1.4426950408889634f;
constexpr float LN2 = 0.6931471805599453f;

using bf16 = __nv_bfloat16;

// element offset of (row, 16-byte chunk) in a 64 x 64 bf16 tile
__device__ __forceinline__ int swz(int row, int chunk) {
  return row * HD + ((chunk ^ (row & 7)) << 3);
}

// Loads rows [r0, r0+64) of one 64-wide head slice; rows >= valid are zero.
__device__ __forceinline__ void load_tile(bf16* tile, const bf16* base, int64_t row_stride,
                                          int r0, int valid) {
#pragma unroll
  for (int i = threadIdx.x; i < 64 * 8; i += NTHR) {
    const int r = i >> 3, c = i & 7;
    const bool ok = r0 + r < valid;
    const bf16* src = ok ? base + (int64_t)(r0 + r) * row_stride + c * 8 : base;
    ptx::cp_async_16(ptx::smem_u32(tile + swz(r, c)), src, ok ? 16u : 0u);
  }
}

// A-operand fragment (16 rows starting at r0, k-step kk) from a swizzled tile.
__device__ __forceinline__ void frag_a(uint32_t (&a)[4], const bf16* tile, int r0, int kk) {
  const int l = threadIdx.x & 31;
  const int row = r0 + (l & 7) + 8 * ((l >> 3) & 1);
  const int chunk = 2 * kk + (l >> 4);
  ptx::ldmatrix_x4(a, ptx::smem_u32(tile + swz(row, chunk)));
}
// B fragments for two n-tiles (rows n0..n0+15 of the tile are the n index,
// tile columns are k): b[0],b[1] for n-tile n0, b[2],b[3] for n0+8.
__device__ __forceinline__ void frag_b_rows(uint32_t (&b)[4], const bf16* tile, int n0, int kk) {
  const int l = threadIdx.x & 31;
  const int row = n0 + (l & 7) + 8 * (l >> 4);
  const int chunk = 2 * kk + ((l >> 3) & 1);
  ptx::ldmatrix_x4(b, ptx::smem_u32(tile + swz(row, chunk)));
}
// B fragments when tile rows are the k index and tile columns the n index:
// k rows k0..k0+15, n columns d0..d0+15 (two n-tiles).
__device__ __forceinline__ void frag_b_cols(uint32_t (&b)[4], const bf16* tile, int k0, int d0) {
  const int l = threadIdx.x & 31;
  const int row = k0 + (l & 7) + 8 * ((l >> 3) & 1);
  const int chunk = (d0 >> 3) + (l >> 4);
  ptx::ldmatrix_x4_trans(b, ptx::smem_u32(tile + swz(row, chunk)));
}

__device__ __forceinline__ int checked_len(const int32_t* lens, int b, int S, int32_t* status) {
  int n = lens[b];
  if (n < 1 || n > S) {
    if (status && threadIdx.x == 0) atomicOr(status, kStatusBadLength);
    n = n < 1 ? 1 : S;
  }
  return n;
}

// ------------------------------------------------------------------ forward
__global__ void __launch_bounds__(NTHR) attn_fwd_bf16(const bf16* __restrict__ qkv,
                                                      const int32_t* __restrict__ lens, int S,
                                                      int H, bf16* __restrict__ ctx,
                                                      float* __restrict__ lse, int32_t* status) {
  __shared__ __align__(128) bf16 sQ[TQ * HD];
  __shared__ __align__(128) bf16 sK[2][TKV * HD];
  __shared__ __align__(128) bf16 sV[2][TKV * HD];
  const int qt = blockIdx.x, a = blockIdx.y, b = blockIdx.z;
  const int A = gridDim.y;
  const int warp = threadIdx.x >> 5, l = threadIdx.x & 31;
  const int g = l >> 2, t = l & 3;
  const int len = checked_len(lens, b, S, status);
  const int64_t rs = 3 * (int64_t)H;
  const bf16* base = qkv + (int64_t)b * S * rs + a * HD;
  const int q0 = qt * TQ;
  const int n_kt = (len + TKV - 1) / TKV;
  const float sl2 = LOG2E * rsqrtf((float)HD);

  load_tile(sQ, base, rs, q0, S);
  load_tile(sK[0], base + H, rs, 0, len);
  load_tile(sV[0], base + 2 * H, rs, 0, len);
  ptx::cp_async_commit();

  uint32_t qf[4][4];
  float o[8][4] = {};
  float m_r[2] = {-INFINITY, -INFINITY}, l_r[2] = {0.f, 0.f};

  for (int kt = 0; kt < n_kt; ++kt) {
    const int cur = kt & 1;
    if (kt + 1 < n_kt) {
      load_tile(sK[cur ^ 1], base + H, rs, (kt + 1) * TKV, len);
      load_tile(sV[cur ^ 1], base + 2 * H, rs, (kt + 1) * TKV, len);
    }
    ptx::cp_async_commit();
    ptx::cp_async_wait<1>();
    __syncthreads();
    if (kt == 0) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) frag_a(qf[kk], sQ, warp * 16, kk);
    }
    float s[8][4] = {};
#pragma unroll
    for (int j = 0; j < 8; j += 2) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t bb[4];
        frag_b_rows(bb, sK[cur], j * 8, kk);
        ptx::mma_bf16_16816(s[j], qf[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(s[j + 1], qf[kk], bb[2], bb[3]);
      }
    }
    // scale to log2 units, mask, online softmax
    float mx[2] = {m_r[0], m_r[1]};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int key = kt * TKV + j * 8 + 2 * t;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const bool valid = key + (e & 1) < len;
        s[j][e] = valid ? s[j][e] * sl2 : -INFINITY;
        mx[e >> 1] = fmaxf(mx[e >> 1], s[j][e]);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
    }
    float corr[2], rsum[2] = {0.f, 0.f};
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      corr[r] = exp2f(m_r[r] - mx[r]);
      m_r[r] = mx[r];
    }
    uint32_t pf[4][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        s[j][e] = exp2f(s[j][e] - m_r[e >> 1]);
        rsum[e >> 1] += s[j][e];
      }
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      pf[kk][0] = ptx::pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      pf[kk][1] = ptx::pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      pf[kk][2] = ptx::pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      pf[kk][3] = ptx::pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) l_r[r] = l_r[r] * corr[r] + rsum[r];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      o[j][0] *= corr[0]; o[j][1] *= corr[0];
      o[j][2] *= corr[1]; o[j][3] *= corr[1];
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int j = 0; j < 8; j += 2) {
        uint32_t bb[4];
        frag_b_cols(bb, sV[cur], kk * 16, j * 8);
        ptx::mma_bf16_16816(o[j], pf[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(o[j + 1], pf[kk], bb[2], bb[3]);
      }
    }
    __syncthreads();
  }
  // quad-reduce the row sums, normalise, store
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    l_r[r] += __shfl_xor_sync(0xffffffffu, l_r[r], 1);
    l_r[r] += __shfl_xor_sync(0xffffffffu, l_r[r], 2);
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int q = q0 + warp * 16 + g + 8 * r;
    if (q >= S) continue;
    const float inv = 1.f / l_r[r];
    bf16* out = ctx + ((int64_t)b * S + q) * H + a * HD;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      *reinterpret_cast<uint32_t*>(out + j * 8 + 2 * t) =
          ptx::pack_bf16(o[j][2 * r] * inv, o[j][2 * r + 1] * inv);
    if (t == 0) lse[((int64_t)b * A + a) * S + q] = (m_r[r] + log2f(l_r[r])) * LN2;
  }
}

// delta[b,a,s] = sum_d dctx[b,s,a,d] * ctx[b,s,a,d]  (equals sum_j P_sj dP_sj)
// One warp per token row; each lane takes 8 consecutive elements (16 bytes
// of bf16) per step, and the 8 lanes covering one 64-wide head reduce with
// shuffles.  Requires D == 64.
__global__ void attn_delta_bf16(const bf16* __restrict__ ctx, const bf16* __restrict__ dctx, int S,
                                int H, int A, int64_t rows, float* __restrict__ delta) {
  const int64_t row = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int l = threadIdx.x & 31;
  if (row >= rows) return;
  const int64_t b = row / S, s = row % S;
  for (int c0 = 0; c0 < H; c0 += 256) {
    const int col = c0 + l * 8;
    float acc = 0.f;
    if (col < H) {
      const uint4 x = *reinterpret_cast<const uint4*>(ctx + row * H + col);
      const uint4 y = *reinterpret_cast<const uint4*>(dctx + row * H + col);
      const __nv_bfloat162* xs = reinterpret_cast<const __nv_bfloat162*>(&x);
      const __nv_bfloat162* ys = reinterpret_cast<const __nv_bfloat162*>(&y);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 p = __bfloat1622float2(xs[i]), q = __bfloat1622float2(ys[i]);
        acc += p.x * q.x + p.y * q.y;
      }
    }
    acc += __shfl_xor_sync(0xffffffffu, acc, 1);
    acc += __shfl_xor_sync(0xffffffffu, acc, 2);
    acc += __shfl_xor_sync(0xffffffffu, acc, 4);
    if ((l & 7) == 0 && col < H) delta[(b * A + col / HD) * S + s] = acc;
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

// ---------------------------------------------------------- backward dK, dV
__global__ void __launch_bounds__(NTHR) attn_bwd_dkdv_bf16(
    const bf16* __restrict__ qkv, const bf16* __restrict__ dctx, const float* __restrict__ lse,
    const float* __restrict__ delta, const int32_t* __restrict__ lens, int S, int H,
    bf16* __restrict__ dqkv, int32_t* status) {
  __shared__ __align__(128) bf16 sKV[TKV * HD];  // K tile, then V tile
  __shared__ __align__(128) bf16 sQ[2][TQ * HD];
  __shared__ __align__(128) bf16 sO[2][TQ * HD];  // dO = dctx tiles
  __shared__ float sL[2][TQ], sD[2][TQ];
  const int kt = blockIdx.x, a = blockIdx.y, b = blockIdx.z;
  const int A = gridDim.y;
  const int warp = threadIdx.x >> 5, l = threadIdx.x & 31;
  const int g = l >> 2, t = l & 3;
  const int len = checked_len(lens, b, S, status);
  const int64_t rs = 3 * (int64_t)H;
  const bf16* base = qkv + (int64_t)b * S * rs + a * HD;
  const bf16* obase = dctx + (int64_t)b * S * H + a * HD;
  const int k0 = kt * TKV;
  bf16* dk_out = dqkv + (int64_t)b * S * rs + H + a * HD;
  bf16* dv_out = dk_out + H;
  if (k0 >= len) {  // keys of this tile are all padding: zero gradients
    for (int i = threadIdx.x; i < TKV * 8; i += NTHR) {
      const int r = i >> 3, c = i & 7;
      if (k0 + r < S) {
        *reinterpret_cast<uint4*>(dk_out + (int64_t)(k0 + r) * rs + c * 8) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(dv_out + (int64_t)(k0 + r) * rs + c * 8) = make_uint4(0, 0, 0, 0);
      }
    }
    return;
  }
  const float sl2 = LOG2E * rsqrtf((float)HD);
  const float* lse_b = lse + ((int64_t)b * A + a) * S;
  const float* del_b = delta + ((int64_t)b * A + a) * S;
  const int n_qt = (S + TQ - 1) / TQ;

  uint32_t kf[4][4], vf[4][4];
  load_tile(sKV, base + H, rs, k0, len);
  ptx::cp_async_commit();
  ptx::cp_async_wait<0>();
  __syncthreads();
#pragma unroll
  for (int kk = 0; kk < 4; ++kk) frag_a(kf[kk], sKV, warp * 16, kk);
  __syncthreads();
  load_tile(sKV, base + 2 * H, rs, k0, len);
  ptx::cp_async_commit();
  ptx::cp_async_wait<0>();
  __syncthreads();
#pragma unroll
  for (int kk = 0; kk < 4; ++kk) frag_a(vf[kk], sKV, warp * 16, kk);

  auto stage_q = [&](int buf, int qt) {
    load_tile(sQ[buf], base, rs, qt * TQ, S);
    load_tile(sO[buf], obase, H, qt * TQ, S);
    for (int i = threadIdx.x; i < TQ; i += NTHR) {
      const int q = qt * TQ + i;
      sL[buf][i] = q < S ? lse_b[q] * LOG2E : INFINITY;
      sD[buf][i] = q < S ? del_b[q] : 0.f;
    }
  };
  stage_q(0, 0);
  ptx::cp_async_commit();

  float dk[8][4] = {}, dv[8][4] = {};
  const int key_r0 = k0 + warp * 16 + g;  // this thread's key rows: key_r0, key_r0 + 8
  for (int qt = 0; qt < n_qt; ++qt) {
    const int cur = qt & 1;
    __syncthreads();  // everyone is done with buffer cur^1
    if (qt + 1 < n_qt) stage_q(cur ^ 1, qt + 1);
    ptx::cp_async_commit();
    ptx::cp_async_wait<1>();
    __syncthreads();
    // S^T = K Q^T : 16 keys x 64 queries
    float st[8][4] = {};
#pragma unroll
    for (int j = 0; j < 8; j += 2) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t bb[4];
        frag_b_rows(bb, sQ[cur], j * 8, kk);
        ptx::mma_bf16_16816(st[j], kf[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(st[j + 1], kf[kk], bb[2], bb[3]);
      }
    }
    // P^T = exp(S^T / sqrt(D) - lse_q), zero for padded keys
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = key_r0 + 8 * (e >> 1);
        const int qi = j * 8 + 2 * t + (e & 1);
        st[j][e] = key < len ? exp2f(st[j][e] * sl2 - sL[cur][qi]) : 0.f;
      }
    }
    uint32_t pf[4][4];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      pf[kk][0] = ptx::pack_bf16(st[2 * kk][0], st[2 * kk][1]);
      pf[kk][1] = ptx::pack_bf16(st[2 * kk][2], st[2 * kk][3]);
      pf[kk][2] = ptx::pack_bf16(st[2 * kk + 1][0], st[2 * kk + 1][1]);
      pf[kk][3] = ptx::pack_bf16(st[2 * kk + 1][2], st[2 * kk + 1][3]);
    }
    // dV += P^T dO
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int j = 0; j < 8; j += 2) {
        uint32_t bb[4];
        frag_b_cols(bb, sO[cur], kk * 16, j * 8);
        ptx::mma_bf16_16816(dv[j], pf[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(dv[j + 1], pf[kk], bb[2], bb[3]);
      }
    }
    // dP^T = V dO^T
    float dpt[8][4] = {};
#pragma unroll
    for (int j = 0; j < 8; j += 2) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t bb[4];
        frag_b_rows(bb, sO[cur], j * 8, kk);
        ptx::mma_bf16_16816(dpt[j], vf[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(dpt[j + 1], vf[kk], bb[2], bb[3]);
      }
    }
    // dS^T = P^T (dP^T - delta_q)
    uint32_t sf[4][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int qi = j * 8 + 2 * t + (e & 1);
        dpt[j][e] = st[j][e] * (dpt[j][e] - sD[cur][qi]);
      }
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      sf[kk][0] = ptx::pack_bf16(dpt[2 * kk][0], dpt[2 * kk][1]);
      sf[kk][1] = ptx::pack_bf16(dpt[2 * kk][2], dpt[2 * kk][3]);
      sf[kk][2] = ptx::pack_bf16(dpt[2 * kk + 1][0], dpt[2 * kk + 1][1]);
      sf[kk][3] = ptx::pack_bf16(dpt[2 * kk + 1][2], dpt[2 * kk + 1][3]);
    }
    // dK += dS^T Q
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int j = 0; j < 8; j += 2) {
        uint32_t bb[4];
        frag_b_cols(bb, sQ[cur], kk * 16, j * 8);
        ptx::mma_bf16_16816(dk[j], sf[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(dk[j + 1], sf[kk], bb[2], bb[3]);
      }
    }
  }
  const float sc = rsqrtf((float)HD);
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int key = key_r0 + 8 * r;
    if (key >= S) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      *reinterpret_cast<uint32_t*>(dk_out + (int64_t)key * rs + j * 8 + 2 * t) =
          ptx::pack_bf16(dk[j][2 * r] * sc, dk[j][2 * r + 1] * sc);
      *reinterpret_cast<uint32_t*>(dv_out + (int64_t)key * rs + j * 8 + 2 * t) =
          ptx::pack_bf16(dv[j][2 * r], dv[j][2 * r + 1]);
    }
  }
}

// --------------------------------------------------------------- backward dQ
__global__ void __launch_bounds__(NTHR) attn_bwd_dq_bf16(
    const bf16* __restrict__ qkv, const bf16* __restrict__ dctx, const float* __restrict__ lse,
    const float* __restrict__ delta, const int32_t* __restrict__ lens, int S, int H,
    bf16* __restrict__ dqkv, int32_t* status) {
  __shared__ __align__(128) bf16 sQ[TQ * HD];  // Q tile, then dO tile
  __shared__ __align__(128) bf16 sK[2][TKV * HD];
  __shared__ __align__(128) bf16 sV[2][TKV * HD];
  const int qt = blockIdx.x, a = blockIdx.y, b = blockIdx.z;
  const int A = gridDim.y;
  const int warp = threadIdx.x >> 5, l = threadIdx.x & 31;
  const int g = l >> 2, t = l & 3;
  const int len = checked_len(lens, b, S, status);
  const int64_t rs = 3 * (int64_t)H;
  const bf16* base = qkv + (int64_t)b * S * rs + a * HD;
  const bf16* obase = dctx + (int64_t)b * S * H + a * HD;
  const int q0 = qt * TQ;
  const int n_kt = (len + TKV - 1) / TKV;
  const float sl2 = LOG2E * rsqrtf((float)HD);

  uint32_t qf[4][4], of[4][4];
  load_tile(sQ, base, rs, q0, S);
  ptx::cp_async_commit();
  ptx::cp_async_wait<0>();
  __syncthreads();
#pragma unroll
  for (int kk = 0; kk < 4; ++kk) frag_a(qf[kk], sQ, warp * 16, kk);
  __syncthreads();
  load_tile(sQ, obase, H, q0, S);
  load_tile(sK[0], base + H, rs, 0, len);
  load_tile(sV[0], base + 2 * H, rs, 0, len);
  ptx::cp_async_commit();
  ptx::cp_async_wait<0>();
  __syncthreads();
#pragma unroll
  for (int kk = 0; kk < 4; ++kk) frag_a(of[kk], sQ, warp * 16, kk);

  float lq[2], dq_del[2];
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int q = q0 + warp * 16 + g + 8 * r;
    const int64_t idx = ((int64_t)b * A + a) * S + (q < S ? q : 0);
    lq[r] = q < S ? lse[idx] * LOG2E : INFINITY;
    dq_del[r] = q < S ? delta[idx] : 0.f;
  }
  float dq[8][4] = {};
  for (int kt = 0; kt < n_kt; ++kt) {
    const int cur = kt & 1;
    if (kt + 1 < n_kt) {
      load_tile(sK[cur ^ 1], base + H, rs, (kt + 1) * TKV, len);
      load_tile(sV[cur ^ 1], base + 2 * H, rs, (kt + 1) * TKV, len);
    }
    ptx::cp_async_commit();
    ptx::cp_async_wait<1>();
    __syncthreads();
    float s[8][4] = {}, dp[8][4] = {};
#pragma unroll
    for (int j = 0; j < 8; j += 2) {
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t bb[4];
        frag_b_rows(bb, sK[cur], j * 8, kk);
        ptx::mma_bf16_16816(s[j], qf[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(s[j + 1], qf[kk], bb[2], bb[3]);
        frag_b_rows(bb, sV[cur], j * 8, kk);
        ptx::mma_bf16_16816(dp[j], of[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(dp[j + 1], of[kk], bb[2], bb[3]);
      }
    }
    uint32_t sf[4][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int key = kt * TKV + j * 8 + 2 * t;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int r = e >> 1;
        const float p = key + (e & 1) < len ? exp2f(s[j][e] * sl2 - lq[r]) : 0.f;
        s[j][e] = p * (dp[j][e] - dq_del[r]);
      }
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      sf[kk][0] = ptx::pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      sf[kk][1] = ptx::pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      sf[kk][2] = ptx::pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      sf[kk][3] = ptx::pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int j = 0; j < 8; j += 2) {
        uint32_t bb[4];
        frag_b_cols(bb, sK[cur], kk * 16, j * 8);
        ptx::mma_bf16_16816(dq[j], sf[kk], bb[0], bb[1]);
        ptx::mma_bf16_16816(dq[j + 1], sf[kk], bb[2], bb[3]);
      }
    }
    __syncthreads();
  }
  const float sc = rsqrtf((float)HD);
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int q = q0 + warp * 16 + g + 8 * r;
    if (q >= S) continue;
    bf16* out = dqkv + ((int64_t)b * S + q) * rs + a * HD;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      *reinterpret_cast<uint32_t*>(out + j * 8 + 2 * t) =
          ptx::pack_bf16(dq[j][2 * r] * sc, dq[j][2 * r + 1] * sc);
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
  if (l == 0) lse[((int64_t)b * A + a) * S + i] = mx + logf(sum);
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
      const float p = expf(s * sc - lse_b[i]);
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
        const float p = expf(s * sc - lse_b[i]);
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
sky_status attention_fwd(const void* qkv, const int32_t* lens, int B, int S, int H, int A,
                         sky_dtype dt, void* ctx, float* lse, int32_t* status,
                         cudaStream_t stream) {
  const int D = H / A;
  if (dt == SKY_DTYPE_BF16) {
    SKY_CHECK(D == attn::HD, SKY_ERR_UNSUPPORTED, "bf16 attention needs head dim 64 (got %d)", D);
    dim3 grid(ceil_div(S, attn::TQ), A, B);
    attn::attn_fwd_bf16<<<grid, attn::NTHR, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(qkv), lens, S, H, static_cast<__nv_bfloat16*>(ctx),
        lse, status);
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

size_t attention_bwd_ws(int B, int S, int A) { return (size_t)B * A * S * sizeof(float); }

sky_status attention_bwd(const void* qkv, const void* ctx, const void* dctx, const float* lse,
                         const int32_t* lens, int B, int S, int H, int A, sky_dtype dt, void* dqkv,
                         float* delta, int32_t* status, cudaStream_t stream) {
  const int D = H / A;
  const int64_t rows = (int64_t)B * S;
  const int dblocks = ceil_div(rows * A * 32, 256);
  if (dt == SKY_DTYPE_BF16) {
    SKY_CHECK(D == attn::HD, SKY_ERR_UNSUPPORTED, "bf16 attention needs head dim 64 (got %d)", D);
    attn::attn_delta_bf16<<<ceil_div(rows * 32, 256), 256, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(ctx), static_cast<const __nv_bfloat16*>(dctx), S, H, A,
        rows, delta);
    dim3 grid(ceil_div(S, attn::TQ), A, B);
    const auto* q = static_cast<const __nv_bfloat16*>(qkv);
    const auto* o = static_cast<const __nv_bfloat16*>(dctx);
    auto* dq = static_cast<__nv_bfloat16*>(dqkv);
    attn::attn_bwd_dkdv_bf16<<<grid, attn::NTHR, 0, stream>>>(q, o, lse, delta, lens, S, H, dq,
                                                               status);
    attn::attn_bwd_dq_bf16<<<grid, attn::NTHR, 0, stream>>>(q, o, lse, delta, lens, S, H, dq,
                                                             status);
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
