// Row-wise and element-wise kernels of the encoder layer: residual +
// LayerNorm forward and backward (post-LN placement, biased variance),
// bias + GELU forward and GELU backward, and deterministic column sums (the
// bias / gamma / beta gradients).
//
// All are HBM-bound.  One warp owns one row; every lane moves 16-byte vectors
// (8 bf16 or 4 fp32) so a warp touches 512 contiguous bytes per access; row
// statistics are fp32, two-pass in registers, reduced with warp shuffles.
// Column sums never use floating-point atomics: each CTA writes per-column
// partials, and a second pass adds them in a fixed order.
#include <algorithm>

#include "common.cuh"
#include "ptx.cuh"
#include "gemm.h"
#include "rowwise.h"

namespace sky {
namespace rw {

// 8 consecutive elements <-> fp32 registers (one 16-byte bf16 vector or two
// 16-byte fp32 vectors).
__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
  const float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 raw = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat16* e = reinterpret_cast<const __nv_bfloat16*>(&raw);
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = __bfloat162float(e[i]);
}
__device__ __forceinline__ void store8(float* p, const float (&v)[8]) {
  reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
  reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
}
__device__ __forceinline__ void store8(__nv_bfloat16* p, const float (&v)[8]) {
  uint4 raw;
  __nv_bfloat16* e = reinterpret_cast<__nv_bfloat16*>(&raw);
#pragma unroll
  for (int i = 0; i < 8; ++i) e[i] = __float2bfloat16_rn(v[i]);
  *reinterpret_cast<uint4*>(p) = raw;
}

constexpr int LN_WARPS = 8;
constexpr int V = 8;  // elements per lane per chunk; chunk c of a lane starts at (c*32+lane)*8

// u = a + r (the linear layer's output plus the fp32 residual stream), then
// y = gamma * (u - mean) * rstd + beta.  u is written back (u_out may alias a)
// for the backward pass; y goes to y32 (fp32) and/or yT (slice dtype).
template <typename T, int NV>
__global__ void __launch_bounds__(LN_WARPS * 32) ln_fwd_kernel(
    const float* a, const float* __restrict__ r, const T* __restrict__ gamma,
    const T* __restrict__ beta, int rows, int H, float eps, float* u_out,
    float* __restrict__ y32, T* __restrict__ yT, float* __restrict__ mean_out,
    float* __restrict__ rstd_out) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int warp = blockIdx.x * LN_WARPS + (threadIdx.x >> 5);
  const int nwarps = gridDim.x * LN_WARPS;
  const float invH = 1.f / H;
  for (int row = warp; row < rows; row += nwarps) {
    float x[NV][V];
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < NV; ++c) {
      const int col = (c * 32 + lane) * V;
      if (col < H) {
        const int64_t off = (int64_t)row * H + col;
        load8(a + off, x[c]);
        if (r) {
          float rv[V];
          load8(r + off, rv);
#pragma unroll
          for (int i = 0; i < V; ++i) x[c][i] += rv[i];
        }
#pragma unroll
        for (int i = 0; i < V; ++i) s += x[c][i];
      }
    }
    const float mu = warp_sum(s) * invH;
    float q = 0.f;
#pragma unroll
    for (int c = 0; c < NV; ++c) {
      const int col = (c * 32 + lane) * V;
      if (col < H) {
#pragma unroll
        for (int i = 0; i < V; ++i) {
          const float d = x[c][i] - mu;
          q += d * d;
        }
      }
    }
    const float rs = rsqrtf(warp_sum(q) * invH + eps);
#pragma unroll
    for (int c = 0; c < NV; ++c) {
      const int col = (c * 32 + lane) * V;
      if (col < H) {
        const int64_t off = (int64_t)row * H + col;
        float gm[V], bt[V], o[V];
        load8(gamma + col, gm);
        load8(beta + col, bt);
#pragma unroll
        for (int i = 0; i < V; ++i) o[i] = gm[i] * ((x[c][i] - mu) * rs) + bt[i];
        if (u_out) store8(u_out + off, x[c]);
        if (y32) store8(y32 + off, o);
        if (yT) store8(yT + off, o);
      }
    }
    if (lane == 0) {
      mean_out[row] = mu;
      rstd_out[row] = rs;
    }
  }
}

// du = rstd * (g - mean(g) - xhat * mean(g * xhat)), g = dy * gamma with
// dy = dy + dy2 (the two gradient contributions of a residual branch point,
// dy2 optional), and the per-CTA column partials of dy * xhat, dy and du.
// Each warp keeps its running
// column sums in its own shared-memory rows (red[w][k][:]), which keeps the
// register count low enough for two or more CTAs per SM; at the end the CTA's
// warps are added in order into part[k][blockIdx.x][:].
template <typename TDY, typename T, int NV>
__global__ void __launch_bounds__(LN_WARPS * 32) ln_bwd_kernel(
    const TDY* __restrict__ dy, const float* __restrict__ dy2, const float* __restrict__ u,
    const T* __restrict__ gamma,
    const float* __restrict__ mean, const float* __restrict__ rstd, int rows, int H,
    float* __restrict__ du32, T* __restrict__ duT, float* __restrict__ part) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ float red[];  // [LN_WARPS][3][H]
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const int warp = blockIdx.x * LN_WARPS + wib;
  const int nwarps = gridDim.x * LN_WARPS;
  float* mine = red + (size_t)wib * 3 * H;
  for (int i = lane * 4; i < 3 * H; i += 128) *reinterpret_cast<float4*>(mine + i) = make_float4(0.f, 0.f, 0.f, 0.f);
  __syncwarp();
  const float invH = 1.f / H;
  for (int row = warp; row < rows; row += nwarps) {
    const float mu = mean[row], rs = rstd[row];
    float xh[NV][V], dyv[NV][V];
    float s1 = 0.f, s2 = 0.f;
#pragma unroll
    for (int c = 0; c < NV; ++c) {
      const int col = (c * 32 + lane) * V;
      if (col < H) {
        const int64_t off = (int64_t)row * H + col;
        load8(u + off, xh[c]);
        load8(dy + off, dyv[c]);
        if (dy2) {
          float d2[V];
          load8(dy2 + off, d2);
#pragma unroll
          for (int i = 0; i < V; ++i) dyv[c][i] += d2[i];
        }
      }
    }
#pragma unroll
    for (int c = 0; c < NV; ++c) {
      const int col = (c * 32 + lane) * V;
      if (col < H) {
        float gm[V];
        load8(gamma + col, gm);
#pragma unroll
        for (int i = 0; i < V; ++i) {
          xh[c][i] = (xh[c][i] - mu) * rs;
          const float g = dyv[c][i] * gm[i];
          s1 += g;
          s2 += g * xh[c][i];
        }
      }
    }
    const float mg = warp_sum(s1) * invH, mgx = warp_sum(s2) * invH;
#pragma unroll
    for (int c = 0; c < NV; ++c) {
      const int col = (c * 32 + lane) * V;
      if (col < H) {
        float gm[V], o[V], pg[V], pb[V], pu[V];
        load8(gamma + col, gm);
        load8(mine + col, pg);
        load8(mine + H + col, pb);
        load8(mine + 2 * H + col, pu);
#pragma unroll
        for (int i = 0; i < V; ++i) {
          o[i] = rs * (dyv[c][i] * gm[i] - mg - xh[c][i] * mgx);
          pg[i] += dyv[c][i] * xh[c][i];
          pb[i] += dyv[c][i];
          pu[i] += o[i];
        }
        store8(mine + col, pg);
        store8(mine + H + col, pb);
        store8(mine + 2 * H + col, pu);
        if (du32) store8(du32 + (int64_t)row * H + col, o);
        if (duT) store8(duT + (int64_t)row * H + col, o);
      }
    }
  }
  __syncthreads();
  for (int k = 0; k < 3; ++k) {
    for (int col = threadIdx.x; col < H; col += blockDim.x) {
      float s = 0.f;
      for (int w = 0; w < LN_WARPS; ++w) s += red[((size_t)w * 3 + k) * H + col];
      part[((int64_t)k * gridDim.x + blockIdx.x) * H + col] = s;
    }
  }
}

// out = a + b (fp32 inputs) in fp32 or bf16.
template <typename T>
__global__ void add_kernel(const float* __restrict__ a, const float* __restrict__ b, int64_t n,
                           T* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    out[i] = from_f32<T>(a[i] + b[i]);
}

__global__ void to_bf16_kernel(const float* __restrict__ x, int64_t n,
                               __nv_bfloat16* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    out[i] = __float2bfloat16_rn(x[i]);
}

template <typename T>
__global__ void to_f32_kernel(const T* __restrict__ x, int64_t n, float* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    out[i] = to_f32(x[i]);
}

// LayerNorm backward, streamed through shared memory (bf16 slices, H = 1024
// or less, H % 256 == 0).  One persistent CTA per SM owns a contiguous block
// of rows.  A producer thread keeps RING rows of (u, dy, dy2) in flight with
// 1-D bulk copies into a shared-memory ring; 8 pairs of consumer warps take
// rows round-robin, the two warps of a pair one half of the row's columns
// each (16 per lane, two 8-wide chunks), and compute
//   du = rstd * (g - mean(g) - xhat * mean(g * xhat)),  g = (dy + dy2) * gamma
// The pair adds its two halves' row sums in a fixed order through shared
// memory (one named barrier per row), and each warp keeps the column sums of
// dy*xhat, dy and du for its columns in registers -- 48 a lane, which lets 16
// consumer warps share an SM.  At the end the 8 pairs' sums are added in
// order into part[k][blockIdx.x][:].
constexpr int SB_PAIRS = 8, SB_WARPS = 2 * SB_PAIRS, SB_RING = 16, SB_NV = 2;  // H <= 1024
constexpr int SB_ROW_BYTES = 3 * 1024 * 4;                                     // u, dy, dy2 (fp32)

// part[k][blockIdx.x][:] = sum over the consumer pairs (in order) of acc.
__device__ __forceinline__ void sb_flush(const float (&acc)[SB_NV][8], int k, float* red,
                                         float* __restrict__ part, int H) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp < SB_WARPS) {
    const int pr = warp >> 1, hh = warp & 1, half = H / 2;
#pragma unroll
    for (int c = 0; c < SB_NV; ++c) {
      const int col = (c * 32 + lane) * 8;
      if (col < half) store8(red + pr * H + hh * half + col, acc[c]);
    }
  }
  __syncthreads();
  for (int col = threadIdx.x; col < H; col += blockDim.x) {
    float s = 0.f;
    for (int w = 0; w < SB_PAIRS; ++w) s += red[w * H + col];
    part[(static_cast<int64_t>(k) * gridDim.x + blockIdx.x) * H + col] = s;
  }
  __syncthreads();
}

__device__ __forceinline__ void pair_sync(int pair) {
  asm volatile("bar.sync %0, 64;" ::"r"(1 + pair) : "memory");
}

template <typename TDY>
__global__ void __launch_bounds__(32 * (SB_WARPS + 1), 1) ln_bwd_stream_kernel(
    const TDY* __restrict__ dy, const float* __restrict__ dy2, const float* __restrict__ u,
    const __nv_bfloat16* __restrict__ gamma, const float* __restrict__ mean,
    const float* __restrict__ rstd, int rows, int H, float* __restrict__ du32,
    __nv_bfloat16* __restrict__ duT, float* __restrict__ part, int32_t* status) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ uint8_t sm_raw[];
  uint8_t* sm = sm_raw + ((128 - (ptx::smem_u32(sm_raw) & 127)) & 127);
  uint64_t* full = reinterpret_cast<uint64_t*>(sm + SB_RING * SB_ROW_BYTES);
  uint64_t* empty = full + SB_RING;
  // per pair, row parity and half: {partial sum of g, of g * xhat, ok flag}
  float* xch = reinterpret_cast<float*>(empty + SB_RING);
  float* sgm = xch + SB_PAIRS * 2 * 2 * 4;  // gamma as fp32 [H]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = (rows + gridDim.x - 1) / gridDim.x;
  const int r0 = blockIdx.x * per, r1 = min(rows, r0 + per);
  const int n = r1 > r0 ? r1 - r0 : 0;
  const uint32_t ubytes = H * 4, dbytes = H * sizeof(TDY);
  const uint64_t lim = 2000000000ull;
  for (int c = threadIdx.x; c < H; c += blockDim.x) sgm[c] = __bfloat162float(gamma[c]);
  if (threadIdx.x == 0) {
    for (int s = 0; s < SB_RING; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 64);  // the two warps of the row's pair
    }
    ptx::fence_mbar_init();
    ptx::fence_proxy_async_smem();
  }
  __syncthreads();
  float pg[SB_NV][8] = {}, pb[SB_NV][8] = {}, pu[SB_NV][8] = {};  // column sums (consumers)
  if (warp == SB_WARPS) {
    // producer
    if (lane == 0) {
      for (int i = 0; i < n; ++i) {
        const int s = i % SB_RING;
        if (!ptx::mbar_wait(&empty[s], ((i / SB_RING) & 1) ^ 1u, lim, status, 5000)) break;
        uint8_t* slot = sm + s * SB_ROW_BYTES;
        const int64_t row = r0 + i;
        ptx::mbar_arrive_expect_tx(&full[s], ubytes + dbytes + (dy2 ? ubytes : 0));
        ptx::bulk_load(slot, u + row * H, ubytes, &full[s]);
        ptx::bulk_load(slot + 4096, dy + row * H, dbytes, &full[s]);
        if (dy2) ptx::bulk_load(slot + 8192, dy2 + row * H, ubytes, &full[s]);
      }
    }
    // wait (bounded) for the last copies before the CTA may exit
    if (lane == 0)
      for (int i = n - 1; i >= 0 && i >= n - SB_RING; --i)
        ptx::mbar_wait(&full[i % SB_RING], (i / SB_RING) & 1, lim, status, 5000);
  } else {
    const float invH = 1.f / H;
    const int pr = warp >> 1, hh = warp & 1, half = H / 2;
    for (int i = pr, it = 0; i < n; i += SB_PAIRS, ++it) {
      const int s = i % SB_RING;
      const int64_t row = r0 + i;
      const float mu = mean[row], rs = rstd[row];
      const bool ok = __all_sync(0xffffffffu, ptx::mbar_wait(&full[s], (i / SB_RING) & 1, lim, status, 5000));
      const uint8_t* slot = sm + s * SB_ROW_BYTES;
      const float* su = reinterpret_cast<const float*>(slot) + hh * half;
      const TDY* sdy = reinterpret_cast<const TDY*>(slot + 4096) + hh * half;
      const float* sd2 = reinterpret_cast<const float*>(slot + 8192) + hh * half;
      const float* sg = sgm + hh * half;
      // x-hat and dy (+ dy2) of 8 columns of this warp's half, read from the slot
      auto fetch = [&](int col, float (&xh)[8], float (&d)[8]) {
        load8(su + col, xh);
        load8(sdy + col, d);
        if (dy2) {
          float e[8];
          load8(sd2 + col, e);
#pragma unroll
          for (int k = 0; k < 8; ++k) d[k] += e[k];
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) xh[k] = (xh[k] - mu) * rs;
      };
      float s1 = 0.f, s2 = 0.f;
#pragma unroll
      for (int c = 0; c < SB_NV; ++c) {
        const int col = (c * 32 + lane) * 8;
        if (col < half) {
          float xh[8], d[8], gm[8];
          fetch(col, xh, d);
          load8(sg + col, gm);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float g = d[k] * gm[k];
            s1 += g;
            s2 += g * xh[k];
          }
        }
      }
      s1 = warp_sum(s1);
      s2 = warp_sum(s2);
      // the pair's two halves, added in a fixed order (low half first)
      float* xp = xch + ((pr * 2 + (it & 1)) * 2) * 4;
      if (lane == 0) {
        xp[hh * 4 + 0] = s1;
        xp[hh * 4 + 1] = s2;
        xp[hh * 4 + 2] = ok ? 1.f : 0.f;
      }
      pair_sync(pr);
      if (xp[2] == 0.f || xp[4 + 2] == 0.f) break;  // either warp timed out: the pair stops
      const float mg = (xp[0] + xp[4]) * invH, mgx = (xp[1] + xp[4 + 1]) * invH;
      // second pass re-reads the slot instead of holding the row in registers
#pragma unroll
      for (int c = 0; c < SB_NV; ++c) {
        const int col = (c * 32 + lane) * 8;
        if (col < half) {
          float xh[8], d[8], gm[8], o[8];
          fetch(col, xh, d);
          load8(sg + col, gm);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            o[k] = rs * (d[k] * gm[k] - mg - xh[k] * mgx);
            pg[c][k] += d[k] * xh[k];
            pb[c][k] += d[k];
            pu[c][k] += o[k];
          }
          const int64_t off = row * H + hh * half + col;
          if (du32) store8(du32 + off, o);
          if (duT) store8(duT + off, o);
        }
      }
      __syncwarp();
      ptx::mbar_arrive(&empty[s]);  // slot s may be refilled once both warps are done
    }
  }
  // every row's copy has landed and been consumed: the ring is free for the
  // CTA's fixed-order reduction of the 8 pairs' column sums
  __syncthreads();
  float* red = reinterpret_cast<float*>(sm);  // [SB_PAIRS][H]
  sb_flush(pg, 0, red, part, H);
  sb_flush(pb, 1, red, part, H);
  sb_flush(pu, 2, red, part, H);
}

// out_k[n] = sum_b part[k][b][n] for the non-null outputs, in a fixed order:
// CTA (cx, k) owns 32 columns; warp w of its RP_WARPS warps adds the partial
// rows b = w + RP_WARPS * (4 i + j) into accumulator j (coalesced 128-byte
// reads, four rows in flight per warp), the four accumulators are added as
// (a0 + a1) + (a2 + a3), and the warp sums are added in warp order.
constexpr int RP_WARPS = 16;
__global__ void __launch_bounds__(RP_WARPS * 32) reduce_partials(const float* __restrict__ part,
                                                                 int nblk, int N, float* out0,
                                                                 float* out1, float* out2) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[RP_WARPS][33];
  const int k = blockIdx.y;
  float* out = k == 0 ? out0 : (k == 1 ? out1 : out2);
  if (out == nullptr) return;  // uniform over the CTA
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int n = blockIdx.x * 32 + lane;
  float a[4] = {0.f, 0.f, 0.f, 0.f};
  if (n < N) {
    const float* p = part + (int64_t)k * nblk * N + n;
    int b = w;
    for (; b + 3 * RP_WARPS < nblk; b += 4 * RP_WARPS) {
      float v[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) v[j] = p[(int64_t)(b + j * RP_WARPS) * N];
#pragma unroll
      for (int j = 0; j < 4; ++j) a[j] += v[j];
    }
    // fewer than four rows left: at most three
    if (b < nblk) a[0] += p[(int64_t)b * N];
    if (b + RP_WARPS < nblk) a[1] += p[(int64_t)(b + RP_WARPS) * N];
    if (b + 2 * RP_WARPS < nblk) a[2] += p[(int64_t)(b + 2 * RP_WARPS) * N];
  }
  red[w][lane] = (a[0] + a[1]) + (a[2] + a[3]);
  __syncthreads();
  if (w == 0 && n < N) {
    float t = 0.f;
#pragma unroll
    for (int j = 0; j < RP_WARPS; ++j) t += red[j][lane];
    out[n] = t;
  }
}

// Several fixed-order column reductions in one launch: segment y = blockIdx.y
// computes segs[y].out[n] = sum_b segs[y].part[b][n] over its rows, exactly
// as reduce_partials does (so the same partials give the same bits).
__global__ void __launch_bounds__(RP_WARPS * 32) reduce_segments(const ColSegments segs) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[RP_WARPS][33];
  const ColSegment& sg = segs.seg[blockIdx.y];
  const int N = sg.cols, nblk = sg.rows;
  if (blockIdx.x * 32 >= N) return;  // uniform over the CTA
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int n = blockIdx.x * 32 + lane;
  float a[4] = {0.f, 0.f, 0.f, 0.f};
  if (n < N) {
    const float* p = sg.part + n;
    int b = w;
    for (; b + 3 * RP_WARPS < nblk; b += 4 * RP_WARPS) {
      float v[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) v[j] = p[(int64_t)(b + j * RP_WARPS) * N];
#pragma unroll
      for (int j = 0; j < 4; ++j) a[j] += v[j];
    }
    if (b < nblk) a[0] += p[(int64_t)b * N];
    if (b + RP_WARPS < nblk) a[1] += p[(int64_t)(b + RP_WARPS) * N];
    if (b + 2 * RP_WARPS < nblk) a[2] += p[(int64_t)(b + 2 * RP_WARPS) * N];
  }
  red[w][lane] = (a[0] + a[1]) + (a[2] + a[3]);
  __syncthreads();
  if (w == 0 && n < N) {
    float t = 0.f;
#pragma unroll
    for (int j = 0; j < RP_WARPS; ++j) t += red[j][lane];
    sg.out[n] = t;
  }
}

// Column partial sums of x[T, N] (N % 8 == 0): CTA (cx, g) owns columns
// [256 cx, 256 cx + 256); warp w of the CTA adds rows 8 g + w, + 8 G, ...
// with 16-byte loads (a warp reads 512 contiguous bytes of bf16 per row), the
// CTA's 8 warps are added in order and part[g][n] is written.
template <typename T>
__global__ void __launch_bounds__(256) colsum_partial(const T* __restrict__ x, int rows, int N,
                                                      float* __restrict__ part) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[8][256];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int col = blockIdx.x * 256 + lane * 8;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (col < N) {
    const int step = gridDim.y * 8;
    int r = blockIdx.y * 8 + w;
    for (; r + 3 * step < rows; r += 4 * step) {
      float v[4][8];
#pragma unroll
      for (int k = 0; k < 4; ++k) load8(x + (int64_t)(r + k * step) * N + col, v[k]);
#pragma unroll
      for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] += v[k][i];
    }
    for (; r < rows; r += step) {
      float v[8];
      load8(x + (int64_t)r * N + col, v);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] += v[i];
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) red[w][lane * 8 + i] = acc[i];
  __syncthreads();
  const int c = blockIdx.x * 256 + threadIdx.x;
  if (c < N) {
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) s += red[k][threadIdx.x];
    part[(int64_t)blockIdx.y * N + c] = s;
  }
}

template <typename T>
__global__ void bias_gelu_kernel(const T* __restrict__ z, const T* __restrict__ bias, int64_t n,
                                 int N, T* __restrict__ hpre, T* __restrict__ g) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const float h = to_f32(z[i]) + (bias ? to_f32(bias[i % N]) : 0.f);
    hpre[i] = from_f32<T>(h);
    g[i] = from_f32<T>(gelu_f(h));
  }
}

template <typename T>
__global__ void gelu_bwd_kernel(const T* __restrict__ dg, const T* __restrict__ hpre, int64_t n,
                                T* __restrict__ dh) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    dh[i] = from_f32<T>(to_f32(dg[i]) * gelu_grad_f(to_f32(hpre[i])));
}

int ln_blocks(int rows) {
  const int want = ceil_div(rows, LN_WARPS);
  const int cap = 4 * (sm_count() > 0 ? sm_count() : 148);
  return want < cap ? want : cap;
}
int stream_blocks() { return sm_count() > 0 ? sm_count() : 148; }
// Backward CTAs also write column partials, so fewer, longer-lived CTAs.
int ln_bwd_blocks(int rows) {
  const int want = ceil_div(rows, LN_WARPS);
  const int cap = 2 * (sm_count() > 0 ? sm_count() : 148);
  return want < cap ? want : cap;
}

template <typename T, int NV>
void ln_fwd_launch(const float* a, const float* r, const void* gm, const void* bt, int rows, int H,
                   float eps, float* u_out, float* y32, void* y, float* mean, float* rstd,
                   cudaStream_t st) {
  launch_pdl(ln_fwd_kernel<T, NV>, dim3(ln_blocks(rows)), dim3(LN_WARPS * 32), 0, st, 1, 
      a, r, static_cast<const T*>(gm), static_cast<const T*>(bt), rows, H, eps, u_out, y32,
      static_cast<T*>(y), mean, rstd);
}
template <typename TDY, typename T, int NV>
void ln_bwd_launch(const void* dy, const float* dy2, const float* u, const void* gm,
                   const float* mean, const float* rstd, int rows, int H, float* du32, void* du,
                   float* part, int nblk, cudaStream_t st) {
  const size_t smem = (size_t)LN_WARPS * 3 * H * sizeof(float);
  if (smem > 48 * 1024)
    cudaFuncSetAttribute(ln_bwd_kernel<TDY, T, NV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
  launch_pdl(ln_bwd_kernel<TDY, T, NV>, dim3(nblk), dim3(LN_WARPS * 32), smem, st, 1, 
      static_cast<const TDY*>(dy), dy2, u, static_cast<const T*>(gm), mean, rstd, rows, H, du32,
      static_cast<T*>(du), part);
}

}  // namespace rw

// ------------------------------------------------------------------- host
namespace {
constexpr int kMaxNV = 8;
int lane_vectors(int H) { return ceil_div(H, 32 * rw::V); }
}  // namespace

#define SKY_NV_DISPATCH(NVV, CALL) \
  switch (NVV) {                   \
    case 1: CALL(1); break;        \
    case 2: CALL(2); break;        \
    case 3: CALL(3); break;        \
    case 4: CALL(4); break;        \
    case 5: CALL(5); break;        \
    case 6: CALL(6); break;        \
    case 7: CALL(7); break;        \
    default: CALL(8); break;       \
  }

namespace {
// the row kernels move 16-byte vectors (and bulk-copy rows), so every [rows, H]
// tensor and gamma, beta must start on a 16-byte boundary (null is accepted)
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }
}  // namespace

sky_status layernorm_fwd(const float* a, const float* r, const void* gamma, const void* beta,
                         int rows, int H, float eps, sky_dtype dt, float* u_out, float* y32,
                         void* y, float* mean, float* rstd, cudaStream_t st) {
  SKY_CHECK(aligned16(a) && aligned16(r) && aligned16(gamma) && aligned16(beta) &&
                aligned16(u_out) && aligned16(y32) && aligned16(y),
            SKY_ERR_UNSUPPORTED, "LayerNorm tensors must be 16-byte aligned");
  SKY_CHECK(H % rw::V == 0 && lane_vectors(H) <= kMaxNV && (dt == SKY_DTYPE_BF16 || H <= 1024),
            SKY_ERR_UNSUPPORTED, "LayerNorm width %d unsupported", H);
  SKY_CHECK(y32 || y, SKY_ERR_INVALID_ARG, "LayerNorm forward needs an output");
  const int nv = lane_vectors(H);
  if (dt == SKY_DTYPE_BF16) {
#define LNF(NV) rw::ln_fwd_launch<__nv_bfloat16, NV>(a, r, gamma, beta, rows, H, eps, u_out, y32, y, mean, rstd, st)
    SKY_NV_DISPATCH(nv, LNF)
#undef LNF
  } else {
    // fp32 slices: the dtype output is itself fp32, so one store suffices
    float* only = y32 ? y32 : static_cast<float*>(y);
#define LNF(NV) rw::ln_fwd_launch<float, NV>(a, r, gamma, beta, rows, H, eps, u_out, only, nullptr, mean, rstd, st)
    SKY_NV_DISPATCH(nv, LNF)
#undef LNF
    if (y32 && y && y != y32)
      SKY_CUDA(cudaMemcpyAsync(y, y32, (size_t)rows * H * 4, cudaMemcpyDeviceToDevice, st));
  }
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "layernorm forward launch");
}

size_t layernorm_bwd_ws(int rows, int H) {
  return (size_t)3 * rw::ln_bwd_blocks(rows) * H * sizeof(float);
}

sky_status layernorm_bwd(const void* dy, sky_dtype dy_dt, const float* dy2, const float* u,
                         const void* gamma, const float* mean, const float* rstd, int rows, int H,
                         sky_dtype dt, float* du32, void* du, float* dgamma, float* dbeta,
                         float* dbias, void* ws, size_t ws_bytes, cudaStream_t st,
                         int* deferred_parts, int32_t* status) {
  SKY_CHECK(aligned16(dy) && aligned16(dy2) && aligned16(u) && aligned16(gamma) &&
                aligned16(du32) && aligned16(du),
            SKY_ERR_UNSUPPORTED, "LayerNorm tensors must be 16-byte aligned");
  SKY_CHECK(H % rw::V == 0 && lane_vectors(H) <= kMaxNV && (dt == SKY_DTYPE_BF16 || H <= 1024),
            SKY_ERR_UNSUPPORTED, "LayerNorm width %d unsupported", H);
  SKY_CHECK(du32 || du, SKY_ERR_INVALID_ARG, "LayerNorm backward needs an output");
  const int nblk = rw::ln_bwd_blocks(rows);
  SKY_CHECK(ws && ws_bytes >= (size_t)3 * nblk * H * sizeof(float), SKY_ERR_INVALID_ARG,
            "LayerNorm backward workspace too small");
  float* part = static_cast<float*>(ws);
  const int nv = lane_vectors(H);
  if (dt == SKY_DTYPE_BF16 && H <= 1024 && H % 256 == 0 && rw::stream_blocks() <= nblk) {
    // streamed variant: one CTA per SM, rows staged through shared memory
    const int sb = rw::stream_blocks();
    const size_t fixed = (size_t)rw::SB_RING * rw::SB_ROW_BYTES + 2 * rw::SB_RING * 8 +
                         (size_t)rw::SB_PAIRS * 2 * 2 * 4 * 4 + 128;
    const size_t smem = fixed + (size_t)H * 4;
    // the attribute is set once, for the largest H this variant takes
    const size_t smem_max = fixed + 1024 * 4;
    const int threads = 32 * (rw::SB_WARPS + 1);
    if (dy_dt == SKY_DTYPE_BF16) {
      static cudaError_t a = cudaFuncSetAttribute(rw::ln_bwd_stream_kernel<__nv_bfloat16>,
                                                  cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_max);
      if (a != cudaSuccess) return cuda_fail(a, "LayerNorm backward smem attribute");
      launch_pdl(rw::ln_bwd_stream_kernel<__nv_bfloat16>, dim3(sb), dim3(threads), smem, st, 1, 
          static_cast<const __nv_bfloat16*>(dy), dy2, u, static_cast<const __nv_bfloat16*>(gamma),
          mean, rstd, rows, H, du32, static_cast<__nv_bfloat16*>(du), part, status);
    } else {
      static cudaError_t a = cudaFuncSetAttribute(rw::ln_bwd_stream_kernel<float>,
                                                  cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_max);
      if (a != cudaSuccess) return cuda_fail(a, "LayerNorm backward smem attribute");
      launch_pdl(rw::ln_bwd_stream_kernel<float>, dim3(sb), dim3(threads), smem, st, 1, 
          static_cast<const float*>(dy), dy2, u, static_cast<const __nv_bfloat16*>(gamma), mean,
          rstd, rows, H, du32, static_cast<__nv_bfloat16*>(du), part, status);
    }
    count_launches(1);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "layernorm backward launch");
    if (deferred_parts) {
      *deferred_parts = sb;
      return SKY_OK;
    }
    return layernorm_bwd_reduce(part, sb, H, dgamma, dbeta, dbias, st);
  }
  if (dt == SKY_DTYPE_BF16) {
    if (dy_dt == SKY_DTYPE_BF16) {
#define LNB(NV) rw::ln_bwd_launch<__nv_bfloat16, __nv_bfloat16, NV>(dy, dy2, u, gamma, mean, rstd, rows, H, du32, du, part, nblk, st)
      SKY_NV_DISPATCH(nv, LNB)
#undef LNB
    } else {
#define LNB(NV) rw::ln_bwd_launch<float, __nv_bfloat16, NV>(dy, dy2, u, gamma, mean, rstd, rows, H, du32, du, part, nblk, st)
      SKY_NV_DISPATCH(nv, LNB)
#undef LNB
    }
  } else {
    float* only = du32 ? du32 : static_cast<float*>(du);
#define LNB(NV) rw::ln_bwd_launch<float, float, NV>(dy, dy2, u, gamma, mean, rstd, rows, H, only, nullptr, part, nblk, st)
    SKY_NV_DISPATCH(nv, LNB)
#undef LNB
    if (du32 && du && du != du32)
      SKY_CUDA(cudaMemcpyAsync(du, du32, (size_t)rows * H * 4, cudaMemcpyDeviceToDevice, st));
  }
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "layernorm backward launch");
  if (deferred_parts) {
    *deferred_parts = nblk;
    return SKY_OK;
  }
  return layernorm_bwd_reduce(part, nblk, H, dgamma, dbeta, dbias, st);
}

sky_status layernorm_bwd_reduce(const void* ws, int parts, int H, float* dgamma, float* dbeta,
                                float* dbias, cudaStream_t st) {
  dim3 grid(ceil_div(H, 32), 3);
  launch_pdl(rw::reduce_partials, dim3(grid), dim3(rw::RP_WARPS * 32), 0, st, 1, static_cast<const float*>(ws), parts, H, dgamma,
                                            dbeta, dbias);
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "layernorm backward reduce launch");
}

sky_status reduce_column_segments(const ColSegments& segs, cudaStream_t st) {
  if (segs.n <= 0) return SKY_OK;
  int max_cols = 0;
  for (int i = 0; i < segs.n; ++i) max_cols = std::max(max_cols, segs.seg[i].cols);
  launch_pdl(rw::reduce_segments, dim3(ceil_div(max_cols, 32), segs.n), dim3(rw::RP_WARPS * 32), 0,
             st, 1, segs);
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "column-segment reduce launch");
}

namespace gemm {
cudaError_t reduce_rows_f32(const float* part, int rows, int N, float* out, cudaStream_t stream) {
  launch_pdl(rw::reduce_partials, dim3(dim3(ceil_div(N, 32), 1)), dim3(rw::RP_WARPS * 32), 0, stream, 1, part, rows, N, out, nullptr,
                                                                  nullptr);
  count_launches(1);
  return cudaGetLastError();
}
}  // namespace gemm

sky_status add_f32(const float* a, const float* b, int64_t n, sky_dtype out_dt, void* out,
                   cudaStream_t st) {
  if (n <= 0) return SKY_OK;
  const int blocks = (int)std::min<int64_t>(ceil_div(n, 256), 8 * 148);
  if (out_dt == SKY_DTYPE_BF16)
    launch_pdl(rw::add_kernel<__nv_bfloat16>, dim3(blocks), dim3(256), 0, st, 1, a, b, n, static_cast<__nv_bfloat16*>(out));
  else
    launch_pdl(rw::add_kernel<float>, dim3(blocks), dim3(256), 0, st, 1, a, b, n, static_cast<float*>(out));
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "add launch");
}

sky_status f32_to_bf16(const float* x, int64_t n, void* out, cudaStream_t st) {
  if (n <= 0) return SKY_OK;
  const int blocks = (int)std::min<int64_t>(ceil_div(n, 256), 8 * 148);
  launch_pdl(rw::to_bf16_kernel, dim3(blocks), dim3(256), 0, st, 1, x, n, static_cast<__nv_bfloat16*>(out));
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "narrow launch");
}

sky_status to_f32(const void* x, int64_t n, sky_dtype dt, float* out, cudaStream_t st) {
  if (n <= 0) return SKY_OK;
  const int blocks = (int)std::min<int64_t>(ceil_div(n, 256), 8 * 148);
  if (dt == SKY_DTYPE_BF16)
    launch_pdl(rw::to_f32_kernel<__nv_bfloat16>, dim3(blocks), dim3(256), 0, st, 1, 
        static_cast<const __nv_bfloat16*>(x), n, out);
  else
    launch_pdl(rw::to_f32_kernel<float>, dim3(blocks), dim3(256), 0, st, 1, static_cast<const float*>(x), n, out);
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "widen launch");
}

namespace {
int colsum_row_groups(int rows, int N) {
  const int cb = ceil_div(N, 256);
  int g = 2 * (sm_count() > 0 ? sm_count() : 148) / cb;
  const int max_g = ceil_div(rows, 8);
  if (g > max_g) g = max_g;
  if (g > 65535) g = 65535;
  return g < 1 ? 1 : g;
}
}  // namespace

size_t column_sum_ws(int rows, int N) {
  return (size_t)colsum_row_groups(rows, N) * N * sizeof(float);
}

sky_status column_sum(const void* x, int rows, int N, sky_dtype dt, float* out, void* ws,
                      size_t ws_bytes, cudaStream_t st) {
  SKY_CHECK(N % 8 == 0, SKY_ERR_UNSUPPORTED, "column sum needs N %% 8 == 0 (got %d)", N);
  const int groups = colsum_row_groups(rows, N);
  SKY_CHECK(ws && ws_bytes >= (size_t)groups * N * sizeof(float), SKY_ERR_INVALID_ARG,
            "column-sum workspace too small");
  float* part = static_cast<float*>(ws);
  dim3 grid(ceil_div(N, 256), groups);
  if (dt == SKY_DTYPE_BF16)
    launch_pdl(rw::colsum_partial<__nv_bfloat16>, dim3(grid), dim3(256), 0, st, 1, 
        static_cast<const __nv_bfloat16*>(x), rows, N, part);
  else
    launch_pdl(rw::colsum_partial<float>, dim3(grid), dim3(256), 0, st, 1, static_cast<const float*>(x), rows, N, part);
  launch_pdl(rw::reduce_partials, dim3(dim3(ceil_div(N, 32), 1)), dim3(rw::RP_WARPS * 32), 0, st, 1, part, groups, N, out, nullptr,
                                                                nullptr);
  count_launches(2);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "column sum launch");
}

sky_status bias_gelu_fwd(const void* z, const void* bias, int rows, int N, sky_dtype dt,
                         void* hpre, void* g, cudaStream_t st) {
  const int64_t n = (int64_t)rows * N;
  const int blocks = (int)std::min<int64_t>(ceil_div(n, 256), 8 * 148);
  if (dt == SKY_DTYPE_BF16)
    rw::bias_gelu_kernel<__nv_bfloat16><<<blocks, 256, 0, st>>>(
        static_cast<const __nv_bfloat16*>(z), static_cast<const __nv_bfloat16*>(bias), n, N,
        static_cast<__nv_bfloat16*>(hpre), static_cast<__nv_bfloat16*>(g));
  else
    rw::bias_gelu_kernel<float><<<blocks, 256, 0, st>>>(static_cast<const float*>(z),
                                                        static_cast<const float*>(bias), n, N,
                                                        static_cast<float*>(hpre),
                                                        static_cast<float*>(g));
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "bias+GELU launch");
}

sky_status gelu_bwd(const void* dg, const void* hpre, int rows, int N, sky_dtype dt, void* dh,
                    cudaStream_t st) {
  const int64_t n = (int64_t)rows * N;
  const int blocks = (int)std::min<int64_t>(ceil_div(n, 256), 8 * 148);
  if (dt == SKY_DTYPE_BF16)
    rw::gelu_bwd_kernel<__nv_bfloat16><<<blocks, 256, 0, st>>>(
        static_cast<const __nv_bfloat16*>(dg), static_cast<const __nv_bfloat16*>(hpre), n,
        static_cast<__nv_bfloat16*>(dh));
  else
    rw::gelu_bwd_kernel<float><<<blocks, 256, 0, st>>>(static_cast<const float*>(dg),
                                                       static_cast<const float*>(hpre), n,
                                                       static_cast<float*>(dh));
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "GELU backward launch");
}

}  // namespace sky
