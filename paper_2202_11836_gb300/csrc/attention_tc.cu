// Masked scaled dot-product attention (Eq. 1) forward on the 5th-generation
// tensor cores, bf16, head dim D = 64.
//
// One CTA owns 128 query rows of one (sequence b, head a).  Per 64-key tile j
// (only tiles below len[b] are visited):
//   S_j = Q K_j^T                  tcgen05.mma M=128 N=64 K=64 -> TMEM
//   softmax (4 warps, thread = query row = TMEM lane): row max over the
//     valid keys, P_j = exp2(S_j log2(e)/sqrt(D) - m) written as bf16 to
//     shared memory in the 128-byte-swizzled K-major operand layout
//   O += P_j V_j                   tcgen05.mma M=128 N=64 K=64 -> TMEM
// Q, K and V come straight out of the packed QKV activations by TMA (one
// tensor map, per-head column offsets).  Because a thread owns a whole query
// row, the row max and row sum need no shuffles.  When a row's running max
// rises, that row of O is rescaled in TMEM (tcgen05.ld / st) before the next
// P V product is issued; the final O is divided by the row sum and the
// log-sum-exp is kept for the backward pass.  Everything in one CTA is
// sequential; three CTAs per SM (64 KB shared memory, 128 TMEM columns each)
// overlap one CTA's softmax with another's MMAs.  All mbarrier waits are
// time-bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "ptx.cuh"

namespace sky {
namespace attn_tc {

constexpr int BQ = 128, BKV = 64, HD = 64;
constexpr int Q_BYTES = BQ * HD * 2;    // 16 KiB
constexpr int KV_BYTES = BKV * HD * 2;  // 8 KiB per K or V tile
constexpr int P_BYTES = BQ * BKV * 2;   // 16 KiB
constexpr int STAGES = 2;
constexpr int Q_OFF = 0;
constexpr int K_OFF = Q_OFF + Q_BYTES;
constexpr int V_OFF = K_OFF + STAGES * KV_BYTES;
constexpr int P_OFF = V_OFF + STAGES * KV_BYTES;
constexpr int BAR_OFF = P_OFF + P_BYTES;
constexpr int SMEM_BYTES = BAR_OFF + 128 + 1024;
constexpr int TMEM_COLS = 128;  // S: columns [0, 64), O: [64, 128)
constexpr int NTHR = 192;       // warp 0 TMA, warp 1 MMA, warps 2..5 softmax
constexpr float LOG2E = 1.4426950408889634f;
constexpr float LN2 = 0.6931471805599453f;
// Suspend-time hint (ns) of every mbarrier wait: a waiting thread sleeps
// until the phase completes instead of spinning on issue slots that the
// softmax warps (the critical path) share with the producer and MMA threads.
constexpr uint32_t kWaitHint = 10000;

struct FwdParams {
  int S, H, A;
  const int32_t* lens;
  __nv_bfloat16* ctx;
  float* lse;
  int32_t* status;
  uint64_t timeout_ns;
};

__global__ void __launch_bounds__(NTHR, 2) attn_fwd_tc(const __grid_constant__ CUtensorMap tmQ,
                                                    const __grid_constant__ CUtensorMap tmKV,
                                                    const FwdParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + BAR_OFF);
  uint64_t* kv_full = q_full + 1;
  uint64_t* kv_empty = kv_full + STAGES;
  uint64_t* s_full = kv_empty + STAGES;
  uint64_t* p_full = s_full + 1;
  uint64_t* pv_done = p_full + 1;
  uint64_t* done = pv_done + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);

  const int qt = blockIdx.x, a = blockIdx.y, b = blockIdx.z;
  const int S = p.S, H = p.H;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int len = p.lens[b];
  if (len < 1 || len > S) {
    if (p.status && threadIdx.x == 0) atomicOr(p.status, kStatusBadLength);
    len = len < 1 ? 1 : S;
  }
  const int n_kt = (len + BKV - 1) / BKV;
  const int row0 = b * S;  // first token row of this sequence
  const int q0 = qt * BQ;
  const uint64_t lim = p.timeout_ns;

  if (threadIdx.x == 0) {
    ptx::mbar_init(q_full, 1);
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(&kv_full[s], 1);
      ptx::mbar_init(&kv_empty[s], 1);
    }
    ptx::mbar_init(s_full, 1);
    ptx::mbar_init(p_full, 128);
    ptx::mbar_init(pv_done, 1);
    ptx::mbar_init(done, 1);
    ptx::fence_mbar_init();
    ptx::fence_proxy_async_smem();
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, TMEM_COLS);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS = tmem, tO = tmem + 64;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      ptx::mbar_arrive_expect_tx(q_full, Q_BYTES);
      ptx::tma_load_2d(smem + Q_OFF, &tmQ, q_full, a * HD, row0 + q0);
      bool ok = true;
      int issued = 0;
      for (int j = 0; j < n_kt && ok; ++j) {
        const int st = j & 1;
        const uint32_t ph = (j >> 1) & 1;
        if (!ptx::mbar_wait(&kv_empty[st], ph ^ 1u, lim, p.status, kWaitHint)) { ok = false; break; }
        ptx::mbar_arrive_expect_tx(&kv_full[st], 2 * KV_BYTES);
        ptx::tma_load_2d(smem + K_OFF + st * KV_BYTES, &tmKV, &kv_full[st], H + a * HD,
                         row0 + j * BKV);
        ptx::tma_load_2d(smem + V_OFF + st * KV_BYTES, &tmKV, &kv_full[st], 2 * H + a * HD,
                         row0 + j * BKV);
        ++issued;
      }
      // drain: bounded waits for the copies still in flight
      ptx::mbar_wait(q_full, 0, lim, p.status, kWaitHint);
      for (int j = issued - 1; j >= 0 && j >= issued - STAGES; --j)
        ptx::mbar_wait(&kv_full[j & 1], (j >> 1) & 1, lim, p.status, kWaitHint);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issue
    if (lane == 0) {
      constexpr uint32_t idS = ptx::idesc_bf16_f32(BQ, BKV, false, false);
      constexpr uint32_t idO = ptx::idesc_bf16_f32(BQ, HD, false, true);
      const uint32_t sq = ptx::smem_u32(smem + Q_OFF), sp = ptx::smem_u32(smem + P_OFF);
      bool ok = ptx::mbar_wait(q_full, 0, lim, p.status, kWaitHint);
      for (int j = 0; j < n_kt && ok; ++j) {
        const int st = j & 1;
        const uint32_t ph = (j >> 1) & 1;
        if (!ptx::mbar_wait(&kv_full[st], ph, lim, p.status, kWaitHint)) break;
        ptx::tc_fence_after();
        const uint32_t sk = ptx::smem_u32(smem + K_OFF + st * KV_BYTES);
        const uint32_t sv = ptx::smem_u32(smem + V_OFF + st * KV_BYTES);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tS, ptx::smem_desc_sw128(sq + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sk + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
        ptx::tc_commit(s_full);
        if (!ptx::mbar_wait(p_full, j & 1, lim, p.status, kWaitHint)) break;
        ptx::tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < BKV / 16; ++kk)
          ptx::tc_mma_f16(tO, ptx::smem_desc_sw128(sp + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sv + kk * 2048, 8192, 1024), idO,
                          (j > 0 || kk > 0) ? 1u : 0u);
        ptx::tc_commit(pv_done);
        ptx::tc_commit(&kv_empty[st]);
      }
      ptx::tc_commit(done);
      ptx::mbar_wait(done, 0, lim, p.status, kWaitHint);
    }
  } else {
    // --------------------------------------------------- softmax / epilogue
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;  // query row within the tile == TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    const float sl2 = LOG2E * 0.125f;  // log2(e) / sqrt(64)
    uint8_t* prow = smem + P_OFF + r * 128;
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    // every lane waits (bounded); the outcome is made warp-uniform so the
    // warp-collective tcgen05 loads and votes below never see a split warp
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      const bool mine = ptx::mbar_wait(bar, parity, lim, p.status, kWaitHint);
      return __all_sync(0xffffffffu, mine);
    };
    for (int j = 0; j < n_kt; ++j) {
      if (!wait_all(s_full, j & 1)) { ok = false; break; }
      ptx::tc_fence_after();
      const int kbase = j * BKV;
      const bool full_tile = kbase + BKV <= len;  // CTA-uniform: only the last tile is masked
      // pass 1: row max of the raw scores (scaling by log2(e)/sqrt(D) > 0 commutes with max)
      float mx = -INFINITY;
#pragma unroll
      for (int c = 0; c < BKV / 32; ++c) {
        uint32_t v[32];
        ptx::tmem_ld_32x32b_x32(tS + lane_base + c * 32, v);
        ptx::tmem_ld_wait();
        if (full_tile) {
#pragma unroll
          for (int i = 0; i < 32; ++i) mx = fmaxf(mx, __uint_as_float(v[i]));
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (kbase + c * 32 + i < len) mx = fmaxf(mx, __uint_as_float(v[i]));
        }
      }
      mx *= sl2;
      const float m_new = fmaxf(m, mx);
      if (j > 0) {
        // P_{j-1} V_{j-1} must be done: the P buffer is reused and O may be rescaled
        if (!wait_all(pv_done, (j - 1) & 1)) { ok = false; break; }
        ptx::tc_fence_after();
        const bool need = m_new > m;
        if (__any_sync(0xffffffffu, need)) {
          const float alpha = need ? exp2f(m - m_new) : 1.f;
#pragma unroll
          for (int c = 0; c < HD / 32; ++c) {
            uint32_t o[32];
            ptx::tmem_ld_32x32b_x32(tO + lane_base + c * 32, o);
            ptx::tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
            ptx::tmem_st_32x32b_x32(tO + lane_base + c * 32, o);
          }
          ptx::tmem_st_wait();
        }
        l *= exp2f(m - m_new);
      }
      m = m_new;
      // pass 2: P = exp2(s * sl2 - m) as bf16, row r of the swizzled K-major tile
      const float nm = -m;
#pragma unroll
      for (int c = 0; c < BKV / 32; ++c) {
        uint32_t v[32];
        ptx::tmem_ld_32x32b_x32(tS + lane_base + c * 32, v);
        ptx::tmem_ld_wait();
        float pv[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) pv[i] = ptx::ex2_ftz(fmaf(__uint_as_float(v[i]), sl2, nm));
        if (!full_tile) {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (kbase + c * 32 + i >= len) pv[i] = 0.f;
        }
        uint32_t pk[16];
        float ls = 0.f;
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          ls += pv[i] + pv[i + 1];
          pk[i >> 1] = ptx::pack_bf16(pv[i], pv[i + 1]);
        }
        l += ls;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int unit = c * 4 + u;  // 16-byte unit (8 keys) within the 128-byte row
          *reinterpret_cast<uint4*>(prow + ((unit ^ (r & 7)) << 4)) =
              make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
        }
      }
      ptx::fence_proxy_async_smem();
      ptx::tc_fence_before();
      ptx::mbar_arrive(p_full);
    }
    // epilogue: O / l -> ctx (bf16), log-sum-exp
    if (ok && wait_all(pv_done, (n_kt - 1) & 1)) {
      ptx::tc_fence_after();
      const float inv = 1.f / l;
      const int q = q0 + r;
      __nv_bfloat16* out = p.ctx + (static_cast<int64_t>(row0) + q) * H + a * HD;
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t o[32];
        ptx::tmem_ld_32x32b_x32(tO + lane_base + c * 32, o);
        ptx::tmem_ld_wait();
        if (q < S) {
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            uint32_t w[4];
#pragma unroll
            for (int t = 0; t < 4; ++t)
              w[t] = ptx::pack_bf16(__uint_as_float(o[8 * u + 2 * t]) * inv,
                                    __uint_as_float(o[8 * u + 2 * t + 1]) * inv);
            *reinterpret_cast<uint4*>(out + c * 32 + u * 8) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
      }
      if (q < S) p.lse[(static_cast<int64_t>(b) * p.A + a) * S + q] = (m + log2f(l)) * LN2;
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, TMEM_COLS);
  }
}

// ----------------------------------------------------------- backward, dQ
// One CTA per 128 query rows of (b, a); per 64-key tile j < len:
//   S = Q K_j^T, dP = dO V_j^T (TMEM); thread = query row:
//   P = exp2(S log2(e)/sqrt(D) - lse2), dS = P (dP - delta) -> smem (bf16)
//   dQ += dS K_j (TMEM); finally dQ / sqrt(D) -> dQKV[:, Q block].
constexpr int DQ_QD_BYTES = 2 * Q_BYTES;  // Q and dO tiles (128 x 64 each)
constexpr int DQ_Q_OFF = 0, DQ_DO_OFF = Q_BYTES;
constexpr int DQ_K_OFF = DQ_QD_BYTES;
constexpr int DQ_V_OFF = DQ_K_OFF + STAGES * KV_BYTES;
constexpr int DQ_DS_OFF = DQ_V_OFF + STAGES * KV_BYTES;
constexpr int DQ_BAR_OFF = DQ_DS_OFF + P_BYTES;
constexpr int DQ_SMEM = DQ_BAR_OFF + 128 + 1024;

struct BwdParams {
  int S, H, A;
  const int32_t* lens;
  const float* lse;
  const float* delta;
  __nv_bfloat16* dqkv;
  int32_t* status;
  uint64_t timeout_ns;
};

__global__ void __launch_bounds__(NTHR, 2) attn_bwd_dq_tc(const __grid_constant__ CUtensorMap tmQ,
                                                          const __grid_constant__ CUtensorMap tmKV,
                                                          const __grid_constant__ CUtensorMap tmO,
                                                          const BwdParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
  uint64_t* qd_full = reinterpret_cast<uint64_t*>(smem + DQ_BAR_OFF);
  uint64_t* kv_full = qd_full + 1;
  uint64_t* kv_empty = kv_full + STAGES;
  uint64_t* s_full = kv_empty + STAGES;
  uint64_t* ds_full = s_full + 1;
  uint64_t* dq_done = ds_full + 1;
  uint64_t* done = dq_done + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);

  const int qt = blockIdx.x, a = blockIdx.y, b = blockIdx.z;
  const int S = p.S, H = p.H;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int len = p.lens[b];
  if (len < 1 || len > S) {
    if (p.status && threadIdx.x == 0) atomicOr(p.status, kStatusBadLength);
    len = len < 1 ? 1 : S;
  }
  const int n_kt = (len + BKV - 1) / BKV;
  const int row0 = b * S, q0 = qt * BQ;
  const uint64_t lim = p.timeout_ns;

  if (threadIdx.x == 0) {
    ptx::mbar_init(qd_full, 1);
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(&kv_full[s], 1);
      ptx::mbar_init(&kv_empty[s], 1);
    }
    ptx::mbar_init(s_full, 1);
    ptx::mbar_init(ds_full, 128);
    ptx::mbar_init(dq_done, 1);
    ptx::mbar_init(done, 1);
    ptx::fence_mbar_init();
    ptx::fence_proxy_async_smem();
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, 256);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS = tmem, tdP = tmem + 64, tdQ = tmem + 128;

  if (warp == 0) {
    if (lane == 0) {
      ptx::mbar_arrive_expect_tx(qd_full, DQ_QD_BYTES);
      ptx::tma_load_2d(smem + DQ_Q_OFF, &tmQ, qd_full, a * HD, row0 + q0);
      ptx::tma_load_2d(smem + DQ_DO_OFF, &tmO, qd_full, a * HD, row0 + q0);
      int issued = 0;
      for (int j = 0; j < n_kt; ++j) {
        const int st = j & 1;
        if (!ptx::mbar_wait(&kv_empty[st], ((j >> 1) & 1) ^ 1u, lim, p.status, kWaitHint)) break;
        ptx::mbar_arrive_expect_tx(&kv_full[st], 2 * KV_BYTES);
        ptx::tma_load_2d(smem + DQ_K_OFF + st * KV_BYTES, &tmKV, &kv_full[st], H + a * HD,
                         row0 + j * BKV);
        ptx::tma_load_2d(smem + DQ_V_OFF + st * KV_BYTES, &tmKV, &kv_full[st], 2 * H + a * HD,
                         row0 + j * BKV);
        ++issued;
      }
      ptx::mbar_wait(qd_full, 0, lim, p.status, kWaitHint);
      for (int j = issued - 1; j >= 0 && j >= issued - STAGES; --j)
        ptx::mbar_wait(&kv_full[j & 1], (j >> 1) & 1, lim, p.status, kWaitHint);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = ptx::idesc_bf16_f32(BQ, BKV, false, false);
      constexpr uint32_t idQ = ptx::idesc_bf16_f32(BQ, HD, false, true);
      const uint32_t sq = ptx::smem_u32(smem + DQ_Q_OFF), so = ptx::smem_u32(smem + DQ_DO_OFF);
      const uint32_t sds = ptx::smem_u32(smem + DQ_DS_OFF);
      bool ok = ptx::mbar_wait(qd_full, 0, lim, p.status, kWaitHint);
      for (int j = 0; j < n_kt && ok; ++j) {
        const int st = j & 1;
        if (!ptx::mbar_wait(&kv_full[st], (j >> 1) & 1, lim, p.status, kWaitHint)) break;
        ptx::tc_fence_after();
        const uint32_t sk = ptx::smem_u32(smem + DQ_K_OFF + st * KV_BYTES);
        const uint32_t sv = ptx::smem_u32(smem + DQ_V_OFF + st * KV_BYTES);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tS, ptx::smem_desc_sw128(sq + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sk + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tdP, ptx::smem_desc_sw128(so + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sv + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
        ptx::tc_commit(s_full);
        if (!ptx::mbar_wait(ds_full, j & 1, lim, p.status, kWaitHint)) break;
        ptx::tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < BKV / 16; ++kk)
          ptx::tc_mma_f16(tdQ, ptx::smem_desc_sw128(sds + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sk + kk * 2048, 8192, 1024), idQ,
                          (j > 0 || kk > 0) ? 1u : 0u);
        ptx::tc_commit(dq_done);
        ptx::tc_commit(&kv_empty[st]);
      }
      ptx::tc_commit(done);
      ptx::mbar_wait(done, 0, lim, p.status, kWaitHint);
    }
  } else {
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;
    const int q = q0 + r;
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    const float sl2 = LOG2E * 0.125f;
    const int64_t sidx = (static_cast<int64_t>(b) * p.A + a) * S + (q < S ? q : 0);
    const float nlse2 = q < S ? -p.lse[sidx] * LOG2E : -INFINITY;  // P = 0 on rows past S
    const float dl = q < S ? p.delta[sidx] : 0.f;
    uint8_t* drow = smem + DQ_DS_OFF + r * 128;
    bool ok = true;
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      const bool mine = ptx::mbar_wait(bar, parity, lim, p.status, kWaitHint);
      return __all_sync(0xffffffffu, mine);
    };
    for (int j = 0; j < n_kt; ++j) {
      if (!wait_all(s_full, j & 1)) { ok = false; break; }
      if (j > 0 && !wait_all(dq_done, (j - 1) & 1)) { ok = false; break; }
      ptx::tc_fence_after();
      const int kbase = j * BKV;
      const bool full_tile = kbase + BKV <= len;
#pragma unroll
      for (int c = 0; c < BKV / 32; ++c) {
        uint32_t sv[32], dv[32];
        ptx::tmem_ld_32x32b_x32(tS + lane_base + c * 32, sv);
        ptx::tmem_ld_32x32b_x32(tdP + lane_base + c * 32, dv);
        ptx::tmem_ld_wait();
        float ds[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float pr = ptx::ex2_ftz(fmaf(__uint_as_float(sv[i]), sl2, nlse2));
          ds[i] = pr * (__uint_as_float(dv[i]) - dl);
        }
        if (!full_tile) {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (kbase + c * 32 + i >= len) ds[i] = 0.f;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int unit = c * 4 + u;
          *reinterpret_cast<uint4*>(drow + ((unit ^ (r & 7)) << 4)) =
              make_uint4(ptx::pack_bf16(ds[8 * u], ds[8 * u + 1]),
                         ptx::pack_bf16(ds[8 * u + 2], ds[8 * u + 3]),
                         ptx::pack_bf16(ds[8 * u + 4], ds[8 * u + 5]),
                         ptx::pack_bf16(ds[8 * u + 6], ds[8 * u + 7]));
        }
      }
      ptx::fence_proxy_async_smem();
      ptx::tc_fence_before();
      ptx::mbar_arrive(ds_full);
    }
    if (ok && wait_all(dq_done, (n_kt - 1) & 1)) {
      ptx::tc_fence_after();
      __nv_bfloat16* out = p.dqkv + (static_cast<int64_t>(row0) + q) * (3 * H) + a * HD;
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t o[32];
        ptx::tmem_ld_32x32b_x32(tdQ + lane_base + c * 32, o);
        ptx::tmem_ld_wait();
        if (q < S) {
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            uint32_t w[4];
#pragma unroll
            for (int t = 0; t < 4; ++t)
              w[t] = ptx::pack_bf16(__uint_as_float(o[8 * u + 2 * t]) * 0.125f,
                                    __uint_as_float(o[8 * u + 2 * t + 1]) * 0.125f);
            *reinterpret_cast<uint4*>(out + c * 32 + u * 8) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
      }
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 256);
  }
}

// --------------------------------------------------------- backward, dK dV
// One CTA per 128 keys of (b, a) (tiles at or past len[b] only write zeros);
// per 64-query tile i over all S queries:
//   S^T = K Q_i^T, dP^T = V dO_i^T (TMEM); thread = key row:
//   P^T = exp2(S^T log2(e)/sqrt(D) - lse2_q), dS^T = P^T (dP^T - delta_q) -> smem
//   dV += P^T dO_i, dK += dS^T Q_i (TMEM); finally dK / sqrt(D), dV -> dQKV.
// The Q_i / dO_i tiles serve both as K-major operands (S^T, dP^T) and as
// MN-major operands (dK, dV).
constexpr int BK2 = 128, BQ2 = 64;
constexpr int KV2_BYTES = BK2 * HD * 2;    // 16 KiB (K or V of 128 keys)
constexpr int QO2_BYTES = BQ2 * HD * 2;    // 8 KiB  (Q or dO of 64 queries)
constexpr int PS2_BYTES = BK2 * BQ2 * 2;   // 16 KiB (P^T or dS^T)
constexpr int KV_K_OFF = 0, KV_V_OFF = KV2_BYTES;
constexpr int KV_Q_OFF = 2 * KV2_BYTES;
constexpr int KV_O_OFF = KV_Q_OFF + STAGES * QO2_BYTES;
constexpr int KV_P_OFF = KV_O_OFF + STAGES * QO2_BYTES;
constexpr int KV_DS_OFF = KV_P_OFF + PS2_BYTES;
constexpr int KV_LD_OFF = KV_DS_OFF + PS2_BYTES;   // [STAGES][2][64] floats: lse2, delta
constexpr int KV_BAR_OFF = KV_LD_OFF + STAGES * 2 * BQ2 * 4;
constexpr int KV_SMEM = KV_BAR_OFF + 128 + 1024;

__global__ void __launch_bounds__(NTHR, 2) attn_bwd_dkdv_tc(const __grid_constant__ CUtensorMap tmK,
                                                            const __grid_constant__ CUtensorMap tmQ,
                                                            const __grid_constant__ CUtensorMap tmO,
                                                            const BwdParams p) {
  extern __shared__ uint8_t smem_raw[];
  const int kt = blockIdx.x, a = blockIdx.y, b = blockIdx.z;
  const int S = p.S, H = p.H;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int len = p.lens[b];
  if (len < 1 || len > S) {
    if (p.status && threadIdx.x == 0) atomicOr(p.status, kStatusBadLength);
    len = len < 1 ? 1 : S;
  }
  const int row0 = b * S, k0 = kt * BK2;
  const int64_t rs = 3 * static_cast<int64_t>(H);
  if (k0 >= len) {  // keys of this tile are all padding: zero gradients
    for (int i = threadIdx.x; i < BK2 * 8; i += NTHR) {
      const int rr = i >> 3, c = i & 7;
      if (k0 + rr < S) {
        __nv_bfloat16* base = p.dqkv + (static_cast<int64_t>(row0) + k0 + rr) * rs + a * HD + c * 8;
        *reinterpret_cast<uint4*>(base + H) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(base + 2 * H) = make_uint4(0, 0, 0, 0);
      }
    }
    return;
  }
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
  float* ldst = reinterpret_cast<float*>(smem + KV_LD_OFF);
  uint64_t* kv_full = reinterpret_cast<uint64_t*>(smem + KV_BAR_OFF);
  uint64_t* q_full = kv_full + 1;
  uint64_t* q_empty = q_full + STAGES;
  uint64_t* s_full = q_empty + STAGES;
  uint64_t* pds_full = s_full + 1;
  uint64_t* mm_done = pds_full + 1;
  uint64_t* done = mm_done + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  const int n_qt = (S + BQ2 - 1) / BQ2;
  const uint64_t lim = p.timeout_ns;

  if (threadIdx.x == 0) {
    ptx::mbar_init(kv_full, 1);
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(&q_full[s], 32);  // lane 0's expect_tx + 31 lanes' lse/delta stores
      ptx::mbar_init(&q_empty[s], 1);
    }
    ptx::mbar_init(s_full, 1);
    ptx::mbar_init(pds_full, 128);
    ptx::mbar_init(mm_done, 1);
    ptx::mbar_init(done, 1);
    ptx::fence_mbar_init();
    ptx::fence_proxy_async_smem();
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, 256);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tST = tmem, tdPT = tmem + 64, tdV = tmem + 128, tdK = tmem + 192;

  if (warp == 0) {
    // producer: K, V once; per query tile Q_i, dO_i by TMA and lse2 / delta by the warp
    if (lane == 0) {
      ptx::mbar_arrive_expect_tx(kv_full, 2 * KV2_BYTES);
      ptx::tma_load_2d(smem + KV_K_OFF, &tmK, kv_full, H + a * HD, row0 + k0);
      ptx::tma_load_2d(smem + KV_V_OFF, &tmK, kv_full, 2 * H + a * HD, row0 + k0);
    }
    const float* lse_b = p.lse + (static_cast<int64_t>(b) * p.A + a) * S;
    const float* del_b = p.delta + (static_cast<int64_t>(b) * p.A + a) * S;
    int issued = 0;
    for (int i = 0; i < n_qt; ++i) {
      const int st = i & 1;
      bool ok = true;
      if (lane == 0) ok = ptx::mbar_wait(&q_empty[st], ((i >> 1) & 1) ^ 1u, lim, p.status, kWaitHint);
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;
      float* l2 = ldst + st * 2 * BQ2;
      for (int t = lane; t < BQ2; t += 32) {
        const int q = i * BQ2 + t;
        l2[t] = q < S ? lse_b[q] * LOG2E : INFINITY;  // rows past S get P = 0
        l2[BQ2 + t] = q < S ? del_b[q] : 0.f;
      }
      if (lane == 0) {
        ptx::mbar_arrive_expect_tx(&q_full[st], 2 * QO2_BYTES);
        ptx::tma_load_2d(smem + KV_Q_OFF + st * QO2_BYTES, &tmQ, &q_full[st], a * HD,
                         row0 + i * BQ2);
        ptx::tma_load_2d(smem + KV_O_OFF + st * QO2_BYTES, &tmO, &q_full[st], a * HD,
                         row0 + i * BQ2);
      } else {
        ptx::mbar_arrive(&q_full[st]);
      }
      ++issued;
    }
    if (lane == 0) {
      ptx::mbar_wait(kv_full, 0, lim, p.status, kWaitHint);
      for (int i = issued - 1; i >= 0 && i >= issued - STAGES; --i)
        ptx::mbar_wait(&q_full[i & 1], (i >> 1) & 1, lim, p.status, kWaitHint);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = ptx::idesc_bf16_f32(BK2, BQ2, false, false);
      constexpr uint32_t idG = ptx::idesc_bf16_f32(BK2, HD, false, true);
      const uint32_t sk = ptx::smem_u32(smem + KV_K_OFF), sv = ptx::smem_u32(smem + KV_V_OFF);
      const uint32_t sp = ptx::smem_u32(smem + KV_P_OFF), sds = ptx::smem_u32(smem + KV_DS_OFF);
      bool ok = ptx::mbar_wait(kv_full, 0, lim, p.status, kWaitHint);
      for (int i = 0; i < n_qt && ok; ++i) {
        const int st = i & 1;
        if (!ptx::mbar_wait(&q_full[st], (i >> 1) & 1, lim, p.status, kWaitHint)) break;
        ptx::tc_fence_after();
        const uint32_t sq = ptx::smem_u32(smem + KV_Q_OFF + st * QO2_BYTES);
        const uint32_t so = ptx::smem_u32(smem + KV_O_OFF + st * QO2_BYTES);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tST, ptx::smem_desc_sw128(sk + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sq + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tdPT, ptx::smem_desc_sw128(sv + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(so + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
        ptx::tc_commit(s_full);
        if (!ptx::mbar_wait(pds_full, i & 1, lim, p.status, kWaitHint)) break;
        ptx::tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < BQ2 / 16; ++kk) {
          ptx::tc_mma_f16(tdV, ptx::smem_desc_sw128(sp + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(so + kk * 2048, 8192, 1024), idG,
                          (i > 0 || kk > 0) ? 1u : 0u);
          ptx::tc_mma_f16(tdK, ptx::smem_desc_sw128(sds + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sq + kk * 2048, 8192, 1024), idG,
                          (i > 0 || kk > 0) ? 1u : 0u);
        }
        ptx::tc_commit(mm_done);
        ptx::tc_commit(&q_empty[st]);
      }
      ptx::tc_commit(done);
      ptx::mbar_wait(done, 0, lim, p.status, kWaitHint);
    }
  } else {
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;  // key row within the tile == TMEM lane
    const int key = k0 + r;
    const bool kvalid = key < len;
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    const float sl2 = LOG2E * 0.125f;
    uint8_t* prow = smem + KV_P_OFF + r * 128;
    uint8_t* drow = smem + KV_DS_OFF + r * 128;
    bool ok = true;
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      const bool mine = ptx::mbar_wait(bar, parity, lim, p.status, kWaitHint);
      return __all_sync(0xffffffffu, mine);
    };
    for (int i = 0; i < n_qt; ++i) {
      const int st = i & 1;
      if (!wait_all(&q_full[st], (i >> 1) & 1)) { ok = false; break; }
      if (!wait_all(s_full, i & 1)) { ok = false; break; }
      if (i > 0 && !wait_all(mm_done, (i - 1) & 1)) { ok = false; break; }
      ptx::tc_fence_after();
      const float* l2 = ldst + st * 2 * BQ2;
#pragma unroll
      for (int c = 0; c < BQ2 / 32; ++c) {
        uint32_t sv[32], dv[32];
        ptx::tmem_ld_32x32b_x32(tST + lane_base + c * 32, sv);
        ptx::tmem_ld_32x32b_x32(tdPT + lane_base + c * 32, dv);
        ptx::tmem_ld_wait();
        float pt[32], ds[32];
#pragma unroll
        for (int t = 0; t < 32; ++t) {
          const int qq = c * 32 + t;
          pt[t] = kvalid ? ptx::ex2_ftz(fmaf(__uint_as_float(sv[t]), sl2, -l2[qq])) : 0.f;
          ds[t] = pt[t] * (__uint_as_float(dv[t]) - l2[BQ2 + qq]);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int unit = c * 4 + u;
          const int pos = (unit ^ (r & 7)) << 4;
          *reinterpret_cast<uint4*>(prow + pos) =
              make_uint4(ptx::pack_bf16(pt[8 * u], pt[8 * u + 1]),
                         ptx::pack_bf16(pt[8 * u + 2], pt[8 * u + 3]),
                         ptx::pack_bf16(pt[8 * u + 4], pt[8 * u + 5]),
                         ptx::pack_bf16(pt[8 * u + 6], pt[8 * u + 7]));
          *reinterpret_cast<uint4*>(drow + pos) =
              make_uint4(ptx::pack_bf16(ds[8 * u], ds[8 * u + 1]),
                         ptx::pack_bf16(ds[8 * u + 2], ds[8 * u + 3]),
                         ptx::pack_bf16(ds[8 * u + 4], ds[8 * u + 5]),
                         ptx::pack_bf16(ds[8 * u + 6], ds[8 * u + 7]));
        }
      }
      ptx::fence_proxy_async_smem();
      ptx::tc_fence_before();
      ptx::mbar_arrive(pds_full);
    }
    if (ok && wait_all(mm_done, (n_qt - 1) & 1)) {
      ptx::tc_fence_after();
      __nv_bfloat16* outk = p.dqkv + (static_cast<int64_t>(row0) + key) * rs + H + a * HD;
      __nv_bfloat16* outv = outk + H;
#pragma unroll
      for (int which = 0; which < 2; ++which) {
        const uint32_t tacc = which == 0 ? tdK : tdV;
        const float sc = which == 0 ? 0.125f : 1.f;
        __nv_bfloat16* out = which == 0 ? outk : outv;
#pragma unroll
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t o[32];
          ptx::tmem_ld_32x32b_x32(tacc + lane_base + c * 32, o);
          ptx::tmem_ld_wait();
          if (key < S) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              uint32_t w[4];
#pragma unroll
              for (int t = 0; t < 4; ++t)
                w[t] = ptx::pack_bf16(__uint_as_float(o[8 * u + 2 * t]) * sc,
                                      __uint_as_float(o[8 * u + 2 * t + 1]) * sc);
              *reinterpret_cast<uint4*>(out + c * 32 + u * 8) = make_uint4(w[0], w[1], w[2], w[3]);
            }
          }
        }
      }
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 256);
  }
}

namespace {
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

// [T, W] bf16 activations, box {64 columns (one head), rows}, 128B swizzle.
bool head_map(CUtensorMap* map, const void* base, int64_t T, int W, int rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(W), static_cast<cuuint64_t>(T)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(W) * 2};
  cuuint32_t box[2] = {64u, static_cast<cuuint32_t>(rows)};
  cuuint32_t estr[2] = {1u, 1u};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
}  // namespace

}  // namespace attn_tc

// Forward launcher used by the bf16 attention path (D = 64).
sky_status attention_fwd_tc(const void* qkv, const int32_t* lens, int B, int S, int H, int A,
                            void* ctx, float* lse, int32_t* status, uint64_t timeout_ns,
                            cudaStream_t stream) {
  using namespace attn_tc;
  SKY_CHECK(H == A * HD, SKY_ERR_UNSUPPORTED, "tensor-core attention needs head dim 64");
  SKY_CHECK((reinterpret_cast<uintptr_t>(qkv) & 15) == 0 && (reinterpret_cast<uintptr_t>(ctx) & 15) == 0,
            SKY_ERR_UNSUPPORTED, "attention buffers must be 16-byte aligned");
  CUtensorMap tq, tkv;
  const int64_t T = static_cast<int64_t>(B) * S;
  SKY_CHECK(head_map(&tq, qkv, T, 3 * H, BQ) && head_map(&tkv, qkv, T, 3 * H, BKV), SKY_ERR_CUDA,
            "cuTensorMapEncodeTiled failed for the attention operands");
  static cudaError_t attr = cudaFuncSetAttribute(attn_fwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 SMEM_BYTES);
  if (attr != cudaSuccess) return cuda_fail(attr, "attention smem attribute");
  FwdParams p{S, H, A, lens, static_cast<__nv_bfloat16*>(ctx), lse, status, timeout_ns};
  dim3 grid(ceil_div(S, BQ), A, B);
  attn_fwd_tc<<<grid, NTHR, SMEM_BYTES, stream>>>(tq, tkv, p);
  count_launches(1);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "tensor-core attention forward launch");
}

// Backward launchers (bf16, D = 64): delta must already hold rowsum(dO * O).
sky_status attention_bwd_tc(const void* qkv, const void* dctx, const float* lse, const float* delta,
                            const int32_t* lens, int B, int S, int H, int A, void* dqkv,
                            int32_t* status, uint64_t timeout_ns, cudaStream_t stream) {
  using namespace attn_tc;
  SKY_CHECK(H == A * HD, SKY_ERR_UNSUPPORTED, "tensor-core attention needs head dim 64");
  const int64_t T = static_cast<int64_t>(B) * S;
  CUtensorMap tq128, tkv64, to128, tk128, tq64, to64;
  SKY_CHECK(head_map(&tq128, qkv, T, 3 * H, BQ) && head_map(&tkv64, qkv, T, 3 * H, BKV) &&
                head_map(&to128, dctx, T, H, BQ) && head_map(&tk128, qkv, T, 3 * H, BK2) &&
                head_map(&tq64, qkv, T, 3 * H, BQ2) && head_map(&to64, dctx, T, H, BQ2),
            SKY_ERR_CUDA, "cuTensorMapEncodeTiled failed for the attention backward operands");
  static cudaError_t a1 = cudaFuncSetAttribute(attn_bwd_dq_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, DQ_SMEM);
  static cudaError_t a2 = cudaFuncSetAttribute(attn_bwd_dkdv_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, KV_SMEM);
  if (a1 != cudaSuccess) return cuda_fail(a1, "attention dQ smem attribute");
  if (a2 != cudaSuccess) return cuda_fail(a2, "attention dK/dV smem attribute");
  BwdParams p{S, H, A, lens, lse, delta, static_cast<__nv_bfloat16*>(dqkv), status, timeout_ns};
  attn_bwd_dkdv_tc<<<dim3(ceil_div(S, BK2), A, B), NTHR, KV_SMEM, stream>>>(tk128, tq64, to64, p);
  attn_bwd_dq_tc<<<dim3(ceil_div(S, BQ), A, B), NTHR, DQ_SMEM, stream>>>(tq128, tkv64, to128, p);
  count_launches(2);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "tensor-core attention backward launch");
}

}  // namespace sky
