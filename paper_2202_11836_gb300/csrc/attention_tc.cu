// Masked scaled dot-product attention (Eq. 1) forward and backward on the
// 5th-generation tensor cores, bf16, head dim D = 64.
//
// Forward: one CTA owns 128 query rows of one (sequence b, head a).  Per
// 64-key tile j (only tiles below len[b] are visited):
//   S_j = Q K_j^T                  tcgen05.mma M=128 N=64 K=64 -> TMEM
//   softmax (4 warps, thread = query row = TMEM lane): row max over the
//     valid keys, P_j = exp2(S_j log2(e)/sqrt(D) - m) written as bf16 pairs
//     back to tensor memory (tcgen05.st), where the next product reads it
//   O += P_j V_j                   tcgen05.mma M=128 N=64 K=64, A = P_j from
//                                  TMEM, B = V_j from shared memory -> TMEM
// Q, K and V come straight out of the packed QKV activations by TMA (one
// tensor map, per-head column offsets), and O / l leaves by TMA from shared
// memory.  Because a thread owns a whole query row, the row max and row sum
// need no shuffles.
//
// The steps are pipelined inside the CTA: S and P have two TMEM buffers each,
// so the MMA warp computes S_{j+1} (issued one tile
// ahead) and P_{j-1} V_{j-1} while the softmax warps work on tile j, and K/V
// tiles stream through a 3-stage TMA ring.  The exponent offset m of a row
// is only raised when the tile's max exceeds it by more than 2^8 (a factor
// 256 in P): then O and the row sum are rescaled in TMEM once the pending
// P V product has landed.  Otherwise P may exceed 1 by at most that factor,
// which bf16 and the fp32 sums carry with the same relative precision; the
// final O / l and the log-sum-exp do not depend on m.  The log-sum-exp is
// kept in base-2 units, lse2 = log2 sum_j exp2(S_ij log2(e)/sqrt(D)), which
// is what the backward kernels subtract in the exponent.  All mbarrier
// waits are time-bounded.
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
// forward CTA: warp 0 TMA and O += P V issue, warp 1 S = Q K^T issue,
// warps 2..5 softmax
constexpr int NTHR = 192;
// The backward kernels run eight softmax warps: warps w and w + 4 share TMEM
// lane quarter w % 4 and take the low / high 32 columns of each 64-wide tile.
constexpr int NSM_B = 256;              // softmax threads in the backward kernels
// Backward CTAs: warp 0 TMA, warp 1 issues the score products (S and dP),
// warps 2..9 softmax, warp 10 issues the accumulating products (dQ, or dV
// and dK).  One thread issues a tcgen05.mma only about every 100 cycles,
// while an M=128, N=64, K=16 product keeps the tensor pipe busy for about
// 32, so the two kinds of product are issued side by side by two warps.
constexpr int NTHR_B = 352;
constexpr float LOG2E = 1.4426950408889634f;
// Suspend-time hint (ns) of every mbarrier wait: a waiting thread sleeps
// until the phase completes instead of spinning on issue slots that the
// softmax warps (the critical path) share with the producer and MMA threads.
constexpr uint32_t kWaitHint = 10000;

// forward shared-memory layout (offsets from a 1024-byte aligned base)
constexpr int F_STAGES = 3;
constexpr int F_Q_OFF = 0;
constexpr int F_KV_OFF = F_Q_OFF + Q_BYTES;                  // [F_STAGES] x {K, V}
constexpr int F_BAR_OFF = F_KV_OFF + F_STAGES * 2 * KV_BYTES;
constexpr int F_SMEM = F_BAR_OFF + 256 + 1024;
// S_0: [0, 64), S_1: [64, 128), O: [128, 192), P_0: [192, 224), P_1: [224, 256)
// (P as bf16 pairs: the A operand of P V read from tensor memory)
constexpr int F_TMEM_COLS = 256;
constexpr float kRescaleLog2 = 8.f;

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
                                                    const __grid_constant__ CUtensorMap tmOut,
                                                    const FwdParams p) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + F_BAR_OFF);
  uint64_t* kv_full = q_full + 1;
  uint64_t* kv_empty = kv_full + F_STAGES;
  uint64_t* s_full = kv_empty + F_STAGES;  // [2]
  uint64_t* s_free = s_full + 2;           // [2]
  uint64_t* p_full = s_free + 2;           // [2]
  uint64_t* pv_done = p_full + 2;          // [2]
  uint64_t* done = pv_done + 2;            // [2], one per issuing warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 2);

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
    for (int s = 0; s < F_STAGES; ++s) {
      ptx::mbar_init(&kv_full[s], 1);
      ptx::mbar_init(&kv_empty[s], 2);  // S_j has read K_j, P_j V_j has read V_j
    }
    for (int s = 0; s < 2; ++s) {
      ptx::mbar_init(&s_full[s], 1);
      ptx::mbar_init(&s_free[s], 128);
      ptx::mbar_init(&p_full[s], 128);
      ptx::mbar_init(&pv_done[s], 1);
    }
    ptx::mbar_init(&done[0], 1);
    ptx::mbar_init(&done[1], 1);
    ptx::fence_mbar_init();
    ptx::fence_proxy_async_smem();
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, F_TMEM_COLS);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS = tmem, tO = tmem + 128, tP = tmem + 192;

  if (warp == 0) {
    // --------------------------------- producer and O += P V issue (warp 0)
    // Loads Q and the first F_STAGES K/V tiles, then per tile j: issues
    // O += P_j V_j once the softmax warps have written P_j, and refills the
    // ring slot of tile j with tile j + F_STAGES once S_j and P_j V_j have
    // read it.  (Two threads issue this CTA's MMAs: one thread issues a
    // tcgen05.mma only about every 100 cycles.)
    if (lane == 0) {
      constexpr uint32_t idO = ptx::idesc_bf16_f32(BQ, HD, false, true);
      const uint32_t skv = ptx::smem_u32(smem + F_KV_OFF);
      auto load_kv = [&](int j) {
        const int st = j % F_STAGES;
        uint8_t* kv = smem + F_KV_OFF + st * 2 * KV_BYTES;
        ptx::mbar_arrive_expect_tx(&kv_full[st], 2 * KV_BYTES);
        ptx::tma_load_2d(kv, &tmKV, &kv_full[st], H + a * HD, row0 + j * BKV);
        ptx::tma_load_2d(kv + KV_BYTES, &tmKV, &kv_full[st], 2 * H + a * HD, row0 + j * BKV);
      };
      ptx::mbar_arrive_expect_tx(q_full, Q_BYTES);
      ptx::tma_load_2d(smem + F_Q_OFF, &tmQ, q_full, a * HD, row0 + q0);
      int issued = 0;
      for (; issued < n_kt && issued < F_STAGES; ++issued) load_kv(issued);
      for (int j = 0; j < n_kt; ++j) {
        if (!ptx::mbar_wait(&p_full[j & 1], (j >> 1) & 1, lim, p.status, kWaitHint)) break;
        if (!ptx::mbar_wait(&kv_full[j % F_STAGES], (j / F_STAGES) & 1, lim, p.status, kWaitHint))
          break;
        ptx::tc_fence_after();
        const uint32_t sv = skv + (j % F_STAGES) * 2 * KV_BYTES + KV_BYTES;
        const uint32_t tpj = tP + (j & 1) * (BKV / 2);
#pragma unroll
        for (int kk = 0; kk < BKV / 16; ++kk)
          ptx::tc_mma_f16_tmem_a(tO, tpj + kk * 8, ptx::smem_desc_sw128(sv + kk * 2048, 8192, 1024),
                                 idO, (j > 0 || kk > 0) ? 1u : 0u);
        ptx::tc_commit(&pv_done[j & 1]);
        ptx::tc_commit(&kv_empty[j % F_STAGES]);
        if (issued < n_kt) {  // the slot of tile j takes tile j + F_STAGES
          const int st = issued % F_STAGES;
          if (!ptx::mbar_wait(&kv_empty[st], ((issued / F_STAGES) & 1) ^ 1u, lim, p.status, kWaitHint))
            break;
          load_kv(issued++);
        }
      }
      ptx::tc_commit(&done[1]);
      ptx::mbar_wait(&done[1], 0, lim, p.status, kWaitHint);
      // drain: bounded waits for the copies still in flight
      ptx::mbar_wait(q_full, 0, lim, p.status, kWaitHint);
      for (int j = issued - 1; j >= 0 && j >= issued - F_STAGES; --j)
        ptx::mbar_wait(&kv_full[j % F_STAGES], (j / F_STAGES) & 1, lim, p.status, kWaitHint);
    }
  } else if (warp == 1) {
    // --------------------------------------------- S = Q K^T issue (warp 1)
    // S_j goes into buffer j & 1 as soon as K_j has landed and the softmax
    // warps hold S_{j-2} in registers (s_free)
    if (lane == 0) {
      constexpr uint32_t idS = ptx::idesc_bf16_f32(BQ, BKV, false, false);
      const uint32_t sq = ptx::smem_u32(smem + F_Q_OFF);
      const uint32_t skv = ptx::smem_u32(smem + F_KV_OFF);
      bool ok = ptx::mbar_wait(q_full, 0, lim, p.status, kWaitHint);
      for (int j = 0; j < n_kt && ok; ++j) {
        if (j >= 2 && !ptx::mbar_wait(&s_free[j & 1], ((j - 2) >> 1) & 1, lim, p.status, kWaitHint))
          break;
        if (!ptx::mbar_wait(&kv_full[j % F_STAGES], (j / F_STAGES) & 1, lim, p.status, kWaitHint))
          break;
        ptx::tc_fence_after();
        const uint32_t sk = skv + (j % F_STAGES) * 2 * KV_BYTES;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tS + (j & 1) * BKV, ptx::smem_desc_sw128(sq + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sk + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
        ptx::tc_commit(&s_full[j & 1]);
        ptx::tc_commit(&kv_empty[j % F_STAGES]);
      }
      ptx::tc_commit(&done[0]);
      ptx::mbar_wait(&done[0], 0, lim, p.status, kWaitHint);
    }
  } else {
    // --------------------------------------------------- softmax / epilogue
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;  // query row within the tile == TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    const float sl2 = LOG2E * 0.125f;  // log2(e) / sqrt(64)
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    // every lane waits (bounded); the outcome is made warp-uniform so the
    // warp-collective tcgen05 loads and votes below never see a split warp
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      const bool mine = ptx::mbar_wait(bar, parity, lim, p.status, kWaitHint);
      return __all_sync(0xffffffffu, mine);
    };
    for (int j = 0; j < n_kt; ++j) {
      if (!wait_all(&s_full[j & 1], (j >> 1) & 1)) { ok = false; break; }
      ptx::tc_fence_after();
      uint32_t v[BKV];
      {
        uint32_t (&v0)[32] = *reinterpret_cast<uint32_t(*)[32]>(&v[0]);
        uint32_t (&v1)[32] = *reinterpret_cast<uint32_t(*)[32]>(&v[32]);
        ptx::tmem_ld_32x32b_x32(tS + (j & 1) * BKV + lane_base, v0);
        ptx::tmem_ld_32x32b_x32(tS + (j & 1) * BKV + lane_base + 32, v1);
      }
      ptx::tmem_ld_wait();
      // S_j is in registers: its buffer may take S_{j+2}
      ptx::tc_fence_before();
      ptx::mbar_arrive(&s_free[j & 1]);
      const int kbase = j * BKV;
      if (kbase + BKV > len) {  // CTA-uniform: only the last tile holds masked keys
#pragma unroll
        for (int i = 0; i < BKV; ++i)
          if (kbase + i >= len) v[i] = 0xff800000u;  // -inf: excluded from the max, P = 0
      }
      // row max of the raw scores (scaling by log2(e)/sqrt(D) > 0 commutes with max)
      float mx8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx8[i] = __uint_as_float(v[i]);
#pragma unroll
      for (int i = 8; i < BKV; ++i) mx8[i & 7] = fmaxf(mx8[i & 7], __uint_as_float(v[i]));
      const float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                             fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7]))) * sl2;
      if (j == 0) {
        m = mx;
      } else if (__any_sync(0xffffffffu, mx > m + kRescaleLog2)) {
        // O must hold P_{j-1} V_{j-1} before it is rescaled
        if (!wait_all(&pv_done[(j - 1) & 1], ((j - 1) >> 1) & 1)) { ok = false; break; }
        ptx::tc_fence_after();
        const float m_new = fmaxf(m, mx);
        const float alpha = exp2f(m - m_new);
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
        l *= alpha;
        m = m_new;
      }
      // P = exp2(s * sl2 - m) as bf16 pairs into this row's lane of P buffer
      // j & 1 in tensor memory
      const float nm = -m;
      float ls = 0.f;
      uint32_t pk[BKV / 2];
#pragma unroll
      for (int u = 0; u < BKV / 8; ++u) {
        float e[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) e[t] = ptx::ex2_ftz(fmaf(__uint_as_float(v[8 * u + t]), sl2, nm));
        ls += ((e[0] + e[1]) + (e[2] + e[3])) + ((e[4] + e[5]) + (e[6] + e[7]));
#pragma unroll
        for (int t = 0; t < 4; ++t) pk[4 * u + t] = ptx::pack_bf16(e[2 * t], e[2 * t + 1]);
      }
      l += ls;
      // P buffer j & 1 was last read by P_{j-2} V_{j-2}
      if (j >= 2 && !wait_all(&pv_done[j & 1], ((j - 2) >> 1) & 1)) { ok = false; break; }
      ptx::tmem_st_32x32b_x32(tP + (j & 1) * (BKV / 2) + lane_base, pk);
      ptx::tmem_st_wait();
      ptx::tc_fence_before();
      ptx::mbar_arrive(&p_full[j & 1]);
    }
    // epilogue: O / l -> ctx (bf16) as 128-byte-swizzled rows over the Q
    // tile (the last S product has read it), stored by one TMA that drops the
    // rows past S; the log-sum-exp directly
    if (ok && wait_all(&pv_done[(n_kt - 1) & 1], ((n_kt - 1) >> 1) & 1)) {
      ptx::tc_fence_after();
      const float inv = 1.f / l;
      const int q = q0 + r;
      const uint32_t orow = ptx::smem_u32(smem + F_Q_OFF) + r * 128;
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t o[32];
        ptx::tmem_ld_32x32b_x32(tO + lane_base + c * 32, o);
        ptx::tmem_ld_wait();
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          uint32_t w[4];
#pragma unroll
          for (int t = 0; t < 4; ++t)
            w[t] = ptx::pack_bf16(__uint_as_float(o[8 * u + 2 * t]) * inv,
                                  __uint_as_float(o[8 * u + 2 * t + 1]) * inv);
          ptx::st_shared_v4(orow + (((c * 4 + u) ^ (r & 7)) << 4), w[0], w[1], w[2], w[3]);
        }
      }
      if (q < S) p.lse[(static_cast<int64_t>(b) * p.A + a) * S + q] = m + log2f(l);
    }
    ptx::fence_proxy_async_smem();  // the staged rows -> the TMA store
    asm volatile("bar.sync 1, 128;" ::: "memory");  // the four softmax warps
    if (warp == 2 && lane == 0) {
      ptx::tma_store_3d(&tmOut, smem + F_Q_OFF, a * HD, q0, b);
      ptx::bulk_commit_group();
      ptx::bulk_wait_group_read0();  // before the CTA's memory goes
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, F_TMEM_COLS);
  }
}

// ----------------------------------------------------------- backward, dQ
// One CTA per 128 query rows of (b, a); per 64-key tile j < len:
//   S = Q K_j^T, dP = dO V_j^T (TMEM); thread = query row:
//   P = exp2(S log2(e)/sqrt(D) - lse2), dS = P (dP - delta) -> TMEM as bf16
//   pairs, the A operand of
//   dQ += dS K_j (TMEM); finally dQ / sqrt(D) -> dQKV[:, Q block].
// Pipelining: the softmax warps release S / dP as soon as they hold them in
// registers (s_free), so S_{j+1} and dP_{j+1} run on the tensor cores while
// dS_j is formed; K / V tiles stream through a 3-stage TMA ring.
constexpr int DQ_STAGES = 3;
constexpr int DQ_QD_BYTES = 2 * Q_BYTES;  // Q and dO tiles (128 x 64 each)
constexpr int DQ_Q_OFF = 0, DQ_DO_OFF = Q_BYTES;
constexpr int DQ_KV_OFF = DQ_QD_BYTES;                           // [DQ_STAGES] x {K, V}
constexpr int DQ_BAR_OFF = DQ_KV_OFF + DQ_STAGES * 2 * KV_BYTES;
constexpr int DQ_SMEM = DQ_BAR_OFF + 256 + 1024;

struct BwdParams {
  int S, H, A;
  const int32_t* lens;
  const float* lse;
  const float* delta;
  const uint4* xtab;  // dK/dV per-query rows: [B*A][2][S] x 16 bytes (attn_delta_bf16)
  __nv_bfloat16* dqkv;
  // optional: column sums of the stored dQKV, one row per 128-row tile of a
  // sequence: colpart[b * ceil(S/128) + tile][3H]
  float* colpart;
  int32_t* status;
  uint64_t timeout_ns;
};

// v[j] of lane l -> after the call, v[0] of lane l holds the sum over the
// warp's 32 lanes of v[l]: a butterfly in which every lane keeps the half of
// its columns given by its lane bit and receives the partner's half (31
// shuffles for 32 columns).
__device__ __forceinline__ void lanes_column_sum(float (&v)[32], int lane) {
#pragma unroll
  for (int k = 16; k >= 1; k >>= 1) {
    const bool upper = (lane & k) != 0;
#pragma unroll
    for (int j = 0; j < k; ++j) {
      const float send = upper ? v[j] : v[j + k];
      const float keep = upper ? v[j + k] : v[j];
      v[j] = keep + __shfl_xor_sync(0xffffffffu, send, k);
    }
  }
}
__device__ __forceinline__ float bf16_round(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}
// The 8 softmax warps of a backward kernel (256 threads) meet here.
__device__ __forceinline__ void softmax_warps_sync() {
  asm volatile("bar.sync 1, 256;" ::: "memory");
}

__global__ void __maxnreg__(80) attn_bwd_dq_tc(const __grid_constant__ CUtensorMap tmQ,
                                                          const __grid_constant__ CUtensorMap tmKV,
                                                          const __grid_constant__ CUtensorMap tmO,
                                                          const __grid_constant__ CUtensorMap tmOut,
                                                          const BwdParams p) {
  // Launched right behind the dK/dV kernel, which it does not depend on (it
  // writes the other columns of dQKV): it starts once every dK/dV CTA has
  // started -- and so has seen the delta pre-pass complete -- runs beside it,
  // and waits for it only before exiting, so the next kernel, which waits
  // for this one, also sees dK and dV.
  pdl_trigger();
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
  uint64_t* qd_full = reinterpret_cast<uint64_t*>(smem + DQ_BAR_OFF);
  uint64_t* kv_full = qd_full + 1;
  uint64_t* kv_empty = kv_full + DQ_STAGES;
  uint64_t* s_full = kv_empty + DQ_STAGES;
  uint64_t* s_free = s_full + 1;
  uint64_t* ds_full = s_free + 1;
  uint64_t* dq_done = ds_full + 1;
  uint64_t* done = dq_done + 1;  // [2], one per issuing warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 2);

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
    for (int s = 0; s < DQ_STAGES; ++s) {
      ptx::mbar_init(&kv_full[s], 1);
      ptx::mbar_init(&kv_empty[s], 2);  // the tile's S / dP products and its dQ product
    }
    ptx::mbar_init(s_full, 1);
    ptx::mbar_init(s_free, NSM_B);
    ptx::mbar_init(ds_full, NSM_B);
    ptx::mbar_init(dq_done, 1);
    ptx::mbar_init(&done[0], 1);
    ptx::mbar_init(&done[1], 1);
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
  // S: [0, 64), dP: [64, 128), dQ: [128, 192), dS as bf16 pairs (the A
  // operand of dS K, read from tensor memory): [192, 224)
  const uint32_t tS = tmem, tdP = tmem + 64, tdQ = tmem + 128, tdS = tmem + 192;

  if (warp == 0) {
    if (lane == 0) {
      ptx::prefetch_tensormap(&tmQ);
      ptx::prefetch_tensormap(&tmO);
      ptx::prefetch_tensormap(&tmKV);
      ptx::mbar_arrive_expect_tx(qd_full, DQ_QD_BYTES);
      ptx::tma_load_2d(smem + DQ_Q_OFF, &tmQ, qd_full, a * HD, row0 + q0);
      ptx::tma_load_2d(smem + DQ_DO_OFF, &tmO, qd_full, a * HD, row0 + q0);
      int issued = 0;
      for (int j = 0; j < n_kt; ++j) {
        const int st = j % DQ_STAGES;
        if (!ptx::mbar_wait(&kv_empty[st], ((j / DQ_STAGES) & 1) ^ 1u, lim, p.status, kWaitHint))
          break;
        uint8_t* kv = smem + DQ_KV_OFF + st * 2 * KV_BYTES;
        ptx::mbar_arrive_expect_tx(&kv_full[st], 2 * KV_BYTES);
        ptx::tma_load_2d(kv, &tmKV, &kv_full[st], H + a * HD, row0 + j * BKV);
        ptx::tma_load_2d(kv + KV_BYTES, &tmKV, &kv_full[st], 2 * H + a * HD, row0 + j * BKV);
        ++issued;
      }
      ptx::mbar_wait(qd_full, 0, lim, p.status, kWaitHint);
      for (int j = issued - 1; j >= 0 && j >= issued - DQ_STAGES; --j)
        ptx::mbar_wait(&kv_full[j % DQ_STAGES], (j / DQ_STAGES) & 1, lim, p.status, kWaitHint);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = ptx::idesc_bf16_f32(BQ, BKV, false, false);
      const uint32_t sq = ptx::smem_u32(smem + DQ_Q_OFF), so = ptx::smem_u32(smem + DQ_DO_OFF);
      const uint32_t skv = ptx::smem_u32(smem + DQ_KV_OFF);
      // S_j = Q K_j^T and dP_j = dO V_j^T, as soon as the softmax warps hold
      // S_{j-1} / dP_{j-1} in registers (s_free) and K_j / V_j have landed
      bool ok = ptx::mbar_wait(qd_full, 0, lim, p.status, kWaitHint);
      for (int j = 0; j < n_kt && ok; ++j) {
        if (j >= 1 && !ptx::mbar_wait(s_free, (j - 1) & 1, lim, p.status, kWaitHint)) break;
        if (!ptx::mbar_wait(&kv_full[j % DQ_STAGES], (j / DQ_STAGES) & 1, lim, p.status, kWaitHint))
          break;
        ptx::tc_fence_after();
        const uint32_t sk = skv + (j % DQ_STAGES) * 2 * KV_BYTES, sv = sk + KV_BYTES;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tS, ptx::smem_desc_sw128(sq + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sk + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tdP, ptx::smem_desc_sw128(so + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sv + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
        ptx::tc_commit(s_full);
        ptx::tc_commit(&kv_empty[j % DQ_STAGES]);
      }
      ptx::tc_commit(&done[0]);
      ptx::mbar_wait(&done[0], 0, lim, p.status, kWaitHint);
    }
  } else if (warp == 10) {
    // dQ += dS_j K_j, in tile order, from a warp of its own: one thread
    // issues a tcgen05.mma only about every 100 cycles, so the dQ products
    // and the score products of the next tile go in side by side
    if (lane == 0) {
      constexpr uint32_t idQ = ptx::idesc_bf16_f32(BQ, HD, false, true);
      const uint32_t skv = ptx::smem_u32(smem + DQ_KV_OFF);
      for (int j = 0; j < n_kt; ++j) {
        if (!ptx::mbar_wait(ds_full, j & 1, lim, p.status, kWaitHint)) break;
        if (!ptx::mbar_wait(&kv_full[j % DQ_STAGES], (j / DQ_STAGES) & 1, lim, p.status, kWaitHint))
          break;
        ptx::tc_fence_after();
        const uint32_t sk = skv + (j % DQ_STAGES) * 2 * KV_BYTES;
#pragma unroll
        for (int kk = 0; kk < BKV / 16; ++kk)
          ptx::tc_mma_f16_tmem_a(tdQ, tdS + kk * 8, ptx::smem_desc_sw128(sk + kk * 2048, 8192, 1024),
                                 idQ, (j > 0 || kk > 0) ? 1u : 0u);
        ptx::tc_commit(dq_done);
        ptx::tc_commit(&kv_empty[j % DQ_STAGES]);
      }
      ptx::tc_commit(&done[1]);
      ptx::mbar_wait(&done[1], 0, lim, p.status, kWaitHint);
    }
  } else {
    const int q4 = warp & 3;
    const int hf = (warp - 2) >> 2;  // column half: keys [32 hf, 32 hf + 32) of a tile
    const int r = q4 * 32 + lane;
    const int q = q0 + r;
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    const float sl2 = LOG2E * 0.125f;
    const int64_t sidx = (static_cast<int64_t>(b) * p.A + a) * S + (q < S ? q : 0);
    const float nlse2 = q < S ? -p.lse[sidx] : -INFINITY;  // P = 0 on rows past S
    const float dl = q < S ? p.delta[sidx] : 0.f;
    bool ok = true;
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      const bool mine = ptx::mbar_wait(bar, parity, lim, p.status, kWaitHint);
      return __all_sync(0xffffffffu, mine);
    };
    for (int j = 0; j < n_kt; ++j) {
      if (!wait_all(s_full, j & 1)) { ok = false; break; }
      ptx::tc_fence_after();
      uint32_t sv[32], dv[32];
      ptx::tmem_ld_32x32b_x32(tS + lane_base + hf * 32, sv);
      ptx::tmem_ld_32x32b_x32(tdP + lane_base + hf * 32, dv);
      ptx::tmem_ld_wait();
      ptx::tc_fence_before();
      ptx::mbar_arrive(s_free);
      const int kbase = j * BKV + hf * 32;
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        float ds2[2];
#pragma unroll
        for (int t = 0; t < 2; ++t) {
          const float pr = ptx::ex2_ftz(fmaf(__uint_as_float(sv[i + t]), sl2, nlse2));
          ds2[t] = pr * (__uint_as_float(dv[i + t]) - dl);
        }
        pk[i >> 1] = ptx::pack_bf16(ds2[0], ds2[1]);
      }
      if (kbase + 32 > len) {  // warp-uniform: only the last tile holds masked keys
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          const uint32_t lo = kbase + i < len ? 0x0000ffffu : 0u;
          const uint32_t hi = kbase + i + 1 < len ? 0xffff0000u : 0u;
          pk[i >> 1] &= lo | hi;
        }
      }
      // the dS buffer was last read by the dQ product of tile j - 1
      if (j >= 1 && !wait_all(dq_done, (j - 1) & 1)) { ok = false; break; }
      {  // this half's 32 keys = 16 columns of the row's lane
        uint32_t (&p0)[16] = *reinterpret_cast<uint32_t(*)[16]>(&pk[0]);
        ptx::tmem_st_32x32b_x16(tdS + hf * 16 + lane_base, p0);
      }
      ptx::tmem_st_wait();
      ptx::tc_fence_before();
      ptx::mbar_arrive(ds_full);
    }
    // epilogue: each half stages 32 of the 64 dQ columns as 128-byte-swizzled
    // bf16 rows over the Q tile (the last S product has read it); one thread
    // then stores the tile by TMA, which drops the rows past S
    float* red = reinterpret_cast<float*>(smem + DQ_KV_OFF);  // [4 row quarters][64]: ring is idle
    if (ok && wait_all(dq_done, (n_kt - 1) & 1)) {
      ptx::tc_fence_after();
      const uint32_t orow = ptx::smem_u32(smem + DQ_Q_OFF) + r * 128;
      uint32_t o[32];
      ptx::tmem_ld_32x32b_x32(tdQ + lane_base + hf * 32, o);
      ptx::tmem_ld_wait();
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        uint32_t w[4];
#pragma unroll
        for (int t = 0; t < 4; ++t)
          w[t] = ptx::pack_bf16(__uint_as_float(o[8 * u + 2 * t]) * 0.125f,
                                __uint_as_float(o[8 * u + 2 * t + 1]) * 0.125f);
        ptx::st_shared_v4(orow + (((hf * 4 + u) ^ (r & 7)) << 4), w[0], w[1], w[2], w[3]);
      }
      if (p.colpart) {  // column sums of the stored values over this warp's 32 rows
        float v[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = q < S ? bf16_round(__uint_as_float(o[j]) * 0.125f) : 0.f;
        lanes_column_sum(v, lane);
        red[q4 * 64 + hf * 32 + lane] = v[0];
      }
    } else if (p.colpart) {
      red[q4 * 64 + hf * 32 + lane] = 0.f;
    }
    ptx::fence_proxy_async_smem();  // the staged rows -> the TMA store
    softmax_warps_sync();
    if (warp == 2 && lane == 0) {
      ptx::tma_store_3d(&tmOut, smem + DQ_Q_OFF, a * HD, q0, b);
      ptx::bulk_commit_group();
    }
    if (p.colpart && q4 == 0) {  // the four row quarters, added in order, by the quarter-0 warps
      const int c = hf * 32 + lane;
      const float sum = ((red[c] + red[64 + c]) + red[128 + c]) + red[192 + c];
      p.colpart[(static_cast<int64_t>(b) * gridDim.x + qt) * (3 * H) + a * HD + c] = sum;
    }
    if (warp == 2 && lane == 0) ptx::bulk_wait_group_read0();  // before the CTA's memory goes
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 256);
  }
  pdl_wait();
}

// --------------------------------------------------------- backward, dK dV
// One CTA per 128 keys of (b, a) (tiles at or past len[b] only write zeros);
// per 64-query tile i over all S queries:
//   S^T = K Q_i^T, dP^T = V dO_i^T (TMEM); thread = key row:
//   P^T = exp2(S^T log2(e)/sqrt(D) - lse2_q), dS^T = P^T (dP^T - delta_q),
//   written back to TMEM over the S^T / dP^T columns they came from;
//   dV += P^T dO_i, dK += dS^T Q_i with P^T, dS^T as TMEM A operands;
//   finally dK / sqrt(D), dV -> dQKV.
// Keeping P^T and dS^T in TMEM takes their 32 KiB of shared-memory stores and
// the accumulating products' 32 KiB of A-operand reads off the shared-memory
// port per tile, which the score products' operand reads otherwise saturate.
// The price is order within a CTA: S^T_{i+1} waits until dV_i has read P^T_i
// (and dP^T_{i+1} until dK_i has read dS^T_i), so the two CTAs on an SM take
// turns on the tensor pipe rather than one CTA overlapping itself.
// The Q_i / dO_i tiles serve both as K-major operands (S^T, dP^T) and as
// MN-major operands (dK, dV).
constexpr int BK2 = 128, BQ2 = 64;
constexpr int KV2_BYTES = BK2 * HD * 2;    // 16 KiB (K or V of 128 keys)
constexpr int QO2_BYTES = BQ2 * HD * 2;    // 8 KiB  (Q or dO of 64 queries)
constexpr int KV_STAGES = 3;               // Q / dO ring
constexpr int KV_K_OFF = 0, KV_V_OFF = KV2_BYTES;
constexpr int KV_Q_OFF = 2 * KV2_BYTES;
constexpr int KV_O_OFF = KV_Q_OFF + KV_STAGES * QO2_BYTES;
// The per-query terms enter the score products as one more K = 16 step:
// S^T - lse2 / c = [K | E] [Q | X_lse]^T and dP^T - delta = [V | E] [dO | X_delta]^T,
// with c = log2(e)/sqrt(D), E the 128 x 16 matrix whose first two columns are
// ones, and X the 64 x 16 per-tile matrix whose first two columns hold the
// negated term split into a bf16 high part and a bf16 low part (exact to
// about 2^-17 relative).  The softmax threads then need no per-query loads.
// E and X are K-major without swizzling, built from 8-row x 16-byte core
// matrices: a row's K columns 0..7 are 16 contiguous bytes (row groups 128
// bytes apart), and columns 8..15, all zero, come from one shared zero block
// (the descriptors' K-direction offset points there).  So an X tile is 64
// rows of 16 bytes, one bulk copy of the table the delta pre-pass writes.
constexpr int XROW_BYTES = 16;
constexpr int X_BYTES = BQ2 * XROW_BYTES;                      // 1 KiB: X of one product
constexpr int KV_E_OFF = KV_O_OFF + KV_STAGES * QO2_BYTES;     // E: 2 KiB
constexpr int KV_X_OFF = KV_E_OFF + BK2 * XROW_BYTES;          // [KV_STAGES][2 products] X
constexpr int KV_Z_OFF = KV_X_OFF + KV_STAGES * 2 * X_BYTES;   // zeros: 2 KiB
constexpr int KV_RED_OFF = KV_Z_OFF + BK2 * XROW_BYTES;  // [2 halves][4 quarters][64] floats
constexpr int KV_BAR_OFF = KV_RED_OFF + 2 * 4 * 64 * 4;
// 91 KiB: more than a third of the SM's shared memory, so at most two CTAs
// share an SM, as their 256 TMEM columns each require.
constexpr int KV_SMEM = KV_BAR_OFF + 128 + 1024;
static_assert(3 * (KV_SMEM + 1024) > 233472 && 2 * (KV_SMEM + 1024) <= 233472,
              "exactly two dK/dV CTAs per SM");

__global__ void __maxnreg__(80) attn_bwd_dkdv_tc(const __grid_constant__ CUtensorMap tmK,
                                                            const __grid_constant__ CUtensorMap tmQ,
                                                            const __grid_constant__ CUtensorMap tmO,
                                                            const __grid_constant__ CUtensorMap tmOut,
                                                            const BwdParams p) {
  // wait first, then let the dQ kernel start: once every CTA here has passed
  // the wait, the delta pre-pass (and everything before it) is complete
  pdl_wait();
  pdl_trigger();
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
    for (int i = threadIdx.x; i < BK2 * 8; i += NTHR_B) {
      const int rr = i >> 3, c = i & 7;
      if (k0 + rr < S) {
        __nv_bfloat16* base = p.dqkv + (static_cast<int64_t>(row0) + k0 + rr) * rs + a * HD + c * 8;
        *reinterpret_cast<uint4*>(base + H) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(base + 2 * H) = make_uint4(0, 0, 0, 0);
      }
    }
    if (p.colpart && threadIdx.x < 2 * HD) {  // and zero column sums
      const int hf = threadIdx.x / HD, c = threadIdx.x % HD;
      p.colpart[(static_cast<int64_t>(b) * gridDim.x + kt) * rs + (1 + hf) * H + a * HD + c] = 0.f;
    }
    return;
  }
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
  uint64_t* kv_full = reinterpret_cast<uint64_t*>(smem + KV_BAR_OFF);
  uint64_t* q_full = kv_full + 1;
  uint64_t* q_empty = q_full + KV_STAGES;
  uint64_t* st_full = q_empty + KV_STAGES;  // S^T_i complete
  uint64_t* dpt_full = st_full + 1;         // dP^T_i complete
  uint64_t* pds_full = dpt_full + 1;        // P^T_i, dS^T_i stored to TMEM
  uint64_t* dv_done = pds_full + 1;         // dV += P^T_i dO_i complete: S^T columns free
  uint64_t* dk_done = dv_done + 1;          // dK += dS^T_i Q_i complete: dP^T columns free
  uint64_t* done = dk_done + 1;             // [2], one per issuing warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 2);
  const int n_qt = (S + BQ2 - 1) / BQ2;
  const uint64_t lim = p.timeout_ns;

  if (threadIdx.x == 0) {
    ptx::mbar_init(kv_full, 1);
    for (int s = 0; s < KV_STAGES; ++s) {
      ptx::mbar_init(&q_full[s], 1);  // lane 0's expect_tx (Q_i, dO_i, both X)
      ptx::mbar_init(&q_empty[s], 2);  // the tile's dV and dK products (each after its score product)
    }
    ptx::mbar_init(st_full, 1);
    ptx::mbar_init(dpt_full, 1);
    ptx::mbar_init(pds_full, NSM_B);
    ptx::mbar_init(dv_done, 1);
    ptx::mbar_init(dk_done, 1);
    ptx::mbar_init(&done[0], 1);
    ptx::mbar_init(&done[1], 1);
    ptx::fence_mbar_init();
    ptx::fence_proxy_async_smem();
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, 256);
    ptx::tmem_relinquish();
  }
  // E: rows [1, 1, 0 x 6] (bf16); the X ring and the zero block: zeros
  for (int w = threadIdx.x; w < (KV_RED_OFF - KV_E_OFF) / 16; w += NTHR_B)
    *reinterpret_cast<uint4*>(smem + KV_E_OFF + w * 16) =
        make_uint4(w < BK2 ? 0x3F803F80u : 0u, 0u, 0u, 0u);
  ptx::fence_proxy_async_smem();
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // S^T (then P^T, bf16 pairs), dP^T (then dS^T), dV, dK accumulators.  The
  // column half hf of S^T (queries 32 hf ..) holds that half's P^T in its
  // first 16 columns, so the two halves never write columns the other reads.
  const uint32_t tST = tmem, tdPT = tmem + 64, tdV = tmem + 128, tdK = tmem + 192;

  if (warp == 0) {
    // producer: K, V once; per query tile Q_i, dO_i by TMA and the tile's
    // two X matrices by bulk copy, all completing on q_full
    if (lane == 0) {
      ptx::prefetch_tensormap(&tmK);
      ptx::prefetch_tensormap(&tmQ);
      ptx::prefetch_tensormap(&tmO);
      ptx::mbar_arrive_expect_tx(kv_full, 2 * KV2_BYTES);
      ptx::tma_load_2d(smem + KV_K_OFF, &tmK, kv_full, H + a * HD, row0 + k0);
      ptx::tma_load_2d(smem + KV_V_OFF, &tmK, kv_full, 2 * H + a * HD, row0 + k0);
    }
    // this (sequence, head)'s X_lse rows, followed by its X_delta rows
    const uint4* xs_b = p.xtab + (static_cast<int64_t>(b) * p.A + a) * 2 * S;
    int issued = 0;
    for (int i = 0; i < n_qt && lane == 0; ++i) {
      const int st = i % KV_STAGES;
      if (!ptx::mbar_wait(&q_empty[st], ((i / KV_STAGES) & 1) ^ 1u, lim, p.status, kWaitHint)) break;
      const uint32_t xbytes = static_cast<uint32_t>(min(BQ2, S - i * BQ2)) * XROW_BYTES;
      ptx::mbar_arrive_expect_tx(&q_full[st], 2 * QO2_BYTES + 2 * xbytes);
      ptx::tma_load_2d(smem + KV_Q_OFF + st * QO2_BYTES, &tmQ, &q_full[st], a * HD, row0 + i * BQ2);
      ptx::tma_load_2d(smem + KV_O_OFF + st * QO2_BYTES, &tmO, &q_full[st], a * HD, row0 + i * BQ2);
      uint8_t* x = smem + KV_X_OFF + st * 2 * X_BYTES;
      ptx::bulk_load(x, xs_b + i * BQ2, xbytes, &q_full[st]);
      ptx::bulk_load(x + X_BYTES, xs_b + S + i * BQ2, xbytes, &q_full[st]);
      ++issued;
    }
    if (lane == 0) {
      ptx::mbar_wait(kv_full, 0, lim, p.status, kWaitHint);
      for (int i = issued - 1; i >= 0 && i >= issued - KV_STAGES; --i)
        ptx::mbar_wait(&q_full[i % KV_STAGES], (i / KV_STAGES) & 1, lim, p.status, kWaitHint);
    }
  } else if (warp == 1 || warp == 10) {
    // Warp 1: S^T_i = K Q_i^T, then dV += P^T_i dO_i.  Warp 10: dP^T_i =
    // V dO_i^T, then dK += dS^T_i Q_i.  Each warp's score product of tile i
    // goes in once its accumulating product of tile i - 1 has read the
    // columns it overwrites; the accumulating product once the softmax warps
    // have stored P^T_i / dS^T_i.
    if (lane == 0) {
      const bool v_side = warp == 1;
      constexpr uint32_t idS = ptx::idesc_bf16_f32(BK2, BQ2, false, false);
      constexpr uint32_t idG = ptx::idesc_bf16_f32(BK2, HD, false, true);
      const uint32_t skv = ptx::smem_u32(smem + (v_side ? KV_K_OFF : KV_V_OFF));
      const uint32_t tscore = v_side ? tST : tdPT, tacc = v_side ? tdV : tdK;
      uint64_t* score_full = v_side ? st_full : dpt_full;
      uint64_t* acc_done = v_side ? dv_done : dk_done;
      // K-major operand of the score product (Q_i or dO_i) and MN-major
      // operand of the accumulating product (dO_i or Q_i)
      const int score_off = v_side ? KV_Q_OFF : KV_O_OFF, acc_off = v_side ? KV_O_OFF : KV_Q_OFF;
      const uint32_t se = ptx::smem_u32(smem + KV_E_OFF), sz = ptx::smem_u32(smem + KV_Z_OFF);
      const uint32_t sx = ptx::smem_u32(smem + KV_X_OFF + (v_side ? 0 : X_BYTES));
      bool ok = ptx::mbar_wait(kv_full, 0, lim, p.status, kWaitHint);
      for (int i = 0; i < n_qt && ok; ++i) {
        const int st = i % KV_STAGES;
        if (i >= 1 && !ptx::mbar_wait(acc_done, (i - 1) & 1, lim, p.status, kWaitHint)) break;
        if (!ptx::mbar_wait(&q_full[st], (i / KV_STAGES) & 1, lim, p.status, kWaitHint)) break;
        ptx::tc_fence_after();
        const uint32_t sb = ptx::smem_u32(smem + score_off + st * QO2_BYTES);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          ptx::tc_mma_f16(tscore, ptx::smem_desc_sw128(skv + kk * 32, 16, 1024),
                          ptx::smem_desc_sw128(sb + kk * 32, 16, 1024), idS, kk > 0 ? 1u : 0u);
        // the per-query term: E X^T
        const uint32_t sxs = sx + st * 2 * X_BYTES;
        ptx::tc_mma_f16(tscore, ptx::smem_desc_noswizzle(se, sz - se, 128),
                        ptx::smem_desc_noswizzle(sxs, sz - sxs, 128), idS, 1u);
        ptx::tc_commit(score_full);
        if (!ptx::mbar_wait(pds_full, i & 1, lim, p.status, kWaitHint)) break;
        ptx::tc_fence_after();
        const uint32_t sa = ptx::smem_u32(smem + acc_off + st * QO2_BYTES);
#pragma unroll
        for (int kk = 0; kk < BQ2 / 16; ++kk)  // queries 16 kk ..: half kk / 2, packed column 8 (kk % 2)
          ptx::tc_mma_f16_tmem_a(tacc, tscore + (kk >> 1) * 32 + (kk & 1) * 8,
                                 ptx::smem_desc_sw128(sa + kk * 2048, 8192, 1024), idG,
                                 (i > 0 || kk > 0) ? 1u : 0u);
        ptx::tc_commit(acc_done);
        ptx::tc_commit(&q_empty[st]);
      }
      uint64_t* fin = &done[v_side ? 0 : 1];
      ptx::tc_commit(fin);
      ptx::mbar_wait(fin, 0, lim, p.status, kWaitHint);
    }
  } else {
    const int q4 = warp & 3;
    const int hf = (warp - 2) >> 2;  // column half: queries [32 hf, 32 hf + 32) of a tile
    const int r = q4 * 32 + lane;    // key row within the tile == TMEM lane
    const int key = k0 + r;
    const bool kvalid = key < len;
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    const float sl2 = LOG2E * 0.125f;
    bool ok = true;
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      const bool mine = ptx::mbar_wait(bar, parity, lim, p.status, kWaitHint);
      return __all_sync(0xffffffffu, mine);
    };
    for (int i = 0; i < n_qt; ++i) {
      if (!wait_all(st_full, i & 1) || !wait_all(dpt_full, i & 1)) { ok = false; break; }
      ptx::tc_fence_after();
      uint32_t sv[32], dv[32];
      ptx::tmem_ld_32x32b_x32(tST + lane_base + hf * 32, sv);
      ptx::tmem_ld_32x32b_x32(tdPT + lane_base + hf * 32, dv);
      ptx::tmem_ld_wait();
      // sv = S^T - lse2 / c and dv = dP^T - delta, the terms added by the MMAs
      uint32_t pp[16], dd[16];
#pragma unroll
      for (int t = 0; t < 32; t += 2) {
        float pt[2], ds[2];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          pt[e] = kvalid ? ptx::ex2_ftz(__uint_as_float(sv[t + e]) * sl2) : 0.f;
          ds[e] = pt[e] * __uint_as_float(dv[t + e]);
        }
        pp[t >> 1] = ptx::pack_bf16(pt[0], pt[1]);
        dd[t >> 1] = ptx::pack_bf16(ds[0], ds[1]);
      }
      const int nq = S - i * BQ2 - hf * 32;  // queries of this half inside the sequence
      if (nq < 32) {  // warp-uniform: queries past S
#pragma unroll
        for (int t = 0; t < 32; t += 2) {
          const uint32_t keep = (t < nq ? 0x0000ffffu : 0u) | (t + 1 < nq ? 0xffff0000u : 0u);
          pp[t >> 1] &= keep;
          dd[t >> 1] &= keep;
        }
      }
      // over the columns this thread has just read: P^T_i, dS^T_i as bf16 pairs
      ptx::tmem_st_32x32b_x16(tST + lane_base + hf * 32, pp);
      ptx::tmem_st_32x32b_x16(tdPT + lane_base + hf * 32, dd);
      ptx::tmem_st_wait();
      ptx::tc_fence_before();
      ptx::mbar_arrive(pds_full);
    }
    // epilogue: the low-half warps stage dK / sqrt(D), the high-half warps dV,
    // as 128-byte-swizzled bf16 rows over the K / V tiles (the last score
    // products have read them); one thread then stores both tiles by TMA
    // through a [B][S][3H] map, which drops the rows past S.
    float* red = reinterpret_cast<float*>(smem + KV_RED_OFF);  // [2 halves][4 quarters][64]
    if (ok && wait_all(dv_done, (n_qt - 1) & 1) && wait_all(dk_done, (n_qt - 1) & 1)) {
      ptx::tc_fence_after();
      const uint32_t tacc = hf == 0 ? tdK : tdV;
      const float sc = hf == 0 ? 0.125f : 1.f;
      const uint32_t orow = ptx::smem_u32(smem + (hf == 0 ? KV_K_OFF : KV_V_OFF)) + r * 128;
      uint32_t o[2][32];
      ptx::tmem_ld_32x32b_x32(tacc + lane_base, o[0]);
      ptx::tmem_ld_32x32b_x32(tacc + lane_base + 32, o[1]);
      ptx::tmem_ld_wait();
#pragma unroll
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          uint32_t w[4];
#pragma unroll
          for (int t = 0; t < 4; ++t)
            w[t] = ptx::pack_bf16(__uint_as_float(o[c][8 * u + 2 * t]) * sc,
                                  __uint_as_float(o[c][8 * u + 2 * t + 1]) * sc);
          ptx::st_shared_v4(orow + (((c * 4 + u) ^ (r & 7)) << 4), w[0], w[1], w[2], w[3]);
        }
      if (p.colpart) {  // column sums of the stored values over this warp's 32 rows
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = key < S ? bf16_round(__uint_as_float(o[c][j]) * sc) : 0.f;
          lanes_column_sum(v, lane);
          red[(hf * 4 + q4) * 64 + c * 32 + lane] = v[0];
        }
      }
    } else if (p.colpart) {
      red[(hf * 4 + q4) * 64 + lane] = 0.f;
      red[(hf * 4 + q4) * 64 + 32 + lane] = 0.f;
    }
    ptx::fence_proxy_async_smem();  // the staged rows -> the TMA store
    softmax_warps_sync();
    if (warp == 2 && lane == 0) {
      ptx::tma_store_3d(&tmOut, smem + KV_K_OFF, H + a * HD, k0, b);
      ptx::tma_store_3d(&tmOut, smem + KV_V_OFF, 2 * H + a * HD, k0, b);
      ptx::bulk_commit_group();
    }
    if (p.colpart && q4 == 0) {  // the four row quarters, added in order, by the quarter-0 warps
      const float* rh = red + hf * 4 * 64;
      float* dst = p.colpart + (static_cast<int64_t>(b) * gridDim.x + kt) * rs + (1 + hf) * H + a * HD;
#pragma unroll
      for (int c = lane; c < 64; c += 32)
        dst[c] = ((rh[c] + rh[64 + c]) + rh[128 + c]) + rh[192 + c];
    }
    if (warp == 2 && lane == 0) ptx::bulk_wait_group_read0();  // before the CTA's memory goes
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

// dQKV as [B][S][3H] bf16 for the dK/dV tile stores: box {64 columns, 128
// rows of one sequence}, 128B swizzle; rows past S fall outside the tensor.
bool seq_map(CUtensorMap* map, void* base, int B, int S, int W, int rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(W), static_cast<cuuint64_t>(S),
                        static_cast<cuuint64_t>(B)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(W) * 2, static_cast<cuuint64_t>(W) * 2 * S};
  cuuint32_t box[3] = {64u, static_cast<cuuint32_t>(rows), 1u};
  cuuint32_t estr[3] = {1u, 1u, 1u};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
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
  CUtensorMap tq, tkv, tout;
  const int64_t T = static_cast<int64_t>(B) * S;
  SKY_CHECK(head_map(&tq, qkv, T, 3 * H, BQ) && head_map(&tkv, qkv, T, 3 * H, BKV) &&
                seq_map(&tout, ctx, B, S, H, BQ),
            SKY_ERR_CUDA,
            "cuTensorMapEncodeTiled failed for the attention operands");
  static cudaError_t attr = cudaFuncSetAttribute(attn_fwd_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 F_SMEM);
  if (attr != cudaSuccess) return cuda_fail(attr, "attention smem attribute");
  FwdParams p{S, H, A, lens, static_cast<__nv_bfloat16*>(ctx), lse, status, timeout_ns};
  dim3 grid(ceil_div(S, BQ), A, B);
  const cudaError_t e = launch_pdl(attn_fwd_tc, grid, dim3(NTHR), F_SMEM, stream, 1, tq, tkv, tout, p);
  count_launches(1);
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "tensor-core attention forward launch");
}

// Backward launchers (bf16, D = 64): delta must already hold rowsum(dO * O).
sky_status attention_bwd_tc(const void* qkv, const void* dctx, const float* lse, const float* delta,
                            const uint4* xtab, const int32_t* lens, int B, int S, int H, int A, void* dqkv,
                            int32_t* status, uint64_t timeout_ns, cudaStream_t stream,
                            float* colpart) {
  using namespace attn_tc;
  SKY_CHECK(H == A * HD, SKY_ERR_UNSUPPORTED, "tensor-core attention needs head dim 64");
  const int64_t T = static_cast<int64_t>(B) * S;
  CUtensorMap tq128, tkv64, to128, tk128, tq64, to64, tout;
  SKY_CHECK(head_map(&tq128, qkv, T, 3 * H, BQ) && head_map(&tkv64, qkv, T, 3 * H, BKV) &&
                head_map(&to128, dctx, T, H, BQ) && head_map(&tk128, qkv, T, 3 * H, BK2) &&
                head_map(&tq64, qkv, T, 3 * H, BQ2) && head_map(&to64, dctx, T, H, BQ2) &&
                seq_map(&tout, dqkv, B, S, 3 * H, BK2),
            SKY_ERR_CUDA, "cuTensorMapEncodeTiled failed for the attention backward operands");
  static cudaError_t a1 = cudaFuncSetAttribute(attn_bwd_dq_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, DQ_SMEM);
  static cudaError_t a2 = cudaFuncSetAttribute(attn_bwd_dkdv_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, KV_SMEM);
  if (a1 != cudaSuccess) return cuda_fail(a1, "attention dQ smem attribute");
  if (a2 != cudaSuccess) return cuda_fail(a2, "attention dK/dV smem attribute");
  SKY_CHECK((reinterpret_cast<uintptr_t>(xtab) & 15) == 0, SKY_ERR_INVALID_ARG,
            "attention backward workspace must be 16-byte aligned");
  BwdParams p{S, H, A, lens, lse, delta, xtab, static_cast<__nv_bfloat16*>(dqkv), colpart, status,
              timeout_ns};
  cudaError_t e = launch_pdl(attn_bwd_dkdv_tc, dim3(ceil_div(S, BK2), A, B), dim3(NTHR_B), KV_SMEM,
                             stream, 1, tk128, tq64, to64, tout, p);
  if (e == cudaSuccess)
    e = launch_pdl(attn_bwd_dq_tc, dim3(ceil_div(S, BQ), A, B), dim3(NTHR_B), DQ_SMEM, stream, 1,
                   tq128, tkv64, to128, tout, p);
  count_launches(2);
  return e == cudaSuccess ? SKY_OK : cuda_fail(e, "tensor-core attention backward launch");
}

}  // namespace sky
