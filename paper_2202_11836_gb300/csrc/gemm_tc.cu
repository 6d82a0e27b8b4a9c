// bf16 GEMMs of the encoder layer on the 5th-generation tensor cores.
//
// The linear maps of Sec. II-C (Q/K/V projection, attention-output dense,
// intermediate and output layers) and their input and weight gradients are
// the dense contractions of the slice.  One persistent, warp-specialised
// kernel serves all three contraction forms:
//   warp 0      TMA producer: 128-byte-swizzled tiles of A and B into a
//               STAGES-deep shared-memory ring (mbarrier complete_tx),
//   warp 1      MMA issuer: one thread issues tcgen05.mma (M=128, N=256,
//               K=16) into a TMEM accumulator; two accumulators (512 TMEM
//               columns) let the epilogue of one tile overlap the next,
//   warps 2..9  epilogue (two warps per TMEM lane quarter, one per half of
//               the tile's columns; 2..17 and a quarter of the columns each
//               for bias + GELU): tcgen05.ld of the accumulator, a
//               transpose through shared memory so stores coalesce, fused
//               bias / GELU, store to global memory.  The forward GELU
//               epilogue also stores GELU'(z) (fp16); the backward epilogue
//               multiplies by it, loading it for the whole tile before the
//               accumulator is waited on so its latency hides under the
//               tile's main loop.
// K-major operands (x and W in y = x W^T) and MN-major operands (W in
// dy W, and both operands of dy^T x) are read directly through the
// descriptors' major-ness bit, so no transpose pass exists.
// Large problems run the CTA-pair variant: a cluster of two CTAs on two SMs
// computes a 256 x 256 tile with tcgen05.mma.cta_group::2 (M = 256); each CTA
// loads its 128 rows of A and half of the tile's B columns, so every SM moves
// a third less operand data per FLOP through shared memory and L2 than with
// the single-CTA 128 x 256 tile.  The leader CTA's thread issues the MMAs;
// both CTAs' TMA loads complete on the leader's stage barrier, and the
// leader's commits arrive on both CTAs' stage-empty and accumulator barriers.
// Weight gradients (fp32 output) may split the token dimension over CTAs;
// partials go to a workspace and are summed in a fixed order, so results are
// deterministic.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include <cuda_fp16.h>

#include "common.cuh"
#include "gemm.h"
#include "ptx.cuh"

namespace sky {
namespace gemm {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;        // 16 KiB
constexpr int NUM_EPI_WARPS = 8;            // two per TMEM lane quarter (default)
constexpr int MN_CHUNK_BYTES = 64 * BK * 2; // one 64-wide MN-major box: 8 KiB
// CTA-pair variant: per CTA and stage A 128 x 64 + B 128 x 64 (32 KiB).  Six
// stages (192 KiB) for every epilogue but the GELU' data gradient, which
// keeps five: with six, its kernel ran 5 us slower (its epilogue prefetches
// the whole tile's GELU'(z) and competes for bandwidth with the deeper
// ring), while the others ran 1-2 us faster and the step 0.7% faster.
constexpr int PAIR_STAGES = 5;
constexpr int PAIR_STAGES_WIDE = 6;  // all but the GELU' data-gradient epilogue

// Launch shape per instantiation: epilogue warps (a multiple of 4, one group
// per TMEM lane quarter), epilogue chunk width, ring stages and shared memory.
// The bias+GELU epilogue is bound by its own math: it runs 16 warps (four per
// lane quarter, 64 columns each) on 16-column chunks, which keeps it at about
// 100 registers a thread (576 threads leave 112).
// TBN: the tile's width (256, or 192 for K-major B operands whose output
// width fills the SM pairs better in 192-wide tiles).
template <int EPI, bool PAIR, int TBN = BN>
struct Shape {
  static constexpr int EW = EPI == SKY_EPI_BIAS_GELU ? 16 : NUM_EPI_WARPS;
  static constexpr int CW = EW == 16 ? 16 : 32;              // epilogue chunk width (columns)
  static constexpr int THREADS = 64 + 32 * EW;
  static constexpr int NST = PAIR ? (EPI == SKY_EPI_GELU_BWD ? PAIR_STAGES : PAIR_STAGES_WIDE) : STAGES;
  static constexpr int SBYTES = A_BYTES + (PAIR ? TBN / 2 : TBN) * BK * 2;
  // two fp32 accumulators of 128 x TBN, in a power-of-two TMEM allocation
  static constexpr int TMEM_ALLOC = 2 * TBN <= 256 ? 256 : 512;
  static constexpr int EPI_OFF = NST * SBYTES;               // per epilogue warp: 32 x CW fp32 staging
  static constexpr int BAR_OFF = EPI_OFF + EW * 32 * CW * 4;
  static constexpr int SMEM = BAR_OFF + 256 /*barriers*/ + 1024 /*alignment slack*/;
  static_assert(SMEM <= 232448, "shared memory per CTA");
};
constexpr uint32_t kSleepNs = 20000;         // suspend hint of the epilogue's accumulator wait

struct Params {
  int M, N, K;
  int m_tiles, n_tiles, splits, kb_per_split, k_blocks;
  void* C;                        // bf16 [M,N], fp32 [M,N], or fp32 [splits][M][N]
  const __nv_bfloat16* bias;      // [N] or null
  const __half* aux;              // [M,N] GELU'(z) (GELU_BWD) or null
  __half* aux_out;                // [M,N] GELU'(z) (BIAS_GELU) or null
  float* colpart;                 // [m_tiles * 4][N] per-warp column sums of C, or null
  const float* resid;             // [M,N] fp32 added after the bias (fp32 outputs), or null
  const float* ln_mean;           // [M] with ln_rstd, ln_gamma, ln_beta: resid is the
  const float* ln_rstd;           //   pre-LayerNorm sum u and LN(u) is added, or null
  const __nv_bfloat16* ln_gamma;  // [N]
  const __nv_bfloat16* ln_beta;   // [N]
  int32_t* status;
  uint64_t timeout_ns;
  int skip_loads;                 // fault injection: producer never issues TMA
};

// 8-byte read-only load that does not allocate in L1 (streamed once).
__device__ __forceinline__ uint2 ld_nc_u2(const void* p) {
  uint2 v;
  asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0, %1}, [%2];"
               : "=r"(v.x), "=r"(v.y)
               : "l"(p));
  return v;
}
__device__ __forceinline__ float4 ld_nc_f4(const float* p) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p));
  return v;
}

// ---- work schedule ------------------------------------------------------
// Every persistent CTA (pair) walks the same list of work units cid, cid +
// ncl, cid + 2 ncl, ... of the tiles * splits (split-major): unit u is tile
// u % tiles over the k-blocks of split u / tiles.
struct Work {
  int tile, split, kb0, kb1;
};
struct Sched {
  int tiles, units, kbps, kbs, ncl, cid;
};
__device__ __forceinline__ bool work_item(const Sched& sched, int it, Work& w) {
  const int u = sched.cid + it * sched.ncl;
  if (u >= sched.units) return false;
  w.split = u / sched.tiles;
  w.tile = u - w.split * sched.tiles;
  w.kb0 = w.split * sched.kbps;
  w.kb1 = min(sched.kbs, w.kb0 + sched.kbps);
  return true;
}

// PAIR: the CTA-pair variant (launched in clusters of two; p.m_tiles counts
// 256-row tiles).
template <bool A_MN, bool B_MN, int EPI, bool OUT_F32, bool PAIR, int TBN = BN>
__global__ void __launch_bounds__(Shape<EPI, PAIR, TBN>::THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA,
                   const __grid_constant__ CUtensorMap tmB, const Params p) {
  using SH = Shape<EPI, PAIR, TBN>;
  constexpr int NST = SH::NST;
  constexpr int SBYTES = SH::SBYTES;
  constexpr int EW = SH::EW;
  constexpr int B_ROWS = PAIR ? TBN / 2 : TBN;  // B rows (tile columns) this CTA loads
  static_assert(!B_MN || B_ROWS % 64 == 0, "MN-major B is loaded in 64-column boxes");
  constexpr int TILE_M = PAIR ? 2 * BM : BM;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + SH::BAR_OFF);
  uint64_t* empty = full + NST;
  uint64_t* tfull = empty + NST;
  uint64_t* tempty = tfull + 2;
  uint64_t* done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);

  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = PAIR ? ptx::cluster_ctarank() : 0u;
  const bool leader = rank == 0;
  const int cid = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int ncl = PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
  if (threadIdx.x == 0) {
    for (int s = 0; s < NST; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(&tfull[a], 1);
      ptx::mbar_init(&tempty[a], (PAIR ? 2 : 1) * 32 * EW);
    }
    ptx::mbar_init(done, 1);
    if constexpr (PAIR) ptx::fence_mbar_init_cluster();
    else ptx::fence_mbar_init();
    ptx::fence_proxy_async_smem();
    ptx::prefetch_tensormap(&tmA);
    ptx::prefetch_tensormap(&tmB);
  }
  if (warp == 1) {
    if constexpr (PAIR) {
      ptx::tmem_alloc_pair(tmem_slot, SH::TMEM_ALLOC);
      ptx::tmem_relinquish_pair();
    } else {
      ptx::tmem_alloc(tmem_slot, SH::TMEM_ALLOC);
      ptx::tmem_relinquish();
    }
  }
  ptx::tc_fence_before();
  __syncwarp();
  if constexpr (PAIR) ptx::cluster_sync();  // barriers of both CTAs initialised
  else __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();  // the set-up above overlapped the previous kernel; its outputs are visible now

  const uint64_t lim = p.timeout_ns;
  const Sched sched{p.m_tiles * p.n_tiles, p.m_tiles * p.n_tiles * p.splits, p.kb_per_split,
                    p.k_blocks, ncl, cid};
  Work w;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      bool ok = true;
      for (int it = 0; ok && work_item(sched, it, w); ++it) {
        const int m0 = (w.tile / p.n_tiles) * TILE_M + static_cast<int>(rank) * BM;
        const int n0 = (w.tile % p.n_tiles) * TBN + static_cast<int>(rank) * (TBN - B_ROWS);
        for (int kb = w.kb0; kb < w.kb1; ++kb) {
          if (!ptx::mbar_wait(&empty[stage], phase ^ 1u, lim, p.status)) { ok = false; break; }
          uint8_t* sa = smem + stage * SBYTES;
          uint8_t* sb = sa + A_BYTES;
          // the leader's stage barrier expects both CTAs' bytes
          if (leader) ptx::mbar_arrive_expect_tx(&full[stage], (PAIR ? 2 : 1) * SBYTES);
          if (!p.skip_loads) {
            const int k0 = kb * BK;
            auto load = [&](void* dst, const CUtensorMap* map, int c0, int c1) {
              if constexpr (PAIR)
                ptx::tma_load_2d_pair(dst, map, ptx::mapa_shared(ptx::smem_u32(&full[stage]), 0),
                                      c0, c1);
              else
                ptx::tma_load_2d(dst, map, &full[stage], c0, c1);
            };
            if (A_MN) {
              load(sa, &tmA, m0, k0);
              load(sa + MN_CHUNK_BYTES, &tmA, m0 + 64, k0);
            } else {
              load(sa, &tmA, k0, m0);
            }
            if (B_MN) {
#pragma unroll
              for (int j = 0; j < B_ROWS / 64; ++j)
                load(sb + j * MN_CHUNK_BYTES, &tmB, n0 + 64 * j, k0);
            } else {
              load(sb, &tmB, k0, n0);
            }
          }
          ++issued;
          if (++stage == NST) { stage = 0; phase ^= 1u; }
        }
      }
      // Drain: wait (bounded) for the loads still in flight before exiting.
      // The leader's stage barriers count the peer's loads too; the peer
      // stays resident until the leader has drained (final cluster barrier).
      const int n_tail = !leader ? 0 : (issued < NST ? issued : NST);
      for (int i = 0; i < n_tail; ++i) {
        if (--stage < 0) { stage = NST - 1; phase ^= 1u; }
        ptx::mbar_wait(&full[stage], phase, lim, p.status);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issue
    if (lane == 0 && leader) {
      constexpr uint32_t idesc = ptx::idesc_bf16_f32(TILE_M, TBN, A_MN, B_MN);
      auto commit = [&](uint64_t* bar) {  // to this barrier in both CTAs of a pair
        if constexpr (PAIR) ptx::tc_commit_pair(bar, 3);
        else ptx::tc_commit(bar);
      };
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t aphase = 0;
      bool ok = true;
      for (int it = 0; ok && work_item(sched, it, w); ++it) {
        // both CTAs' epilogues have drained this accumulator
        if (!(PAIR ? ptx::mbar_wait_cluster(&tempty[acc], aphase ^ 1u, lim, p.status)
                   : ptx::mbar_wait(&tempty[acc], aphase ^ 1u, lim, p.status)))
          break;
        ptx::tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * TBN;
        for (int kb = w.kb0; kb < w.kb1; ++kb) {
          if (!ptx::mbar_wait(&full[stage], phase, lim, p.status)) { ok = false; break; }
          ptx::tc_fence_after();
          const uint32_t sa = ptx::smem_u32(smem + stage * SBYTES);
          const uint32_t sb = sa + A_BYTES;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint64_t ad = A_MN ? ptx::smem_desc_sw128(sa + kk * 2048, MN_CHUNK_BYTES, 1024)
                                     : ptx::smem_desc_sw128(sa + kk * 32, 16, 1024);
            const uint64_t bd = B_MN ? ptx::smem_desc_sw128(sb + kk * 2048, MN_CHUNK_BYTES, 1024)
                                     : ptx::smem_desc_sw128(sb + kk * 32, 16, 1024);
            if constexpr (PAIR)
              ptx::tc_mma_f16_pair(d_tmem, ad, bd, idesc, (kb > w.kb0 || kk > 0) ? 1u : 0u);
            else
              ptx::tc_mma_f16(d_tmem, ad, bd, idesc, (kb > w.kb0 || kk > 0) ? 1u : 0u);
          }
          commit(&empty[stage]);
          if (++stage == NST) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        commit(&tfull[acc]);
        if (++acc == 2) { acc = 0; aphase ^= 1u; }
      }
      // All issued MMAs must finish before TMEM is released.
      if constexpr (PAIR) ptx::tc_commit_pair(done, 1);
      else ptx::tc_commit(done);
      ptx::mbar_wait(done, 0, lim, p.status);
    }
  } else {
    // -------------------------------------------------------------- epilogue
    // Warp w owns TMEM lanes [32q, 32q+32) (q = w % 4: rows m0+32q..) and the
    // column half hf of the tile.  Per 32-column chunk: tcgen05.ld (thread =
    // row) -> XOR-swizzled smem tile -> read back so that 8 lanes cover one
    // row's 32 columns, then the fused epilogue and coalesced stores.
    constexpr int HALF = TBN / (EW / 4), CHUNKS = HALF / 32;  // columns of a warp, 32-column chunks
    const int q = warp & 3, hf = (warp - 2) >> 2;
    float* stage = reinterpret_cast<float*>(smem + SH::EPI_OFF) + (warp - 2) * 32 * SH::CW;
    const int c4 = lane & 7;          // this lane's 4-column group in a chunk
    const int rsub = lane >> 3;       // row within each group of 4 rows
    int acc = 0;
    uint32_t aphase = 0;
    // hands the accumulator back to the MMA issuer (both CTAs' epilogues arrive
    // on the leader's barrier)
    auto release_acc = [&]() {
      ptx::tc_fence_before();
      if (leader) ptx::mbar_arrive(&tempty[acc]);
      else ptx::mbar_arrive_cluster(ptx::mapa_shared(ptx::smem_u32(&tempty[acc]), 0));
      if (++acc == 2) { acc = 0; aphase ^= 1u; }
    };
    for (int it = 0; work_item(sched, it, w); ++it) {
      const int m0 = (w.tile / p.n_tiles) * TILE_M + static_cast<int>(rank) * BM;
      const int n0 = (w.tile % p.n_tiles) * TBN + hf * HALF;
      // GELU' input of this warp's whole sub-tile, fetched before the wait
      uint2 pre[EPI == SKY_EPI_GELU_BWD ? CHUNKS : 1][8];
      if constexpr (EPI == SKY_EPI_GELU_BWD) {
#pragma unroll
        for (int cc = 0; cc < CHUNKS; ++cc) {
          const int col = n0 + cc * 32 + 4 * c4;
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int row = m0 + q * 32 + 4 * i + rsub;
            pre[cc][i] = (col < p.N && row < p.M)
                                            ? ld_nc_u2(p.aux + static_cast<int64_t>(row) * p.N + col)
                             : make_uint2(0u, 0u);
          }
        }
      }
      // fp32 residual (post-LN residual branch), one 32-column chunk ahead:
      // chunk 0 before the accumulator wait, chunk cc+1 while cc is stored
      const float* rp = OUT_F32 ? p.resid : nullptr;
      float4 res[OUT_F32 ? 8 : 1];
      auto load_res = [&](int cc, float4* d) {
        const int col = n0 + cc * 32 + 4 * c4;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int row = m0 + q * 32 + 4 * i + rsub;
          d[i] = (col < p.N && row < p.M) ? ld_nc_f4(rp + static_cast<int64_t>(row) * p.N + col)
                                          : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      };
      if constexpr (OUT_F32) {
        if (rp) load_res(0, res);
      }
      // LayerNorm residual: this lane's 8 rows' statistics (the same rows in
      // every chunk)
      const bool ln = OUT_F32 && rp && p.ln_mean;
      float mu[OUT_F32 ? 8 : 1], rs[OUT_F32 ? 8 : 1];
      if constexpr (OUT_F32) {
        if (ln) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int row = m0 + q * 32 + 4 * i + rsub;
            mu[i] = row < p.M ? __ldg(p.ln_mean + row) : 0.f;
            rs[i] = row < p.M ? __ldg(p.ln_rstd + row) : 0.f;
          }
        }
      }
      if (!ptx::mbar_wait(&tfull[acc], aphase, lim, p.status, kSleepNs)) break;
      ptx::tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + acc * TBN + hf * HALF;
      float* outf = OUT_F32 ? static_cast<float*>(p.C) +
                                  static_cast<int64_t>(w.split) * p.M * static_cast<int64_t>(p.N)
                            : nullptr;
      if constexpr (EPI == SKY_EPI_BIAS_GELU) {
        // CW-column chunks: LPR lanes cover a row's CW columns, RPI rows per step
        constexpr int CW = SH::CW, LPR = CW / 4, RPI = 32 / LPR, NI = 32 / RPI;
        const int g4 = lane % LPR, grs = lane / LPR;
        auto swz = [](int row) { return CW == 32 ? (row & 7) : ((row >> 1) & 3); };
#pragma unroll 1
        for (int c = 0; c < HALF; c += CW) {
          uint32_t r[CW];
          __syncwarp();
          if constexpr (CW == 16) ptx::tmem_ld_32x32b_x16(taddr + c, *reinterpret_cast<uint32_t(*)[16]>(r));
          else ptx::tmem_ld_32x32b_x32(taddr + c, *reinterpret_cast<uint32_t(*)[32]>(r));
          ptx::tmem_ld_wait();
          if (n0 + c >= p.N) continue;  // warp-uniform
#pragma unroll
          for (int j = 0; j < CW / 4; ++j)
            *reinterpret_cast<float4*>(stage + lane * CW + ((j ^ swz(lane)) << 2)) =
                make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                            __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
          __syncwarp();
          const int col = n0 + c + 4 * g4;
          if (col >= p.N) continue;
          const uint2 braw = *reinterpret_cast<const uint2*>(p.bias + col);
          const __nv_bfloat162* bh = reinterpret_cast<const __nv_bfloat162*>(&braw);
          const float2 bf0 = __bfloat1622float2(bh[0]), bf1 = __bfloat1622float2(bh[1]);
          const float b4[4] = {bf0.x, bf0.y, bf1.x, bf1.y};
#pragma unroll
          for (int i = 0; i < NI; ++i) {
            const int rl = RPI * i + grs;
            const float4 t4 = *reinterpret_cast<const float4*>(stage + rl * CW + ((g4 ^ swz(rl)) << 2));
            float z[4] = {t4.x + b4[0], t4.y + b4[1], t4.z + b4[2], t4.w + b4[3]}, gp[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) gelu_and_grad_as(z[j], z[j], gp[j]);
            const int row = m0 + q * 32 + rl;
            if (row < p.M) {
              const int64_t off = static_cast<int64_t>(row) * p.N + col;
              const __half2 h0 = __floats2half2_rn(gp[0], gp[1]), h1 = __floats2half2_rn(gp[2], gp[3]);
              *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.C) + off) =
                  make_uint2(ptx::pack_bf16(z[0], z[1]), ptx::pack_bf16(z[2], z[3]));
              // GELU'(z) is read again only by the backward pass: a streaming
              // store keeps it from displacing G, which FFN2 reads next, in L2
              __stcs(reinterpret_cast<uint2*>(p.aux_out + off),
                     make_uint2(*reinterpret_cast<const uint32_t*>(&h0),
                                *reinterpret_cast<const uint32_t*>(&h1)));
            }
          }
        }
      } else
#pragma unroll CHUNKS
      for (int cc = 0; cc < CHUNKS; ++cc) {
        const int c = cc * 32;
        uint32_t r[32];
        __syncwarp();
        ptx::tmem_ld_32x32b_x32(taddr + c, r);
        ptx::tmem_ld_wait();
        if (n0 + c >= p.N) continue;  // warp-uniform
        // stage: row `lane`, 16-byte chunk j at position j ^ (lane & 7)
#pragma unroll
        for (int j = 0; j < 8; ++j)
          *reinterpret_cast<float4*>(stage + lane * 32 + ((j ^ (lane & 7)) << 2)) =
              make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                          __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
        __syncwarp();
        const int col = n0 + c + 4 * c4;
        const bool col_ok = col < p.N;
        float b4[4] = {0.f, 0.f, 0.f, 0.f};
        if (p.bias && col_ok) {
          const uint2 raw = *reinterpret_cast<const uint2*>(p.bias + col);
          const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&raw);
          const float2 f0 = __bfloat1622float2(h[0]), f1 = __bfloat1622float2(h[1]);
          b4[0] = f0.x; b4[1] = f0.y; b4[2] = f1.x; b4[3] = f1.y;
        }
        // all 8 rows x 4 columns first (independent, branch-free), then the
        // bounds-checked stores
        float4 nxt[OUT_F32 ? 8 : 1];
        if constexpr (OUT_F32) {
          if (rp && cc + 1 < CHUNKS) load_res(cc + 1, nxt);
        }
        float v[8][4];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int rl = 4 * i + rsub;
          const float4 t4 = *reinterpret_cast<const float4*>(stage + rl * 32 + ((c4 ^ (rl & 7)) << 2));
          v[i][0] = t4.x + b4[0]; v[i][1] = t4.y + b4[1]; v[i][2] = t4.z + b4[2]; v[i][3] = t4.w + b4[3];
        }
        if constexpr (OUT_F32) {
          if (ln) {
            float g4[4] = {0.f, 0.f, 0.f, 0.f}, e4[4] = {0.f, 0.f, 0.f, 0.f};
            if (col_ok) {
              const uint2 gr = *reinterpret_cast<const uint2*>(p.ln_gamma + col);
              const uint2 er = *reinterpret_cast<const uint2*>(p.ln_beta + col);
              const __nv_bfloat162* gh = reinterpret_cast<const __nv_bfloat162*>(&gr);
              const __nv_bfloat162* eh = reinterpret_cast<const __nv_bfloat162*>(&er);
              const float2 g0 = __bfloat1622float2(gh[0]), g1 = __bfloat1622float2(gh[1]);
              const float2 e0 = __bfloat1622float2(eh[0]), e1 = __bfloat1622float2(eh[1]);
              g4[0] = g0.x; g4[1] = g0.y; g4[2] = g1.x; g4[3] = g1.y;
              e4[0] = e0.x; e4[1] = e0.y; e4[2] = e1.x; e4[3] = e1.y;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const float u4[4] = {res[i].x, res[i].y, res[i].z, res[i].w};
#pragma unroll
              for (int j = 0; j < 4; ++j) v[i][j] += g4[j] * ((u4[j] - mu[i]) * rs[i]) + e4[j];
              res[i] = nxt[i];
            }
          } else if (rp) {
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              v[i][0] += res[i].x; v[i][1] += res[i].y; v[i][2] += res[i].z; v[i][3] += res[i].w;
              res[i] = nxt[i];
            }
          }
        }
        if constexpr (EPI == SKY_EPI_GELU_BWD) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const __half2* h = reinterpret_cast<const __half2*>(&pre[cc][i]);
            const float2 f0 = __half22float2(h[0]), f1 = __half22float2(h[1]);
            v[i][0] *= f0.x; v[i][1] *= f0.y; v[i][2] *= f1.x; v[i][3] *= f1.y;
          }
        }
        uint2 gq[EPI == SKY_EPI_BIAS_GELU ? 8 : 1];
        if constexpr (EPI == SKY_EPI_BIAS_GELU) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            float gp[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) gelu_and_grad_as(v[i][j], v[i][j], gp[j]);
            const __half2 h0 = __floats2half2_rn(gp[0], gp[1]), h1 = __floats2half2_rn(gp[2], gp[3]);
            gq[i] = make_uint2(*reinterpret_cast<const uint32_t*>(&h0),
                               *reinterpret_cast<const uint32_t*>(&h1));
          }
        }
        if (p.colpart) {
          // column sums of this warp's 32 rows (the bias gradient), fixed order
          float cs[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int i = 0; i < 8; ++i)
            if (m0 + q * 32 + 4 * i + rsub < p.M) {
#pragma unroll
              for (int j = 0; j < 4; ++j) cs[j] += v[i][j];
            }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            cs[j] += __shfl_xor_sync(0xffffffffu, cs[j], 8);
            cs[j] += __shfl_xor_sync(0xffffffffu, cs[j], 16);
          }
          if (rsub == 0 && col_ok)
            *reinterpret_cast<float4*>(p.colpart + (static_cast<int64_t>(m0 / 32 + q)) * p.N + col) =
                make_float4(cs[0], cs[1], cs[2], cs[3]);
        }
        if (col_ok) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int row = m0 + q * 32 + 4 * i + rsub;
            if (row >= p.M) continue;
            const int64_t off = static_cast<int64_t>(row) * p.N + col;
            if constexpr (OUT_F32) {
              *reinterpret_cast<float4*>(outf + off) = make_float4(v[i][0], v[i][1], v[i][2], v[i][3]);
            } else {
              *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.C) + off) =
                  make_uint2(ptx::pack_bf16(v[i][0], v[i][1]), ptx::pack_bf16(v[i][2], v[i][3]));
              if constexpr (EPI == SKY_EPI_BIAS_GELU)
                __stcs(reinterpret_cast<uint2*>(p.aux_out + off), gq[i]);
            }
          }
        }
      }
      release_acc();
    }
  }

  ptx::tc_fence_before();
  __syncwarp();
  if constexpr (PAIR) ptx::cluster_sync();  // no CTA leaves while its peer may still signal it
  else __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    if constexpr (PAIR) ptx::tmem_dealloc_pair(tmem_base, SH::TMEM_ALLOC);
    else ptx::tmem_dealloc(tmem_base, SH::TMEM_ALLOC);
  }
}

// Fixed-order sum of split-K partials: out[i] = sum_s ws[s][i], added in
// split order.  SPLITS > 0: every split's load of a vector is issued before
// the first add (a loop over a run-time count would wait for each load in
// turn); SPLITS == 0: any count.
template <int SPLITS>
__global__ void splitk_reduce_kernel(const float* __restrict__ ws, int splits, int64_t n,
                                     float* __restrict__ out) {
  pdl_trigger();
  pdl_wait();
  const int64_t n4 = n / 4;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4;
       i += (int64_t)gridDim.x * blockDim.x) {
    float4 acc;
    if constexpr (SPLITS > 0) {
      float4 v[SPLITS];
#pragma unroll
      for (int s = 0; s < SPLITS; ++s) v[s] = reinterpret_cast<const float4*>(ws + s * n)[i];
      acc = v[0];
#pragma unroll
      for (int s = 1; s < SPLITS; ++s) {
        acc.x += v[s].x; acc.y += v[s].y; acc.z += v[s].z; acc.w += v[s].w;
      }
    } else {
      acc = reinterpret_cast<const float4*>(ws)[i];
      for (int s = 1; s < splits; ++s) {
        const float4 v = reinterpret_cast<const float4*>(ws + s * n)[i];
        acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
      }
    }
    reinterpret_cast<float4*>(out)[i] = acc;
  }
  for (int64_t i = n4 * 4 + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    float acc = ws[i];
    for (int s = 1; s < splits; ++s) acc += ws[s * n + i];
    out[i] = acc;
  }
}

// ------------------------------------------------------------------- host
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

// 2-D bf16 tensor map over a row-major [rows, cols] matrix, box {64, box_rows},
// 128-byte swizzle; out-of-range elements read as zero.
bool make_map(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {64u, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1u, 1u};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Launches the product's work units on a persistent grid: one CTA per SM, or
// for the pair variant one two-CTA cluster per SM pair, capped by how many
// such clusters the device holds at once (a single wave).
template <bool A_MN, bool B_MN, int EPI, bool OUT_F32, bool PAIR, int TBN = BN>
cudaError_t launch_variant(const Params& p, int sms, const CUtensorMap& ta, const CUtensorMap& tb,
                           cudaStream_t stream) {
  auto kern = gemm_tc_kernel<A_MN, B_MN, EPI, OUT_F32, PAIR, TBN>;
  using SH = Shape<EPI, PAIR, TBN>;
  static cudaError_t attr =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SH::SMEM);
  if (attr != cudaSuccess) return attr;
  int ctas = sms;
  if constexpr (PAIR) {
    static int max_clusters = [&] {
      cudaLaunchConfig_t q = {};
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 2;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      q.blockDim = dim3(SH::THREADS);
      q.dynamicSmemBytes = SH::SMEM;
      q.attrs = at;
      q.numAttrs = 1;
      q.gridDim = dim3(2 * (sms / 2));
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, kern, &q) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
      }
      return n;
    }();
    if (max_clusters < 1) return cudaErrorLaunchOutOfResources;
    ctas = max_clusters;
  }
  const int units = p.m_tiles * p.n_tiles * p.splits;
  const int grid = units < ctas ? units : ctas;
  return launch_pdl(kern, dim3((PAIR ? 2 : 1) * grid), dim3(SH::THREADS), SH::SMEM, stream,
                    PAIR ? 2 : 1, ta, tb, p);
}

// One instantiation per (operand majorness, epilogue, output type, pairing)
// keeps every kernel's code to the epilogue it runs.
template <bool A_MN, bool B_MN, bool PAIR>
cudaError_t launch_form(const Params& p, int sms, const CUtensorMap& ta, const CUtensorMap& tb,
                        int epi, bool out_f32, cudaStream_t stream) {
  if (out_f32)
    return launch_variant<A_MN, B_MN, SKY_EPI_STORE, true, PAIR>(p, sms, ta, tb, stream);
  switch (epi) {
    case SKY_EPI_BIAS_GELU:
      return launch_variant<A_MN, B_MN, SKY_EPI_BIAS_GELU, false, PAIR>(p, sms, ta, tb, stream);
    case SKY_EPI_GELU_BWD:
      return launch_variant<A_MN, B_MN, SKY_EPI_GELU_BWD, false, PAIR>(p, sms, ta, tb, stream);
    default:
      return launch_variant<A_MN, B_MN, SKY_EPI_STORE, false, PAIR>(p, sms, ta, tb, stream);
  }
}

// The pair variant serves every problem with at least one full 256-row tile.
bool use_pair(int M, int /*epi*/) { return M >= 2 * BM; }

uint64_t g_timeout_ns = 2000000000ull;  // 2 s per wait
int g_skip_loads = 0;
}  // namespace

void set_debug(uint64_t timeout_ns, int skip_loads) {
  g_timeout_ns = timeout_ns ? timeout_ns : 2000000000ull;
  g_skip_loads = skip_loads;
}

int colpart_rows_max(int M) {
  return std::max(ceil_div(M, BM) * 4, ceil_div(M, 2 * BM) * 8);
}

int choose_splits(int tiles, int k_blocks, int sms) {
  // Estimated makespan (in k-block units) of `tiles * s` units on `sms` CTAs
  // plus a small per-unit cost; the fixed-order reduce is charged per split.
  int best = 1;
  double best_cost = 1e30;
  for (int s = 1; s <= 32 && s <= k_blocks; ++s) {
    const int per = ceil_div(k_blocks, s);
    const int s_eff = ceil_div(k_blocks, per);
    const int waves = ceil_div((int64_t)tiles * s_eff, sms);
    const double cost = waves * (per + 4.0) + (s_eff > 1 ? 2.0 + 0.5 * s_eff : 0.0);
    if (cost < best_cost - 1e-9) { best_cost = cost; best = s_eff; }
  }
  return best;
}

size_t workspace_bytes(sky_gemm_form form, int M, int N, int K, bool out_f32) {
  if (!out_f32) return 0;
  const bool pair = use_pair(M, SKY_EPI_STORE);  // fp32 outputs use the STORE epilogue
  const int tiles = ceil_div(M, pair ? 2 * BM : BM) * ceil_div(N, BN);
  const int kb = ceil_div(K, BK);
  const int sms = sm_count() > 0 ? sm_count() : 148;
  const int s = choose_splits(tiles, kb, pair ? sms / 2 : sms);
  (void)form;
  return s > 1 ? static_cast<size_t>(s) * M * N * sizeof(float) : 0;
}

sky_status launch_bf16(sky_gemm_form form, int M, int N, int K, const void* A, const void* B,
                       void* C, bool out_f32, int epi, const void* bias, const void* aux,
                       void* aux_out, void* ws, size_t ws_bytes, int32_t* status,
                       cudaStream_t stream, float* colsum, float* colpart, size_t colpart_bytes,
                       int* deferred_rows, const float* resid, const LnResid* ln) {
  // TMA row pitches and the 16-byte epilogue stores need the contiguous
  // dimensions to be multiples of 8 elements; the token dimension is free.
  const bool dims_ok = N % 8 == 0 && (form == SKY_GEMM_XTW ? M % 8 == 0 : K % 8 == 0);
  SKY_CHECK(dims_ok, SKY_ERR_UNSUPPORTED,
            "bf16 GEMM form %d: contiguous dimensions must be multiples of 8 (M=%d N=%d K=%d)",
            (int)form, M, N, K);
  SKY_CHECK(M > 0 && N > 0 && K > 0, SKY_ERR_INVALID_ARG, "GEMM sizes must be positive");
  SKY_CHECK((reinterpret_cast<uintptr_t>(A) & 15) == 0 && (reinterpret_cast<uintptr_t>(B) & 15) == 0,
            SKY_ERR_UNSUPPORTED, "bf16 GEMM operands must be 16-byte aligned");
  SKY_CHECK(reinterpret_cast<uintptr_t>(C) % 16 == 0, SKY_ERR_UNSUPPORTED,
            "GEMM output must be 16-byte aligned");
  SKY_CHECK(epi == SKY_EPI_STORE || epi == SKY_EPI_BIAS_GELU || epi == SKY_EPI_GELU_BWD,
            SKY_ERR_INVALID_ARG, "unknown epilogue %d", epi);
  SKY_CHECK(!out_f32 || epi == SKY_EPI_STORE, SKY_ERR_UNSUPPORTED,
            "fp32-output GEMM supports the STORE epilogue");
  SKY_CHECK(epi != SKY_EPI_BIAS_GELU || (bias && aux_out), SKY_ERR_INVALID_ARG,
            "BIAS_GELU epilogue needs bias and aux_out");
  SKY_CHECK(epi != SKY_EPI_GELU_BWD || aux, SKY_ERR_INVALID_ARG, "GELU' epilogue needs aux");
  SKY_CHECK(!resid || (out_f32 && epi == SKY_EPI_STORE && !colsum && !deferred_rows &&
                       (reinterpret_cast<uintptr_t>(resid) & 15) == 0),
            SKY_ERR_UNSUPPORTED, "a residual needs a 16-byte aligned fp32 output of the STORE epilogue");
  SKY_CHECK(!ln || (resid && ln->mean && ln->rstd && ln->gamma && ln->beta &&
                    (reinterpret_cast<uintptr_t>(ln->gamma) & 7) == 0 &&
                    (reinterpret_cast<uintptr_t>(ln->beta) & 7) == 0),
            SKY_ERR_INVALID_ARG, "a LayerNorm residual needs u, mean, rstd and 8-byte aligned gamma, beta");
  const int sms = sm_count();
  SKY_CHECK(sms > 0, SKY_ERR_CUDA, "no CUDA device");

  CUtensorMap ta, tb;
  const bool a_mn = form == SKY_GEMM_XTW;
  const bool b_mn = form != SKY_GEMM_XWT;
  const bool pair = use_pair(M, epi);
  // 192-wide pair tiles for K-major B and the plain-store epilogue (bf16 or
  // fp32 output, bias and residual allowed; no split-K) when the product is
  // less than one wave of 256-wide tiles and still one wave of 192-wide ones:
  // more SM pairs then share it.  (Over several waves the narrower tile's
  // main loop, which reuses each A tile for fewer columns, lost more than
  // the fuller last wave gained: QKV at T = 8192 took 47.1 instead of 43.1 us.)
  const int clusters = sms / 2;
  const int64_t m_t = ceil_div(M, pair ? 2 * BM : BM);
  // 192-wide pair tiles for K-major B and the plain-store epilogue when the
  // product is less than one wave of 256-wide tiles and still one wave of
  // 192-wide ones: more SM pairs then share it.  (Over several waves the
  // narrower tile's main loop, which reuses each A tile for fewer columns,
  // lost more than the fuller last wave gained: QKV at T = 8192 took 47.1
  // instead of 43.1 us.)
  const bool may_split = out_f32 && epi == SKY_EPI_STORE && bias == nullptr && resid == nullptr;
  const bool narrow = pair && form == SKY_GEMM_XWT && epi == SKY_EPI_STORE && !may_split &&
                      !colsum && !deferred_rows && N % 192 == 0 &&
                      m_t * ceil_div(N, BN) < clusters && m_t * (N / 192) <= clusters;
  const int tbn = narrow ? 192 : BN;
  bool ok = a_mn ? make_map(&ta, A, K, M, 64) : make_map(&ta, A, M, K, BM);
  ok = ok && (b_mn ? make_map(&tb, B, K, N, 64) : make_map(&tb, B, N, K, pair ? tbn / 2 : tbn));
  SKY_CHECK(ok, SKY_ERR_CUDA, "cuTensorMapEncodeTiled failed (M=%d N=%d K=%d)", M, N, K);

  Params p{};
  p.M = M; p.N = N; p.K = K;
  p.m_tiles = static_cast<int>(m_t);
  p.n_tiles = ceil_div(N, tbn);
  p.k_blocks = ceil_div(K, BK);
  p.splits = may_split ? choose_splits(p.m_tiles * p.n_tiles, p.k_blocks, pair ? sms / 2 : sms) : 1;
  if (p.splits > 1) {  // never more partials than the workspace holds
    const size_t cap = ws_bytes / (static_cast<size_t>(M) * N * sizeof(float));
    p.splits = cap < 2 ? 1 : (p.splits < (int)cap ? p.splits : (int)cap);
  }
  p.kb_per_split = ceil_div(p.k_blocks, p.splits);
  p.splits = ceil_div(p.k_blocks, p.kb_per_split);
  const size_t need = p.splits > 1 ? static_cast<size_t>(p.splits) * M * N * sizeof(float) : 0;
  SKY_CHECK(ws_bytes >= need && (need == 0 || ws), SKY_ERR_INVALID_ARG,
            "GEMM workspace too small (%zu < %zu)", ws_bytes, need);
  p.C = p.splits > 1 ? ws : C;
  // optional fused column sum of C (bf16 outputs only): per-warp partials in
  // the workspace, added in a fixed order after the kernel
  const int colpart_rows = p.m_tiles * (pair ? 8 : 4);  // one per 32 rows of every tile
  if (colsum || deferred_rows) {
    SKY_CHECK(!out_f32 && p.splits == 1, SKY_ERR_UNSUPPORTED, "fused column sum needs a bf16 output");
    float* buf = deferred_rows ? colpart : static_cast<float*>(ws);
    const size_t cap = deferred_rows ? colpart_bytes : ws_bytes;
    SKY_CHECK(buf && cap >= static_cast<size_t>(colpart_rows) * N * sizeof(float),
              SKY_ERR_INVALID_ARG, "GEMM column-sum workspace too small");
    p.colpart = buf;
    if (deferred_rows) *deferred_rows = colpart_rows;
  }
  p.bias = static_cast<const __nv_bfloat16*>(bias);
  p.resid = resid;
  if (ln) {
    p.ln_mean = ln->mean;
    p.ln_rstd = ln->rstd;
    p.ln_gamma = static_cast<const __nv_bfloat16*>(ln->gamma);
    p.ln_beta = static_cast<const __nv_bfloat16*>(ln->beta);
  }
  p.aux = epi == SKY_EPI_GELU_BWD ? static_cast<const __half*>(aux) : nullptr;
  p.aux_out = static_cast<__half*>(aux_out);
  p.status = status;
  p.timeout_ns = g_timeout_ns;
  p.skip_loads = g_skip_loads;

  cudaError_t e;
  if (narrow) {
    e = out_f32 ? launch_variant<false, false, SKY_EPI_STORE, true, true, 192>(p, sms, ta, tb, stream)
                : launch_variant<false, false, SKY_EPI_STORE, false, true, 192>(p, sms, ta, tb, stream);
  } else if (pair) {
    if (form == SKY_GEMM_XWT)
      e = launch_form<false, false, true>(p, sms, ta, tb, epi, out_f32, stream);
    else if (form == SKY_GEMM_XW)
      e = launch_form<false, true, true>(p, sms, ta, tb, epi, out_f32, stream);
    else
      e = launch_form<true, true, true>(p, sms, ta, tb, epi, out_f32, stream);
  } else {
    if (form == SKY_GEMM_XWT)
      e = launch_form<false, false, false>(p, sms, ta, tb, epi, out_f32, stream);
    else if (form == SKY_GEMM_XW)
      e = launch_form<false, true, false>(p, sms, ta, tb, epi, out_f32, stream);
    else
      e = launch_form<true, true, false>(p, sms, ta, tb, epi, out_f32, stream);
  }
  count_launches(1);
  if (e != cudaSuccess) return cuda_fail(e, "gemm_tc_kernel launch");
  if (colsum && !deferred_rows) {
    e = reduce_rows_f32(p.colpart, colpart_rows, N, colsum, stream);
    if (e != cudaSuccess) return cuda_fail(e, "column-sum reduce launch");
  }
  if (p.splits > 1) {
    const int64_t n = static_cast<int64_t>(M) * N;
    const int blocks = static_cast<int>(std::min<int64_t>(ceil_div(n / 4 + 1, 256), sms * 8));
    const float* wsf = static_cast<const float*>(ws);
    float* cf = static_cast<float*>(C);
    switch (p.splits) {
      case 2: e = launch_pdl(splitk_reduce_kernel<2>, dim3(blocks), dim3(256), 0, stream, 1, wsf, p.splits, n, cf); break;
      case 3: e = launch_pdl(splitk_reduce_kernel<3>, dim3(blocks), dim3(256), 0, stream, 1, wsf, p.splits, n, cf); break;
      case 4: e = launch_pdl(splitk_reduce_kernel<4>, dim3(blocks), dim3(256), 0, stream, 1, wsf, p.splits, n, cf); break;
      case 5: e = launch_pdl(splitk_reduce_kernel<5>, dim3(blocks), dim3(256), 0, stream, 1, wsf, p.splits, n, cf); break;
      case 6: e = launch_pdl(splitk_reduce_kernel<6>, dim3(blocks), dim3(256), 0, stream, 1, wsf, p.splits, n, cf); break;
      case 8: e = launch_pdl(splitk_reduce_kernel<8>, dim3(blocks), dim3(256), 0, stream, 1, wsf, p.splits, n, cf); break;
      default: e = launch_pdl(splitk_reduce_kernel<0>, dim3(blocks), dim3(256), 0, stream, 1, wsf, p.splits, n, cf); break;
    }
    count_launches(1);
    if (e != cudaSuccess) return cuda_fail(e, "splitk_reduce launch");
  }
  return SKY_OK;
}

}  // namespace gemm
}  // namespace sky
