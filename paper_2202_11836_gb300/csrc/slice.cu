// Slice runtime and the C ABI (sky_slice.h, sky_ops.h).
//
// A slice owns the layers [l0, l1) of the encoder (the partition unit of
// Sec. IV-D).  At create it makes one device allocation holding, per layer,
// the 12 parameters (slice dtype), their fp32 gradients and the activation
// stash the backward pass needs (Sec. IV-B counts exactly these: inputs,
// weights, gradients and outputs), plus one shared workspace.  forward runs
// the layers in order and leaves each layer's intermediates in its stash;
// backward walks the layers in reverse (Sec. III) reading that stash.  Every
// launch goes on the caller's stream; nothing synchronises the host except the
// calls documented as synchronous.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdlib>
#include <cstring>
#include <exception>
#include <new>
#include <string>
#include <vector>

#include "common.cuh"
#include "gemm.h"
#include "optimizer.h"
#include "rowwise.h"

namespace sky {

constexpr int kMaxStashSlots = 64;
constexpr uint64_t kMaxDelayNs = 10ull * 1000 * 1000 * 1000;  // sky_device_delay: 10 s

namespace {
thread_local std::string g_last_error;
uint64_t g_alloc_cap = 0;
std::atomic<int64_t> g_launches{0};
}  // namespace

bool pdl_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("SKY_PDL");
    return !(v && v[0] == '0');
  }();
  return on;
}

void count_launches(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

void set_error(const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
}

sky_status cuda_fail(cudaError_t e, const char* what) {
  set_error("%s: %s", what, cudaGetErrorString(e));
  return e == cudaErrorMemoryAllocation ? SKY_ERR_OOM : SKY_ERR_CUDA;
}

int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  static int cache[64] = {0};
  if (dev < 0 || dev >= 64) return 0;
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    cache[dev] = n;
  }
  return cache[dev];
}

// ---------------------------------------------------------------- profiling
struct ProfRecord {
  int cat;
  cudaEvent_t start, stop;
  double flops, bytes;
};
enum ProfCat { P_GEMM_FWD, P_GEMM_DGRAD, P_GEMM_WGRAD, P_ATTN_FWD, P_ATTN_BWD, P_LN_FWD,
               P_LN_BWD, P_COLSUM, P_COPY, P_NCAT };
static const char* kCatNames[P_NCAT] = {"gemm_fwd", "gemm_dgrad", "gemm_wgrad", "attn_fwd",
                                        "attn_bwd", "ln_fwd", "ln_bwd", "colsum", "copy"};

// Per-layer parameters, gradients and the activation stash.  The residual
// sums U1 and U2 are kept in fp32.  bf16 slices keep the LayerNorm outputs
// (X1 and the next layer's X) only as the bf16 copies the contractions read:
// the residual branch that adds them in fp32 recomputes them from U and the
// row statistics in the GEMM epilogue.  fp32 slices keep X and X1 in fp32.
struct LayerBufs {
  void* p[SKY_NUM_PARAMS];
  float* g[SKY_NUM_PARAMS];
  void *Xb, *QKV, *ctx, *X1b, *Gp, *G;  // Gp = GELU'(Z) (fp16 in bf16 slices)
  float *U1, *U2;
  float *lse, *mean1, *rstd1, *mean2, *rstd2;
};

}  // namespace sky

struct sky_slice {
  sky_slice_config cfg;
  int L, H, A, F, D;
  size_t esz;
  int64_t maxT;
  int device;
  void* arena = nullptr;
  uint64_t param_bytes = 0, grad_bytes = 0, stash_bytes = 0, ws_bytes_total = 0;
  std::vector<sky::LayerBufs> layers;
  // fp32 gradient stream; k alternates per layer.  bf16: dP[k] holds the
  // whole input gradient dQKV Wqkv + dU1 (the GEMM epilogue adds dR[k] = dU1).
  // fp32: it travels as the two terms dP[k], dR[k] that the next LayerNorm
  // backward adds.
  float *dP[2], *dR[2], *dU2_32, *dP1;
  void *dU2b, *dU1b, *dH, *dctx, *dqkv;           // dtype copies / branch gradients
  float* delta;
  void* ws;
  size_t ws_bytes;
  int32_t* d_status;
  // bf16 slices: the first layer's fp32 residual input (the caller's x when it
  // is fp32 and 16-byte aligned, else the fp32 copy x32 made at the start of
  // the forward)
  float* x32 = nullptr;
  const float* res0 = nullptr;
  // Weight-gradient GEMMs of a bf16 backward run on a second stream, so they
  // fill the SMs that the data-gradient chain leaves idle.  ev_in[j]: input j
  // of the side stream (dU2, dZ, dU1, dQKV) is ready on the caller's stream;
  // ev_out[j]: the side GEMM reading input j is done, so the next layer may
  // overwrite that buffer; ev_out_live[j]: ev_out[j] was recorded by the
  // current backward call (earlier records are already ordered by that
  // call's final join, and waiting on them would tie a captured backward
  // pass to work outside its CUDA graph).  ws2: the side GEMMs' split-K
  // scratch.
  cudaStream_t side = nullptr;
  cudaEvent_t ev_in[4] = {}, ev_out[4] = {}, ev_join = nullptr;
  bool ev_out_live[4] = {};
  void* ws2 = nullptr;
  size_t ws2_bytes = 0;
  // Column partials whose fixed-order reduction (a bias / LayerNorm-parameter
  // gradient, needed by nothing downstream) also runs on the side stream:
  // lnp[k][0] / lnp[k][1] of the LN2 / LN1 backward, db1p[k] of the fused
  // db1.  Two sets, k = the layer's parity, so that a layer's partials are
  // still intact when its one batched reduction runs on the weight-gradient
  // stream while the data-gradient chain moves on to the next layer.
  // ev_red[k]: that reduction is done (the layer two further down may reuse
  // set k); ev_red_live[k]: recorded by the current backward call.
  void* lnp[2][2] = {};
  size_t lnp_bytes = 0;
  float* db1p[2] = {};
  size_t db1p_bytes = 0;
  cudaEvent_t ev_red[2] = {};
  bool ev_red_live[2] = {};
  // column partials of dQKV written by the attention backward kernels (one
  // row per 128-row tile of every sequence), summed into dbqkv on the side
  // stream
  float* qkvp[2] = {};
  size_t qkvp_bytes = 0;
  // local parameter update (Sec. III): fp32 master weights and state in one
  // allocation, the tensor and chunk tables the update kernel walks
  bool opt_ready = false;
  sky_optimizer_config opt_cfg{};
  int64_t opt_t = 0;
  void* opt_mem = nullptr;
  std::vector<sky::opt::Tensor> opt_tensors;
  sky::opt::Tensor* d_opt_tensors = nullptr;
  sky::opt::Chunk* d_opt_chunks = nullptr;
  int opt_chunks = 0;
  // Activation stashes: slot m holds everything the backward pass of the
  // micro-batch whose forward used slot m needs (stash_slots of them, so
  // that several forwards can precede their backwards, as in a micro-batched
  // pipeline).  slot_layers[m][i] has layer i's parameter and gradient
  // pointers (shared by all slots) and slot m's stash pointers; `layers` is
  // the view of the slot the current call uses.
  int n_slots = 1;
  std::vector<std::vector<sky::LayerBufs>> slot_layers;
  // per slot: the batch shape and lengths of its most recent forward
  std::vector<char> slot_fwd;
  std::vector<int> slot_B, slot_S;
  std::vector<const int32_t*> slot_len;
  // gradient accumulation: a backward with accumulate = 1 writes each
  // layer's gradients into this scratch set and adds it into the layer's
  // gradients on the weight-gradient stream (one layer's worth, reused)
  float* gscr[SKY_NUM_PARAMS] = {};
  bool accumulate = false;
  // layer_cost / profiled step graph: timing events are being captured
  bool marks_in_graph = false;
  // per-kernel records of a step graph captured with profiling on, and the
  // events they use (taken out of the pool, owned until the graph goes)
  std::vector<sky::ProfRecord> graph_recs;
  std::vector<cudaEvent_t> graph_events;
  // batch shape and lengths of the pass in progress (the slot in use)
  int B = 0, S = 0;
  const int32_t* d_len = nullptr;
  cudaStream_t last_stream = nullptr;
  // one captured training step (forward + backward) as an executable CUDA
  // graph, the private stream it was captured on, the kernel launches it
  // holds and the batch shape and lengths it was captured with
  cudaGraphExec_t step_exec = nullptr;
  cudaStream_t cap_stream = nullptr;
  int64_t step_launches = 0;
  int step_B = 0, step_S = 0;
  const int32_t* step_len = nullptr;
  // profiling
  bool prof = false;
  std::vector<sky::ProfRecord> recs;
  std::vector<cudaEvent_t> event_pool;
  size_t event_next = 0;
  double cat_ms[sky::P_NCAT] = {0};
  double cat_flops[sky::P_NCAT] = {0};
  double cat_bytes[sky::P_NCAT] = {0};
  int64_t cat_n[sky::P_NCAT] = {0};
};

namespace sky {
namespace {

size_t param_elems(const sky_slice* s, int k) {
  const size_t H = s->H, F = s->F;
  switch (k) {
    case 0: return 3 * H * H;
    case 1: return 3 * H;
    case 2: return H * H;
    case 6: return F * H;
    case 7: return F;
    case 8: return H * F;
    default: return H;
  }
}

size_t align_up(size_t x) { return (x + 255) & ~size_t(255); }

// Scratch needed by the backward pass at T tokens (shared by all steps).
size_t workspace_need(const sky_slice* s, int64_t T) {
  const int H = s->H, F = s->F;
  size_t need = 0;
  if (s->cfg.dtype == SKY_DTYPE_BF16) {
    const int64_t shapes[4][2] = {{3 * H, H}, {H, H}, {F, H}, {H, F}};
    for (auto& sh : shapes)
      need = std::max(need, gemm::workspace_bytes(SKY_GEMM_XTW, (int)sh[0], (int)sh[1], (int)T, true));
  }
  need = std::max(need, layernorm_bwd_ws((int)T, H));
  need = std::max(need, (size_t)ceil_div(T, 128) * 4 * F * sizeof(float));  // fused db1 partials
  need = std::max(need, column_sum_ws((int)T, F));
  need = std::max(need, column_sum_ws((int)T, 3 * H));
  return need;
}

// Split-K scratch of the weight-gradient GEMMs (their own, so they can run
// beside the main stream's kernels).
size_t side_workspace_need(const sky_slice* s, int64_t T) {
  const int H = s->H, F = s->F;
  size_t need = column_sum_ws((int)T, 3 * H);  // dbqkv
  const int64_t shapes[4][2] = {{3 * H, H}, {H, H}, {F, H}, {H, F}};
  for (auto& sh : shapes)
    need = std::max(need, gemm::workspace_bytes(SKY_GEMM_XTW, (int)sh[0], (int)sh[1], (int)T, true));
  return need;
}

cudaEvent_t next_event(sky_slice* s) {
  if (s->event_next == s->event_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    s->event_pool.push_back(e);
  }
  return s->event_pool[s->event_next++];
}

// Brackets one launch with CUDA events when profiling is on.
struct Timed {
  sky_slice* s;
  cudaStream_t st;
  ProfRecord r{};
  Timed(sky_slice* s_, cudaStream_t st_, int cat, double flops, double bytes) : s(s_), st(st_) {
    if (!s->prof) return;
    r.cat = cat; r.flops = flops; r.bytes = bytes;
    r.start = next_event(s);
    r.stop = next_event(s);
    if (r.start) record(r.start);
  }
  ~Timed() {
    if (!s->prof || !r.start || !r.stop) return;
    record(r.stop);
    s->recs.push_back(r);
  }
  // inside a stream capture the records become event record nodes that every
  // replay of the graph records
  void record(cudaEvent_t e) {
    if (s->marks_in_graph) cudaEventRecordWithFlags(e, st, cudaEventRecordExternal);
    else cudaEventRecord(e, st);
  }
};

sky_status run_gemm(sky_slice* s, cudaStream_t st, int cat, sky_gemm_form form, int M, int N,
                    int K, const void* A, const void* Bm, void* C, bool out_f32, int epi,
                    const void* bias, const void* aux, void* aux_out, float* colsum = nullptr,
                    void* ws = nullptr, size_t ws_bytes = 0, const float* resid = nullptr,
                    const gemm::LnResid* ln = nullptr) {
  Timed t(s, st, cat, 2.0 * M * N * K, 0);
  if (!ws) {
    ws = s->ws;
    ws_bytes = s->ws_bytes;
  }
  if (s->cfg.dtype == SKY_DTYPE_BF16)
    return gemm::launch_bf16(form, M, N, K, A, Bm, C, out_f32, epi, bias, aux, aux_out, ws,
                             ws_bytes, s->d_status, st, colsum, nullptr, 0, nullptr, resid, ln);
  return gemm::launch_f32(form, M, N, K, static_cast<const float*>(A),
                          static_cast<const float*>(Bm), static_cast<float*>(C), epi,
                          static_cast<const float*>(bias), static_cast<const float*>(aux),
                          static_cast<float*>(aux_out), st);
}

#define SKY_TRY(call)                   \
  do {                                  \
    sky_status st_ = (call);            \
    if (st_ != SKY_OK) return st_;      \
  } while (0)

// ------------------------------------------------------------------ forward
// One layer, steps a1..a8.  y_out == nullptr: write the next layer's Xb.
sky_status forward_layer(sky_slice* s, int i, void* y_out, cudaStream_t st) {
  LayerBufs& Lb = s->layers[i];
  const int B = s->B, S = s->S, H = s->H, A = s->A, F = s->F;
  const int T = B * S;
  const sky_dtype dt = s->cfg.dtype;
  const double e = (double)s->esz;
  // a1: QKV = X Wqkv^T + bqkv
  SKY_TRY(run_gemm(s, st, P_GEMM_FWD, SKY_GEMM_XWT, T, 3 * H, H, Lb.Xb, Lb.p[0], Lb.QKV, false,
                   SKY_EPI_STORE, Lb.p[1], nullptr, nullptr));
  // a2: masked scaled dot-product attention (Eq. 1)
  {
    Timed t(s, st, P_ATTN_FWD, 4.0 * H * S * (double)T, e * T * 4.0 * H);
    SKY_TRY(attention_fwd(Lb.QKV, s->d_len, B, S, H, A, dt, Lb.ctx, Lb.lse, s->d_status, st));
  }
  // a3 + a4: U1 = ctx Wo^T + bo + X (fp32).  bf16: the residual X is added
  // by the GEMM epilogue (for layers after the first, as LN2 of the previous
  // layer's U2, recomputed there); fp32: by the LayerNorm.  X1 = LN(U1)
  const bool bf = dt == SKY_DTYPE_BF16;
  {
    const gemm::LnResid* ln = nullptr;
    gemm::LnResid prev{};
    const float* r = s->res0;
    if (bf && i > 0) {
      const LayerBufs& Pv = s->layers[i - 1];
      prev = gemm::LnResid{Pv.mean2, Pv.rstd2, Pv.p[10], Pv.p[11]};
      ln = &prev;
      r = Pv.U2;
    }
    SKY_TRY(run_gemm(s, st, P_GEMM_FWD, SKY_GEMM_XWT, T, H, H, Lb.ctx, Lb.p[2], Lb.U1, true,
                     SKY_EPI_STORE, Lb.p[3], nullptr, nullptr, nullptr, nullptr, 0,
                     bf ? r : nullptr, ln));
  }
  {
    Timed t(s, st, P_LN_FWD, 0, (bf ? 4.0 + e : 16.0) * T * H + 8.0 * T);
    SKY_TRY(layernorm_fwd(Lb.U1, bf ? nullptr : static_cast<const float*>(Lb.Xb), Lb.p[4],
                          Lb.p[5], T, H, s->cfg.ln_eps, dt, bf ? nullptr : Lb.U1, nullptr,
                          Lb.X1b, Lb.mean1, Lb.rstd1, st));
  }
  // a5 + a6: Z = X1 W1^T + b1; G = GELU(Z) and GELU'(Z) for the backward (fused epilogue)
  SKY_TRY(run_gemm(s, st, P_GEMM_FWD, SKY_GEMM_XWT, T, F, H, Lb.X1b, Lb.p[6], Lb.G, false,
                   SKY_EPI_BIAS_GELU, Lb.p[7], nullptr, Lb.Gp));
  // a7 + a8: U2 = G W2^T + b2 + X1 (fp32; the residual as in a3, X1 = LN1(U1)
  // recomputed in the bf16 epilogue).  Y = LN(U2) -> next layer's input (its
  // dtype copy) or the caller's y
  {
    const gemm::LnResid ln1{Lb.mean1, Lb.rstd1, Lb.p[4], Lb.p[5]};
    SKY_TRY(run_gemm(s, st, P_GEMM_FWD, SKY_GEMM_XWT, T, H, F, Lb.G, Lb.p[8], Lb.U2, true,
                     SKY_EPI_STORE, Lb.p[9], nullptr, nullptr, nullptr, nullptr, 0,
                     bf ? Lb.U1 : nullptr, bf ? &ln1 : nullptr));
  }
  {
    const bool f32 = bf && y_out && s->cfg.io_fp32;
    Timed t(s, st, P_LN_FWD, 0, (bf ? 4.0 + (f32 ? 4.0 : e) : 16.0) * T * H + 8.0 * T);
    const float* r2 = bf ? nullptr : static_cast<const float*>(Lb.X1b);
    float* u2 = bf ? nullptr : Lb.U2;
    if (y_out) {
      SKY_TRY(layernorm_fwd(Lb.U2, r2, Lb.p[10], Lb.p[11], T, H, s->cfg.ln_eps, dt, u2,
                            f32 ? static_cast<float*>(y_out) : nullptr, f32 ? nullptr : y_out,
                            Lb.mean2, Lb.rstd2, st));
    } else {
      LayerBufs& Nx = s->layers[i + 1];
      SKY_TRY(layernorm_fwd(Lb.U2, r2, Lb.p[10], Lb.p[11], T, H, s->cfg.ln_eps, dt, u2,
                            nullptr, Nx.Xb, Lb.mean2, Lb.rstd2, st));
    }
  }
  return SKY_OK;
}

// ----------------------------------------------------------------- backward
// One layer, steps a9..a16.  The upstream gradient is dY + dY2: dY in dy_dt
// (the caller's dy for the top layer) and dY2 fp32 or null.  Outputs go to
// dP[k] (bf16: the whole input gradient) and dR[k] (fp32: the second term);
// for the slice's first layer they end in dx.
sky_status backward_layer(sky_slice* s, int i, const void* dY, sky_dtype dy_dt, const float* dY2,
                          int k, void* dx, cudaStream_t st, cudaStream_t sw) {
  LayerBufs& Lb = s->layers[i];
  // gradients go to the layer's buffers, or with accumulation to the scratch
  // set that is added into them at the end of the layer
  float* const* G = s->accumulate ? s->gscr : Lb.g;
  const int B = s->B, S = s->S, H = s->H, A = s->A, F = s->F;
  const int T = B * S;
  const sky_dtype dt = s->cfg.dtype;
  const bool bf = dt == SKY_DTYPE_BF16;
  const double e = (double)s->esz;
  const double dye = (dy_dt == SKY_DTYPE_BF16 ? 2.0 : 4.0) + (dY2 ? 4.0 : 0.0);
  void* dU1b = bf ? s->dU1b : s->dR[k];
  // Weight gradients go to stream sw (== st when they run in line).  fork(j)
  // hands input j to sw; reuse(j) makes st wait until the previous layer's
  // weight-gradient GEMM has finished reading buffer j before st overwrites it;
  // done(j) marks that GEMM's completion.
  const bool two = sw != st;
  auto fork = [&](int j) -> sky_status {
    if (!two) return SKY_OK;
    SKY_CUDA(cudaEventRecord(s->ev_in[j], st));
    SKY_CUDA(cudaStreamWaitEvent(sw, s->ev_in[j], 0));
    return SKY_OK;
  };
  auto reuse = [&](int j) -> sky_status {
    if (two && s->ev_out_live[j]) SKY_CUDA(cudaStreamWaitEvent(st, s->ev_out[j], 0));
    return SKY_OK;
  };
  auto done = [&](int j) -> sky_status {
    if (two) {
      SKY_CUDA(cudaEventRecord(s->ev_out[j], sw));
      s->ev_out_live[j] = true;
    }
    return SKY_OK;
  };
  void* ws2 = bf ? s->ws2 : nullptr;
  const size_t ws2b = s->ws2_bytes;
  // bf16: the column sums behind this layer's bias and LayerNorm-parameter
  // gradients (LN2 and LN1 partials per CTA, db1 partials per 32 rows from
  // the FFN2 data-gradient epilogue, dbqkv partials per 128-row tile from the
  // attention backward) land in partial buffers of set k and are added up by
  // one fixed-order launch on sw at the end of the layer.  Set k was last
  // used by the layer two above; wait for its reduction before reusing it.
  int ln2_parts = 0, ln1_parts = 0, db1_rows = 0;
  if (bf && two && s->ev_red_live[k]) SKY_CUDA(cudaStreamWaitEvent(st, s->ev_red[k], 0));
  // a9: LN2 backward -> dU2 (fp32 + dtype), dgamma2, dbeta2, db2
  SKY_TRY(reuse(0));
  {
    Timed t(s, st, P_LN_BWD, 0, (dye + 4.0 + 4.0 + (bf ? e : 0.0)) * T * H + 8.0 * T);
    SKY_TRY(layernorm_bwd(dY, dy_dt, dY2, Lb.U2, Lb.p[10], Lb.mean2, Lb.rstd2, T, H, dt,
                          bf ? s->dU2_32 : nullptr, s->dU2b, G[10], G[11], G[9],
                          bf ? s->lnp[k][0] : s->ws, bf ? s->lnp_bytes : s->ws_bytes, st,
                          bf ? &ln2_parts : nullptr, s->d_status));
  }
  SKY_TRY(fork(0));
  // a10 + a11: dW2 = dU2^T G (on sw, beside the data gradient);
  //            dZ = (dU2 W2) * GELU'(Z);
  //            db1 = sum_rows dZ (fused into the bf16 epilogue; a column-sum pass for fp32)
  SKY_TRY(run_gemm(s, sw, P_GEMM_WGRAD, SKY_GEMM_XTW, H, F, T, s->dU2b, Lb.G, G[8], true,
                   SKY_EPI_STORE, nullptr, nullptr, nullptr, nullptr, ws2, ws2b));
  SKY_TRY(done(0));
  SKY_TRY(reuse(1));
  if (bf) {
    Timed t(s, st, P_GEMM_DGRAD, 2.0 * T * F * H, 0);
    SKY_TRY(gemm::launch_bf16(SKY_GEMM_XW, T, F, H, s->dU2b, Lb.p[8], s->dH, false,
                              SKY_EPI_GELU_BWD, nullptr, Lb.Gp, nullptr, s->ws, s->ws_bytes,
                              s->d_status, st, nullptr, s->db1p[k], s->db1p_bytes, &db1_rows));
  } else {
    SKY_TRY(run_gemm(s, st, P_GEMM_DGRAD, SKY_GEMM_XW, T, F, H, s->dU2b, Lb.p[8], s->dH, false,
                     SKY_EPI_GELU_BWD, nullptr, Lb.Gp, nullptr));
    Timed t(s, st, P_COLSUM, 0, e * T * F);
    SKY_TRY(column_sum(s->dH, T, F, dt, G[7], s->ws, s->ws_bytes, st));
  }
  SKY_TRY(fork(1));
  // a12: dX1 = dZ W1 + dU2 (fp32; bf16: dU2 added by the GEMM epilogue, fp32:
  // by the LN1 backward);  dW1 = dZ^T X1
  SKY_TRY(run_gemm(s, st, P_GEMM_DGRAD, SKY_GEMM_XW, T, H, F, s->dH, Lb.p[6], s->dP1, true,
                   SKY_EPI_STORE, nullptr, nullptr, nullptr, nullptr, nullptr, 0,
                   bf ? s->dU2_32 : nullptr));
  SKY_TRY(run_gemm(s, sw, P_GEMM_WGRAD, SKY_GEMM_XTW, F, H, T, s->dH, Lb.X1b, G[6], true,
                   SKY_EPI_STORE, nullptr, nullptr, nullptr, nullptr, ws2, ws2b));
  SKY_TRY(done(1));
  // a13: LN1 backward of dX1 = P1 + dU2 -> dU1 (fp32 + dtype), dgamma1, dbeta1, dbo
  SKY_TRY(reuse(2));
  {
    Timed t(s, st, P_LN_BWD, 0, (bf ? 4.0 : 8.0) * T * H + (4.0 + 4.0 + (bf ? e : 0.0)) * T * H + 8.0 * T);
    SKY_TRY(layernorm_bwd(s->dP1, SKY_DTYPE_FP32, bf ? nullptr : static_cast<float*>(s->dU2b),
                          Lb.U1, Lb.p[4], Lb.mean1, Lb.rstd1, T, H, dt, bf ? s->dR[k] : nullptr,
                          dU1b, G[4], G[5], G[3], bf ? s->lnp[k][1] : s->ws,
                          bf ? s->lnp_bytes : s->ws_bytes, st, bf ? &ln1_parts : nullptr,
                          s->d_status));
  }
  SKY_TRY(fork(2));
  // a14: dctx = dU1 Wo;  dWo = dU1^T ctx
  SKY_TRY(run_gemm(s, st, P_GEMM_DGRAD, SKY_GEMM_XW, T, H, H, dU1b, Lb.p[2], s->dctx, false,
                   SKY_EPI_STORE, nullptr, nullptr, nullptr));
  SKY_TRY(run_gemm(s, sw, P_GEMM_WGRAD, SKY_GEMM_XTW, H, H, T, dU1b, Lb.ctx, G[2], true,
                   SKY_EPI_STORE, nullptr, nullptr, nullptr, nullptr, ws2, ws2b));
  SKY_TRY(done(2));
  // a15: attention backward -> dQKV
  SKY_TRY(reuse(3));
  {
    Timed t(s, st, P_ATTN_BWD, 8.0 * H * S * (double)T, e * T * 8.0 * H);
    SKY_TRY(attention_bwd(Lb.QKV, Lb.ctx, s->dctx, Lb.lse, s->d_len, B, S, H, A, dt, s->dqkv,
                          s->delta, s->d_status, st, bf ? s->qkvp[k] : nullptr));
  }
  SKY_TRY(fork(3));
  if (bf) {
    // the layer's eight column reductions in one fixed-order launch on sw:
    // dgamma2, dbeta2, db2 and dgamma1, dbeta1, dbo from the LayerNorm
    // partials, db1 from the FFN2 data-gradient partials, dbqkv from the
    // attention backward's partials
    const int qkv_rows = B * ceil_div(S, 128);
    const float* l2 = static_cast<const float*>(s->lnp[k][0]);
    const float* l1 = static_cast<const float*>(s->lnp[k][1]);
    ColSegments sg{};
    sg.seg[0] = {l2, G[10], ln2_parts, H};
    sg.seg[1] = {l2 + (size_t)ln2_parts * H, G[11], ln2_parts, H};
    sg.seg[2] = {l2 + 2 * (size_t)ln2_parts * H, G[9], ln2_parts, H};
    sg.seg[3] = {l1, G[4], ln1_parts, H};
    sg.seg[4] = {l1 + (size_t)ln1_parts * H, G[5], ln1_parts, H};
    sg.seg[5] = {l1 + 2 * (size_t)ln1_parts * H, G[3], ln1_parts, H};
    sg.seg[6] = {s->db1p[k], G[7], db1_rows, F};
    sg.seg[7] = {s->qkvp[k], G[1], qkv_rows, 3 * H};
    sg.n = 8;
    Timed t(s, sw, P_COLSUM, 0,
            4.0 * (3.0 * (ln2_parts + ln1_parts) * H + (double)db1_rows * F + qkv_rows * 3.0 * H));
    SKY_TRY(reduce_column_segments(sg, sw));
    if (two) {
      SKY_CUDA(cudaEventRecord(s->ev_red[k], sw));
      s->ev_red_live[k] = true;
    }
  } else {  // dbqkv = column sums of dQKV
    Timed t(s, sw, P_COLSUM, 0, e * T * 3.0 * H);
    SKY_TRY(column_sum(s->dqkv, T, 3 * H, dt, G[1], s->ws, s->ws_bytes, sw));
  }
  // a16: dX = dQKV Wqkv + dU1;  dWqkv = dQKV^T X.  bf16: dU1 is added by the
  // GEMM epilogue (straight into dx for the slice's first layer with fp32
  // I/O); fp32: by the next LayerNorm backward, or here for the first layer
  const bool direct = bf && dx && s->cfg.io_fp32 && (reinterpret_cast<uintptr_t>(dx) & 15) == 0;
  SKY_TRY(run_gemm(s, st, P_GEMM_DGRAD, SKY_GEMM_XW, T, H, 3 * H, s->dqkv, Lb.p[0],
                   direct ? dx : s->dP[k], true, SKY_EPI_STORE, nullptr, nullptr, nullptr, nullptr,
                   nullptr, 0, bf ? s->dR[k] : nullptr));
  if (dx && !direct) {
    const sky_dtype odt = s->cfg.io_fp32 ? SKY_DTYPE_FP32 : dt;
    Timed t(s, st, P_COPY, 0, ((bf ? 4.0 : 8.0) + (odt == SKY_DTYPE_BF16 ? 2.0 : 4.0)) * T * H);
    if (!bf)
      SKY_TRY(add_f32(s->dP[k], s->dR[k], (int64_t)T * H, odt, dx, st));
    else if (odt == SKY_DTYPE_BF16)
      SKY_TRY(f32_to_bf16(s->dP[k], (int64_t)T * H, dx, st));
    else
      SKY_CUDA(cudaMemcpyAsync(dx, s->dP[k], (size_t)T * H * 4, cudaMemcpyDeviceToDevice, st));
  }
  SKY_TRY(run_gemm(s, sw, P_GEMM_WGRAD, SKY_GEMM_XTW, 3 * H, H, T, s->dqkv, Lb.Xb, G[0], true,
                   SKY_EPI_STORE, nullptr, nullptr, nullptr, nullptr, ws2, ws2b));
  SKY_TRY(done(3));
  if (s->accumulate) {  // Lb.g += scratch: both are the 12 tensors laid out alike, contiguous
    const int64_t n = (Lb.g[SKY_NUM_PARAMS - 1] + param_elems(s, SKY_NUM_PARAMS - 1)) - Lb.g[0];
    Timed t(s, sw, P_COPY, 0, 12.0 * n);
    SKY_TRY(add_f32(Lb.g[0], s->gscr[0], n, SKY_DTYPE_FP32, Lb.g[0], sw));
  }
  return SKY_OK;
}

// A per-layer timing mark.  Inside a stream capture it becomes an event
// record node that a replay of the graph records.
sky_status record_mark(sky_slice* s, cudaEvent_t ev, cudaStream_t st) {
  if (s->marks_in_graph)
    SKY_CUDA(cudaEventRecordWithFlags(ev, st, cudaEventRecordExternal));
  else
    SKY_CUDA(cudaEventRecord(ev, st));
  return SKY_OK;
}

sky_status forward_all(sky_slice* s, const void* x, void* y, cudaStream_t st,
                       std::vector<cudaEvent_t>* marks) {
  const int64_t n = (int64_t)s->B * s->S * s->H;
  {
    LayerBufs& L0 = s->layers[0];
    s->res0 = nullptr;
    if (s->cfg.dtype == SKY_DTYPE_BF16 && s->cfg.io_fp32) {
      // the first layer's residual branch reads x in place; its bf16 copy
      // feeds the QKV projection
      const bool in_place = (reinterpret_cast<uintptr_t>(x) & 15) == 0;
      Timed t(s, st, P_COPY, 0, (in_place ? 6.0 : 14.0) * n);
      if (!in_place)
        SKY_CUDA(cudaMemcpyAsync(s->x32, x, n * 4, cudaMemcpyDeviceToDevice, st));
      s->res0 = in_place ? static_cast<const float*>(x) : s->x32;
      SKY_TRY(f32_to_bf16(s->res0, n, L0.Xb, st));
    } else {
      Timed t(s, st, P_COPY, 0, (2.0 * s->esz + (s->esz == 2 ? 6.0 : 0.0)) * n);
      SKY_CUDA(cudaMemcpyAsync(L0.Xb, x, n * s->esz, cudaMemcpyDeviceToDevice, st));
      if (s->cfg.dtype == SKY_DTYPE_BF16) {
        SKY_TRY(to_f32(x, n, s->cfg.dtype, s->x32, st));
        s->res0 = s->x32;
      }
    }
  }
  for (int i = 0; i < s->L; ++i) {
    if (marks) SKY_TRY(record_mark(s, (*marks)[2 * i], st));
    SKY_TRY(forward_layer(s, i, i + 1 < s->L ? nullptr : y, st));
    if (marks) SKY_TRY(record_mark(s, (*marks)[2 * i + 1], st));
  }
  return SKY_OK;
}

sky_status backward_all(sky_slice* s, const void* dy, void* dx, cudaStream_t st,
                        std::vector<cudaEvent_t>* marks) {
  const void* cur = dy;
  const float* cur2 = nullptr;
  sky_dtype cur_dt = s->cfg.io_fp32 ? SKY_DTYPE_FP32 : s->cfg.dtype;
  // The side stream is used unless kernels are being timed one by one.  It
  // joins the caller's stream at the end, so the caller's stream still orders
  // everything the backward pass does.
  cudaStream_t sw = (s->side && !s->prof) ? s->side : st;
  auto join = [&]() -> sky_status {
    if (sw == st) return SKY_OK;
    SKY_CUDA(cudaEventRecord(s->ev_join, sw));
    SKY_CUDA(cudaStreamWaitEvent(st, s->ev_join, 0));
    return SKY_OK;
  };
  for (bool& live : s->ev_out_live) live = false;
  for (bool& live : s->ev_red_live) live = false;
  if (sw != st) {  // the side stream starts after everything before this call
    SKY_CUDA(cudaEventRecord(s->ev_join, st));
    SKY_CUDA(cudaStreamWaitEvent(sw, s->ev_join, 0));
  }
  for (int i = s->L - 1; i >= 0; --i) {
    const int k = (s->L - 1 - i) & 1;
    if (marks) SKY_TRY(record_mark(s, (*marks)[2 * i], st));
    const sky_status rc = backward_layer(s, i, cur, cur_dt, cur2, k, i == 0 ? dx : nullptr, st, sw);
    if (rc != SKY_OK) {
      join();
      return rc;
    }
    if (marks) {
      // per-layer marks on the caller's stream only: a layer's weight
      // gradients on the second stream overlap the next layer's interval, as
      // in a step, and the slice's first layer (the last one here) takes the
      // final join, so the per-layer times add up to the backward pass
      if (i == 0) SKY_TRY(join());
      SKY_TRY(record_mark(s, (*marks)[2 * i + 1], st));
    }
    cur = s->dP[k];
    cur2 = s->cfg.dtype == SKY_DTYPE_BF16 ? nullptr : s->dR[k];  // bf16: already in dP[k]
    cur_dt = SKY_DTYPE_FP32;
  }
  return join();
}

int layer_index(const sky_slice* s, int32_t layer) {
  if (layer < s->cfg.layer_begin || layer >= s->cfg.layer_end) return -1;
  return layer - s->cfg.layer_begin;
}

__global__ void fill_pattern(void* p, int64_t n, int bf16, float scale, uint32_t seed) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    uint32_t h = (uint32_t)i * 2654435761u ^ seed;
    h ^= h >> 15; h *= 2246822519u; h ^= h >> 13; h *= 3266489917u; h ^= h >> 16;
    const float v = scale * ((h & 0xFFFFFF) / 8388608.0f - 1.0f);
    if (bf16) static_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
    else static_cast<float*>(p)[i] = v;
  }
}

// Occupies the stream for `ns` nanoseconds of wall time (one thread polling
// the global timer, sleeping between polls), then returns.
__global__ void delay_kernel(uint64_t ns) {
  if (threadIdx.x != 0) return;
  uint64_t t0, t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  do {
    __nanosleep(2000);
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  } while (t - t0 < ns);
}

}  // namespace
}  // namespace sky

using namespace sky;

#define ABI_GUARD_BEGIN try {
#define ABI_GUARD_END                                              \
  }                                                                \
  catch (const std::bad_alloc&) {                                  \
    set_error("host allocation failed");                           \
    return SKY_ERR_OOM;                                            \
  }                                                                \
  catch (const std::exception& ex) {                               \
    set_error("internal error: %s", ex.what());                    \
    return SKY_ERR_CUDA;                                           \
  }                                                                \
  catch (...) {                                                    \
    set_error("internal error");                                   \
    return SKY_ERR_CUDA;                                           \
  }

extern "C" {

void sky_debug_set_alloc_cap(uint64_t bytes) { g_alloc_cap = bytes; }

int64_t sky_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

const char* sky_status_string(sky_status st) {
  switch (st) {
    case SKY_OK: return "SKY_OK";
    case SKY_ERR_INVALID_ARG: return "SKY_ERR_INVALID_ARG";
    case SKY_ERR_OOM: return "SKY_ERR_OOM";
    case SKY_ERR_CUDA: return "SKY_ERR_CUDA";
    case SKY_ERR_STATE: return "SKY_ERR_STATE";
    case SKY_ERR_TIMEOUT: return "SKY_ERR_TIMEOUT";
    case SKY_ERR_UNSUPPORTED: return "SKY_ERR_UNSUPPORTED";
    case SKY_ERR_INFEASIBLE: return "SKY_ERR_INFEASIBLE";
  }
  return "SKY_ERR_UNKNOWN";
}

const char* sky_last_error(void) { return g_last_error.c_str(); }

int32_t sky_device_sm_count(void) { return sm_count(); }

void sky_debug_gemm_fault(uint64_t limit_ns, int32_t skip_loads) {
  gemm::set_debug(limit_ns, skip_loads);
}

// Sizes of the arena carved at create, computed on the host only.
static sky_status plan_slice(sky_slice* s, size_t* total) {
  const sky_slice_config& c = s->cfg;
  const int64_t T = (int64_t)c.max_batch * c.max_seq;
  s->maxT = T;
  size_t pb = 0, gb = 0;
  for (int k = 0; k < SKY_NUM_PARAMS; ++k) {
    pb += align_up(param_elems(s, k) * s->esz);
    gb += align_up(param_elems(s, k) * 4);
  }
  const size_t th = align_up((size_t)T * s->H * s->esz);
  const size_t t32 = align_up((size_t)T * s->H * 4);
  const bool bf = c.dtype == SKY_DTYPE_BF16;
  const size_t lse = align_up((size_t)c.max_batch * s->A * c.max_seq * 4);
  // Xb ctx X1b | QKV | Gp G | U1 U2 | lse | 4 stats
  const size_t stash = 3 * th + align_up((size_t)T * 3 * s->H * s->esz) +
                       2 * align_up((size_t)T * s->F * s->esz) + 2 * t32 + lse +
                       4 * align_up((size_t)T * 4);
  s->param_bytes = pb * s->L;
  s->grad_bytes = gb * s->L;
  s->stash_bytes = stash * s->L * s->n_slots;
  s->ws_bytes = align_up(workspace_need(s, T));
  s->ws2_bytes = bf ? align_up(side_workspace_need(s, T)) : 0;
  s->lnp_bytes = bf ? align_up(layernorm_bwd_ws((int)T, s->H)) : 0;
  s->db1p_bytes = bf ? align_up((size_t)gemm::colpart_rows_max((int)T) * s->F * 4) : 0;
  s->qkvp_bytes = bf ? align_up((size_t)c.max_batch * ceil_div(c.max_seq, 128) * 3 * s->H * 4) : 0;
  // dP[2] dR[2] dU2_32 dP1 | dU2b dU1b dctx (bf16) | dH | dqkv | delta | ws | ws2 | lnp[2] |
  // db1p | qkvp | status | x32 (bf16)
  const size_t wk = (bf ? 7 : 6) * t32 + (bf ? 3 : 1) * th + align_up((size_t)T * s->F * s->esz) +
                    align_up((size_t)T * 3 * s->H * s->esz) +
                    align_up(attention_bwd_ws(c.max_batch, c.max_seq, s->A)) + s->ws_bytes +
                    s->ws2_bytes + 4 * s->lnp_bytes + 2 * s->db1p_bytes + 2 * s->qkvp_bytes + 256 +
                    (s->n_slots > 1 ? gb : 0);  // gradient-accumulation scratch (one layer)
  s->ws_bytes_total = wk;
  *total = s->param_bytes + s->grad_bytes + s->stash_bytes + wk;
  return SKY_OK;
}

sky_status sky_slice_create(const sky_slice_config* cfg, sky_slice** out) {
  ABI_GUARD_BEGIN
  SKY_CHECK(cfg && out, SKY_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  const sky_slice_config& c = *cfg;
  SKY_CHECK(c.width > 0 && c.heads > 0 && c.ffn > 0 && c.max_batch > 0 && c.max_seq > 0,
            SKY_ERR_INVALID_ARG, "sizes must be positive");
  SKY_CHECK(c.width % c.heads == 0, SKY_ERR_INVALID_ARG, "width %d not divisible by heads %d",
            c.width, c.heads);
  SKY_CHECK(c.layer_begin >= 0 && c.layer_begin < c.layer_end, SKY_ERR_INVALID_ARG,
            "need 0 <= layer_begin < layer_end");
  SKY_CHECK(c.dtype == SKY_DTYPE_BF16 || c.dtype == SKY_DTYPE_FP32, SKY_ERR_INVALID_ARG,
            "unknown dtype");
  SKY_CHECK(c.ln_eps >= 0.f, SKY_ERR_INVALID_ARG, "ln_eps must be >= 0");
  SKY_CHECK(c.io_fp32 == 0 || c.io_fp32 == 1, SKY_ERR_INVALID_ARG, "io_fp32 must be 0 or 1");
  SKY_CHECK(c.stash_slots >= 0 && c.stash_slots <= kMaxStashSlots, SKY_ERR_INVALID_ARG,
            "stash_slots must be in [0, %d]", kMaxStashSlots);
  const int D = c.width / c.heads;
  if (c.dtype == SKY_DTYPE_BF16) {
    SKY_CHECK(D == 64, SKY_ERR_UNSUPPORTED, "bf16 slices need head dim 64 (got %d)", D);
    SKY_CHECK(c.width % 8 == 0 && c.ffn % 8 == 0, SKY_ERR_UNSUPPORTED,
              "bf16 slices need width and ffn multiples of 8");
    SKY_CHECK(c.width <= 2048, SKY_ERR_UNSUPPORTED, "width above 2048 not supported");
  } else {
    SKY_CHECK(D <= 128 && c.width % 4 == 0 && c.width <= 1024, SKY_ERR_UNSUPPORTED,
              "fp32 slices need head dim <= 128 and width <= 1024, multiple of 4");
  }
  SKY_CHECK((int64_t)c.max_batch * c.max_seq <= (int64_t)1 << 30, SKY_ERR_INVALID_ARG,
            "max_batch * max_seq too large");
  auto* s = new sky_slice();
  s->cfg = c;
  s->L = c.layer_end - c.layer_begin;
  s->H = c.width; s->A = c.heads; s->F = c.ffn; s->D = D;
  s->esz = c.dtype == SKY_DTYPE_BF16 ? 2 : 4;
  s->n_slots = c.stash_slots > 1 ? c.stash_slots : 1;
  size_t total = 0;
  plan_slice(s, &total);
  if (g_alloc_cap && total > g_alloc_cap) {
    set_error("slice needs %zu bytes, above the allocation cap %llu", total,
              (unsigned long long)g_alloc_cap);
    delete s;
    return SKY_ERR_OOM;
  }
  if (cudaGetDevice(&s->device) != cudaSuccess) {
    set_error("no CUDA device");
    delete s;
    return SKY_ERR_CUDA;
  }
  cudaError_t e = cudaMalloc(&s->arena, total);
  if (e != cudaSuccess) {
    cudaGetLastError();
    set_error("cudaMalloc(%zu): %s", total, cudaGetErrorString(e));
    delete s;
    return e == cudaErrorMemoryAllocation ? SKY_ERR_OOM : SKY_ERR_CUDA;
  }
  e = cudaMemset(s->arena, 0, total);
  if (e != cudaSuccess) {
    cudaFree(s->arena);
    delete s;
    return cuda_fail(e, "cudaMemset");
  }
  char* p = static_cast<char*>(s->arena);
  auto take = [&](size_t bytes) {
    void* r = p;
    p += align_up(bytes);
    return r;
  };
  const int64_t T = s->maxT;
  const size_t th = (size_t)T * s->H * s->esz;
  const size_t t32 = (size_t)T * s->H * 4;
  const bool bf = c.dtype == SKY_DTYPE_BF16;
  const size_t lse_b = (size_t)c.max_batch * s->A * c.max_seq * 4;
  auto take_stash = [&](LayerBufs& Lb) {
    Lb.Xb = take(th); Lb.ctx = take(th); Lb.X1b = take(th);
    Lb.QKV = take((size_t)T * 3 * s->H * s->esz);
    Lb.Gp = take((size_t)T * s->F * s->esz);
    Lb.G = take((size_t)T * s->F * s->esz);
    Lb.U1 = static_cast<float*>(take(t32));
    Lb.U2 = static_cast<float*>(take(t32));
    Lb.lse = static_cast<float*>(take(lse_b));
    Lb.mean1 = static_cast<float*>(take((size_t)T * 4));
    Lb.rstd1 = static_cast<float*>(take((size_t)T * 4));
    Lb.mean2 = static_cast<float*>(take((size_t)T * 4));
    Lb.rstd2 = static_cast<float*>(take((size_t)T * 4));
  };
  s->layers.resize(s->L);
  for (auto& Lb : s->layers) {
    for (int k = 0; k < SKY_NUM_PARAMS; ++k) Lb.p[k] = take(param_elems(s, k) * s->esz);
    for (int k = 0; k < SKY_NUM_PARAMS; ++k) Lb.g[k] = static_cast<float*>(take(param_elems(s, k) * 4));
    take_stash(Lb);
  }
  for (int k = 0; k < 2; ++k) {
    s->dP[k] = static_cast<float*>(take(t32));
    s->dR[k] = static_cast<float*>(take(t32));
  }
  s->dU2_32 = static_cast<float*>(take(t32));
  s->dP1 = static_cast<float*>(take(t32));
  s->dU2b = bf ? take(th) : s->dU2_32;
  s->dU1b = bf ? take(th) : nullptr;  // fp32 slices use dR[k] directly
  s->dctx = take(th);
  s->dH = take((size_t)T * s->F * s->esz);
  s->dqkv = take((size_t)T * 3 * s->H * s->esz);
  s->delta = static_cast<float*>(take(attention_bwd_ws(c.max_batch, c.max_seq, s->A)));
  s->ws = take(s->ws_bytes);
  if (s->ws2_bytes) s->ws2 = take(s->ws2_bytes);
  for (int k = 0; k < 2; ++k) {
    if (s->lnp_bytes) {
      s->lnp[k][0] = take(s->lnp_bytes);
      s->lnp[k][1] = take(s->lnp_bytes);
    }
    if (s->db1p_bytes) s->db1p[k] = static_cast<float*>(take(s->db1p_bytes));
    if (s->qkvp_bytes) s->qkvp[k] = static_cast<float*>(take(s->qkvp_bytes));
  }
  s->d_status = static_cast<int32_t*>(take(4));
  if (bf) s->x32 = static_cast<float*>(take(t32));
  // further stash slots (parameters and gradients are shared), and the
  // gradient-accumulation scratch, laid out like one layer's gradients
  s->slot_layers.assign(s->n_slots, s->layers);
  for (int m = 1; m < s->n_slots; ++m)
    for (auto& Lb : s->slot_layers[m]) take_stash(Lb);
  if (s->n_slots > 1)
    for (int k = 0; k < SKY_NUM_PARAMS; ++k) s->gscr[k] = static_cast<float*>(take(param_elems(s, k) * 4));
  s->slot_fwd.assign(s->n_slots, 0);
  s->slot_B.assign(s->n_slots, 0);
  s->slot_S.assign(s->n_slots, 0);
  s->slot_len.assign(s->n_slots, nullptr);
  if (bf) {
    // the weight-gradient side stream and its events
    bool ok = cudaStreamCreateWithFlags(&s->side, cudaStreamNonBlocking) == cudaSuccess;
    for (int j = 0; j < 4 && ok; ++j)
      ok = cudaEventCreateWithFlags(&s->ev_in[j], cudaEventDisableTiming) == cudaSuccess &&
           cudaEventCreateWithFlags(&s->ev_out[j], cudaEventDisableTiming) == cudaSuccess;
    if (ok) ok = cudaEventCreateWithFlags(&s->ev_join, cudaEventDisableTiming) == cudaSuccess;
    for (int k = 0; k < 2 && ok; ++k)
      ok = cudaEventCreateWithFlags(&s->ev_red[k], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
      const cudaError_t ce = cudaGetLastError();
      sky_slice_destroy(s);
      return cuda_fail(ce, "side stream / events");
    }
  }
  *out = s;
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_destroy(sky_slice* s) {
  ABI_GUARD_BEGIN
  if (!s) return SKY_OK;
  cudaDeviceSynchronize();
  // the graph first: its nodes use the slice's events
  if (s->step_exec) cudaGraphExecDestroy(s->step_exec);
  s->step_exec = nullptr;
  for (auto e : s->event_pool) cudaEventDestroy(e);
  for (auto e : s->graph_events) cudaEventDestroy(e);
  for (int j = 0; j < 4; ++j) {
    if (s->ev_in[j]) cudaEventDestroy(s->ev_in[j]);
    if (s->ev_out[j]) cudaEventDestroy(s->ev_out[j]);
  }
  if (s->ev_join) cudaEventDestroy(s->ev_join);
  for (int k = 0; k < 2; ++k)
    if (s->ev_red[k]) cudaEventDestroy(s->ev_red[k]);
  if (s->cap_stream) cudaStreamDestroy(s->cap_stream);
  if (s->side) cudaStreamDestroy(s->side);
  if (s->opt_mem) cudaFree(s->opt_mem);
  if (s->arena) cudaFree(s->arena);
  delete s;
  return SKY_OK;
  ABI_GUARD_END
}

static sky_status copy_tensors(sky_slice* s, int32_t layer, const void* const* src,
                               void* const* dst, int on_device, bool to_slice, bool grads) {
  SKY_CHECK(s && (to_slice ? (const void*)src : (const void*)dst), SKY_ERR_INVALID_ARG,
            "null argument");
  const int li = layer_index(s, layer);
  SKY_CHECK(li >= 0, SKY_ERR_INVALID_ARG, "layer %d outside [%d, %d)", layer,
            s->cfg.layer_begin, s->cfg.layer_end);
  if (s->last_stream) SKY_CUDA(cudaStreamSynchronize(s->last_stream));
  SKY_CUDA(cudaDeviceSynchronize());
  LayerBufs& Lb = s->layers[li];
  for (int k = 0; k < SKY_NUM_PARAMS; ++k) {
    const size_t bytes = param_elems(s, k) * (grads ? 4 : s->esz);
    void* dev = grads ? (void*)Lb.g[k] : Lb.p[k];
    if (to_slice) {
      SKY_CHECK(src[k], SKY_ERR_INVALID_ARG, "tensor %d is null", k);
      SKY_CUDA(cudaMemcpy(dev, src[k], bytes,
                          on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice));
    } else {
      SKY_CHECK(dst[k], SKY_ERR_INVALID_ARG, "tensor %d is null", k);
      SKY_CUDA(cudaMemcpy(dst[k], dev, bytes,
                          on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost));
    }
  }
  return SKY_OK;
}

sky_status sky_slice_set_params(sky_slice* s, int32_t layer, const void* const* tensors,
                                int on_device) {
  ABI_GUARD_BEGIN
  return copy_tensors(s, layer, tensors, nullptr, on_device, true, false);
  ABI_GUARD_END
}

sky_status sky_slice_get_params(sky_slice* s, int32_t layer, void* const* tensors, int on_device) {
  ABI_GUARD_BEGIN
  return copy_tensors(s, layer, nullptr, tensors, on_device, false, false);
  ABI_GUARD_END
}

sky_status sky_slice_sync(sky_slice* s) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s, SKY_ERR_INVALID_ARG, "null handle");
  if (s->last_stream) SKY_CUDA(cudaStreamSynchronize(s->last_stream));
  SKY_CUDA(cudaDeviceSynchronize());
  int32_t st = 0;
  SKY_CUDA(cudaMemcpy(&st, s->d_status, 4, cudaMemcpyDeviceToHost));
  SKY_CUDA(cudaMemset(s->d_status, 0, 4));
  if (st & kStatusTimeout) {
    set_error("a bounded device wait timed out");
    return SKY_ERR_TIMEOUT;
  }
  if (st & kStatusBadLength) {
    set_error("a sequence length was outside [1, S]");
    return SKY_ERR_INVALID_ARG;
  }
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_get_grads(sky_slice* s, int32_t layer, void* const* tensors, int on_device) {
  ABI_GUARD_BEGIN
  SKY_TRY(copy_tensors(s, layer, nullptr, tensors, on_device, false, true));
  return sky_slice_sync(s);
  ABI_GUARD_END
}

sky_status sky_slice_forward_slot(sky_slice* s, const void* x, const int32_t* d_len, int32_t B,
                                  int32_t S, void* y, int32_t slot, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s && x && d_len && y, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CHECK(slot >= 0 && slot < s->n_slots, SKY_ERR_INVALID_ARG, "slot %d outside [0, %d)", slot,
            s->n_slots);
  SKY_CHECK(B >= 1 && S >= 1, SKY_ERR_INVALID_ARG, "B and S must be >= 1 (got %d, %d)", B, S);
  SKY_CHECK(B <= s->cfg.max_batch && S <= s->cfg.max_seq, SKY_ERR_INVALID_ARG,
            "B=%d S=%d exceed max_batch=%d max_seq=%d", B, S, s->cfg.max_batch, s->cfg.max_seq);
  SKY_CHECK(x != y, SKY_ERR_INVALID_ARG, "x and y must not alias");
  SKY_CHECK((reinterpret_cast<uintptr_t>(y) & 15) == 0, SKY_ERR_UNSUPPORTED,
            "y must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  s->layers = s->slot_layers[slot];
  s->B = B; s->S = S; s->d_len = d_len; s->last_stream = st;
  s->slot_fwd[slot] = 0;
  SKY_TRY(forward_all(s, x, y, st, nullptr));
  s->slot_fwd[slot] = 1;
  s->slot_B[slot] = B; s->slot_S[slot] = S; s->slot_len[slot] = d_len;
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_backward_slot(sky_slice* s, const void* dy, void* dx, int32_t slot,
                                   int32_t accumulate, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s && dy && dx, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CHECK(slot >= 0 && slot < s->n_slots, SKY_ERR_INVALID_ARG, "slot %d outside [0, %d)", slot,
            s->n_slots);
  SKY_CHECK(accumulate == 0 || accumulate == 1, SKY_ERR_INVALID_ARG, "accumulate must be 0 or 1");
  SKY_CHECK(!accumulate || s->n_slots > 1, SKY_ERR_UNSUPPORTED,
            "gradient accumulation needs a slice created with stash_slots >= 2");
  SKY_CHECK(s->slot_fwd[slot], SKY_ERR_STATE, "backward needs a forward into slot %d first", slot);
  SKY_CHECK((reinterpret_cast<uintptr_t>(dy) & 15) == 0, SKY_ERR_UNSUPPORTED,
            "dy must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  s->layers = s->slot_layers[slot];
  s->B = s->slot_B[slot]; s->S = s->slot_S[slot]; s->d_len = s->slot_len[slot];
  s->last_stream = st;
  s->accumulate = accumulate != 0;
  const sky_status rc = backward_all(s, dy, dx, st, nullptr);
  s->accumulate = false;
  return rc;
  ABI_GUARD_END
}

sky_status sky_slice_forward(sky_slice* s, const void* x, const int32_t* d_len, int32_t B,
                             int32_t S, void* y, void* stream) {
  return sky_slice_forward_slot(s, x, d_len, B, S, y, 0, stream);
}

sky_status sky_device_delay(uint64_t ns, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(ns <= kMaxDelayNs, SKY_ERR_INVALID_ARG, "delay of %llu ns above the %llu ns limit",
            (unsigned long long)ns, (unsigned long long)kMaxDelayNs);
  if (ns == 0) return SKY_OK;
  delay_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(ns);
  count_launches(1);
  SKY_CUDA(cudaGetLastError());
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_backward(sky_slice* s, const void* dy, void* dx, void* stream) {
  return sky_slice_backward_slot(s, dy, dx, 0, 0, stream);
}

sky_status sky_slice_step_graph_create(sky_slice* s, const void* x, const int32_t* d_len,
                                       int32_t B, int32_t S, void* y, const void* dy, void* dx,
                                       void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s, SKY_ERR_INVALID_ARG, "null handle");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // One step in the ordinary way first: it checks every argument, and any
  // one-time set-up (kernel attributes, occupancy queries) happens outside
  // the capture.
  SKY_TRY(sky_slice_forward(s, x, d_len, B, S, y, stream));
  SKY_TRY(sky_slice_backward(s, dy, dx, stream));
  SKY_CUDA(cudaStreamSynchronize(st));
  if (s->step_exec) {
    SKY_CUDA(cudaGraphExecDestroy(s->step_exec));
    s->step_exec = nullptr;
  }
  for (auto e : s->graph_events) cudaEventDestroy(e);
  s->graph_events.clear();
  s->graph_recs.clear();
  // the direct step's per-kernel records are not kept
  s->recs.clear();
  s->event_next = 0;
  if (!s->cap_stream) SKY_CUDA(cudaStreamCreateWithFlags(&s->cap_stream, cudaStreamNonBlocking));
  cudaStream_t cs = s->cap_stream;
  const int64_t n0 = sky_launch_count();
  SKY_CUDA(cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal));
  s->layers = s->slot_layers[0];
  s->B = B; s->S = S; s->d_len = d_len;
  s->marks_in_graph = s->prof;
  sky_status rc = forward_all(s, x, y, cs, nullptr);
  if (rc == SKY_OK) rc = backward_all(s, dy, dx, cs, nullptr);
  s->marks_in_graph = false;
  if (s->prof) {  // the captured timers now belong to the graph
    s->graph_recs.swap(s->recs);
    s->graph_events.assign(s->event_pool.begin(), s->event_pool.begin() + s->event_next);
    s->event_pool.erase(s->event_pool.begin(), s->event_pool.begin() + s->event_next);
    s->event_next = 0;
  }
  cudaGraph_t graph = nullptr;
  const cudaError_t ec = cudaStreamEndCapture(cs, &graph);
  if (rc != SKY_OK) {
    if (graph) cudaGraphDestroy(graph);
    return rc;
  }
  if (ec != cudaSuccess) return cuda_fail(ec, "cudaStreamEndCapture");
  const cudaError_t ei = cudaGraphInstantiate(&s->step_exec, graph, 0);
  cudaGraphDestroy(graph);
  if (ei != cudaSuccess) {
    s->step_exec = nullptr;
    return cuda_fail(ei, "cudaGraphInstantiate");
  }
  // the captured launches ran nothing yet: they are counted at every replay
  s->step_launches = sky_launch_count() - n0;
  count_launches(-static_cast<int>(s->step_launches));
  s->step_B = B; s->step_S = S; s->step_len = d_len;
  SKY_CUDA(cudaGraphUpload(s->step_exec, st));
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_step_graph_launch(sky_slice* s, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s, SKY_ERR_INVALID_ARG, "null handle");
  SKY_CHECK(s->step_exec, SKY_ERR_STATE, "no step graph: call sky_slice_step_graph_create");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  SKY_CUDA(cudaGraphLaunch(s->step_exec, st));
  count_launches(static_cast<int>(s->step_launches));
  if (s->prof && !s->graph_recs.empty()) {
    // a step graph captured with per-kernel timing: add this replay's times
    SKY_CUDA(cudaStreamSynchronize(st));
    for (const auto& r : s->graph_recs) {
      float ms = 0;
      SKY_CUDA(cudaEventElapsedTime(&ms, r.start, r.stop));
      s->cat_ms[r.cat] += ms;
      s->cat_flops[r.cat] += r.flops;
      s->cat_bytes[r.cat] += r.bytes;
      s->cat_n[r.cat] += 1;
    }
  }
  s->B = s->step_B; s->S = s->step_S; s->d_len = s->step_len;
  s->last_stream = st;
  s->slot_fwd[0] = 1;
  s->slot_B[0] = s->step_B; s->slot_S[0] = s->step_S; s->slot_len[0] = s->step_len;
  return SKY_OK;
  ABI_GUARD_END
}

// Buffers, stream and events of one layer-cost measurement, released on every
// return path.
struct CostScratch {
  void *x = nullptr, *y = nullptr, *dy = nullptr, *dx = nullptr;
  int32_t* len = nullptr;
  cudaStream_t st = nullptr;
  std::vector<cudaEvent_t> ev;
  cudaGraphExec_t exec = nullptr;
  ~CostScratch() {
    if (st) cudaStreamSynchronize(st);
    if (exec) cudaGraphExecDestroy(exec);
    for (auto e : ev)
      if (e) cudaEventDestroy(e);
    if (st) cudaStreamDestroy(st);
    cudaFree(x); cudaFree(y); cudaFree(dy); cudaFree(dx); cudaFree(len);
  }
};

sky_status sky_slice_layer_cost(sky_slice* s, int32_t B, int32_t S, const int32_t* lens,
                                int32_t iters, sky_layer_cost* out, int32_t n_out) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s && out, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CHECK(n_out == s->L, SKY_ERR_INVALID_ARG, "n_out must be %d", s->L);
  SKY_CHECK(iters >= 1 && B >= 1 && S >= 1 && B <= s->cfg.max_batch && S <= s->cfg.max_seq,
            SKY_ERR_INVALID_ARG, "bad B/S/iters");
  std::vector<int32_t> hlen(B, S);
  double sum_len = (double)B * S;
  if (lens) {
    sum_len = 0;
    for (int b = 0; b < B; ++b) {
      SKY_CHECK(lens[b] >= 1 && lens[b] <= S, SKY_ERR_INVALID_ARG,
                "lens[%d] = %d outside [1, %d]", b, lens[b], S);
      hlen[b] = lens[b];
      sum_len += lens[b];
    }
  }
  // The measurement reuses the stash, workspace, gradients and status word:
  // wait for every step already enqueued on this slice (the caller's stream
  // of its last call, and the weight-gradient stream) before touching them.
  if (s->last_stream) SKY_CUDA(cudaStreamSynchronize(s->last_stream));
  if (s->side) SKY_CUDA(cudaStreamSynchronize(s->side));
  SKY_CUDA(cudaDeviceSynchronize());
  const bool io32 = s->cfg.io_fp32 && s->cfg.dtype == SKY_DTYPE_BF16;
  const size_t xb = (size_t)B * S * s->H * (io32 ? 4 : s->esz);
  CostScratch cs;
  SKY_CUDA(cudaMalloc(&cs.x, xb));
  SKY_CUDA(cudaMalloc(&cs.y, xb));
  SKY_CUDA(cudaMalloc(&cs.dy, xb));
  SKY_CUDA(cudaMalloc(&cs.dx, xb));
  SKY_CUDA(cudaMalloc(&cs.len, B * sizeof(int32_t)));
  SKY_CUDA(cudaStreamCreateWithFlags(&cs.st, cudaStreamNonBlocking));
  cudaStream_t st = cs.st;
  SKY_CUDA(cudaMemcpyAsync(cs.len, hlen.data(), B * sizeof(int32_t), cudaMemcpyHostToDevice, st));
  const int64_t n = (int64_t)B * S * s->H;
  const int bf = s->cfg.dtype == SKY_DTYPE_BF16 && !io32;
  fill_pattern<<<256, 256, 0, st>>>(cs.x, n, bf, 1.0f, 1u);
  fill_pattern<<<256, 256, 0, st>>>(cs.dy, n, bf, 1e-3f, 2u);
  count_launches(2);
  cs.ev.assign(4 * s->L, nullptr);
  for (auto& e : cs.ev) SKY_CUDA(cudaEventCreate(&e));
  std::vector<cudaEvent_t> fm(cs.ev.begin(), cs.ev.begin() + 2 * s->L);
  std::vector<cudaEvent_t> bm(cs.ev.begin() + 2 * s->L, cs.ev.end());
  std::vector<std::vector<double>> ft(s->L), bt(s->L);
  s->layers = s->slot_layers[0];
  s->B = B; s->S = S; s->d_len = cs.len; s->last_stream = st;
  const bool prof = s->prof;
  s->prof = false;
  sky_status rc = SKY_OK;
  // two direct passes (one-time set-up happens outside any capture), then
  // one forward + backward with per-layer marks captured as a graph and
  // replayed, as a step is
  for (int it = 0; it < 2 && rc == SKY_OK; ++it) {
    rc = forward_all(s, cs.x, cs.y, st, nullptr);
    if (rc == SKY_OK) rc = backward_all(s, cs.dy, cs.dx, st, nullptr);
    if (rc == SKY_OK && cudaStreamSynchronize(st) != cudaSuccess)
      rc = cuda_fail(cudaGetLastError(), "sync");
  }
  if (rc == SKY_OK) {
    if (cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
      rc = cuda_fail(cudaGetLastError(), "layer-cost capture");
  }
  int64_t captured = 0;
  if (rc == SKY_OK) {
    const int64_t n0 = sky_launch_count();
    s->marks_in_graph = true;
    rc = forward_all(s, cs.x, cs.y, st, &fm);
    if (rc == SKY_OK) rc = backward_all(s, cs.dy, cs.dx, st, &bm);
    s->marks_in_graph = false;
    // the captured launches ran nothing yet: they are counted at every replay
    captured = sky_launch_count() - n0;
    count_launches(-static_cast<int>(captured));
    cudaGraph_t graph = nullptr;
    const cudaError_t ec = cudaStreamEndCapture(st, &graph);
    if (rc == SKY_OK && ec != cudaSuccess) rc = cuda_fail(ec, "layer-cost capture");
    if (rc == SKY_OK) {
      const cudaError_t ei = cudaGraphInstantiate(&cs.exec, graph, 0);
      if (ei != cudaSuccess) rc = cuda_fail(ei, "layer-cost graph instantiate");
    }
    if (graph) cudaGraphDestroy(graph);
  }
  for (int it = 0; it < 1 + iters && rc == SKY_OK; ++it) {
    if (cudaGraphLaunch(cs.exec, st) != cudaSuccess || cudaStreamSynchronize(st) != cudaSuccess) {
      rc = cuda_fail(cudaGetLastError(), "layer-cost replay");
      break;
    }
    count_launches(static_cast<int>(captured));
    if (it < 1) continue;
    for (int i = 0; i < s->L; ++i) {
      float a = 0, b = 0;
      cudaEventElapsedTime(&a, fm[2 * i], fm[2 * i + 1]);
      cudaEventElapsedTime(&b, bm[2 * i], bm[2 * i + 1]);
      ft[i].push_back(a);
      bt[i].push_back(b);
    }
  }
  s->prof = prof;
  s->slot_fwd[0] = 0;
  s->last_stream = nullptr;  // the measuring stream is destroyed with cs
  if (rc != SKY_OK) return rc;
  const double T = (double)B * S, H = s->H, F = s->F;
  const double gemm_fwd = 2.0 * T * (4.0 * H * H + 2.0 * H * F);
  const double attn_fwd = 4.0 * H * S * sum_len;  // all S query rows against the valid keys
  size_t per_param = 0, per_grad = 0;
  for (int k = 0; k < SKY_NUM_PARAMS; ++k) {
    per_param += param_elems(s, k) * s->esz;
    per_grad += param_elems(s, k) * 4;
  }
  for (int i = 0; i < s->L; ++i) {
    auto med = [](std::vector<double>& v) {
      std::sort(v.begin(), v.end());
      return v.empty() ? 0.0 : v[v.size() / 2];
    };
    sky_layer_cost& o = out[i];
    std::memset(&o, 0, sizeof(o));
    o.layer = s->cfg.layer_begin + i;
    o.fwd_ms = med(ft[i]);
    o.bwd_ms = med(bt[i]);
    o.fwd_flops = gemm_fwd + attn_fwd;
    o.bwd_flops = 2.0 * (gemm_fwd + attn_fwd);
    o.param_bytes = per_param;
    o.grad_bytes = per_grad;
    o.stash_bytes = s->stash_bytes / s->L;
    o.workspace_bytes = s->ws_bytes_total / s->L;
  }
  return sky_slice_sync(s);
  ABI_GUARD_END
}

sky_status sky_slice_set_profiling(sky_slice* s, int enable) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s, SKY_ERR_INVALID_ARG, "null handle");
  s->prof = enable != 0;
  s->recs.clear();
  s->event_next = 0;
  for (int k = 0; k < P_NCAT; ++k) {
    s->cat_ms[k] = s->cat_flops[k] = s->cat_bytes[k] = 0;
    s->cat_n[k] = 0;
  }
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_optimizer_init(sky_slice* s, const sky_optimizer_config* cfg) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s && cfg, SKY_ERR_INVALID_ARG, "null argument");
  const sky_optimizer_config c = *cfg;
  SKY_CHECK(c.kind == SKY_OPT_SGD || c.kind == SKY_OPT_ADAMW, SKY_ERR_INVALID_ARG,
            "unknown optimizer kind %d", c.kind);
  SKY_CHECK(c.lr >= 0.f && c.weight_decay >= 0.f, SKY_ERR_INVALID_ARG, "lr and weight_decay must be >= 0");
  SKY_CHECK(c.kind != SKY_OPT_ADAMW || (c.beta1 >= 0.f && c.beta1 < 1.f && c.beta2 >= 0.f &&
                                        c.beta2 < 1.f && c.eps > 0.f),
            SKY_ERR_INVALID_ARG, "AdamW needs beta1, beta2 in [0, 1) and eps > 0");
  SKY_CHECK(c.kind != SKY_OPT_SGD || (c.momentum >= 0.f && c.momentum < 1.f), SKY_ERR_INVALID_ARG,
            "SGD momentum must be in [0, 1)");
  for (int k = 0; k < SKY_NUM_PARAMS; ++k)
    SKY_CHECK(param_elems(s, k) % 4 == 0, SKY_ERR_UNSUPPORTED,
              "parameter %d has %zu elements, not a multiple of 4", k, param_elems(s, k));
  if (s->last_stream) SKY_CUDA(cudaStreamSynchronize(s->last_stream));
  SKY_CUDA(cudaDeviceSynchronize());
  if (s->opt_mem) {
    cudaFree(s->opt_mem);
    s->opt_mem = nullptr;
  }
  s->opt_ready = false;
  const bool bf = s->cfg.dtype == SKY_DTYPE_BF16;
  const int nstate = c.kind == SKY_OPT_ADAMW ? 2 : 1;
  const int copies = nstate + (bf ? 1 : 0);  // fp32 slices update their parameters in place
  size_t per_layer = 0;
  for (int k = 0; k < SKY_NUM_PARAMS; ++k) per_layer += align_up(param_elems(s, k) * 4) * copies;
  const size_t ntens = (size_t)s->L * SKY_NUM_PARAMS;
  std::vector<opt::Tensor> ts;
  ts.reserve(ntens);
  // tables first (sizes known once the tensors are listed), then the tensors
  const size_t state_bytes = per_layer * s->L;
  const size_t tab_bytes = align_up(ntens * sizeof(opt::Tensor));
  // chunk count: one chunk per kChunk float4 groups of every tensor
  size_t nchunks = 0;
  for (int l = 0; l < s->L; ++l)
    for (int k = 0; k < SKY_NUM_PARAMS; ++k)
      nchunks += (size_t)ceil_div((int64_t)param_elems(s, k) / 4, opt::kChunk);
  const size_t total = state_bytes + tab_bytes + align_up(nchunks * sizeof(opt::Chunk));
  if (g_alloc_cap && total > g_alloc_cap) {
    set_error("optimizer state needs %zu bytes, above the allocation cap", total);
    return SKY_ERR_OOM;
  }
  cudaError_t e = cudaMalloc(&s->opt_mem, total);
  if (e != cudaSuccess) {
    cudaGetLastError();
    s->opt_mem = nullptr;
    set_error("cudaMalloc(%zu) for optimizer state: %s", total, cudaGetErrorString(e));
    return e == cudaErrorMemoryAllocation ? SKY_ERR_OOM : SKY_ERR_CUDA;
  }
  SKY_CUDA(cudaMemset(s->opt_mem, 0, state_bytes));
  char* q = static_cast<char*>(s->opt_mem);
  for (int l = 0; l < s->L; ++l) {
    LayerBufs& Lb = s->layers[l];
    for (int k = 0; k < SKY_NUM_PARAMS; ++k) {
      const size_t n = param_elems(s, k);
      auto take = [&]() {
        float* r = reinterpret_cast<float*>(q);
        q += align_up(n * 4);
        return r;
      };
      opt::Tensor t{};
      t.n = (int64_t)n;
      t.g = Lb.g[k];
      if (bf) {
        t.w = take();
        t.p = Lb.p[k];
        SKY_TRY(to_f32(Lb.p[k], (int64_t)n, SKY_DTYPE_BF16, t.w, nullptr));
      } else {
        t.w = static_cast<float*>(Lb.p[k]);
        t.p = nullptr;
      }
      t.s0 = take();
      t.s1 = nstate == 2 ? take() : nullptr;
      t.decay = (k == 0 || k == 2 || k == 6 || k == 8) ? 1 : 0;  // Wqkv, Wo, W1, W2
      ts.push_back(t);
    }
  }
  std::vector<opt::Chunk> chunks;
  opt::make_chunks(ts, &chunks);
  s->d_opt_tensors = reinterpret_cast<opt::Tensor*>(q);
  q += tab_bytes;
  s->d_opt_chunks = reinterpret_cast<opt::Chunk*>(q);
  SKY_CUDA(cudaMemcpy(s->d_opt_tensors, ts.data(), ts.size() * sizeof(opt::Tensor),
                      cudaMemcpyHostToDevice));
  SKY_CUDA(cudaMemcpy(s->d_opt_chunks, chunks.data(), chunks.size() * sizeof(opt::Chunk),
                      cudaMemcpyHostToDevice));
  SKY_CUDA(cudaDeviceSynchronize());
  s->opt_tensors = ts;
  s->opt_chunks = (int)chunks.size();
  s->opt_cfg = c;
  s->opt_t = 0;
  s->opt_ready = true;
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_optimizer_step(sky_slice* s, float lr, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s, SKY_ERR_INVALID_ARG, "null handle");
  SKY_CHECK(s->opt_ready, SKY_ERR_STATE, "optimizer not initialised");
  SKY_CHECK(lr >= 0.f, SKY_ERR_INVALID_ARG, "lr must be >= 0");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const sky_optimizer_config& c = s->opt_cfg;
  s->opt_t += 1;
  s->last_stream = st;
  double bytes = 0;
  for (const auto& t : s->opt_tensors)
    bytes += (double)t.n * (c.kind == SKY_OPT_ADAMW ? 28.0 : 20.0) + (t.p ? 2.0 * t.n : 0.0);
  Timed tm(s, st, P_COPY, 0, bytes);
  if (c.kind == SKY_OPT_ADAMW) {
    opt::AdamArgs a{lr, c.beta1, c.beta2, c.eps, c.weight_decay,
                    (float)(1.0 - std::pow((double)c.beta1, (double)s->opt_t)),
                    (float)(1.0 - std::pow((double)c.beta2, (double)s->opt_t))};
    return opt::launch_adamw(s->d_opt_tensors, s->d_opt_chunks, s->opt_chunks, a, st);
  }
  opt::SgdArgs a{lr, c.momentum, c.weight_decay, s->opt_t == 1 ? 1 : 0};
  return opt::launch_sgd(s->d_opt_tensors, s->d_opt_chunks, s->opt_chunks, a, st);
  ABI_GUARD_END
}

sky_status sky_slice_get_optimizer_state(sky_slice* s, int32_t layer, int32_t which,
                                         void* const* dst) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s && dst, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CHECK(s->opt_ready, SKY_ERR_STATE, "optimizer not initialised");
  const int li = layer_index(s, layer);
  SKY_CHECK(li >= 0, SKY_ERR_INVALID_ARG, "layer %d outside the slice", layer);
  SKY_CHECK(which >= 0 && which <= 2, SKY_ERR_INVALID_ARG, "which must be 0, 1 or 2");
  SKY_CHECK(which != 2 || s->opt_cfg.kind == SKY_OPT_ADAMW, SKY_ERR_INVALID_ARG,
            "SGD keeps one state tensor");
  if (s->last_stream) SKY_CUDA(cudaStreamSynchronize(s->last_stream));
  SKY_CUDA(cudaDeviceSynchronize());
  for (int k = 0; k < SKY_NUM_PARAMS; ++k) {
    const opt::Tensor& t = s->opt_tensors[(size_t)li * SKY_NUM_PARAMS + k];
    const float* src = which == 0 ? t.w : (which == 1 ? t.s0 : t.s1);
    SKY_CHECK(dst[k], SKY_ERR_INVALID_ARG, "tensor %d is null", k);
    SKY_CUDA(cudaMemcpy(dst[k], src, (size_t)t.n * 4, cudaMemcpyDeviceToHost));
  }
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_kernel_stats(sky_slice* s, sky_kernel_stat* out, int32_t n_out,
                                  int32_t* n_written) {
  ABI_GUARD_BEGIN
  SKY_CHECK(s && out && n_written, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CUDA(cudaDeviceSynchronize());
  for (const auto& r : s->recs) {
    float ms = 0;
    SKY_CUDA(cudaEventElapsedTime(&ms, r.start, r.stop));
    s->cat_ms[r.cat] += ms;
    s->cat_flops[r.cat] += r.flops;
    s->cat_bytes[r.cat] += r.bytes;
    s->cat_n[r.cat] += 1;
  }
  s->recs.clear();
  s->event_next = 0;
  int w = 0;
  for (int k = 0; k < P_NCAT && w < n_out; ++k) {
    if (s->cat_n[k] == 0) continue;
    sky_kernel_stat& o = out[w++];
    std::memset(&o, 0, sizeof(o));
    std::snprintf(o.name, sizeof(o.name), "%s", kCatNames[k]);
    o.launches = s->cat_n[k];
    o.total_ms = s->cat_ms[k];
    o.flops = s->cat_flops[k];
    o.bytes = s->cat_bytes[k];
  }
  *n_written = w;
  return SKY_OK;
  ABI_GUARD_END
}

sky_status sky_slice_memory(const sky_slice* s, uint64_t* param_bytes, uint64_t* grad_bytes,
                            uint64_t* stash_bytes, uint64_t* workspace_bytes) {
  SKY_CHECK(s, SKY_ERR_INVALID_ARG, "null handle");
  if (param_bytes) *param_bytes = s->param_bytes;
  if (grad_bytes) *grad_bytes = s->grad_bytes;
  if (stash_bytes) *stash_bytes = s->stash_bytes;
  if (workspace_bytes) *workspace_bytes = s->ws_bytes_total;
  return SKY_OK;
}

// ------------------------------------------------------------- sky_ops.h ABI
size_t sky_gemm_workspace_bytes(sky_gemm_form form, int32_t M, int32_t N, int32_t K,
                                sky_dtype in_dtype, sky_dtype out_dtype) {
  if (in_dtype != SKY_DTYPE_BF16 || out_dtype != SKY_DTYPE_FP32 || M <= 0 || N <= 0 || K <= 0)
    return 0;
  return gemm::workspace_bytes(form, M, N, K, true);
}

sky_status sky_gemm(sky_gemm_form form, int32_t M, int32_t N, int32_t K, sky_dtype in_dtype,
                    const void* A, const void* B, void* C, sky_dtype out_dtype,
                    sky_epilogue epilogue, const void* bias, const void* aux, void* aux_out,
                    void* workspace, size_t workspace_bytes, int32_t* d_status, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(A && B && C, SKY_ERR_INVALID_ARG, "null operand");
  SKY_CHECK(M > 0 && N > 0 && K > 0, SKY_ERR_INVALID_ARG, "sizes must be positive");
  SKY_CHECK(form >= SKY_GEMM_XWT && form <= SKY_GEMM_XTW, SKY_ERR_INVALID_ARG, "bad form");
  SKY_CHECK(epilogue >= SKY_EPI_STORE && epilogue <= SKY_EPI_GELU_BWD, SKY_ERR_INVALID_ARG,
            "bad epilogue");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (in_dtype == SKY_DTYPE_BF16)
    return gemm::launch_bf16(form, M, N, K, A, B, C, out_dtype == SKY_DTYPE_FP32, epilogue, bias,
                             aux, aux_out, workspace, workspace_bytes, d_status, st);
  SKY_CHECK(out_dtype == SKY_DTYPE_FP32, SKY_ERR_UNSUPPORTED, "fp32 input needs fp32 output");
  return gemm::launch_f32(form, M, N, K, static_cast<const float*>(A),
                          static_cast<const float*>(B), static_cast<float*>(C), epilogue,
                          static_cast<const float*>(bias), static_cast<const float*>(aux),
                          static_cast<float*>(aux_out), st);
  ABI_GUARD_END
}

sky_status sky_attention_fwd(const void* qkv, const int32_t* d_len, int32_t B, int32_t S,
                             int32_t H, int32_t A, sky_dtype dtype, void* ctx, float* lse,
                             int32_t* d_status, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(qkv && d_len && ctx && lse, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CHECK(B > 0 && S > 0 && H > 0 && A > 0 && H % A == 0, SKY_ERR_INVALID_ARG, "bad sizes");
  return attention_fwd(qkv, d_len, B, S, H, A, dtype, ctx, lse, d_status,
                       static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

size_t sky_attention_bwd_workspace_bytes(int32_t B, int32_t S, int32_t H, int32_t A) {
  (void)H;
  return attention_bwd_ws(B, S, A);
}

sky_status sky_attention_bwd(const void* qkv, const void* ctx, const void* dctx,
                             const float* lse, const int32_t* d_len, int32_t B, int32_t S,
                             int32_t H, int32_t A, sky_dtype dtype, void* dqkv, void* workspace,
                             size_t workspace_bytes, int32_t* d_status, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(qkv && ctx && dctx && lse && d_len && dqkv && workspace, SKY_ERR_INVALID_ARG,
            "null argument");
  SKY_CHECK(B > 0 && S > 0 && H > 0 && A > 0 && H % A == 0, SKY_ERR_INVALID_ARG, "bad sizes");
  SKY_CHECK(workspace_bytes >= attention_bwd_ws(B, S, A), SKY_ERR_INVALID_ARG,
            "workspace too small");
  return attention_bwd(qkv, ctx, dctx, lse, d_len, B, S, H, A, dtype, dqkv,
                       static_cast<float*>(workspace), d_status, static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

sky_status sky_layernorm_fwd(const float* a, const float* r, const void* gamma,
                             const void* beta, int32_t T, int32_t H, float eps, sky_dtype dtype,
                             float* u_out, float* y32, void* y, float* mean, float* rstd,
                             void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(a && gamma && beta && (y32 || y) && mean && rstd, SKY_ERR_INVALID_ARG,
            "null argument");
  SKY_CHECK(T > 0 && H > 0, SKY_ERR_INVALID_ARG, "bad sizes");
  return layernorm_fwd(a, r, gamma, beta, T, H, eps, dtype, u_out, y32, y, mean, rstd,
                       static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

size_t sky_layernorm_bwd_workspace_bytes(int32_t T, int32_t H) {
  if (T <= 0 || H <= 0) return 0;
  return layernorm_bwd_ws(T, H);
}

sky_status sky_layernorm_bwd(const void* dy, sky_dtype dy_dtype, const float* dy2,
                             const float* u, const void* gamma, const float* mean,
                             const float* rstd, int32_t T, int32_t H, sky_dtype dtype,
                             float* du32, void* du, float* dgamma, float* dbeta, float* dbias,
                             void* workspace, size_t workspace_bytes, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(dy && u && gamma && mean && rstd && (du32 || du), SKY_ERR_INVALID_ARG,
            "null argument");
  SKY_CHECK(T > 0 && H > 0, SKY_ERR_INVALID_ARG, "bad sizes");
  SKY_CHECK(dy_dtype == SKY_DTYPE_FP32 || dy_dtype == dtype, SKY_ERR_INVALID_ARG,
            "dy must be fp32 or the slice dtype");
  return layernorm_bwd(dy, dy_dtype, dy2, u, gamma, mean, rstd, T, H, dtype, du32, du, dgamma,
                       dbeta, dbias, workspace, workspace_bytes, static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

sky_status sky_add_f32(const float* a, const float* b, int64_t n, sky_dtype out_dtype, void* out,
                       void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(a && b && out && n >= 0, SKY_ERR_INVALID_ARG, "bad argument");
  return add_f32(a, b, n, out_dtype, out, static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

sky_status sky_to_f32(const void* x, int64_t n, sky_dtype dtype, float* out, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(x && out && n >= 0, SKY_ERR_INVALID_ARG, "bad argument");
  return to_f32(x, n, dtype, out, static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

sky_status sky_bias_gelu_fwd(const void* z, const void* bias, int32_t T, int32_t N,
                             sky_dtype dtype, void* hpre, void* g, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(z && hpre && g, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CHECK(T > 0 && N > 0, SKY_ERR_INVALID_ARG, "bad sizes");
  return bias_gelu_fwd(z, bias, T, N, dtype, hpre, g, static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

sky_status sky_gelu_bwd(const void* dg, const void* hpre, int32_t T, int32_t N, sky_dtype dtype,
                        void* dh, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(dg && hpre && dh, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CHECK(T > 0 && N > 0, SKY_ERR_INVALID_ARG, "bad sizes");
  return gelu_bwd(dg, hpre, T, N, dtype, dh, static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

size_t sky_column_sum_workspace_bytes(int32_t T, int32_t N) {
  if (T <= 0 || N <= 0) return 0;
  return column_sum_ws(T, N);
}

sky_status sky_column_sum(const void* x, int32_t T, int32_t N, sky_dtype dtype, float* out,
                          void* workspace, size_t workspace_bytes, void* stream) {
  ABI_GUARD_BEGIN
  SKY_CHECK(x && out, SKY_ERR_INVALID_ARG, "null argument");
  SKY_CHECK(T > 0 && N > 0, SKY_ERR_INVALID_ARG, "bad sizes");
  return column_sum(x, T, N, dtype, out, workspace, workspace_bytes,
                    static_cast<cudaStream_t>(stream));
  ABI_GUARD_END
}

}  // extern "C"
