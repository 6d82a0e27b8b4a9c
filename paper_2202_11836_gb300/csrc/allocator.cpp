// Layer allocator of Sky Computing (Sec. IV): even split (Sec. IV-A),
// coarse allocation by memory (Alg. 1), workload fine-tuning (Alg. 2), and
// two exact baselines for the Sec. IV-C model.  Host code only.
//
// Sums are accumulated layer by layer in index order and device by device in
// index order, and every comparison is made on freshly computed sums, so the
// same inputs give the same partition on every machine (the build disables
// floating-point contraction in host code).
#include <algorithm>
#include <cmath>
#include <limits>
#include <numeric>
#include <vector>

#include "../../include/sky_alloc.h"

namespace sky {
void set_error(const char* fmt, ...);

namespace {

using Pi = std::vector<int32_t>;

struct Problem {
  int D, L;
  const double *dt, *dm, *ct, *lf, *lm;
};

bool finite_nonneg(const double* a, int n) {
  for (int i = 0; i < n; ++i)
    if (!std::isfinite(a[i]) || a[i] < 0.0) return false;
  return true;
}

sky_status check(const sky_alloc_problem* p, Problem* out) {
  if (!p || !p->dt || !p->dm || !p->ct || !p->lf || !p->lm) {
    set_error("allocator: null argument");
    return SKY_ERR_INVALID_ARG;
  }
  if (p->devices < 1 || p->layers < p->devices) {
    set_error("allocator: need 1 <= devices <= layers (got D=%d, L=%d)", p->devices, p->layers);
    return SKY_ERR_INVALID_ARG;
  }
  const int D = p->devices, L = p->layers;
  bool ok = finite_nonneg(p->dt, D) && finite_nonneg(p->dm, D) && finite_nonneg(p->ct, D) &&
            finite_nonneg(p->lf, L) && finite_nonneg(p->lm, L);
  for (int i = 0; ok && i < D; ++i) ok = p->dt[i] > 0.0;
  if (!ok) {
    set_error("allocator: inputs must be finite and non-negative (dt positive)");
    return SKY_ERR_INVALID_ARG;
  }
  *out = Problem{D, L, p->dt, p->dm, p->ct, p->lf, p->lm};
  return SKY_OK;
}

bool is_partition(const int32_t* pi, int D, int L) {
  if (pi[0] != 0 || pi[D] != L) return false;
  for (int i = 0; i < D; ++i)
    if (pi[i + 1] <= pi[i]) return false;
  return true;
}

Pi even(int L, int D) {
  Pi pi(D + 1, 0);
  const int base = L / D, extra = L % D;
  for (int i = 0; i < D; ++i) pi[i + 1] = pi[i] + base + (i < extra ? 1 : 0);
  return pi;
}

int layers_of(const Pi& pi, int i) { return pi[i + 1] - pi[i]; }

// memory of device i's layers, summed in layer order
double allocated(const Problem& P, const Pi& pi, int i) {
  double s = 0.0;
  for (int j = pi[i]; j < pi[i + 1]; ++j) s += P.lm[j];
  return s;
}

bool memory_ok(const Problem& P, const Pi& pi) {
  for (int i = 0; i < P.D; ++i)
    if (allocated(P, pi, i) > P.dm[i]) return false;
  return true;
}

// workload of layer j on device i (the text before Alg. 2)
double layer_work(const Problem& P, int i, int j) { return P.dt[i] * P.lf[j] + P.ct[i]; }

double device_work(const Problem& P, const Pi& pi, int i, sky_cost_model m) {
  double s = 0.0;
  if (m == SKY_COST_CT_PER_LAYER) {
    for (int j = pi[i]; j < pi[i + 1]; ++j) s += layer_work(P, i, j);
    return s;
  }
  for (int j = pi[i]; j < pi[i + 1]; ++j) s += P.lf[j];
  return P.dt[i] * s + P.ct[i];
}

// Alg. 1
sky_status coarse(const Problem& P, Pi* out) {
  Pi pi = even(P.L, P.D);
  for (;;) {
    if (memory_ok(P, pi)) {
      *out = pi;
      return SKY_OK;
    }
    const Pi before = pi;
    for (int i = 0; i + 1 < P.D; ++i) {
      while (allocated(P, pi, i) > P.dm[i] && layers_of(pi, i) > 1) --pi[i + 1];
      while (P.dm[i] > allocated(P, pi, i) + P.lm[pi[i + 1]] && layers_of(pi, i + 1) > 1)
        ++pi[i + 1];
    }
    if (pi == before) {
      set_error("allocator: cannot fulfil the memory requirement (Alg. 1 made no progress)");
      return SKY_ERR_INFEASIBLE;
    }
  }
}

// Alg. 2
int finetune(const Problem& P, int max_iter, Pi* pip) {
  Pi& pi = *pip;
  int sweeps = 0;
  while (sweeps < max_iter) {
    double total = 0.0;
    for (int i = 0; i < P.D; ++i) total += device_work(P, pi, i, SKY_COST_CT_PER_LAYER);
    const double target = total / P.D;
    const Pi before = pi;
    for (int i = 0; i + 1 < P.D; ++i) {
      const double w_this = device_work(P, pi, i, SKY_COST_CT_PER_LAYER);
      Pi take = pi;
      ++take[i + 1];
      if (w_this < target && layers_of(pi, i + 1) > 1 && memory_ok(P, take)) {
        pi = take;
        continue;
      }
      const double w_next = device_work(P, pi, i + 1, SKY_COST_CT_PER_LAYER);
      const double w_last = layer_work(P, i, pi[i + 1] - 1);
      Pi give = pi;
      --give[i + 1];
      if (w_next < target && w_this - w_last > target && layers_of(pi, i) > 1 &&
          memory_ok(P, give))
        pi = give;
    }
    if (pi == before) return sweeps + 1;
    ++sweeps;
  }
  return sweeps;
}

// Minimum of max_k cost(order[k], block k) over splits of the layers into
// D consecutive blocks in the given device order (blocks may be empty when
// allow_empty).  cost(i, a, b) = dt_i * (lf[a] + ... + lf[b-1]) + ct_i;
// blocks over dm_i are excluded.  Returns +inf if nothing fits.
double ordered_dp(const Problem& P, const std::vector<int>& order, bool allow_empty, Pi* cut) {
  const int D = P.D, L = P.L;
  const double inf = std::numeric_limits<double>::infinity();
  // f[k][j]: best q for the first k devices covering layers [0, j)
  std::vector<double> f((D + 1) * (L + 1), inf);
  std::vector<int32_t> arg((D + 1) * (L + 1), -1);
  f[0] = 0.0;
  for (int k = 1; k <= D; ++k) {
    const int dev = order[k - 1];
    for (int j = 0; j <= L; ++j) {
      double best = inf;
      int32_t best_a = -1;
      // block [a, j) for device dev
      double flops = 0.0, mem = 0.0;
      const int a_hi = allow_empty ? j : j - 1;
      for (int a = a_hi; a >= 0; --a) {
        if (a < j) {
          flops += P.lf[a];
          mem += P.lm[a];
        }
        if (mem > P.dm[dev]) break;  // longer blocks only need more memory
        const double prev = f[(k - 1) * (L + 1) + a];
        if (prev == inf) continue;
        const double q = std::max(prev, P.dt[dev] * flops + P.ct[dev]);
        if (q < best) {
          best = q;
          best_a = a;
        }
      }
      f[k * (L + 1) + j] = best;
      arg[k * (L + 1) + j] = best_a;
    }
  }
  const double q = f[D * (L + 1) + L];
  if (q < inf && cut) {
    cut->assign(D + 1, 0);
    int j = L;
    for (int k = D; k >= 1; --k) {
      (*cut)[k] = j;
      j = arg[k * (L + 1) + j];
    }
    (*cut)[0] = j;
  }
  return q;
}

}  // namespace
}  // namespace sky

using namespace sky;

#define ALLOC_GUARD_BEGIN try {
#define ALLOC_GUARD_END                      \
  }                                          \
  catch (...) {                              \
    set_error("allocator: internal error");  \
    return SKY_ERR_INVALID_ARG;              \
  }

extern "C" {

sky_status sky_alloc_even(int32_t layers, int32_t devices, int32_t* pi) {
  ALLOC_GUARD_BEGIN
  if (!pi || devices < 1 || layers < devices) {
    set_error("allocator: need a pi buffer and 1 <= devices <= layers");
    return SKY_ERR_INVALID_ARG;
  }
  const Pi p = even(layers, devices);
  std::copy(p.begin(), p.end(), pi);
  return SKY_OK;
  ALLOC_GUARD_END
}

sky_status sky_alloc_coarse(const sky_alloc_problem* p, int32_t* pi) {
  ALLOC_GUARD_BEGIN
  Problem P;
  sky_status st = check(p, &P);
  if (st != SKY_OK) return st;
  if (!pi) {
    set_error("allocator: null pi");
    return SKY_ERR_INVALID_ARG;
  }
  Pi out;
  st = coarse(P, &out);
  if (st == SKY_OK) std::copy(out.begin(), out.end(), pi);
  return st;
  ALLOC_GUARD_END
}

sky_status sky_alloc_finetune(const sky_alloc_problem* p, int32_t max_iter, int32_t* pi,
                              int32_t* sweeps) {
  ALLOC_GUARD_BEGIN
  Problem P;
  sky_status st = check(p, &P);
  if (st != SKY_OK) return st;
  if (!pi || max_iter < 0 || !is_partition(pi, P.D, P.L)) {
    set_error("allocator: finetune needs a partition pi and max_iter >= 0");
    return SKY_ERR_INVALID_ARG;
  }
  Pi cur(pi, pi + P.D + 1);
  const int n = finetune(P, max_iter, &cur);
  std::copy(cur.begin(), cur.end(), pi);
  if (sweeps) *sweeps = n;
  return SKY_OK;
  ALLOC_GUARD_END
}

sky_status sky_alloc_heuristic(const sky_alloc_problem* p, int32_t max_iter, int32_t* pi) {
  ALLOC_GUARD_BEGIN
  Problem P;
  sky_status st = check(p, &P);
  if (st != SKY_OK) return st;
  if (!pi || max_iter < 0) {
    set_error("allocator: heuristic needs a pi buffer and max_iter >= 0");
    return SKY_ERR_INVALID_ARG;
  }
  Pi cur;
  st = coarse(P, &cur);
  if (st != SKY_OK) return st;
  finetune(P, max_iter, &cur);
  std::copy(cur.begin(), cur.end(), pi);
  return SKY_OK;
  ALLOC_GUARD_END
}

sky_status sky_alloc_workloads(const sky_alloc_problem* p, const int32_t* pi, sky_cost_model model,
                               double* w) {
  ALLOC_GUARD_BEGIN
  Problem P;
  sky_status st = check(p, &P);
  if (st != SKY_OK) return st;
  if (!pi || !w || !is_partition(pi, P.D, P.L) ||
      (model != SKY_COST_CT_PER_DEVICE && model != SKY_COST_CT_PER_LAYER)) {
    set_error("allocator: workloads need a partition pi, an output and a known cost model");
    return SKY_ERR_INVALID_ARG;
  }
  const Pi cur(pi, pi + P.D + 1);
  for (int i = 0; i < P.D; ++i) w[i] = device_work(P, cur, i, model);
  return SKY_OK;
  ALLOC_GUARD_END
}

sky_status sky_alloc_best_ordered(const sky_alloc_problem* p, int32_t* pi, double* q) {
  ALLOC_GUARD_BEGIN
  Problem P;
  sky_status st = check(p, &P);
  if (st != SKY_OK) return st;
  if (!pi || !q) {
    set_error("allocator: null output");
    return SKY_ERR_INVALID_ARG;
  }
  std::vector<int> order(P.D);
  std::iota(order.begin(), order.end(), 0);
  Pi cut;
  const double best = ordered_dp(P, order, false, &cut);
  if (!(best < std::numeric_limits<double>::infinity())) {
    set_error("allocator: no partition in device order fits the memory limits");
    return SKY_ERR_INFEASIBLE;
  }
  std::copy(cut.begin(), cut.end(), pi);
  *q = best;
  return SKY_OK;
  ALLOC_GUARD_END
}

sky_status sky_alloc_milp_exact(const sky_alloc_problem* p, int32_t* owner, double* q) {
  ALLOC_GUARD_BEGIN
  Problem P;
  sky_status st = check(p, &P);
  if (st != SKY_OK) return st;
  if (!owner || !q) {
    set_error("allocator: null output");
    return SKY_ERR_INVALID_ARG;
  }
  if (P.D > 8) {
    set_error("allocator: exact model solution limited to 8 devices (got %d)", P.D);
    return SKY_ERR_UNSUPPORTED;
  }
  std::vector<int> order(P.D), best_order;
  std::iota(order.begin(), order.end(), 0);
  double best = std::numeric_limits<double>::infinity();
  Pi best_cut, cut;
  do {
    const double v = ordered_dp(P, order, true, &cut);
    if (v < best) {
      best = v;
      best_cut = cut;
      best_order = order;
    }
  } while (std::next_permutation(order.begin(), order.end()));
  if (!(best < std::numeric_limits<double>::infinity())) {
    set_error("allocator: no assignment fits the memory limits");
    return SKY_ERR_INFEASIBLE;
  }
  for (int k = 0; k < P.D; ++k)
    for (int j = best_cut[k]; j < best_cut[k + 1]; ++j) owner[j] = best_order[k];
  *q = best;
  return SKY_OK;
  ALLOC_GUARD_END
}

}  // extern "C"
