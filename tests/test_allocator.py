"""The C++ layer allocator (include/sky_alloc.h, through the Python binding)
against the plain-Python oracle of Sec. IV (``oracle/allocator.py``).

Partitions are integer outputs: they must match the oracle exactly, including
every tie the floating-point workloads decide (both sides sum in the same
order).  Objective values of the exact baselines are compared to the
oracle's enumeration within 1e-12 relative (the sums are grouped
differently)."""
import itertools
import random
import time

import pytest

from oracle import allocator as A

alloc = pytest.importorskip("paper_2202_11836_gb300.allocator")
from paper_2202_11836_gb300 import _lib as L  # noqa: E402


def random_problem(rng, D, L_, tight=False, equal_layers=False):
    dt = [rng.uniform(1.0, 7.0) for _ in range(D)]
    ct = [rng.uniform(0.0, 0.5) for _ in range(D)]
    if equal_layers:
        lf, lm = [1.0] * L_, [1.0] * L_
    else:
        lf = [rng.uniform(0.5, 2.0) for _ in range(L_)]
        lm = [rng.uniform(0.5, 2.0) for _ in range(L_)]
    lo = 0.3 if tight else 0.8
    dm = [rng.uniform(lo, 1.0) * sum(lm) for _ in range(D)]
    return dt, dm, ct, lf, lm


def test_even_matches_oracle():
    for L_ in range(1, 40):
        for D in range(1, L_ + 1):
            assert alloc.even(L_, D) == A.even_partition(L_, D)


def test_coarse_finetune_heuristic_match_oracle():
    rng = random.Random(11)
    n_feasible = n_infeasible = 0
    for trial in range(600):
        D = rng.randint(1, 8)
        L_ = rng.randint(D, 40)
        prob = random_problem(rng, D, L_, tight=trial % 2 == 0, equal_layers=trial % 5 == 0)
        P = alloc.Problem(*prob)
        dt, dm, ct, lf, lm = prob
        try:
            want = A.coarse_allocation(dm, lm)
        except RuntimeError:
            with pytest.raises(L.SkyError) as e:
                P.coarse()
            assert e.value.status == L.SKY_ERR_INFEASIBLE
            n_infeasible += 1
            continue
        n_feasible += 1
        assert P.coarse() == want
        for max_iter in (0, 1, 3, 100):
            got, sweeps = P.finetune(want, max_iter)
            assert got == A.finetune(dt, dm, ct, lf, lm, want, max_iter), (trial, max_iter)
            assert 0 <= sweeps <= max(max_iter, 1)
        assert P.heuristic(100) == A.heuristic(dt, dm, ct, lf, lm, 100)
        # Alg. 2 from an arbitrary (possibly memory-violating) partition
        cuts = sorted(rng.sample(range(1, L_), D - 1)) if D > 1 else []
        start = [0] + cuts + [L_]
        assert P.finetune(start, 50)[0] == A.finetune(dt, dm, ct, lf, lm, start, 50)
    assert n_feasible > 100 and n_infeasible > 20


def test_workloads_match_oracle():
    rng = random.Random(5)
    for _ in range(100):
        D = rng.randint(1, 6)
        L_ = rng.randint(D, 20)
        prob = random_problem(rng, D, L_)
        dt, dm, ct, lf, lm = prob
        P = alloc.Problem(*prob)
        pi = A.even_partition(L_, D)
        assert P.workloads(pi, ct_per_layer=True) == [A.device_workload(dt, lf, ct, pi, i)
                                                     for i in range(D)]
        q = A.milp_objective(dt, ct, lf, A.partition_owner(pi))
        assert P.makespan(pi) == pytest.approx(q, rel=1e-12)


def ordered_brute_force(dt, dm, ct, lf, lm):
    """Best partition in device order (>= 1 layer each), by enumerating all cuts."""
    D, L_ = len(dt), len(lf)
    best = (float("inf"), None)
    for cuts in itertools.combinations(range(1, L_), D - 1):
        pi = [0, *cuts, L_]
        if not A.memory_satisfied(dm, lm, pi):
            continue
        q = A.milp_objective(dt, ct, lf, A.partition_owner(pi))
        if q < best[0]:
            best = (q, pi)
    return best


def test_exact_baselines_match_enumeration():
    rng = random.Random(21)
    checked = 0
    for trial in range(250):
        D = rng.randint(1, 3)
        L_ = rng.randint(D, 7)
        prob = random_problem(rng, D, L_, tight=trial % 3 == 0)
        dt, dm, ct, lf, lm = prob
        P = alloc.Problem(*prob)
        # best partition in device order
        q_ref, _ = ordered_brute_force(*prob)
        if q_ref == float("inf"):
            with pytest.raises(L.SkyError) as e:
                P.best_ordered()
            assert e.value.status == L.SKY_ERR_INFEASIBLE
        else:
            pi, q = P.best_ordered()
            assert q == pytest.approx(q_ref, rel=1e-12)
            assert A.memory_satisfied(dm, lm, pi) and all(pi[i + 1] > pi[i] for i in range(D))
            assert A.milp_objective(dt, ct, lf, A.partition_owner(pi)) == pytest.approx(q, rel=1e-12)
        # the Sec. IV-C model, device order free, empty devices allowed
        q_ref, _ = A.milp_brute_force(*prob)
        if q_ref == float("inf"):
            with pytest.raises(L.SkyError) as e:
                P.milp_exact()
            assert e.value.status == L.SKY_ERR_INFEASIBLE
            continue
        owner, q = P.milp_exact()
        assert q == pytest.approx(q_ref, rel=1e-12)
        assert A.milp_objective(dt, ct, lf, owner) == pytest.approx(q, rel=1e-12)
        for i in range(D):  # contiguous and within memory
            idx = [j for j in range(L_) if owner[j] == i]
            assert not idx or idx[-1] - idx[0] == len(idx) - 1
            assert sum(lm[j] for j in idx) <= dm[i]
        checked += 1
    assert checked > 100


def test_errors():
    P = alloc.Problem([1.0, 2.0], [10, 10], [0, 0], [1, 1, 1], [1, 1, 1])
    with pytest.raises(L.SkyError) as e:
        P.finetune([0, 3, 3])  # device 1 empty: not a partition
    assert e.value.status == L.SKY_ERR_INVALID_ARG
    with pytest.raises(L.SkyError):
        alloc.Problem([1.0, -1.0], [10, 10], [0, 0], [1, 1, 1], [1, 1, 1]).heuristic()
    with pytest.raises(L.SkyError):
        alloc.Problem([1.0] * 3, [10] * 3, [0] * 3, [1, 1], [1, 1]).heuristic()  # L < D
    with pytest.raises(L.SkyError) as e:
        alloc.Problem([1.0] * 9, [99] * 9, [0] * 9, [1] * 9, [1] * 9).milp_exact()
    assert e.value.status == L.SKY_ERR_UNSUPPORTED
    with pytest.raises(L.SkyError) as e:
        alloc.Problem([1.0, 1.0], [1, 1], [0, 0], [1, 1, 1], [1, 1, 1]).coarse()
    assert e.value.status == L.SKY_ERR_INFEASIBLE


def test_paper_scale_160_layers_64_devices():
    """The paper's largest run: 160 BERT layers on 64 devices whose speeds are
    spread like its slow_down factors (normal, clipped to [1, 7], Sec. V-A).
    The C++ heuristic matches the oracle and its makespan is compared with
    the even split and the exact best partition in device order."""
    rng = random.Random(2022)
    D, L_ = 64, 160
    dt = [min(7.0, max(1.0, rng.gauss(4.0, 1.5))) for _ in range(D)]
    ct = [rng.uniform(0.0, 0.05) for _ in range(D)]
    lf, lm = [1.0] * L_, [1.0] * L_
    dm = [8.0] * D
    P = alloc.Problem(dt, dm, ct, lf, lm)
    t0 = time.perf_counter()
    pi = P.heuristic(100)
    t_cpp = time.perf_counter() - t0
    t0 = time.perf_counter()
    pi_ref = A.heuristic(dt, dm, ct, lf, lm, 100)
    t_py = time.perf_counter() - t0
    assert pi == pi_ref
    q_even = P.makespan(A.even_partition(L_, D))
    q_heur = P.makespan(pi)
    _, q_best = P.best_ordered()
    assert q_best <= q_heur <= q_even
    print(f"\nD={D} L={L_}: even q={q_even:.3f}, heuristic q={q_heur:.3f}, "
          f"best in device order q={q_best:.3f}; heuristic {t_cpp*1e3:.2f} ms (C++) "
          f"vs {t_py*1e3:.1f} ms (oracle)")


def test_gpipe_makespan_closed_forms():
    from paper_2202_11836_gb300.pipeline import gpipe_makespan
    # identical stages: (M + D - 1) forward slots, then (M + D - 1) backward slots
    for D in (1, 2, 5):
        for M in (1, 3, 8):
            assert gpipe_makespan([2.0] * D, [3.0] * D, M) == pytest.approx((M + D - 1) * 5.0)
    # one micro-batch: the devices run one after the other
    assert gpipe_makespan([1.0, 2.0, 4.0], [2.0, 1.0, 3.0], 1) == pytest.approx(13.0)
    # many micro-batches: the slowest stage sets the pace
    t = gpipe_makespan([1.0, 5.0, 1.0], [1.0, 5.0, 1.0], 100)
    assert t == pytest.approx(2 * (5.0 * 100 + 1.0 + 1.0))
