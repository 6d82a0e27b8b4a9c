"""Pins of the allocator oracle (``oracle/allocator.py``) to facts outside it:
hand-worked runs of Alg. 1 and Alg. 2 whose every step is written out below,
closed-form optima of the Sec. IV-C model, and invariants.  Each example
isolates one rule of the algorithms, so dropping or flipping that rule fails
it (the comments name the rule)."""
import random

import pytest

from oracle import allocator as A


def test_even_partition():
    # Sec. IV-A: equal counts; the first L % D devices take the remainder
    assert A.even_partition(10, 4) == [0, 3, 6, 8, 10]
    assert A.even_partition(8, 2) == [0, 4, 8]
    assert A.even_partition(5, 5) == [0, 1, 2, 3, 4, 5]
    with pytest.raises(ValueError):
        A.even_partition(3, 4)


def test_coarse_gives_then_stops_on_strict_fit():
    # dm = [1, 4, 10], six layers of memory 1.  Even start [0,2,4,6], am = [2,2,2].
    # Sweep 1, i=0: am0 = 2 > 1 and device 0 holds 2 -> give: pi1 = 1, am = [1,3,2];
    #   take? dm0 = 1 > am0 + lm = 2: no.
    # i=1: am1 = 3 <= 4; take? dm1 = 4 > am1 + lm = 4: no (strict).
    # Sweep 2 starts with every device within memory -> return.
    assert A.coarse_allocation([1, 4, 10], [1] * 6) == [0, 1, 4, 6]


def test_coarse_takes_while_it_fits():
    # dm = [10, 1]: even [0,2,4], am = [2,2], device 1 over.
    # i=0: am0 fine; take while 10 > am0 + 1 and device 1 keeps a layer:
    #   pi1 = 3 (am [3,1]); next take would empty device 1 -> stop.
    assert A.coarse_allocation([10, 1], [1] * 4) == [0, 3, 4]
    # already feasible: the even partition is returned unchanged (no packing)
    assert A.coarse_allocation([10, 10], [1] * 4) == [0, 2, 4]


def test_coarse_raises_when_stuck():
    # dm = [1, 1], three unit layers: after one give device 1 still holds 2,
    # and no boundary can move again -> the exception of Alg. 1
    with pytest.raises(RuntimeError):
        A.coarse_allocation([1, 1], [1] * 3)


def test_finetune_take():
    # dt = [1, 3], unit layers, ct = 0: even [0,2,4], w = (2, 6), target 4.
    # i=0: w0 < 4, device 1 keeps a layer, memory fine -> take: [0,3,4], w = (3, 3).
    # Sweep 2: target 3; w0 = 3 is not below; w1 = 3 is not below -> unchanged.
    big = [100.0] * 2
    assert A.finetune([1, 3], big, [0, 0], [1] * 4, [1] * 4, [0, 2, 4], 100) == [0, 3, 4]


def test_finetune_give_is_conservative():
    # dt = [4, 1], eight unit layers: even [0,4,8], w = (16, 4), target 10.
    # i=0: w0 not below target; w1 = 4 < 10 and w0 - 4 = 12 > 10 -> give: [0,3,8].
    # Sweep 2: w = (12, 5), target 8.5; give needs 12 - 4 = 8 > 8.5: no -> stop.
    # The result (q = 12) is not the optimum [0,1,8] (q = 7): the give rule only
    # moves a layer while the giver stays above the mean.
    big = [100.0] * 2
    pi = A.finetune([4, 1], big, [0, 0], [1] * 8, [1] * 8, [0, 4, 8], 100)
    assert pi == [0, 3, 8]
    assert A.milp_objective([4, 1], [0, 0], [1] * 8, A.partition_owner(pi)) == 12
    # one sweep allowed: the first give still happens; none allowed: input back
    assert A.finetune([4, 1], big, [0, 0], [1] * 8, [1] * 8, [0, 4, 8], 1) == [0, 3, 8]
    assert A.finetune([4, 1], big, [0, 0], [1] * 8, [1] * 8, [0, 4, 8], 0) == [0, 4, 8]


def test_finetune_memory_guard():
    # as test_finetune_take but device 0 has memory 2: the take would need 3
    assert A.finetune([1, 3], [2, 10], [0, 0], [1] * 4, [1] * 4, [0, 2, 4], 100) == [0, 2, 4]


def test_finetune_keeps_one_layer():
    # dt = [1, 100], two layers: device 0 is far below target but device 1
    # would be emptied by a take -> no move
    assert A.finetune([1, 100], [9, 9], [0, 0], [1, 1], [1, 1], [0, 1, 2], 100) == [0, 1, 2]


def test_finetune_counts_ct_per_layer():
    # dt = [1, 1], ct = [0, 2], six unit layers.  With ct per layer (the text
    # before Alg. 2): w = (3, 9) -> take -> (4, 6) -> take -> (5, 3) -> stop
    # at [0,5,6].  Charging ct once per device would stop at [0,4,6].
    big = [100.0] * 2
    assert A.finetune([1, 1], big, [0, 2], [1] * 6, [1] * 6, [0, 3, 6], 100) == [0, 5, 6]


def test_milp_closed_forms():
    # identical devices, six unit layers on three: q = 2
    q, owner = A.milp_brute_force([1, 1, 1], [9] * 3, [0] * 3, [1] * 6, [1] * 6)
    assert q == 2 and sorted(owner.count(i) for i in range(3)) == [2, 2, 2]
    # the model allows an empty device: with dt = [4, 1] both layers go to the
    # fast device (q = 2) rather than one each (q = 4)
    q, owner = A.milp_brute_force([4, 1], [9, 9], [0, 0], [1, 1], [1, 1])
    assert q == 2 and owner == [1, 1]
    # ct enters once per device: one device holding everything costs 3 * 1 + 5
    q, _ = A.milp_brute_force([1], [9], [5], [1, 1, 1], [1, 1, 1])
    assert q == 8
    # infeasible memory
    q, owner = A.milp_brute_force([1, 1], [1, 1], [0, 0], [1] * 3, [1] * 3)
    assert q == float("inf") and owner is None
    # contiguity: dt = [1, 1], lf = [2, 3, 2].  The split {0, 2} | {1} would
    # give q = 4, but a device's layers must be contiguous: best is 5
    q, owner = A.milp_brute_force([1, 1], [99, 99], [0, 0], [2, 3, 2], [1, 1, 1])
    assert q == 5


def test_heuristic_invariants_random():
    rng = random.Random(3)
    for _ in range(200):
        D = rng.randint(1, 5)
        L = rng.randint(D, 14)
        dt = [rng.uniform(1, 7) for _ in range(D)]
        ct = [rng.uniform(0, 1) for _ in range(D)]
        lf = [rng.uniform(0.5, 2) for _ in range(L)]
        lm = [rng.uniform(0.5, 2) for _ in range(L)]
        dm = [rng.uniform(0.3, 1.0) * sum(lm) for _ in range(D)]
        try:
            pi = A.heuristic(dt, dm, ct, lf, lm)
        except RuntimeError:
            continue
        assert pi[0] == 0 and pi[-1] == L and len(pi) == D + 1
        assert all(pi[i + 1] - pi[i] >= 1 for i in range(D))
        assert A.memory_satisfied(dm, lm, pi)
        q_opt, _ = A.milp_brute_force(dt, dm, ct, lf, lm) if D ** L <= 20000 else (None, None)
        if q_opt is not None:
            # the exact model optimum is never worse than any feasible partition
            assert q_opt <= A.milp_objective(dt, ct, lf, A.partition_owner(pi)) + 1e-12
