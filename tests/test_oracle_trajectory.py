"""Pins of the oracle's planner loop and start orders (Section IV-C).

The invariants of `test_oracle_pins.py` (Theorem 3's bound, monotonicity,
coordinate-wise optimality) hold for any sweep order and any choice of the
reference value an update is compared against.  These tests pin the loop
itself: each start is rebuilt from enumeration only (tests/bruteforce.py:
best parent-closed sets under the Section III-A saving, no marginals and no
DP), visiting the workers in the start's order pi, keeping a new target only
when the saving strictly exceeds the saving right before the update, and
stopping after a sweep that kept nothing.  Every start's objective, sweep
count, accepted-update count and placement must equal the oracle's.  The
same instances are shown to separate the right loop from two plausible
wrong ones (sweeping in worker-id order; comparing against the saving at the
start of the sweep).

The start orders are pinned as well: SplitMix64 against its published
outputs, the Fisher-Yates shuffle it drives for starts s >= 2, and the tie
rule of the standalone-score order (equal scores keep the lower worker id
first; start 1 is the reverse).
"""
import os

import numpy as np
import pytest

from paper_2608_01655_gb300 import workloads as wl
from tests import bruteforce as bf

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _tiny(rng, mode, n_lo=3, n_hi=7, W=None, demand_max=4):
    W = int(rng.integers(2, 4)) if W is None else W
    inst = wl.random_small(rng, int(rng.integers(n_lo, n_hi)), W, mode, k_max=3, w_max=2 if n_hi <= 7 else 1,
                           demand_max=demand_max)
    inst.budget[:] = np.maximum(inst.budget, 1 if n_hi <= 7 else 2)
    return inst


def _trajectory_cases():
    """Tiny instances (n <= 9, W in 2..4) with 2-3 start orders each: small
    trees with weights 1-2 in both modes, then 4-worker source-dependent
    instances on which refinement accepts several updates per start, so that
    the order of a sweep matters."""
    rng = np.random.default_rng(2608)
    cases = []
    for trial in range(42):
        if trial < 12:
            inst = _tiny(rng, trial % 2)
        else:
            inst = _tiny(rng, 1, n_lo=7, n_hi=10, W=4, demand_max=30)
        S = int(rng.integers(2, 4))
        orders = wl.random_orders(inst.W, S, seed=100 + trial)
        if inst.W == 2:
            orders[0] = [1, 0]          # pi differs from the id order
        cases.append((inst, orders))
    return cases


def test_planner_loop_matches_enumerated_trajectory(oracle_lib):
    """Section IV-C / Theorem 3 / Prop. 1: per start, greedy pass then at most R
    sweeps in pi's order with strict acceptance, rebuilt by enumeration."""
    R = 4
    diverge_id_order = diverge_stale = 0
    for inst, orders in _trajectory_cases():
        prob = oracle_lib.Problem.from_instance(inst)
        S = orders.shape[0]
        res = oracle_lib.plan(prob, S, R, orders=orders, threads=1, safeguards=False)
        per_start = []
        for s in range(S):
            pi = [int(h) for h in orders[s]]
            T, sav, sweeps, acc = bf.coordinate_trajectory(inst, pi, R)
            per_start.append(T)
            assert res.per_start_objective[s] == sav, (s, pi)
            assert res.per_start_sweeps[s] == sweeps, (s, pi)
            assert res.per_start_accepted[s] == acc, (s, pi)
            # the two wrong loops, to show these instances tell them apart
            Ti, savi, swi, acci = bf.coordinate_trajectory(inst, pi, R, sweep_order=sorted(pi))
            Tz, savz, swz, accz = bf.coordinate_trajectory(inst, pi, R, stale_reference=True)
            diverge_id_order += (savi, swi, acci) != (sav, sweeps, acc) or not np.array_equal(Ti, T)
            diverge_stale += (savz, swz, accz) != (sav, sweeps, acc) or not np.array_equal(Tz, T)
        best = int(np.argmax([bf.materialisation_saving(inst, T) for T in per_start]))
        assert res.best_start == best
        np.testing.assert_array_equal(res.placement, per_start[best])
    assert diverge_id_order >= 3, "no instance separates pi-order sweeps from id-order sweeps"
    assert diverge_stale >= 3, "no instance separates the per-update reference from a stale one"


def test_greedy_pass_alone_matches_enumeration(oracle_lib):
    """R = 0: only the greedy pass, each worker against its predecessors in pi."""
    rng = np.random.default_rng(77)
    for trial in range(10):
        inst = _tiny(rng, trial % 2)
        orders = wl.random_orders(inst.W, 2, seed=trial)
        res = oracle_lib.plan(oracle_lib.Problem.from_instance(inst), 2, 0, orders=orders, threads=1)
        for s in range(2):
            T, sav, sweeps, acc = bf.coordinate_trajectory(inst, [int(h) for h in orders[s]], 0)
            assert res.per_start_objective[s] == sav
            assert res.per_start_sweeps[s] == 0 and res.per_start_accepted[s] == 0


def _golden_splitmix():
    vals = []
    for line in open(os.path.join(GOLDEN, "splitmix64_seed0.txt")):
        line = line.strip()
        if line and not line.startswith("#"):
            vals.append(int(line, 16))
    return vals


def test_splitmix64_published_outputs(oracle_lib):
    """SplitMix64 (Steele, Lea, Flood 2014) from state 0: the published outputs."""
    want = _golden_splitmix()
    got = [int(x) for x in oracle_lib.splitmix64(0, len(want))]
    assert got == want


def _fisher_yates(W, draws):
    """Durstenfeld's shuffle of 0..W-1: for i = W-1 down to 1 swap i with
    draws[W-1-i] mod (i + 1)."""
    q = list(range(W))
    for x, i in enumerate(range(W - 1, 0, -1)):
        j = int(draws[x] % (i + 1))
        q[i], q[j] = q[j], q[i]
    return q


@pytest.mark.parametrize("W", [3, 8, 16, 32])
def test_shuffled_start_orders(oracle_lib, W):
    """Starts s >= 2: the Fisher-Yates shuffle driven by SplitMix64 seeded with s."""
    rng = np.random.default_rng(W)
    inst = wl.random_small(rng, 12, W, W % 2, k_max=3, w_max=1)
    prob = oracle_lib.Problem.from_instance(inst)
    S = 7
    orders = oracle_lib.default_orders(prob, S)
    for s in range(2, S):
        draws = oracle_lib.splitmix64(s, W - 1)
        assert list(orders[s]) == _fisher_yates(W, draws), s
    # the seed is the start index: neighbouring starts differ
    assert any(list(orders[2]) != list(orders[s]) for s in range(3, S)) or W <= 3


@pytest.mark.parametrize("mode", [0, 1])
def test_standalone_order_tie_rule(oracle_lib, mode):
    """Start 0 sorts the standalone scores (Section IV-C, each a single-worker
    optimum, here by enumeration) in descending order with equal scores in
    ascending worker id; start 1 is its reverse."""
    rng = np.random.default_rng(31 + mode)
    n, W = 6, 5
    base = wl.random_small(rng, n, W, mode, k_max=3, w_max=2, demand_max=6)
    # two classes of identical workers, so scores tie within a class
    cls = [1, 0, 1, 0, 1]
    rows = {c: int(np.flatnonzero(np.array(cls) == c)[0]) for c in (0, 1)}
    for m in range(W):
        r = rows[cls[m]]
        base.demand[m] = base.demand[r]
        base.recompute[m] = base.recompute[r]
        base.budget[m] = max(int(base.budget[r]), 1)
    if mode == 0:
        for m in range(W):
            base.transfer[m] = base.transfer[rows[cls[m]]]
    else:
        base.transfer[:] = base.transfer[0, 1][None, None, :]
    prob = oracle_lib.Problem.from_instance(base)
    scores = [bf.standalone_score(base, h) for h in range(W)]
    assert list(oracle_lib.standalone(prob)) == scores
    assert len(set(scores)) < W                     # some scores tie
    want = sorted(range(W), key=lambda h: (-scores[h], h))
    o = oracle_lib.default_orders(prob, 3)
    assert list(o[0]) == want
    assert list(o[1]) == want[::-1]
    ties_high = sorted(range(W), key=lambda h: (-scores[h], -h))
    assert ties_high != want                        # the rule is observable here
