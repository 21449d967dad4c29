"""Pins of the CPU oracle against what the paper and mathematics fix.

Each test names the passage it checks.  None of them retypes the oracle's own
formula: they compare against exhaustive enumeration, against the more
primitive materialisation rule of Section III-A, against closed forms
(Theorem 2's spider) or against theorems (Lemma 1, Prop. 1, Theorem 3).
"""
import os

import numpy as np
import pytest

from paper_2608_01655_gb300 import workloads as wl
from tests import bruteforce as bf


def _prob(oracle, inst):
    return oracle.Problem.from_instance(inst)


# ---------------------------------------------------------------- preorder ---
def test_preorder_definition(oracle_lib):
    """Section IV-A: preorder numbering and next(i) = first position after subtree."""
    rng = np.random.default_rng(1)
    for trial in range(30):
        inst = wl.random_small(rng, int(rng.integers(1, 40)), 1, 0)
        order, nxt = oracle_lib.preorder(inst.parent)
        assert list(order) == bf.preorder_positions(inst.parent)
        pos = np.empty(inst.n, int)
        pos[order] = np.arange(inst.n)
        # subtree of order[i] is exactly positions [i, next(i))
        for i, v in enumerate(order):
            sub = set()
            stack = [v]
            while stack:
                u = stack.pop()
                sub.add(u)
                stack.extend(np.nonzero(inst.parent == u)[0].tolist())
            assert sorted(pos[list(sub)]) == list(range(i, nxt[i]))


def test_preorder_rejects_cycles(oracle_lib):
    with pytest.raises(ValueError):
        oracle_lib.preorder(np.array([1, 0, -1], np.int32))
    with pytest.raises(ValueError):
        oracle_lib.preorder(np.array([0], np.int32))
    with pytest.raises(ValueError):
        oracle_lib.preorder(np.array([5, -1], np.int32))


# ------------------------------------------------------------- rooted DP ---
@pytest.mark.parametrize("w_max", [1, 4])
@pytest.mark.parametrize("variant", [0, 1])
def test_rooted_dp_vs_bruteforce(oracle_lib, w_max, variant):
    """Eq. 9 / Theorem 1: optimum over all parent-closed sets of weight <= k,
    and the returned set is the lexicographically smallest preorder indicator
    among optima (take only on a strict improvement)."""
    rng = np.random.default_rng(10 + w_max + 7 * variant)
    for trial in range(60):
        n = int(rng.integers(1, 15))
        inst = wl.random_small(rng, n, 1, 0, w_max=w_max)
        # small profit range -> many ties; some zeros and a few negatives
        profit = rng.integers(-2, 6, size=n).astype(np.int64)
        if trial % 3 == 0:
            profit = np.maximum(profit, 0)
        k = int(rng.integers(0, n * w_max + 2))
        best, chosen = oracle_lib.rooted_dp(inst.parent, inst.weight, profit, k, variant)
        bbest, bset = bf.best_parent_closed(inst.parent, inst.weight, profit, k)
        assert best == bbest
        np.testing.assert_array_equal(chosen, bset)


def test_rooted_dp_variants_agree_on_configs(oracle_lib):
    """The full-table and freed-row variants of Eq. 9 agree on real-sized trees."""
    rng = np.random.default_rng(5)
    for cfg in (0, 1):
        inst = wl.make(cfg)
        profit = rng.integers(0, 1000, size=inst.n).astype(np.int64)
        profit[rng.random(inst.n) < 0.5] = 0
        a = oracle_lib.rooted_dp(inst.parent, inst.weight, profit, 300, 0)
        b = oracle_lib.rooted_dp(inst.parent, inst.weight, profit, 300, 1)
        assert a[0] == b[0]
        np.testing.assert_array_equal(a[1], b[1])


def test_rooted_dp_special_cases(oracle_lib):
    rng = np.random.default_rng(3)
    # star forest of unit-weight roots: top-k profits; ties go to the later
    # preorder position because skipping is preferred at the earliest one
    n = 50
    parent = np.full(n, -1, np.int32)
    profit = rng.integers(0, 20, size=n).astype(np.int64)
    for k in (0, 1, 7, 49, 50, 80):
        best, ch = oracle_lib.rooted_dp(parent, np.ones(n, np.int32), profit, k)
        top = sorted(range(n), key=lambda v: (-profit[v], -v))[:k]
        top = [v for v in top if profit[v] > 0]
        assert best == profit[top].sum()
        assert set(np.nonzero(ch)[0]) == set(top)
    # a single chain with non-negative profits: the first min(k, n) nodes,
    # stopping after the last positive one
    parent = np.arange(-1, n - 1, dtype=np.int32)
    for k in (0, 3, 20, 60):
        best, ch = oracle_lib.rooted_dp(parent, np.ones(n, np.int32), profit, k)
        m = min(k, n)
        assert best == profit[:m].sum()
        pos = np.nonzero(profit[:m] > 0)[0]
        last = pos[-1] + 1 if pos.size else 0
        np.testing.assert_array_equal(ch, (np.arange(n) < last).astype(np.uint8))
    # unlimited budget: exactly the nodes whose subtree holds a positive profit
    inst = wl.random_small(rng, 200, 1, 0, w_max=3)
    profit = rng.integers(0, 3, size=200).astype(np.int64) * (rng.random(200) < 0.1)
    best, ch = oracle_lib.rooted_dp(inst.parent, inst.weight, profit, int(inst.weight.sum()))
    need = profit > 0
    for v in range(200):
        if profit[v] > 0:
            u = inst.parent[v]
            while u >= 0:
                need[u] = True
                u = inst.parent[u]
    np.testing.assert_array_equal(ch.astype(bool), need)
    assert best == profit.sum()


# ------------------------------------------------------------ objectives ---
@pytest.mark.parametrize("mode", [0, 1])
def test_objective_equals_materialisation_rule(oracle_lib, mode):
    """Lemma 1 (Eq. 4) and Eq. 6 equal the savings of the Section III-A rule."""
    rng = np.random.default_rng(20 + mode)
    for trial in range(40):
        inst = wl.random_small(rng, int(rng.integers(1, 12)), int(rng.integers(1, 5)), mode)
        prob = _prob(oracle_lib, inst)
        pl = (rng.random((inst.W, inst.n)) < 0.4).astype(np.uint8)
        assert oracle_lib.objective(prob, pl) == bf.materialisation_saving(inst, pl)


def test_lemma1_reduction(oracle_lib):
    """Setting f_{m<-h} = f_m turns Eq. 6 into Eq. 4 (end of Section III-C)."""
    rng = np.random.default_rng(30)
    for trial in range(40):
        inst = wl.random_small(rng, int(rng.integers(1, 15)), int(rng.integers(1, 6)), 0)
        src = wl.Instance(**{**inst.__dict__, "mode": 1,
                             "transfer": np.broadcast_to(inst.transfer[None], (inst.W, inst.W, inst.n)).copy()})
        pl = (rng.random((inst.W, inst.n)) < 0.5).astype(np.uint8)
        assert oracle_lib.objective_F(_prob(oracle_lib, inst), pl) == \
            oracle_lib.objective_Fpair(_prob(oracle_lib, src), pl)


def _golden(name):
    """Key -> value tokens of a fixture under tests/golden/ ('#' starts a comment)."""
    out = {}
    for line in open(os.path.join(os.path.dirname(__file__), "golden", name)):
        line = line.split("#", 1)[0].split()
        if line:
            out[line[0]] = line[1:]
    return out


def test_theorem2_spider_closed_form(oracle_lib):
    """Theorem 2's spider: covering the first x_i chunks of leg i saves
    lambda_i * sum_{d<=x_i}(2d - 1) = x_i^2 / s_i; demand scaled by L = lcm(s_i).
    The instance and its optimum L*q*B are the fixture tests/golden/spider_3partition.txt."""
    g = _golden("spider_3partition.txt")
    s = [int(v) for v in g["legs"]]             # a 3-Partition instance
    q, B = int(g["q"][0]), int(g["B"][0])
    assign = [int(v) for v in g["assignment"]]
    optimum = int(g["optimum"][0])
    L = int(np.lcm.reduce(s))
    assert L * q * B == optimum
    n = sum(s)
    parent, depth, leg = [], [], []
    for i, si in enumerate(s):
        for d in range(1, si + 1):
            parent.append(-1 if d == 1 else len(parent) - 1)
            depth.append(d)
            leg.append(i)
    parent = np.array(parent, np.int32)
    depth = np.array(depth, np.int64)
    W = q + 1                                   # q holders + one requester (the last)
    demand = np.zeros((W, n), np.int64)
    demand[q] = np.array([L // s[leg[b]] for b in range(n)])
    recompute = np.tile(2 * depth, (W, 1))
    budget = np.array([B] * q + [0], np.int32)
    rng = np.random.default_rng(4)
    for mode in (0, 1):
        transfer = np.ones((W, n), np.int64) if mode == 0 else np.ones((W, W, n), np.int64)
        inst = wl.Instance("spider", n, W, parent, np.ones(n, np.int32), demand, recompute,
                           transfer, mode, budget, 1, 1)
        prob = _prob(oracle_lib, inst)
        for trial in range(20):
            x = [int(rng.integers(0, si + 1)) for si in s]
            pl = np.zeros((W, n), np.uint8)
            for b in range(n):
                if depth[b] <= x[leg[b]]:
                    pl[int(rng.integers(q)), b] = 1       # any holder covers it
            expect = sum(L * xi * xi // si for xi, si in zip(x, s))
            assert oracle_lib.objective(prob, pl) == expect
            assert expect <= optimum
        # the fixture's valid 3-partition reaches the optimum
        pl = np.zeros((W, n), np.uint8)
        for b in range(n):
            pl[assign[leg[b]], b] = 1
        assert oracle_lib.objective(prob, pl) == optimum


# ------------------------------------------------------------- marginals ---
@pytest.mark.parametrize("mode", [0, 1])
def test_prop1_marginal_additivity(oracle_lib, mode):
    """Prop. 1 / Eq. 10: G(T_-h, T') - G(T_-h, {}) = sum_{b in T'} p_h(b) for any T'."""
    rng = np.random.default_rng(40 + mode)
    for trial in range(40):
        inst = wl.random_small(rng, int(rng.integers(1, 14)), int(rng.integers(1, 6)), mode)
        prob = _prob(oracle_lib, inst)
        pl = (rng.random((inst.W, inst.n)) < 0.4).astype(np.uint8)
        h = int(rng.integers(inst.W))
        p = oracle_lib.marginal(prob, h, pl)
        pl[h] = 0
        base = bf.materialisation_saving(inst, pl)
        for rep in range(5):
            Tp = (rng.random(inst.n) < 0.5).astype(np.uint8)
            pl2 = pl.copy()
            pl2[h] = Tp
            assert bf.materialisation_saving(inst, pl2) - base == int(p[Tp.astype(bool)].sum())


def test_eq10_equals_eq7_when_source_independent(oracle_lib):
    rng = np.random.default_rng(50)
    for trial in range(40):
        inst = wl.random_small(rng, int(rng.integers(1, 14)), int(rng.integers(1, 6)), 0)
        src = wl.Instance(**{**inst.__dict__, "mode": 1,
                             "transfer": np.broadcast_to(inst.transfer[None], (inst.W, inst.W, inst.n)).copy()})
        pl = (rng.random((inst.W, inst.n)) < 0.4).astype(np.uint8)
        h = int(rng.integers(inst.W))
        np.testing.assert_array_equal(oracle_lib.marginal(_prob(oracle_lib, inst), h, pl),
                                      oracle_lib.marginal(_prob(oracle_lib, src), h, pl))


# -------------------------------------------------- greedy / refinement ---
@pytest.mark.parametrize("mode", [0, 1])
def test_theorem3_half_approximation(oracle_lib, mode):
    """Theorem 3: one fixed-order greedy pass reaches >= OPT / 2; refinement and
    starts never go below it and never above OPT."""
    rng = np.random.default_rng(60 + mode)
    for trial in range(12):
        W = int(rng.integers(2, 4))
        inst = wl.random_small(rng, int(rng.integers(2, 7)), W, mode, k_max=3, w_max=2)
        prob = _prob(oracle_lib, inst)
        opt = bf.joint_optimum(inst)
        orders = wl.random_orders(W, 3, seed=trial)
        greedy = oracle_lib.plan(prob, 3, 0, orders=orders, threads=1)
        full = oracle_lib.plan(prob, 3, 5, orders=orders, threads=1)
        for s in range(3):
            assert 2 * greedy.per_start_objective[s] >= opt
            assert greedy.per_start_objective[s] <= full.per_start_objective[s] <= opt
        assert full.objective == full.per_start_objective.max()
        assert full.objective == bf.materialisation_saving(inst, full.placement)


@pytest.mark.parametrize("cfg", [0, 1])
def test_plan_invariants_on_configs(oracle_lib, cfg):
    """Algorithm 1 on the tiny and RAG workloads: feasible, prefix-complete,
    non-decreasing through refinement, best-of-starts, and coordinate-wise
    optimal when the returned start converged."""
    inst = wl.make(cfg)
    prob = _prob(oracle_lib, inst)
    S = inst.starts
    greedy = oracle_lib.plan(prob, S, 0)
    res = oracle_lib.plan(prob, S, inst.rounds)
    assert res.objective == res.per_start_objective.max()
    assert res.best_start == int(np.argmax(res.per_start_objective))
    assert np.all(res.per_start_objective >= greedy.per_start_objective)
    for m in range(inst.W):
        assert bf.is_parent_closed(inst.parent, res.placement[m])
        assert int(inst.weight[res.placement[m].astype(bool)].sum()) <= inst.budget[m]
    assert oracle_lib.objective(prob, res.placement) == res.objective
    b = res.best_start
    if res.per_start_sweeps[b] < inst.rounds:
        for h in range(inst.W):
            best, p, _ = oracle_lib.worker_update(prob, h, res.placement)
            assert best <= int(p[res.placement[h].astype(bool)].sum())


def test_default_orders_shape(oracle_lib):
    inst = wl.make(1)
    prob = _prob(oracle_lib, inst)
    o = oracle_lib.default_orders(prob, 6)
    for s in range(6):
        assert sorted(o[s]) == list(range(inst.W))
    sc = oracle_lib.standalone(prob)
    assert all(sc[o[0][t]] >= sc[o[0][t + 1]] for t in range(inst.W - 1))
    np.testing.assert_array_equal(o[1], o[0][::-1])
    assert list(oracle_lib.default_orders(prob, 1)[0]) == list(range(inst.W))


# ------------------------------------------------- generator constants ---
def test_generator_constants_match_paper_arithmetic():
    """Fig. 1 and RQ1 figures (fixture tests/golden/paper_constants.txt) that
    the cost generator is built on, recomputed from its constants and compared
    at the printed precision."""
    g = {k: float(v[0]) for k, v in _golden("paper_constants.txt").items()}
    assert wl.CHUNK_BYTES == 512 * 36_864                             # 3B: 36,864 B per token
    assert round(wl.CHUNK_BYTES / 1e6, 1) == g["kv_bytes_3b_chunk_mb"]
    t = int(wl.fetch_us(wl.CHUNK_BYTES, 1_500_000_000))
    assert round(t / 1000, 1) == g["fetch_3b_at_1p5gbps_ms"]
    b7 = 512 * 57_344                                                 # 7B: 57,344 B per token
    assert round(b7 / 1e6, 1) == g["kv_bytes_7b_chunk_mb"]
    assert round(512 * 262_144 / 1e6, 1) == g["kv_bytes_32b_chunk_mb"]
    f7 = int(wl.fetch_us(b7, 3_000_000_000)) / 1000                   # ms at 3 Gb/s
    p_cross = (f7 - g["a100_7b_fit_base_ms"]) / g["a100_7b_fit_slope_ms"]
    assert abs(p_cross - g["a100_7b_crossover_tokens"]) / g["a100_7b_crossover_tokens"] < 0.02
    assert g["l4_7b_fit_base_ms"] > f7                                # L4-7B favors fetching
    # the middle generator class crosses the 1.5 Gb/s fetch near the L4 crossover
    p_mid = (t - wl.BETA_US[1]) / wl.ALPHA_US_PER_TOKEN[1]
    assert abs(p_mid - g["l4_crossover_tokens"]) < 100
    assert wl.ALPHA_US_PER_TOKEN[1] == 3 * wl.ALPHA_US_PER_TOKEN[0]
    assert wl.ALPHA_US_PER_TOKEN[2] == 8 * wl.ALPHA_US_PER_TOKEN[0]


# ------------------------------------------------- safeguard candidates ---
def test_safeguards_match_their_definitions(oracle_lib):
    """Algorithm 1's requester-side safeguards (Section IV-C, comparators of
    Section V-A), each worker's set found by enumeration from the Section III-A
    saving rule rather than from a profit formula:
      Independent  maximises requester m's own saving with no other copy;
      Popularity   maximises requester m's local hits (its demand);
      LocalDedup   in index order, maximises requester m's own saving given
                   the sets of the earlier workers (later ones empty)."""
    rng = np.random.default_rng(71)
    for trial in range(25):
        W = int(rng.integers(1, 4))
        inst = wl.random_small(rng, int(rng.integers(1, 9)), W, 0, k_max=4, w_max=2)
        pl, obj = oracle_lib.safeguards(_prob(oracle_lib, inst))
        n = inst.n
        hits = wl.Instance(**{**inst.__dict__, "recompute": np.ones_like(inst.recompute),
                              "transfer": np.full_like(inst.transfer, 2)})
        dedup = np.zeros((W, n), np.uint8)
        for m in range(W):
            def alone(s, src=inst):
                x = np.zeros((W, n), np.uint8)
                x[m] = s
                return bf.requester_saving(src, x, m)

            def after_earlier(s):
                x = dedup.copy()
                x[m] = s
                return bf.requester_saving(inst, x, m)
            k = int(inst.budget[m])
            np.testing.assert_array_equal(pl[0, m], bf.best_set_by(inst.parent, inst.weight, k, alone))
            np.testing.assert_array_equal(pl[1, m], bf.best_set_by(inst.parent, inst.weight, k,
                                                                   lambda s: alone(s, hits)))
            dedup[m] = bf.best_set_by(inst.parent, inst.weight, k, after_earlier)
        np.testing.assert_array_equal(pl[2], dedup)
        for c in range(3):
            assert obj[c] == bf.materialisation_saving(inst, pl[c])


def test_safeguards_special_cases(oracle_lib):
    """With one worker Independent and LocalDedup coincide (nothing earlier to
    discount); when every fetch costs at least the recomputation the
    discounted value min{w, f} equals w, so LocalDedup is Independent again;
    with unit recomputation cost Independent is Popularity."""
    rng = np.random.default_rng(72)
    for trial in range(20):
        inst = wl.random_small(rng, int(rng.integers(1, 30)), 1, 0, k_max=10, w_max=3)
        pl, _ = oracle_lib.safeguards(_prob(oracle_lib, inst))
        np.testing.assert_array_equal(pl[0], pl[2])
        W = int(rng.integers(2, 5))
        inst = wl.random_small(rng, int(rng.integers(1, 30)), W, 0, k_max=10, w_max=3)
        slow = wl.Instance(**{**inst.__dict__, "transfer": inst.recompute + inst.transfer})
        pl, _ = oracle_lib.safeguards(_prob(oracle_lib, slow))
        np.testing.assert_array_equal(pl[0], pl[2])
        ones = wl.Instance(**{**inst.__dict__, "recompute": np.ones_like(inst.recompute)})
        pl, _ = oracle_lib.safeguards(_prob(oracle_lib, ones))
        np.testing.assert_array_equal(pl[0], pl[1])


def test_plan_never_worse_than_safeguards(oracle_lib):
    """Section IV-C: the returned placement is never worse than Independent,
    Popularity or LocalDedup under the same objective; a safeguard that beats
    every start is returned as candidate S + c; the source-dependent objective
    has no safeguards."""
    rng = np.random.default_rng(73)
    won = 0
    for trial in range(30):
        inst = wl.random_small(rng, int(rng.integers(2, 25)), int(rng.integers(2, 5)), 0, k_max=6, w_max=2)
        prob = _prob(oracle_lib, inst)
        S = int(rng.integers(1, 4))
        with_sg = oracle_lib.plan(prob, S, 3, threads=1)
        without = oracle_lib.plan(prob, S, 3, threads=1, safeguards=False)
        _, obj = oracle_lib.safeguards(prob)
        np.testing.assert_array_equal(with_sg.safeguard_objective, obj)
        assert with_sg.objective == max(without.objective, int(obj.max()))
        assert with_sg.objective == bf.materialisation_saving(inst, with_sg.placement)
        if with_sg.best_start >= S:
            won += 1
            assert obj[with_sg.best_start - S] == with_sg.objective > without.objective
        else:
            assert with_sg.best_start == without.best_start
    src = wl.random_small(rng, 10, 3, 1)
    r = oracle_lib.plan(_prob(oracle_lib, src), 2, 2, threads=1)
    assert r.safeguard_objective is None and r.best_start < 2
    with pytest.raises(ValueError):
        oracle_lib.safeguards(_prob(oracle_lib, src))


# ------------------------------------------------------- epoch updates ---
def _refreshed(rng, inst, kind):
    """Demand after a shift: log-normal popularity noise, or a routing shift
    that moves one worker's demand to another (cf. RQ5's transitions)."""
    dem = inst.demand.copy()
    if kind == 0:
        dem = np.rint(dem * rng.lognormal(0.0, 1.0, dem.shape)).astype(np.int64)
    else:
        a, b = rng.choice(inst.W, 2, replace=False) if inst.W > 1 else (0, 0)
        dem[[a, b]] = dem[[b, a]]
    return wl.Instance(**{**inst.__dict__, "demand": dem})


@pytest.mark.parametrize("mode", [0, 1])
def test_replan_amortisation_rule(oracle_lib, mode):
    """Section IV-D / RQ5: under refreshed demand the incumbent and the
    reoptimised target are both evaluated; the one-time cost of the new chunks
    is the Section III-A materialisation cost under the incumbent; the new
    target is adopted iff gain * horizon > cost * epoch, and break-even
    requests = ceil(cost * epoch / gain)."""
    rng = np.random.default_rng(80 + mode)
    seen = set()
    for trial in range(24):
        W = int(rng.integers(2, 5))
        inst = wl.random_small(rng, int(rng.integers(3, 20)), W, mode, k_max=6, w_max=2, demand_max=40)
        old = oracle_lib.plan(_prob(oracle_lib, inst), 2, 2, threads=1).placement
        new_inst = _refreshed(rng, inst, trial % 2)
        prob = _prob(oracle_lib, new_inst)
        target = oracle_lib.plan(prob, 2, 2, threads=1).placement
        epoch = 30000
        r0 = oracle_lib.replan(prob, old, 2, 2, epoch, 1, threads=1)
        assert r0.incumbent_objective == bf.materialisation_saving(new_inst, old)
        assert r0.new_objective == bf.materialisation_saving(new_inst, target)
        assert r0.materialization_cost == bf.materialisation_cost(new_inst, old, target)
        gain, cost = r0.new_objective - r0.incumbent_objective, r0.materialization_cost
        if gain <= 0:
            assert r0.break_even_requests == -1 and not r0.adopted
            np.testing.assert_array_equal(r0.placement, old)
            seen.add("kept")
            continue
        be = r0.break_even_requests
        assert be == -(-cost * epoch // gain)
        for horizon in (max(be - 1, 0), be, be + 1, 10 * epoch):
            r = oracle_lib.replan(prob, old, 2, 2, epoch, horizon, threads=1)
            adopt = gain * horizon > cost * epoch
            assert r.adopted == adopt
            np.testing.assert_array_equal(r.placement, target if adopt else old)
            seen.add(adopt)
    assert {True, False} <= seen


def test_replan_without_change_keeps_incumbent(oracle_lib):
    """Unchanged demand and the same planner settings reproduce the incumbent:
    no gain, no cost, nothing adopted."""
    rng = np.random.default_rng(82)
    inst = wl.random_small(rng, 40, 4, 0, k_max=10, w_max=2)
    prob = _prob(oracle_lib, inst)
    old = oracle_lib.plan(prob, 3, 3, threads=1).placement
    r = oracle_lib.replan(prob, old, 3, 3, 30000, 10 ** 9, threads=1)
    assert r.incumbent_objective == r.new_objective and r.materialization_cost == 0
    assert not r.adopted and r.break_even_requests == -1


def test_refinement_accepts_only_strict_improvements(oracle_lib):
    """Section IV-C: only strictly improving replacements are accepted, so a
    greedy result that is already coordinate-wise optimal ends after exactly
    one sweep with no accepted update (the DP re-finds an equal-valued set)."""
    rng = np.random.default_rng(70)
    seen = 0
    for trial in range(60):
        mode = trial % 2
        inst = wl.random_small(rng, int(rng.integers(3, 9)), int(rng.integers(2, 4)), mode,
                               k_max=3, w_max=2)
        prob = _prob(oracle_lib, inst)
        orders = wl.random_orders(inst.W, 1, seed=trial)
        g = oracle_lib.plan(prob, 1, 0, orders=orders, threads=1)
        local_opt = True
        for h in range(inst.W):
            best, p, _ = oracle_lib.worker_update(prob, h, g.placement)
            if best > int(p[g.placement[h].astype(bool)].sum()):
                local_opt = False
        r = oracle_lib.plan(prob, 1, 4, orders=orders, threads=1)
        if local_opt:
            seen += 1
            assert r.per_start_sweeps[0] == 1 and r.per_start_accepted[0] == 0
            np.testing.assert_array_equal(r.placement, g.placement)
        else:
            assert r.per_start_accepted[0] >= 1
    assert seen >= 10


def test_replan_break_even_saturates(oracle_lib):
    """Section IV-D break-even requests = ceil(cost * epoch / gain), computed
    here in exact integers; where it does not fit in int64 the oracle reports
    INT64_MAX (the library's reading), elsewhere the exact value."""
    rng = np.random.default_rng(91)
    seen_big = seen_exact = 0
    for trial in range(12):
        # unit demand keeps the gain small next to the one-time cost
        inst = wl.random_small(rng, 30, 3, trial % 2, k_max=8, w_max=1, demand_max=1)
        prob = _prob(oracle_lib, inst)
        old = oracle_lib.plan(prob, 1, 0, orders=np.array([[2, 1, 0]], np.int32), threads=1,
                              safeguards=False).placement
        epoch = (1 << 63) - 1 if trial % 3 else 30000
        r = oracle_lib.replan(prob, old, 2, 2, epoch, 1, threads=1)
        gain = r.new_objective - r.incumbent_objective
        if gain <= 0:
            assert r.break_even_requests == -1
            continue
        exact = -(-(r.materialization_cost * epoch) // gain)
        if exact > (1 << 63) - 1:
            seen_big += 1
            assert r.break_even_requests == (1 << 63) - 1
        else:
            seen_exact += 1
            assert r.break_even_requests == exact
    assert seen_big >= 2 and seen_exact >= 2
