"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Everything is integer, so the bar is bit-exact: profits, DP optima, chosen
sets, objectives and whole plans must be identical.  Inputs come from the
seeded generator only; expected values come from the oracle only.
"""
import numpy as np
import pytest

from paper_2608_01655_gb300 import workloads as wl
from tests import bruteforce as bf

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def pp():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_01655_gb300 import build
    build.build()
    from paper_2608_01655_gb300 import binding
    return binding


def _dev(a, dtype):
    return torch.from_numpy(np.ascontiguousarray(a).astype(dtype)).cuda()


def _tree_instance(pp, parent, weight, W=1, mode=0, k=1):
    n = len(parent)
    inst = wl.Instance("t", n, W, np.asarray(parent, np.int32), np.asarray(weight, np.int32),
                       np.ones((W, n), np.int64), np.ones((W, n), np.int64),
                       np.ones((W, n), np.int64) if mode == 0 else np.ones((W, W, n), np.int64),
                       mode, np.full(W, k, np.int32), 1, 1)
    return pp.Instance.from_workload(inst)


def _dp_batch(pp, ppi, profits, budgets, max_budget):
    B, n = profits.shape
    prof = _dev(profits, np.int64)
    bud = _dev(budgets, np.int32)
    best = torch.zeros(B, dtype=torch.int64, device="cuda")
    bits = torch.zeros(max(pp.pp_dp_bits_size(ppi, B, max_budget) // 4, 1), dtype=torch.int32, device="cuda")
    chosen = torch.zeros((B, n), dtype=torch.uint8, device="cuda")
    pp.pp_tree_dp(ppi, prof, bud, max_budget, best, bits)
    pp.pp_traceback(ppi, bits, bud, max_budget, chosen)
    ppi.sync()
    return best.cpu().numpy(), chosen.cpu().numpy()


def _trees(rng):
    """Small trees of many shapes: random forests (ids relabelled), chains,
    stars, a binary tree and a single node."""
    out = []
    for _ in range(12):
        out.append(wl.random_small(rng, int(rng.integers(1, 120)), 1, 0, w_max=4).parent)
    out.append(np.arange(-1, 99, dtype=np.int32))                        # chain
    out.append(np.full(77, -1, np.int32))                                 # star forest
    out.append(np.array([-1] + [(v - 1) // 2 for v in range(1, 63)], np.int32))   # binary
    out.append(np.array([-1], np.int32))
    return out


def test_tree_dp_and_traceback_small(pp, oracle_lib):
    """Eq. 9 optimum and traced set, bit-exact, on many small trees and budgets
    (k = 0, k inside, k above the total weight), with ties and negatives."""
    rng = np.random.default_rng(100)
    for parent in _trees(rng):
        n = len(parent)
        weight = rng.integers(1, 5, size=n).astype(np.int32)
        ppi = _tree_instance(pp, parent, weight)
        B = 6
        profits = rng.integers(-3, 8, size=(B, n)).astype(np.int64)
        profits[0] = np.maximum(profits[0], 0)
        profits[1] = 0
        tw = int(weight.sum())
        budgets = np.array([0, 1, tw // 3, tw, tw + 7, int(rng.integers(0, tw + 1))], np.int32)
        maxb = int(budgets.max())
        best, chosen = _dp_batch(pp, ppi, profits, budgets, maxb)
        for b in range(B):
            ob, oc = oracle_lib.rooted_dp(parent, weight, profits[b], int(budgets[b]))
            assert best[b] == ob, (n, b)
            np.testing.assert_array_equal(chosen[b], oc)
        ppi.close()


def test_tree_dp_without_pruning(pp, oracle_lib):
    """The sweep over every row (pruning off: the prune kernel then only
    plans the skip-row stack for the whole tree) gives the oracle's optimum
    and set, as the pruned sweep does, on trees with deep stacks and
    zero-profit subtrees."""
    rng = np.random.default_rng(321)
    trees = _trees(rng)[:8]
    trees.append(np.array([-1] + [(v - 1) // 3 for v in range(1, 400)], np.int32))      # ternary
    for parent in trees:
        n = len(parent)
        weight = rng.integers(1, 3, size=n).astype(np.int32)
        ppi = _tree_instance(pp, parent, weight)
        profits = rng.integers(-2, 9, size=(3, n)).astype(np.int64)
        profits[1][rng.random(n) < 0.6] = 0
        tw = int(weight.sum())
        budgets = np.array([tw // 2 + 1, tw, max(tw // 5, 1)], np.int32)
        maxb = int(budgets.max())
        outs = []
        for no_prune in (True, False):
            pp.pp_tune_dp(ppi, 0, 0, False, no_prune)
            try:
                outs.append(_dp_batch(pp, ppi, profits, budgets, maxb))
            finally:
                pp.pp_tune_dp(ppi, 0, 0, False, False)
        for b in range(3):
            ob, oc = oracle_lib.rooted_dp(parent, weight, profits[b], int(budgets[b]))
            for best, chosen in outs:
                assert best[b] == ob, (n, b)
                np.testing.assert_array_equal(chosen[b], oc)
        ppi.close()


@pytest.mark.parametrize("n,wmax,kmax", [(700, 4, 1500), (3000, 4, 5000), (2500, 1, 2047),
                                         (5000, 3, 9000), (1200, 1, 1061)])
def test_tree_dp_multi_column_tiles(pp, oracle_lib, n, wmax, kmax):
    """Budgets that span several columns per thread (C = 2..16) and ragged
    tails (k not a multiple of 32), on deep and bushy trees."""
    rng = np.random.default_rng(n + kmax)
    inst = wl.random_small(rng, n, 1, 0, w_max=wmax)
    parent = inst.parent
    if n == 2500:                                     # deep: long chains with branching
        parent = np.array([-1] + [v - 1 if rng.random() < 0.9 else int(rng.integers(v)) for v in range(1, n)],
                          np.int32)
    weight = inst.weight
    ppi = _tree_instance(pp, parent, weight)
    profits = rng.integers(0, 1000, size=(3, n)).astype(np.int64)
    profits[1][rng.random(n) < 0.7] = 0
    budgets = np.array([kmax, kmax - 13, kmax // 2 + 1], np.int32)
    best, chosen = _dp_batch(pp, ppi, profits, budgets, kmax)
    for b in range(3):
        ob, oc = oracle_lib.rooted_dp(parent, weight, profits[b], int(budgets[b]))
        assert best[b] == ob
        np.testing.assert_array_equal(chosen[b], oc)


def _tile_crossing_trees(rng):
    """Trees whose walks cross the traceback's tiles in every way: a long chain
    (take-runs of 32 along the diagonal, column exits), a broom of chains from
    one root (skips over whole chains, far past the tile below), and a
    caterpillar (a spine whose nodes carry three leaves each: many single
    skips between takes)."""
    chain = np.arange(-1, 2999, dtype=np.int32)
    broom = [-1]
    for _ in range(24):
        broom.append(0)
        broom.extend(range(len(broom) - 1, len(broom) + 148))
    broom = np.asarray(broom, np.int32)
    cater = [-1]
    spine = 0
    for _ in range(600):
        for _ in range(3):
            cater.append(spine)
        cater.append(spine)
        spine = len(cater) - 1
    cater = np.asarray(cater, np.int32)
    return [("chain", chain), ("broom", broom), ("caterpillar", cater)]


@pytest.mark.parametrize("wmax", [1, 4])
def test_traceback_tile_crossings(pp, oracle_lib, wmax):
    """Optimum and traced set, bit-exact, on walks that leave their tile by
    rows, by columns and by skips far past the tile below, with budgets around
    the 32-row run, 64-row tile and 96-column tile boundaries."""
    rng = np.random.default_rng(4242 + wmax)
    for name, parent in _tile_crossing_trees(rng):
        n = len(parent)
        weight = rng.integers(1, wmax + 1, size=n).astype(np.int32)
        ppi = _tree_instance(pp, parent, weight)
        B = 6
        profits = rng.integers(1, 50, size=(B, n)).astype(np.int64)
        if name == "broom":                    # whole chains cheap: the walk skips them
            heads = np.flatnonzero(parent == 0)
            for b in range(0, B, 2):
                for h in heads[rng.random(len(heads)) < 0.5]:
                    profits[b, h:h + 149] = 1
        profits[1] = rng.integers(0, 3, size=n) * 40      # ties and zeros
        tw = int(weight.sum())
        budgets = np.array([min(tw, 2 * n // 3), 31, 32, 64, 96, min(tw, 97 + int(rng.integers(0, 400)))],
                           np.int32)
        maxb = int(budgets.max())
        best, chosen = _dp_batch(pp, ppi, profits, budgets, maxb)
        for b in range(B):
            ob, oc = oracle_lib.rooted_dp(parent, weight, profits[b], int(budgets[b]))
            assert best[b] == ob, (name, b)
            np.testing.assert_array_equal(chosen[b], oc, err_msg=f"{name} item {b}")
        ppi.close()


@pytest.mark.parametrize("mode", [0, 1])
def test_marginals_and_objective(pp, oracle_lib, mode):
    """Eq. 10 / Eq. 7 marginals and Eq. 4 / Eq. 6 objectives, bit-exact."""
    rng = np.random.default_rng(200 + mode)
    for W in (1, 3, 7, 32):
        inst = wl.random_small(rng, int(rng.integers(1, 300)), W, mode, demand_max=50)
        prob = oracle_lib.Problem.from_instance(inst)
        ppi = pp.Instance.from_workload(inst)
        B = 5
        pls = (rng.random((B, W, inst.n)) < rng.random((B, 1, 1))).astype(np.uint8)
        masks = np.zeros((B, inst.n), np.uint32)
        for m in range(W):
            masks |= pls[:, m, :].astype(np.uint32) << np.uint32(m)
        workers = rng.integers(0, W, size=B).astype(np.int32)
        prof = torch.zeros((B, inst.n), dtype=torch.int64, device="cuda")
        pp.pp_marginals(ppi, _dev(workers, np.int32), _dev(masks.view(np.int32), np.int32), prof)
        obj = torch.zeros(B, dtype=torch.int64, device="cuda")
        pp.pp_objective(ppi, _dev(pls, np.uint8), obj)
        ppi.sync()
        prof = prof.cpu().numpy()
        obj = obj.cpu().numpy()
        for b in range(B):
            np.testing.assert_array_equal(prof[b], oracle_lib.marginal(prob, int(workers[b]), pls[b]))
            assert obj[b] == oracle_lib.objective(prob, pls[b])
        ppi.close()


def _compare_plans(g, o):
    np.testing.assert_array_equal(g.placement, o.placement)
    assert g.objective == o.objective
    assert g.best_start == o.best_start
    np.testing.assert_array_equal(g.per_start_objective, o.per_start_objective)
    np.testing.assert_array_equal(g.per_start_sweeps, o.per_start_sweeps)
    np.testing.assert_array_equal(g.per_start_accepted, o.per_start_accepted)
    if o.safeguard_objective is None:
        assert g.safeguard_objective == ()
    else:
        assert list(g.safeguard_objective) == o.safeguard_objective.tolist()


def test_safeguards_match_oracle(pp, oracle_lib):
    """Independent, Popularity and LocalDedup (Algorithm 1, requester-side):
    every worker's set and the three objectives identical to the oracle, on
    random instances (unit to heavy chunks, so both DP kernels run) and on the
    tiny and RAG workloads at full size."""
    rng = np.random.default_rng(900)
    cases = [wl.random_small(rng, int(rng.integers(1, 150)), int(rng.integers(1, 9)), 0,
                             k_max=50, w_max=int(rng.choice([1, 2, 4, 6])), demand_max=40) for _ in range(12)]
    cases += [wl.make(0), wl.make(1)]
    for inst in cases:
        with pp.Instance.from_workload(inst) as ppi:
            gpl, gobj = pp.pp_safeguards(ppi)
        opl, oobj = oracle_lib.safeguards(oracle_lib.Problem.from_instance(inst))
        np.testing.assert_array_equal(gpl, opl)
        np.testing.assert_array_equal(gobj, oobj)


def test_plan_with_and_without_safeguards(pp, oracle_lib):
    """A safeguard that beats every start is returned as candidate S + c, the
    same as the oracle; without safeguards both return the best start; the
    source-dependent objective has none (pp_safeguards refuses it)."""
    rng = np.random.default_rng(901)
    won = 0
    for trial in range(16):
        W = int(rng.integers(2, 6))
        inst = wl.random_small(rng, int(rng.integers(2, 80)), W, 0, k_max=12, w_max=2, demand_max=30)
        prob = oracle_lib.Problem.from_instance(inst)
        S = int(rng.integers(1, 3))
        with pp.Instance.from_workload(inst) as ppi:
            g = pp.pp_plan_run(ppi, S, None, 1)
            g0 = pp.pp_plan_run(ppi, S, None, 1, safeguards=False)
        _compare_plans(g, oracle_lib.plan(prob, S, 1))
        _compare_plans(g0, oracle_lib.plan(prob, S, 1, safeguards=False))
        won += g.best_start >= S
    assert won >= 1                       # the candidate path S + c is exercised
    src = wl.random_small(rng, 30, 3, 1)
    with pp.Instance.from_workload(src) as ppi:
        with pytest.raises(pp.PPError):
            pp.pp_safeguards(ppi)
        assert pp.pp_plan_run(ppi, 2, None, 1).safeguard_objective == ()


@pytest.mark.parametrize("mode", [0, 1])
def test_plan_small_random(pp, oracle_lib, mode):
    """Algorithm 1 end to end on small random instances, explicit and default orders."""
    rng = np.random.default_rng(300 + mode)
    for trial in range(10):
        W = int(rng.integers(1, 9))
        inst = wl.random_small(rng, int(rng.integers(1, 200)), W, mode, k_max=60, w_max=3, demand_max=30)
        prob = oracle_lib.Problem.from_instance(inst)
        S = int(rng.integers(1, 5))
        orders = wl.random_orders(W, S, seed=trial) if trial % 2 else None
        with pp.Instance.from_workload(inst) as ppi:
            g = pp.pp_plan_run(ppi, S, orders, 4)
        o = oracle_lib.plan(prob, S, 4, orders=orders)
        _compare_plans(g, o)
        if orders is None:
            np.testing.assert_array_equal(g.orders, oracle_lib.default_orders(prob, S))


@pytest.mark.parametrize("cfg", [0, 1, 2])
def test_plan_parity_workloads(pp, oracle_lib, cfg):
    """Whole plans on the tiny, RAG and source-dependent workloads at full size:
    placement, objective, per-start objectives, sweeps and accepts identical."""
    inst = wl.make(cfg)
    prob = oracle_lib.Problem.from_instance(inst)
    with pp.Instance.from_workload(inst) as ppi:
        g = pp.pp_plan_run(ppi, inst.starts, None, inst.rounds)
    o = oracle_lib.plan(prob, inst.starts, inst.rounds)
    _compare_plans(g, o)
    # with default orders and several starts, every start's first greedy update
    # (an empty placement) walks the standalone-score DP of its worker instead
    # of running it again: the oracle evaluates those cells, the GPU does not
    reused = sum(inst.n * int(inst.budget[g.orders[x][0]]) for x in range(inst.starts)) if inst.starts > 1 else 0
    assert g.dp_cells == o.cells - reused


def test_plan_top2_marginals(pp, oracle_lib):
    """Source-dependent plans with the marginals taken from top-2 holder tables
    (Section IV-C) and from scanning the holders: both identical to the oracle,
    including dense holder sets (budgets close to n) and ties in g."""
    rng = np.random.default_rng(960)
    cases = []
    for t in range(8):
        n = int(rng.integers(2, 150))
        W = int(rng.integers(2, 9))
        inst = wl.random_small(rng, n, W, 1, k_max=max(2, n), w_max=2, demand_max=20)
        if t % 3 == 0:                                    # many equal gains: ties in the tables
            inst = wl.Instance(**{**inst.__dict__, "transfer": np.minimum(inst.transfer, 3),
                                  "recompute": np.minimum(inst.recompute, 5)})
        cases.append(inst)
    cases.append(wl.make(2))
    for inst in cases:
        prob = oracle_lib.Problem.from_instance(inst)
        S = min(inst.starts, 3) if inst.starts > 1 else 2
        o = oracle_lib.plan(prob, S, 3)
        with pp.Instance.from_workload(inst) as ppi:
            for mode in (1, 2):
                g = pp.pp_plan_run(ppi, S, None, 3, marginals=mode)
                assert g.used_top2 == (mode == 2)
                _compare_plans(g, o)


def test_plan_matches_oracle_digests(pp):
    """Whole plans at the paper-scale and stress sizes against the oracle's own
    plans, stored as digests by tests/golden/make_plan_digests.py (the oracle
    needs minutes on many cores there): objective, returned candidate and the
    SHA-256 of the placement identical."""
    import hashlib
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "plan_digests.txt")
    rows = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    assert rows
    cfg_of = {c["name"]: k for k, c in wl.CONFIGS.items()}
    for name, obj, best, digest in rows:
        inst = wl.make(cfg_of[name])
        with pp.Instance.from_workload(inst) as ppi:
            g = pp.pp_plan_run(ppi, inst.starts, None, inst.rounds)
        assert g.objective == int(obj)
        assert g.best_start == int(best)
        assert hashlib.sha256(g.placement.astype(np.uint8).tobytes()).hexdigest() == digest


def _shifted(rng, inst, kind):
    dem = inst.demand.copy()
    if kind == 0:
        dem = np.rint(dem * rng.lognormal(0.0, 1.0, dem.shape)).astype(np.int64)
    else:
        a, b = rng.choice(inst.W, 2, replace=False)
        dem[[a, b]] = dem[[b, a]]
    return wl.Instance(**{**inst.__dict__, "demand": dem})


@pytest.mark.parametrize("mode", [0, 1])
def test_replan_matches_oracle(pp, oracle_lib, mode):
    """Epoch update (Section IV-D, RQ5): incumbent and new objectives,
    materialisation cost, break-even requests, the adoption decision and the
    returned placement identical to the oracle, for several horizons."""
    rng = np.random.default_rng(950 + mode)
    cases = [wl.random_small(rng, int(rng.integers(2, 120)), int(rng.integers(2, 7)), mode, k_max=30,
                             w_max=2, demand_max=40) for _ in range(6)]
    if mode == 0:
        cases.append(wl.make(1))
    for t, inst in enumerate(cases):
        S, R = min(inst.starts, 4) if inst.starts > 1 else 2, 2
        old = oracle_lib.plan(oracle_lib.Problem.from_instance(inst), S, R).placement
        new = _shifted(rng, inst, t % 2)
        prob = oracle_lib.Problem.from_instance(new)
        o = oracle_lib.replan(prob, old, S, R, 30000, 1)
        horizons = [1, 10 ** 9] + ([o.break_even_requests, o.break_even_requests + 1]
                                   if o.break_even_requests > 0 else [])
        with pp.Instance.from_workload(new) as ppi:
            for h in horizons:
                g = pp.pp_replan(ppi, old, S, R, 30000, h)
                o = oracle_lib.replan(prob, old, S, R, 30000, h)
                assert (g.incumbent_objective, g.new_objective, g.materialization_cost, g.break_even_requests,
                        g.adopted) == (o.incumbent_objective, o.new_objective, o.materialization_cost,
                                       o.break_even_requests, o.adopted)
                np.testing.assert_array_equal(g.placement, o.placement)
            with pytest.raises(pp.PPError):
                pp.pp_replan(ppi, old, S, R, 0, 1)


def test_replan_break_even_saturates_like_oracle(pp, oracle_lib):
    """Break-even requests whose exact ceiling exceeds int64 saturate at
    INT64_MAX on both sides; smaller ones stay exact."""
    rng = np.random.default_rng(91)
    big = 0
    for trial in range(8):
        inst = wl.random_small(rng, 30, 3, trial % 2, k_max=8, w_max=1, demand_max=1)
        prob = oracle_lib.Problem.from_instance(inst)
        old = oracle_lib.plan(prob, 1, 0, orders=np.array([[2, 1, 0]], np.int32), threads=1,
                              safeguards=False).placement
        epoch = (1 << 63) - 1 if trial % 3 else 30000
        o = oracle_lib.replan(prob, old, 2, 2, epoch, 1)
        with pp.Instance.from_workload(inst) as ppi:
            g = pp.pp_replan(ppi, old, 2, 2, epoch, 1)
        assert (g.new_objective, g.materialization_cost, g.break_even_requests, g.adopted) == \
            (o.new_objective, o.materialization_cost, o.break_even_requests, o.adopted)
        big += o.break_even_requests == (1 << 63) - 1
    assert big >= 2


def _random_feasible_placement(rng, inst, frac):
    """Parent-closed, within-budget placement grown top-down (a plausible
    mid-refinement state to sample one update from)."""
    order, nxt = oracle_lib_preorder(inst.parent)
    pl = np.zeros((inst.W, inst.n), np.uint8)
    for m in range(inst.W):
        used = 0
        take = rng.random(inst.n) < frac
        for i, v in enumerate(order):
            p = inst.parent[v]
            if take[v] and (p < 0 or pl[m, p]) and used + inst.weight[v] <= inst.budget[m]:
                pl[m, v] = 1
                used += inst.weight[v]
    return pl


def oracle_lib_preorder(parent):
    import oracle
    return oracle.preorder(parent)


@pytest.mark.parametrize("cfg", [3, 4])
def test_single_update_full_size(pp, oracle_lib, cfg):
    """One per-worker update (marginals -> DP -> traceback) at the full paper-
    scale and stress sizes, against the oracle computing that one update."""
    inst = wl.make(cfg)
    prob = oracle_lib.Problem.from_instance(inst)
    rng = np.random.default_rng(400 + cfg)
    pl = _random_feasible_placement(rng, inst, 0.3)
    h = int(rng.integers(inst.W))
    masks = np.zeros(inst.n, np.uint32)
    for m in range(inst.W):
        masks |= pl[m].astype(np.uint32) << np.uint32(m)
    with pp.Instance.from_workload(inst) as ppi:
        prof = torch.zeros((1, inst.n), dtype=torch.int64, device="cuda")
        pp.pp_marginals(ppi, _dev([h], np.int32), _dev(masks[None].view(np.int32), np.int32), prof)
        k = int(inst.budget[h])
        best = torch.zeros(1, dtype=torch.int64, device="cuda")
        bits = torch.zeros(pp.pp_dp_bits_size(ppi, 1, k) // 4, dtype=torch.int32, device="cuda")
        chosen = torch.zeros((1, inst.n), dtype=torch.uint8, device="cuda")
        bud = _dev([k], np.int32)
        pp.pp_tree_dp(ppi, prof, bud, k, best, bits)
        pp.pp_traceback(ppi, bits, bud, k, chosen)
        ppi.sync()
    ob, oprof, och = oracle_lib.worker_update(prob, h, pl)
    np.testing.assert_array_equal(prof.cpu().numpy()[0], oprof)
    assert int(best.item()) == ob
    np.testing.assert_array_equal(chosen.cpu().numpy()[0], och)


@pytest.mark.parametrize("B", [16, 17])
def test_split_launch_matches_single_launch(pp, oracle_lib, B):
    """A paper-scale batch just above what clusters of 8 CTAs hold at one CTA
    per SM runs as two concurrent launches (the smallest sweeps on narrower
    clusters); optima, decision bits and chosen sets must equal those of one
    launch of the same shape, and the oracle's on sampled items."""
    inst = wl.make(3)
    prob = oracle_lib.Problem.from_instance(inst)
    rng = np.random.default_rng(77 + B)
    pls = [_random_feasible_placement(rng, inst, float(f)) for f in (0.0, 0.15, 0.3)]
    workers = [b % inst.W for b in range(B)]
    masks = np.zeros((B, inst.n), np.uint32)
    for b in range(B):
        pl = pls[b % len(pls)]
        for m in range(inst.W):
            if m != workers[b]:
                masks[b] |= pl[m].astype(np.uint32) << np.uint32(m)
    k = int(inst.budget[0])
    with pp.Instance.from_workload(inst) as ppi:
        split = pp.pp_dp_split(ppi, B, k)
        if torch.cuda.get_device_properties(0).multi_processor_count == 152:
            assert split["wide_items"] == 15 and split["narrow_cluster_ctas"] == 4, split
        prof = torch.zeros((B, inst.n), dtype=torch.int64, device="cuda")
        pp.pp_marginals(ppi, _dev(workers, np.int32), _dev(masks.view(np.int32), np.int32), prof)
        bud = _dev(np.full(B, k), np.int32)
        outs = []
        for tune in [(0, 0), (8, 4)]:               # automatic (split), then one launch
            pp.pp_tune_dp(ppi, *tune, False, False)
            try:
                best = torch.zeros(B, dtype=torch.int64, device="cuda")
                bits = torch.zeros(pp.pp_dp_bits_size(ppi, B, k) // 4, dtype=torch.int32, device="cuda")
                chosen = torch.zeros((B, inst.n), dtype=torch.uint8, device="cuda")
                pp.pp_tree_dp(ppi, prof, bud, k, best, bits)
                pp.pp_traceback(ppi, bits, bud, k, chosen)
                ppi.sync()
            finally:
                pp.pp_tune_dp(ppi, 0, 0, False, False)
            outs.append((best.cpu().numpy(), bits.cpu().numpy(), chosen.cpu().numpy()))
    np.testing.assert_array_equal(outs[0][0], outs[1][0])
    np.testing.assert_array_equal(outs[0][1], outs[1][1])
    np.testing.assert_array_equal(outs[0][2], outs[1][2])
    for b in (0, B - 1):
        ob, _, och = oracle_lib.worker_update(prob, workers[b], pls[b % len(pls)])
        assert int(outs[0][0][b]) == ob
        np.testing.assert_array_equal(outs[0][2][b], och)


def test_batch_of_16_with_stack_spill(pp, oracle_lib):
    """A 16-item batch on a tree whose skip-row stack is deeper than shared
    memory holds: the automatic shape (with these shared-memory needs, one
    CTA per SM, so clusters narrower than 8 rather than a split) and a forced
    8-CTA shape both spill stack levels to scratch; results equal each other
    and the oracle."""
    rng = np.random.default_rng(4242)
    parent = [-1]
    spine = 0
    for _ in range(70):                 # a spine whose nodes also have a leaf child: stack ~70 deep
        nxt = len(parent)
        parent.append(spine)
        parent.append(spine)
        spine = nxt
    for _ in range(4000):
        parent.append(int(rng.integers(len(parent))))
    parent = np.asarray(parent, np.int32)
    n = len(parent)
    weight = np.ones(n, np.int32)
    B, k = 16, 4096
    ppi = _tree_instance(pp, parent, weight)
    order, nxt, depth = ppi.preorder()
    geo = pp.pp_dp_geometry(ppi, B, k)
    assert geo["stack_levels_smem"] < depth, (geo, depth)
    profits = rng.integers(0, 1000, size=(B, n)).astype(np.int64)
    profits[:, rng.random(n) < 0.3] = 0
    budgets = rng.integers(k // 2, k + 1, size=B).astype(np.int32)
    outs = []
    for tune in [(0, 0), (8, 4)]:
        pp.pp_tune_dp(ppi, *tune, False, False)
        try:
            outs.append(_dp_batch(pp, ppi, profits, budgets, k))
        finally:
            pp.pp_tune_dp(ppi, 0, 0, False, False)
    np.testing.assert_array_equal(outs[0][0], outs[1][0])
    np.testing.assert_array_equal(outs[0][1], outs[1][1])
    for b in (0, 7, 15):
        ob, oc = oracle_lib.rooted_dp(parent, weight, profits[b], int(budgets[b]))
        assert int(outs[0][0][b]) == ob
        np.testing.assert_array_equal(outs[0][1][b], oc)
    ppi.close()


@pytest.mark.parametrize("cfg", [1, 2])
def test_plan_per_start_streams_match_lockstep(pp, cfg):
    """The per-start-stream schedule (each start on its own stream, never
    waiting for a slower one) and the lock-step schedule (one batched launch
    per step) give the same plan, statistics included."""
    inst = wl.make(cfg)
    with pp.Instance.from_workload(inst) as ppi:
        a = pp.pp_plan_run(ppi, inst.starts, None, inst.rounds, schedule=2)
        b = pp.pp_plan_run(ppi, inst.starts, None, inst.rounds, schedule=1)
        with pytest.raises(pp.PPError):
            pp.pp_plan_run(ppi, inst.starts, None, inst.rounds, schedule=3)
    assert (a.schedule, b.schedule) == (2, 1)
    assert a.objective == b.objective and a.best_start == b.best_start
    np.testing.assert_array_equal(a.placement, b.placement)
    np.testing.assert_array_equal(a.per_start_objective, b.per_start_objective)
    np.testing.assert_array_equal(a.per_start_sweeps, b.per_start_sweeps)
    np.testing.assert_array_equal(a.per_start_accepted, b.per_start_accepted)
    assert (a.dp_count, a.dp_cells, a.dp_rows_swept) == (b.dp_count, b.dp_cells, b.dp_rows_swept)


def test_plan_16_starts_with_stack_spill(pp, oracle_lib):
    """16 starts on a tree whose skip-row stack spills out of shared memory:
    the per-start schedule (one stack slot per start, each start's DP CTAs
    reserving more than half an SM) and lock step give the oracle's plan."""
    rng = np.random.default_rng(1616)
    parent = [-1]
    spine = 0
    for _ in range(70):                 # a spine whose nodes also have a leaf child: stack ~70 deep
        nxt = len(parent)
        parent.append(spine)
        parent.append(spine)
        spine = nxt
    for _ in range(4000):
        parent.append(int(rng.integers(len(parent))))
    parent = np.asarray(parent, np.int32)
    n, W, S, k = len(parent), 4, 16, 4096
    base = wl.random_small(rng, n, W, 0, k_max=1, w_max=1, demand_max=30)
    inst = wl.Instance("deep16", n, W, parent, np.ones(n, np.int32), base.demand,
                       rng.integers(1000, 90000, size=(W, n)).astype(np.int64),
                       rng.integers(500, 60000, size=(W, n)).astype(np.int64), 0,
                       np.full(W, k, np.int32), S, 2)
    o = oracle_lib.plan(oracle_lib.Problem.from_instance(inst), S, 2, safeguards=False)
    with pp.Instance.from_workload(inst) as ppi:
        order, nxt, depth = ppi.preorder()
        assert pp.pp_dp_geometry(ppi, S, k)["stack_levels_smem"] < depth
        a = pp.pp_plan_run(ppi, S, None, 2, safeguards=False, schedule=2)
        assert pp.pp_dp_stack_bytes(ppi) > 0
        b = pp.pp_plan_run(ppi, S, None, 2, safeguards=False, schedule=1)
    assert (a.schedule, b.schedule) == (2, 1)
    for g in (a, b):
        assert g.objective == o.objective and g.best_start == o.best_start
        np.testing.assert_array_equal(g.placement, o.placement)
        np.testing.assert_array_equal(g.per_start_objective, o.per_start_objective)
        np.testing.assert_array_equal(g.per_start_sweeps, o.per_start_sweeps)
        np.testing.assert_array_equal(g.per_start_accepted, o.per_start_accepted)


def test_plan_paper_scale_properties(pp, oracle_lib):
    """The n=50,000 / 16-worker / 16-start plan the benchmark times: every
    target prefix-complete and within budget, objective equal to the oracle's
    evaluation of the returned placement, best-of-starts, and (for the returned
    start, when it converged) no worker can strictly improve (Section IV-C)."""
    inst = wl.make(3)
    prob = oracle_lib.Problem.from_instance(inst)
    with pp.Instance.from_workload(inst) as ppi:
        g = pp.pp_plan_run(ppi, inst.starts, None, inst.rounds)
    for m in range(inst.W):
        assert bf.is_parent_closed(inst.parent, g.placement[m])
        assert int(inst.weight[g.placement[m].astype(bool)].sum()) <= inst.budget[m]
    assert oracle_lib.objective(prob, g.placement) == g.objective
    assert g.objective == g.per_start_objective.max()
    assert np.all(g.per_start_sweeps <= inst.rounds)
    if g.per_start_sweeps[g.best_start] < inst.rounds:
        for h in range(inst.W):
            best, p, _ = oracle_lib.worker_update(prob, h, g.placement)
            assert best <= int(p[g.placement[h].astype(bool)].sum())


def test_degenerate_instances(pp, oracle_lib):
    """n = 0, W = 1, every budget 0, a single chunk."""
    for n, W, k in [(0, 2, 5), (1, 1, 1), (5, 3, 0), (1, 32, 3)]:
        rng = np.random.default_rng(n * 10 + W)
        inst = wl.random_small(rng, n, W, 1, k_max=k) if n else wl.Instance(
            "empty", 0, W, np.zeros(0, np.int32), np.zeros(0, np.int32), np.zeros((W, 0), np.int64),
            np.zeros((W, 0), np.int64), np.zeros((W, W, 0), np.int64), 1, np.full(W, k, np.int32), 1, 1)
        if k == 0:
            inst.budget[:] = 0
        with pp.Instance.from_workload(inst) as ppi:
            g = pp.pp_plan_run(ppi, 2, None, 2)
        assert g.placement.shape == (W, n)
        if n == 0 or k == 0:
            assert g.objective == 0 and g.placement.sum() == 0
        else:
            o = oracle_lib.plan(oracle_lib.Problem.from_instance(inst), 2, 2)
            _compare_plans(g, o)


def test_degenerate_safeguards_and_epoch_updates(pp, oracle_lib):
    """Requester-side n = 0, all budgets 0, one worker and one chunk: safeguard
    candidates, plans with them and epoch updates agree with the oracle."""
    for n, W, k in [(0, 2, 5), (1, 1, 1), (6, 3, 0), (1, 32, 3), (4, 1, 2)]:
        rng = np.random.default_rng(n * 7 + W)
        inst = wl.random_small(rng, n, W, 0, k_max=max(k, 1)) if n else wl.Instance(
            "empty", 0, W, np.zeros(0, np.int32), np.zeros(0, np.int32), np.zeros((W, 0), np.int64),
            np.zeros((W, 0), np.int64), np.zeros((W, 0), np.int64), 0, np.full(W, k, np.int32), 1, 1)
        if k == 0:
            inst.budget[:] = 0
        prob = oracle_lib.Problem.from_instance(inst)
        old = np.zeros((W, n), np.uint8)
        with pp.Instance.from_workload(inst) as ppi:
            gpl, gobj = pp.pp_safeguards(ppi)
            g = pp.pp_plan_run(ppi, 2, None, 2)
            r = pp.pp_replan(ppi, old, 2, 2, 30000, 30000)
        opl, oobj = oracle_lib.safeguards(prob)
        np.testing.assert_array_equal(gpl, opl)
        np.testing.assert_array_equal(gobj, oobj)
        _compare_plans(g, oracle_lib.plan(prob, 2, 2))
        o = oracle_lib.replan(prob, old, 2, 2, 30000, 30000)
        assert (r.incumbent_objective, r.new_objective, r.materialization_cost, r.break_even_requests,
                r.adopted) == (o.incumbent_objective, o.new_objective, o.materialization_cost,
                               o.break_even_requests, o.adopted)
        np.testing.assert_array_equal(r.placement, o.placement)


def test_device_bounds_errors(pp):
    """A budget above the declared bound and a worker id out of range are
    reported through the status word, not by faulting."""
    inst = wl.random_small(np.random.default_rng(7), 30, 3, 0)
    with pp.Instance.from_workload(inst) as ppi:
        prof = torch.ones((1, 30), dtype=torch.int64, device="cuda")
        best = torch.zeros(1, dtype=torch.int64, device="cuda")
        bits = torch.zeros(pp.pp_dp_bits_size(ppi, 1, 4) // 4, dtype=torch.int32, device="cuda")
        pp.pp_tree_dp(ppi, prof, _dev([9], np.int32), 4, best, bits)
        with pytest.raises(pp.PPError) as e:
            ppi.sync()
        assert e.value.status == pp.PP_EBOUNDS
        ppi.sync()                                    # the word was cleared
        out = torch.zeros((1, 30), dtype=torch.int64, device="cuda")
        pp.pp_marginals(ppi, _dev([5], np.int32), torch.zeros((1, 30), dtype=torch.int32, device="cuda"), out)
        with pytest.raises(pp.PPError) as e:
            ppi.sync()
        assert e.value.status == pp.PP_EBOUNDS
        with pytest.raises(pp.PPError):
            pp.pp_tree_dp(ppi, prof, _dev([1], np.int32), -1, best, bits)


def test_flat_kernel_for_heavy_chunks(pp, oracle_lib):
    """Chunk weights above 4 use the one-CTA kernel; same bits layout and traceback."""
    rng = np.random.default_rng(500)
    for n, wmax in [(400, 6), (1500, 9)]:
        inst = wl.random_small(rng, n, 1, 0, w_max=wmax)
        ppi = _tree_instance(pp, inst.parent, inst.weight)
        profits = rng.integers(0, 50, size=(3, n)).astype(np.int64)
        tw = int(inst.weight.sum())
        budgets = np.array([tw // 4, tw // 2 + 3, 1500], np.int32)
        best, chosen = _dp_batch(pp, ppi, profits, budgets, int(budgets.max()))
        for b in range(3):
            ob, oc = oracle_lib.rooted_dp(inst.parent, inst.weight, profits[b], int(budgets[b]))
            assert best[b] == ob
            np.testing.assert_array_equal(chosen[b], oc)


def test_bounded_wait_reports_timeout(pp, oracle_lib):
    """A chain warp that never publishes makes its neighbour's wait run out:
    the launch ends with PP_ETIMEOUT (no fault), and the next launch is exact."""
    rng = np.random.default_rng(600)
    n, k = 600, 1024
    inst = wl.random_small(rng, n, 1, 0)
    ppi = _tree_instance(pp, inst.parent, inst.weight)
    profits = rng.integers(0, 100, size=(1, n)).astype(np.int64)
    try:
        pp.pp_test_inject(1, 3)
        with pytest.raises(pp.PPError) as e:
            _dp_batch(pp, ppi, profits, np.array([k], np.int32), k)
        assert e.value.status == pp.PP_ETIMEOUT
    finally:
        pp.pp_test_inject(1, -1)
    best, chosen = _dp_batch(pp, ppi, profits, np.array([k], np.int32), k)
    ob, oc = oracle_lib.rooted_dp(inst.parent, inst.weight, profits[0], k)
    assert best[0] == ob
    np.testing.assert_array_equal(chosen[0], oc)


def test_default_orders_match_oracle(pp, oracle_lib):
    """pp_default_orders (used to split starts across processes) equals the
    oracle's start orders: standalone-score order, reverse, SplitMix64 shuffles."""
    for cfg in (0, 1):
        inst = wl.make(cfg)
        with pp.Instance.from_workload(inst) as ppi:
            for S in (1, 2, 7):
                np.testing.assert_array_equal(pp.pp_default_orders(ppi, S),
                                              oracle_lib.default_orders(oracle_lib.Problem.from_instance(inst), S))
