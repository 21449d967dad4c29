"""The allocation-free DP entry point gives exactly what pp_tree_dp gives.

pp_tree_dp_noalloc serves callers that cannot let the planner allocate device
memory mid-run (a latency-bound serving loop, or a process whose memory is
owned by its own caching allocator).  It keeps the skip-row stack levels that
do not fit in shared memory in a fixed 16 MiB device array.  These checks
compare it with pp_tree_dp on launches that really spill stack levels to that
array, twice in a row (the second call must not be disturbed by what the
first left in the array), that the call leaves the instance without stack
scratch of its own, that a batch pp_tree_dp would split runs as one launch
with the same results, and check the size limit.  This file sorts last so
that a run stopping at the first failure has run every other test before it.
"""
import numpy as np
import pytest

from paper_2608_01655_gb300 import workloads as wl

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


def _deep_stack_tree(rng, depth, extra, w_max):
    """A spine whose every node's last child is a leaf: each level keeps one
    more pending skip row, so the skip-row stack is about `depth` deep."""
    parent = [-1]
    spine = 0
    for _ in range(depth):
        nxt = len(parent)
        parent.append(spine)            # next spine node: the smaller id, visited first
        parent.append(spine)            # a leaf: the last child of the spine node
        spine = nxt
    for _ in range(extra):
        parent.append(int(rng.integers(len(parent))))
    n = len(parent)
    return np.asarray(parent, np.int32), rng.integers(1, w_max + 1, size=n).astype(np.int32)


def _instance(pp, parent, weight, k):
    n = len(parent)
    inst = wl.Instance("deep", n, 1, parent, weight, np.ones((1, n), np.int64), np.ones((1, n), np.int64),
                       np.ones((1, n), np.int64), 0, np.array([k], np.int32), 1, 1)
    return pp.Instance.from_workload(inst)


def _run(pp, ppi, fn, profits, budgets, k):
    B, n = profits.shape
    prof = torch.from_numpy(profits).cuda()
    bud = torch.from_numpy(budgets).cuda()
    best = torch.zeros(B, dtype=torch.int64, device="cuda")
    bits = torch.zeros(pp.pp_dp_bits_size(ppi, B, k) // 4, dtype=torch.int32, device="cuda")
    chosen = torch.zeros((B, n), dtype=torch.uint8, device="cuda")
    fn(ppi, prof, bud, k, best, bits)
    pp.pp_traceback(ppi, bits, bud, k, chosen)
    ppi.sync()
    return best.cpu().numpy(), bits.cpu().numpy(), chosen.cpu().numpy()


@pytest.mark.parametrize("w_max,tune", [(6, (0, 0)), (1, (1, 8))])
def test_noalloc_matches_tree_dp_twice(pp, oracle_lib, w_max, tune):
    rng = np.random.default_rng(900 + w_max)
    parent, weight = _deep_stack_tree(rng, 60, 3000, w_max)
    k = 4096
    ppi = _instance(pp, parent, weight, k)
    pp.pp_tune_dp(ppi, *tune)
    order, nxt, depth = ppi.preorder()
    geo = pp.pp_dp_geometry(ppi, 2, k)
    assert geo["stack_levels_smem"] < depth, (geo, depth)      # the fixed array is really used
    budgets = np.array([k, k // 2 + 5], np.int32)
    for call in range(2):
        profits = rng.integers(0, 1000, size=(2, len(parent))).astype(np.int64)
        profits[:, rng.random(len(parent)) < 0.3] = 0
        # on the fresh instance the allocation-free call runs first: it must
        # leave the instance without stack scratch of its own
        got = _run(pp, ppi, pp.pp_tree_dp_noalloc, profits, budgets, k)
        if call == 0:
            assert pp.pp_dp_stack_bytes(ppi) == 0
        ref = _run(pp, ppi, pp.pp_tree_dp, profits, budgets, k)
        assert pp.pp_dp_stack_bytes(ppi) > 0                 # pp_tree_dp spilled to its own scratch
        if call == 0:                   # the spilling launch against the oracle itself
            for b in range(2):
                ob, oc = oracle_lib.rooted_dp(parent, weight, profits[b], int(budgets[b]))
                assert int(got[0][b]) == ob
                np.testing.assert_array_equal(got[2][b], oc)
        np.testing.assert_array_equal(got[0], ref[0])
        np.testing.assert_array_equal(got[1], ref[1])
        np.testing.assert_array_equal(got[2], ref[2])
    ppi.close()


def test_noalloc_runs_a_split_geometry_as_one_launch(pp, oracle_lib):
    """A batch that pp_tree_dp splits into two concurrent launches (16 items:
    15 on clusters of 8 CTAs, one on a narrower cluster beside them) runs as
    one launch in the allocation-free call; values, decision bits and chosen
    sets are the same.  (A split is only chosen when the wide clusters' stack
    fits in less than half an SM's shared memory, so it never spills.)"""
    if torch.cuda.get_device_properties(0).multi_processor_count != 152:
        pytest.skip("the split is sized for a 152-SM GB300")
    inst = wl.make(3)
    rng = np.random.default_rng(961)
    B, k = 16, int(inst.budget[0])
    n = inst.n
    ppi = _instance(pp, inst.parent, inst.weight, k)
    assert pp.pp_dp_split(ppi, B, k)["wide_items"] > 0
    profits = rng.integers(0, 10 ** 6, size=(B, n)).astype(np.int64)
    profits[:, rng.random(n) < 0.5] = 0
    budgets = rng.integers(k // 2, k + 1, size=B).astype(np.int32)
    for call in range(2):
        got = _run(pp, ppi, pp.pp_tree_dp_noalloc, profits, budgets, k)
        ref = _run(pp, ppi, pp.pp_tree_dp, profits, budgets, k)
        np.testing.assert_array_equal(got[0], ref[0])
        np.testing.assert_array_equal(got[1], ref[1])
        np.testing.assert_array_equal(got[2], ref[2])
        if call == 0:
            for b in (0, B - 1):
                ob, oc = oracle_lib.rooted_dp(inst.parent, inst.weight, profits[b], int(budgets[b]))
                assert int(got[0][b]) == ob
                np.testing.assert_array_equal(got[2][b], oc)
        profits = profits[::-1].copy()
    ppi.close()


def test_noalloc_rejects_oversized_launch(pp):
    rng = np.random.default_rng(950)
    parent, weight = _deep_stack_tree(rng, 60, 3000, 6)
    k = 4096
    ppi = _instance(pp, parent, weight, k)
    B = 64                                  # 64 * (levels beyond shared memory) * 4096 * 8 B > 16 MiB
    prof = torch.zeros((B, len(parent)), dtype=torch.int64, device="cuda")
    bud = torch.full((B,), k, dtype=torch.int32, device="cuda")
    best = torch.zeros(B, dtype=torch.int64, device="cuda")
    bits = torch.zeros(pp.pp_dp_bits_size(ppi, B, k) // 4, dtype=torch.int32, device="cuda")
    with pytest.raises(pp.PPError) as e:
        pp.pp_tree_dp_noalloc(ppi, prof, bud, k, best, bits)
    assert e.value.status == pp.PP_EINVAL and "16777216" in str(e.value)
    ppi.sync()
    ppi.close()
