"""The allocation-free DP entry point gives exactly what pp_tree_dp gives.

pp_tree_dp_noalloc serves callers that cannot let the planner allocate device
memory mid-run (a latency-bound serving loop, or a process whose memory is
owned by its own caching allocator).  It keeps the skip-row stack levels that
do not fit in shared memory in a fixed 16 MiB device array.  These checks
compare it with pp_tree_dp on launches that really spill stack levels to that
array, twice in a row (the second call must not be disturbed by what the
first left in the array), and check the size limit.  This file sorts last so
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
    pp.pp_tune_dp(*tune)
    try:
        ppi = _instance(pp, parent, weight, k)
        order, nxt, depth = ppi.preorder()
        geo = pp.pp_dp_geometry(ppi, 2, k)
        assert geo["stack_levels_smem"] < depth, (geo, depth)      # the fixed array is really used
        budgets = np.array([k, k // 2 + 5], np.int32)
        for call in range(2):
            profits = rng.integers(0, 1000, size=(2, len(parent))).astype(np.int64)
            profits[:, rng.random(len(parent)) < 0.3] = 0
            ref = _run(pp, ppi, pp.pp_tree_dp, profits, budgets, k)
            got = _run(pp, ppi, pp.pp_tree_dp_noalloc, profits, budgets, k)
            if call == 0:                   # the spilling launch against the oracle itself
                for b in range(2):
                    ob, oc = oracle_lib.rooted_dp(parent, weight, profits[b], int(budgets[b]))
                    assert int(ref[0][b]) == ob
                    np.testing.assert_array_equal(ref[2][b], oc)
            np.testing.assert_array_equal(got[0], ref[0])
            np.testing.assert_array_equal(got[1], ref[1])
            np.testing.assert_array_equal(got[2], ref[2])
        ppi.close()
    finally:
        pp.pp_tune_dp(0, 0, False, False)


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
