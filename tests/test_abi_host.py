"""CPU checks of the C-ABI library: it loads, exports every declared entry
point, and its host-side logic (validation, preorder, skip-row stack plan)
is right.  No call here reaches a CUDA kernel."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2608_01655_gb300 import build as ppbuild
from paper_2608_01655_gb300 import workloads as wl
from tests import bruteforce as bf

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    ppbuild.build()
    from paper_2608_01655_gb300 import binding
    return binding


def _declared(header):
    txt = open(os.path.join(ROOT, "include", header)).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return set(re.findall(r"\b(pp_\w+)\s*\(", txt))


def test_library_exports_every_declared_symbol(lib):
    """Every entry point of include/prefixplace.h is exported by
    libprefixplace.so, and the benchmark probe of include/pp_probe.h by
    libpp_probe.so (and not by the planner's library)."""
    headers = sorted(f for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h"))
    assert headers == ["pp_probe.h", "prefixplace.h"]
    declared = _declared("prefixplace.h")
    assert len(declared) >= 12
    so = ctypes.CDLL(lib.LIB_PATH)
    missing = [n for n in sorted(declared) if not hasattr(so, n)]
    assert not missing, missing
    probe = ctypes.CDLL(ppbuild.PROBE_LIB)
    assert _declared("pp_probe.h") == {"pp_probe_read"}
    assert hasattr(probe, "pp_probe_read") and not hasattr(so, "pp_probe_read")


def _create(lib, **kw):
    inst = wl.random_small(np.random.default_rng(0), 6, 2, 0)
    args = dict(n=inst.n, W=inst.W, parent=inst.parent, weight=inst.weight, demand=inst.demand,
                recompute=inst.recompute, transfer=inst.transfer, mode=0, budget=inst.budget)
    args.update(kw)
    a = {k: (np.ascontiguousarray(v) if isinstance(v, np.ndarray) else v) for k, v in args.items()}
    h = ctypes.c_void_p()
    P = lambda x: x.ctypes.data_as(ctypes.c_void_p)
    st = lib._lib.pp_instance_create(a["n"], a["W"], P(a["parent"].astype(np.int32)),
                                     P(a["weight"].astype(np.int32)), P(a["demand"].astype(np.int64)),
                                     P(a["recompute"].astype(np.int64)), P(a["transfer"].astype(np.int64)),
                                     a["mode"], P(a["budget"].astype(np.int32)), None, ctypes.byref(h))
    return st


def test_create_validation_is_host_side(lib):
    """Invalid instances are rejected before any CUDA call (Section III-A
    feasibility data: a forest, weights >= 1, non-negative demand and costs)."""
    assert _create(lib, parent=np.array([1, 2, 0, -1, -1, -1], np.int32)) == lib.PP_ENOTTREE
    assert _create(lib, parent=np.array([0, -1, -1, -1, -1, -1], np.int32)) == lib.PP_ENOTTREE
    assert _create(lib, parent=np.array([9, -1, -1, -1, -1, -1], np.int32)) == lib.PP_ENOTTREE
    assert _create(lib, weight=np.array([1, 0, 1, 1, 1, 1], np.int32)) == lib.PP_EINVAL
    dem = np.ones((2, 6), np.int64)
    dem[1, 3] = -1
    assert _create(lib, demand=dem) == lib.PP_EINVAL
    assert _create(lib, W=0, budget=np.zeros(0, np.int32)) == lib.PP_EINVAL
    assert _create(lib, W=33, budget=np.zeros(33, np.int32)) == lib.PP_EINVAL
    assert _create(lib, mode=2) == lib.PP_EINVAL
    assert _create(lib, budget=np.array([1, -1], np.int32)) == lib.PP_EINVAL
    big = np.full((2, 6), 1 << 30, np.int64)       # 12 products of 2^60 > 2^62
    assert _create(lib, demand=big, recompute=big) == lib.PP_EOVERFLOW
    assert "2^62" in lib.last_error()
    # the Popularity safeguard's DP values (profit Lambda) stay bounded even
    # where w = 0 makes every Lambda * w vanish
    huge = np.full((2, 6), 1 << 59, np.int64)      # 12 x 2^59 > 2^62
    assert _create(lib, demand=huge, recompute=np.zeros((2, 6), np.int64)) == lib.PP_EOVERFLOW
    assert "sum of demand" in lib.last_error()
    # the epoch update's one-time cost (one w per newly held (m, b)) stays
    # bounded even where Lambda = 0
    assert _create(lib, demand=np.zeros((2, 6), np.int64), recompute=huge) == lib.PP_EOVERFLOW
    assert "recompute" in lib.last_error()
    # just inside every bound: accepted up to the CUDA part of the call
    edge = np.full((2, 6), (1 << 62) // 12, np.int64)
    st = _create(lib, demand=edge, recompute=np.zeros((2, 6), np.int64))
    assert st != lib.PP_EOVERFLOW


def test_create_validation_large_and_extreme(lib):
    """The cost arrays' checks hold where they are split over host threads
    (W^2 n transfer costs above 2^20 values) and where the sum of products
    would leave every 128-bit range (products near 2^126)."""
    top = np.full((2, 6), (1 << 63) - 1, np.int64)
    assert _create(lib, demand=top, recompute=top) == lib.PP_EOVERFLOW
    W, n = 16, 4096
    base = dict(n=n, W=W, parent=np.full(n, -1, np.int32), weight=np.ones(n, np.int32),
                demand=np.ones((W, n), np.int64), recompute=np.ones((W, n), np.int64),
                transfer=np.ones((W, W, n), np.int64), mode=1, budget=np.full(W, 8, np.int32))
    tr = base["transfer"].copy()
    tr[W - 1, W - 2, n - 3] = -5                     # in the last thread's slice
    assert _create(lib, **{**base, "transfer": tr}) == lib.PP_EINVAL
    assert "transfer" in lib.last_error()
    dem = base["demand"].copy()
    dem[W // 2, n // 2] = -1
    assert _create(lib, **{**base, "demand": dem}) == lib.PP_EINVAL
    assert "demand" in lib.last_error()
    # the tree's tables are built while the costs are checked: a cost error
    # is still the one reported when the tree is bad as well
    cyc = base["parent"].copy()
    cyc[:3] = [1, 2, 0]
    assert _create(lib, **{**base, "parent": cyc}) == lib.PP_ENOTTREE
    assert _create(lib, **{**base, "parent": cyc, "demand": dem}) == lib.PP_EINVAL
    assert "demand" in lib.last_error()
    # every slice's partial sum is below 2^62, their total above
    spread = np.full((W, n), (1 << 62) // (W * n // 2), np.int64)
    assert _create(lib, **{**base, "demand": spread, "recompute": np.zeros((W, n), np.int64)}) == lib.PP_EOVERFLOW
    assert "sum of demand" in lib.last_error()


def test_row_plan_preorder_matches_definition(lib):
    """The library's preorder (independent of the oracle's) follows Section IV-A."""
    rng = np.random.default_rng(2)
    for trial in range(40):
        inst = wl.random_small(rng, int(rng.integers(1, 60)), 1, 0)
        order, nxt, skip, push, depth = lib.pp_row_plan(inst.parent)
        assert list(order) == bf.preorder_positions(inst.parent)
        size = {v: 1 for v in range(inst.n)}
        for v in reversed(order):
            if inst.parent[v] >= 0:
                size[inst.parent[v]] += size[v]
        assert list(nxt) == [i + size[v] for i, v in enumerate(order)]
    with pytest.raises(lib.PPError):
        lib.pp_row_plan(np.array([1, 0], np.int32))


def _row_stack_dp(parent, weight, profit, k, plan):
    """Eq. 9 swept exactly as the kernel does, driven by the row plan:
    registers hold row i+1, the skip branch reads the code's source."""
    order, nxt, skip, push, depth = plan
    n = len(order)
    cur = np.zeros(k + 1, np.int64)
    stack = [None] * max(depth, 1)
    for i in range(n - 1, -1, -1):
        b = order[i]
        s = cur.copy() if skip[i] == -1 else (np.zeros(k + 1, np.int64) if skip[i] == -2 else stack[skip[i]].copy())
        new = s.copy()
        w = weight[b]
        for j in range(1, k + 1):
            if j >= w:
                t = profit[b] + cur[j - w]
                if t > s[j]:
                    new[j] = t
        new[0] = 0
        cur = new
        if push[i] >= 0:
            stack[push[i]] = cur.copy()
    return int(cur[k])


def test_row_plan_reproduces_the_dp(lib, oracle_lib):
    """The skip-row stack plan feeds every row exactly the D[next(i)] of Eq. 9."""
    rng = np.random.default_rng(3)
    for trial in range(40):
        n = int(rng.integers(1, 50))
        inst = wl.random_small(rng, n, 1, 0, w_max=3)
        profit = rng.integers(0, 20, size=n).astype(np.int64)
        k = int(rng.integers(0, 12))
        plan = lib.pp_row_plan(inst.parent)
        best, _ = oracle_lib.rooted_dp(inst.parent, inst.weight, profit, k)
        assert _row_stack_dp(inst.parent, inst.weight, profit, k, plan) == best


def test_row_plan_stack_depth_on_workloads(lib):
    """The stack stays shallow on the workload trees (depth <= tree depth)."""
    for cfg in (0, 1, 3):
        inst = wl.make(cfg)
        order, nxt, skip, push, depth = lib.pp_row_plan(inst.parent)
        assert 1 <= depth <= inst.profile["max_depth"] + 1
        # every stack read is preceded by a push to that level
        live = set()
        for i in range(inst.n - 1, -1, -1):
            if skip[i] >= 0:
                assert skip[i] in live
            if push[i] >= 0:
                live.add(push[i])


def _register_dp(parent, weight, profit, k, order, code):
    """Eq. 9 swept with the register-resident plan: `cur` is row i+1, `top`
    the stack top (zero row when empty), saved levels in a list."""
    n = len(order)
    cur = np.zeros(k + 1, np.int64)
    top = np.zeros(k + 1, np.int64)
    levels = {}
    for i in range(n - 1, -1, -1):
        c = int(code[i])
        w = (c & 7) + 1
        kind = (c >> 3) & 3
        assert w == min(int(weight[order[i]]), 8)
        s = cur.copy() if kind == 0 else top.copy()
        assert kind in (0, 2)
        new = s.copy()
        for j in range(1, k + 1):
            if j >= w and profit[order[i]] + cur[j - w] > s[j]:
                new[j] = profit[order[i]] + cur[j - w]
        cur = new
        lvl = (c >> 16) & 0xFFFF
        if c & (1 << 6):
            levels[lvl] = cur.copy()
            top = cur.copy()
        elif c & (1 << 5):
            top = levels[lvl].copy()
        elif c & (1 << 7):
            top = np.zeros(k + 1, np.int64)
    return int(cur[k])


def test_register_row_plan_reproduces_the_dp(lib, oracle_lib):
    """The register-resident plan (stack top in registers, zero row as the
    empty stack's top) feeds every row the D[next(i)] of Eq. 9."""
    rng = np.random.default_rng(4)
    for trial in range(60):
        n = int(rng.integers(1, 60))
        inst = wl.random_small(rng, n, 1, 0, w_max=3)
        profit = rng.integers(0, 20, size=n).astype(np.int64)
        k = int(rng.integers(0, 14))
        order, *_ = lib.pp_row_plan(inst.parent)
        code = lib.pp_row_plan_registers(inst.parent, inst.weight)
        best, _ = oracle_lib.rooted_dp(inst.parent, inst.weight, profit, k)
        assert _register_dp(inst.parent, inst.weight, profit, k, order, code) == best, trial
