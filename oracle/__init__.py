"""CPU oracle for PrefixPlace -- TEST INFRASTRUCTURE, NOT PART OF THE PRODUCT.

A plain, slow restatement of the paper's planner (arXiv 2608.01655) in C
(``pp_oracle.c``), loaded through ctypes.  Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
this package.  It shares no code with the CUDA library and never imports it.

Passages followed (each C function names its own):
  * Section IV-A        preorder and next(i)
  * Lemma 1 / Eq. 4     requester-side objective F
  * Eq. 6               source-dependent objective F_pair
  * Eq. 10, Eq. 7       per-worker marginals (Prop. 1)
  * Eq. 9 / Theorem 1   RootedDP with backtracking
  * Algorithm 1         WorkerGreedy, coordinate refinement, starts
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pp_oracle.c")
_LIB = os.path.join(_HERE, "libpp_oracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, pthreads).  Returns the library path."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-Wall", "-shared", "-fPIC", "-pthread",
                               "-o", tmp, _SRC])
        os.replace(tmp, _LIB)
    return _LIB


class _Inst(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int32), ("W", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("parent", ctypes.c_void_p), ("weight", ctypes.c_void_p),
                ("demand", ctypes.c_void_p), ("recompute", ctypes.c_void_p),
                ("transfer", ctypes.c_void_p), ("budget", ctypes.c_void_p)]


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i32, i64 = ctypes.c_int32, ctypes.c_int64
        sig = {
            "or_preorder": (ctypes.c_int, [i32, P, P, P]),
            "or_objective_F": (i64, [P, P]),
            "or_objective_Fpair": (i64, [P, P]),
            "or_objective": (i64, [P, P]),
            "or_marginal": (None, [P, i32, P, P]),
            "or_rooted_dp": (i64, [i32, P, P, P, i32, P, ctypes.c_int]),
            "or_standalone": (ctypes.c_int, [P, P]),
            "or_default_orders": (ctypes.c_int, [P, i32, P]),
            "or_plan": (i32, [P, i32, P, i32, i32, P, P, P, P, P, P, ctypes.c_int, P]),
            "or_safeguards": (ctypes.c_int, [P, P, P]),
            "or_replan": (ctypes.c_int, [P, P, i32, P, i32, i64, i64, i32, ctypes.c_int, P, P]),
            "or_worker_update": (i64, [P, i32, P, P, P]),
            "or_splitmix64": (None, [ctypes.c_uint64, i32, P]),
        }
        for name, (res, args) in sig.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


class Problem:
    """Holds one planner instance in the layout the C oracle reads.

    parent [n] int32 (-1 = top level), weight [n] int32, demand / recompute
    [W][n] int64, transfer [W][n] (mode 0) or [W_src][W_req][n] (mode 1) int64,
    budget [W] int32.
    """

    def __init__(self, parent, weight, demand, recompute, transfer, mode, budget):
        self.parent = _c(parent, np.int32)
        self.weight = _c(weight, np.int32)
        self.demand = _c(demand, np.int64)
        self.recompute = _c(recompute, np.int64)
        self.transfer = _c(transfer, np.int64)
        self.budget = _c(budget, np.int32)
        self.mode = int(mode)
        self.n = int(self.parent.shape[0])
        self.W = int(self.budget.shape[0])
        self._s = _Inst(self.n, self.W, self.mode, self.parent.ctypes.data, self.weight.ctypes.data,
                        self.demand.ctypes.data, self.recompute.ctypes.data,
                        self.transfer.ctypes.data, self.budget.ctypes.data)

    @classmethod
    def from_instance(cls, inst):
        return cls(inst.parent, inst.weight, inst.demand, inst.recompute, inst.transfer,
                   inst.mode, inst.budget)

    @property
    def ref(self):
        return ctypes.byref(self._s)


def preorder(parent):
    parent = _c(parent, np.int32)
    n = parent.shape[0]
    order = np.zeros(max(n, 1), np.int32)
    nxt = np.zeros(max(n, 1), np.int32)
    rc = _load().or_preorder(n, _ptr(parent), _ptr(order), _ptr(nxt))
    if rc != 0:
        raise ValueError("parent array is not a forest")
    return order[:n], nxt[:n]


def objective(prob: Problem, placement) -> int:
    pl = _c(placement, np.uint8)
    return int(_load().or_objective(prob.ref, _ptr(pl)))


def objective_F(prob: Problem, placement) -> int:
    pl = _c(placement, np.uint8)
    return int(_load().or_objective_F(prob.ref, _ptr(pl)))


def objective_Fpair(prob: Problem, placement) -> int:
    pl = _c(placement, np.uint8)
    return int(_load().or_objective_Fpair(prob.ref, _ptr(pl)))


def marginal(prob: Problem, h: int, placement) -> np.ndarray:
    pl = _c(placement, np.uint8)
    out = np.zeros(max(prob.n, 1), np.int64)
    _load().or_marginal(prob.ref, int(h), _ptr(pl), _ptr(out))
    return out[:prob.n]


def rooted_dp(parent, weight, profit, k: int, variant: int = -1):
    """Eq. 9 DP + backtrack.  Returns (optimum, chosen[n] uint8 by node id)."""
    parent = _c(parent, np.int32)
    weight = _c(weight, np.int32)
    profit = _c(profit, np.int64)
    n = parent.shape[0]
    chosen = np.zeros(max(n, 1), np.uint8)
    best = _load().or_rooted_dp(n, _ptr(parent), _ptr(weight), _ptr(profit), int(k),
                                _ptr(chosen), int(variant))
    if best == np.iinfo(np.int64).min:
        raise ValueError("parent array is not a forest")
    return int(best), chosen[:n]


def standalone(prob: Problem) -> np.ndarray:
    out = np.zeros(prob.W, np.int64)
    if _load().or_standalone(prob.ref, _ptr(out)) != 0:
        raise ValueError("parent array is not a forest")
    return out


def splitmix64(seed: int, count: int) -> np.ndarray:
    """The first `count` outputs of the oracle's SplitMix64 from state `seed`."""
    out = np.zeros(max(count, 1), np.uint64)
    _load().or_splitmix64(int(seed), int(count), _ptr(out))
    return out[:count]


def default_orders(prob: Problem, S: int) -> np.ndarray:
    out = np.zeros((S, prob.W), np.int32)
    if _load().or_default_orders(prob.ref, int(S), _ptr(out)) != 0:
        raise ValueError("parent array is not a forest")
    return out


@dataclass
class PlanResult:
    placement: np.ndarray      # [W][n] uint8
    objective: int
    best_start: int
    per_start_objective: np.ndarray
    per_start_sweeps: np.ndarray
    per_start_accepted: np.ndarray
    cells: int
    safeguard_objective: np.ndarray | None = None   # [3] when the safeguards took part


def safeguards(prob: Problem):
    """Independent, Popularity and LocalDedup placements (requester-side only).

    Returns (placement [3][W][n] uint8, objective [3] int64)."""
    pl = np.zeros((3, prob.W, max(prob.n, 1)), np.uint8)
    obj = np.zeros(3, np.int64)
    r = _load().or_safeguards(prob.ref, _ptr(pl), _ptr(obj))
    if r == -2:
        raise ValueError("safeguard candidates are defined for the requester-side objective only")
    if r != 0:
        raise ValueError("parent array is not a forest")
    return pl[:, :, :prob.n].copy(), obj


def plan(prob: Problem, S: int, R: int, orders=None, threads: int | None = None,
         safeguards: bool = True) -> PlanResult:
    """Algorithm 1 over S starts and at most R refinement sweeps; with the
    requester-side objective the safeguard candidates join as indices S..S+2
    unless safeguards=False."""
    if threads is None:
        threads = min(S, os.cpu_count() or 1)
    pl = np.zeros((prob.W, max(prob.n, 1)), np.uint8)
    obj = ctypes.c_int64(0)
    per = np.zeros(S, np.int64)
    sw = np.zeros(S, np.int32)
    acc = np.zeros(S, np.int32)
    cells = ctypes.c_int64(0)
    op = None
    if orders is not None:
        orders = _c(orders, np.int32)
        assert orders.shape == (S, prob.W)
        op = _ptr(orders)
    sg = np.zeros(3, np.int64)
    best = _load().or_plan(prob.ref, int(S), op, int(R), int(threads), _ptr(pl), ctypes.byref(obj),
                           _ptr(per), _ptr(sw), _ptr(acc), ctypes.byref(cells), int(bool(safeguards)),
                           _ptr(sg))
    if best < 0:
        raise ValueError("parent array is not a forest")
    used = bool(safeguards) and prob.mode == 0
    return PlanResult(pl[:, :prob.n].copy(), int(obj.value), int(best), per, sw, acc, int(cells.value),
                      sg if used else None)


@dataclass
class ReplanResult:
    placement: np.ndarray      # [W][n] uint8, the adopted target
    incumbent_objective: int
    new_objective: int
    materialization_cost: int
    break_even_requests: int   # -1 without a gain
    adopted: bool


def replan(prob: Problem, incumbent, S: int, R: int, epoch_requests: int, horizon_requests: int,
           orders=None, threads: int | None = None, safeguards: bool = True) -> ReplanResult:
    """Epoch update with the amortisation rule (Section IV-D, RQ5)."""
    if threads is None:
        threads = min(S, os.cpu_count() or 1)
    inc = _c(incumbent, np.uint8)
    assert inc.shape == (prob.W, prob.n)
    pl = np.zeros((prob.W, max(prob.n, 1)), np.uint8)
    out = np.zeros(5, np.int64)
    op = None
    if orders is not None:
        orders = _c(orders, np.int32)
        op = _ptr(orders)
    r = _load().or_replan(prob.ref, _ptr(inc), int(S), op, int(R), int(epoch_requests), int(horizon_requests),
                          int(threads), int(bool(safeguards)), _ptr(pl), _ptr(out))
    if r != 0:
        raise ValueError("parent array is not a forest")
    return ReplanResult(pl[:, :prob.n].copy(), int(out[0]), int(out[1]), int(out[2]), int(out[3]), bool(out[4]))


def worker_update(prob: Problem, h: int, placement):
    """Marginals of worker h against `placement`, then RootedDP.

    Returns (optimum, profit[n], chosen[n])."""
    pl = _c(placement, np.uint8)
    profit = np.zeros(max(prob.n, 1), np.int64)
    chosen = np.zeros(max(prob.n, 1), np.uint8)
    best = _load().or_worker_update(prob.ref, int(h), _ptr(pl), _ptr(profit), _ptr(chosen))
    return int(best), profit[:prob.n], chosen[:prob.n]
