"""Thin ctypes binding of libprefixplace.so (include/prefixplace.h).

Argument marshalling only: every step of the planner runs in the library's
CUDA kernels.  Device buffers are torch CUDA tensors (PyTorch provides device
memory and streams, nothing else); host buffers are numpy arrays.  If the
library has not been built, importing this module raises ImportError: there is
no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np

# The plan's per-start schedule puts each start on its own CUDA stream; the
# driver maps streams onto CUDA_DEVICE_MAX_CONNECTIONS hardware queues (8 by
# default), and streams sharing a queue wait on one another's launches.  The
# variable acts when the CUDA context is created, so it is set here, before
# that, unless the caller has chosen a value.
os.environ.setdefault("CUDA_DEVICE_MAX_CONNECTIONS", "32")

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libprefixplace.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with paper_2608_01655_gb300.build.build() "
                      "(there is no CPU fallback)")

_lib = ctypes.CDLL(LIB_PATH)
_P = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_st = ctypes.c_int

PP_OK, PP_EINVAL, PP_ENOTTREE, PP_EOVERFLOW, PP_ENOMEM, PP_ECUDA, PP_ETIMEOUT, PP_EBOUNDS = range(8)
STATUS_NAMES = ["PP_OK", "PP_EINVAL", "PP_ENOTTREE", "PP_EOVERFLOW", "PP_ENOMEM", "PP_ECUDA",
                "PP_ETIMEOUT", "PP_EBOUNDS"]
PP_TRANSFER_REQUESTER, PP_TRANSFER_SOURCE = 0, 1


class PPError(RuntimeError):
    def __init__(self, status: int, msg: str):
        self.status = status
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__(f"{name}: {msg}")


class PlanStats(ctypes.Structure):
    _fields_ = [("per_start_objective", _P), ("per_start_sweeps", _P), ("per_start_accepted", _P),
                ("orders_used", _P), ("best_start", _i32), ("dp_count", _i32), ("dp_cells", _i64),
                ("kernel_launches", _i32), ("dp_rows_swept", _i64), ("time_phases", _i32),
                ("phase_ms", ctypes.c_float * 3), ("dp_launches", _i32), ("no_safeguards", _i32),
                ("safeguard_objective", ctypes.c_int64 * 3), ("marginals", _i32), ("used_top2", _i32),
                ("schedule", _i32), ("hw_queues", _i32)]


_SIGS = {
    "pp_instance_create": [_i32, _i32, _P, _P, _P, _P, _P, _i32, _P, _P, ctypes.POINTER(_P)],
    "pp_instance_destroy": [_P],
    "pp_instance_preorder": [_P, _P, _P, _P],
    "pp_row_plan": [_i32, _P, _P, _P, _P, _P, _P],
    "pp_row_plan_registers": [_i32, _P, _P, _P],
    "pp_instance_sync": [_P, _P],
    "pp_marginals": [_P, _i32, _P, _P, _P, _P],
    "pp_tree_dp": [_P, _i32, _P, _P, _i32, _P, _P, _P],
    "pp_traceback": [_P, _i32, _P, _P, _i32, _P, _P],
    "pp_objective": [_P, _i32, _P, _P, _P],
    "pp_plan_run": [_P, _i32, _P, _i32, _P, _P, ctypes.POINTER(PlanStats), _P],
    "pp_test_inject": [_i32, _i32],
    "pp_dp_geometry": [_P, _i32, _i32, _P],
    "pp_dp_split": [_P, _i32, _i32, _P],
    "pp_tune_dp": [_P, _i32, _i32, _i32, _i32],
    "pp_tree_dp_noalloc": [_P, _i32, _P, _P, _i32, _P, _P, _P],
    "pp_dp_rows_swept": [_P, _i32, _i32, _P, _P, _P],
    "pp_dp_stack_bytes": [_P, ctypes.POINTER(ctypes.c_size_t)],
    "pp_default_orders": [_P, _i32, _P, _P],
    "pp_safeguards": [_P, _P, _P, _P],
    "pp_replan": [_P, _P, _i32, _P, _i32, _i64, _i64, _P, _P, _P, _P],
}
for _name, _args in _SIGS.items():
    _f = getattr(_lib, _name)
    _f.argtypes = _args
    _f.restype = _st
_lib.pp_dp_bits_size.argtypes = [_P, _i32, _i32]
_lib.pp_dp_bits_size.restype = ctypes.c_size_t
_lib.pp_last_error.argtypes = []
_lib.pp_last_error.restype = ctypes.c_char_p


def last_error() -> str:
    return _lib.pp_last_error().decode()


def _check(status: int):
    if status != PP_OK:
        raise PPError(status, last_error())


def _np(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _host(a):
    return a.ctypes.data_as(_P)


def _dev(t):
    """Device pointer of a contiguous CUDA tensor (None -> NULL)."""
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("expected a contiguous CUDA tensor")
    return _P(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return _P(stream.cuda_stream) if hasattr(stream, "cuda_stream") else _P(int(stream))


def pp_row_plan(parent):
    """Host-only preorder and skip-row stack plan.  Returns (order, next, skip_code, push_level, depth)."""
    parent = _np(parent, np.int32)
    n = parent.shape[0]
    outs = [np.zeros(max(n, 1), np.int32) for _ in range(4)]
    depth = _i32(0)
    _check(_lib.pp_row_plan(n, _host(parent), *[_host(o) for o in outs], ctypes.byref(depth)))
    return (*[o[:n] for o in outs], int(depth.value))


def pp_row_plan_registers(parent, weight):
    """Host-only per-row codes of the register-resident row plan (see the header)."""
    parent = _np(parent, np.int32)
    weight = _np(weight, np.int32)
    n = parent.shape[0]
    code = np.zeros(max(n, 1), np.int32)
    _check(_lib.pp_row_plan_registers(n, _host(parent), _host(weight), _host(code)))
    return code[:n]


class Instance:
    """Owns one pp_instance (pp_instance_create / pp_instance_destroy)."""

    def __init__(self, parent, weight, demand, recompute, transfer, mode, budget, stream=None):
        self.parent = _np(parent, np.int32)
        self.n = int(self.parent.shape[0])
        self.budget = _np(budget, np.int32)
        self.W = int(self.budget.shape[0])
        self.mode = int(mode)
        arrays = (self.parent, _np(weight, np.int32), _np(demand, np.int64), _np(recompute, np.int64),
                  _np(transfer, np.int64))
        h = _P()
        _check(_lib.pp_instance_create(self.n, self.W, *[_host(a) for a in arrays], self.mode,
                                       _host(self.budget), _stream(stream), ctypes.byref(h)))
        self._h = h

    @classmethod
    def from_workload(cls, inst, stream=None):
        return cls(inst.parent, inst.weight, inst.demand, inst.recompute, inst.transfer, inst.mode,
                   inst.budget, stream)

    @property
    def handle(self):
        if self._h is None:
            raise RuntimeError("instance destroyed")
        return self._h

    def close(self):
        if getattr(self, "_h", None) is not None:
            _lib.pp_instance_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def preorder(self):
        order = np.zeros(max(self.n, 1), np.int32)
        nxt = np.zeros(max(self.n, 1), np.int32)
        depth = _i32(0)
        _check(_lib.pp_instance_preorder(self.handle, _host(order), _host(nxt), ctypes.byref(depth)))
        return order[:self.n], nxt[:self.n], int(depth.value)

    def sync(self, stream=None):
        _check(_lib.pp_instance_sync(self.handle, _stream(stream)))


def pp_marginals(inst: Instance, worker, holder_mask, profit, stream=None):
    """worker [B] int32, holder_mask [B][n] int32 (bit pattern), profit [B][n] int64: CUDA tensors."""
    _check(_lib.pp_marginals(inst.handle, int(worker.shape[0]), _dev(worker), _dev(holder_mask),
                             _dev(profit), _stream(stream)))


def pp_dp_bits_size(inst: Instance, batch: int, max_budget: int) -> int:
    return int(_lib.pp_dp_bits_size(inst.handle, int(batch), int(max_budget)))


def pp_tree_dp(inst: Instance, profit, budget, max_budget: int, best, bits, stream=None):
    _check(_lib.pp_tree_dp(inst.handle, int(budget.shape[0]), _dev(profit), _dev(budget),
                           int(max_budget), _dev(best), _dev(bits), _stream(stream)))


def pp_tree_dp_noalloc(inst: Instance, profit, budget, max_budget: int, best, bits, stream=None):
    """pp_tree_dp without device allocation (fixed 16 MiB stack scratch per device)."""
    _check(_lib.pp_tree_dp_noalloc(inst.handle, int(budget.shape[0]), _dev(profit), _dev(budget),
                                   int(max_budget), _dev(best), _dev(bits), _stream(stream)))


def pp_dp_rows_swept(inst: Instance, batch: int, max_budget: int, bits, stream=None) -> np.ndarray:
    """Rows each item of the last DP on `bits` swept after pruning."""
    rows = np.zeros(max(int(batch), 1), np.int32)
    _check(_lib.pp_dp_rows_swept(inst.handle, int(batch), int(max_budget), _dev(bits), _host(rows),
                                 _stream(stream)))
    return rows[:int(batch)]


def pp_traceback(inst: Instance, bits, budget, max_budget: int, chosen, stream=None):
    _check(_lib.pp_traceback(inst.handle, int(budget.shape[0]), _dev(bits), _dev(budget),
                             int(max_budget), _dev(chosen), _stream(stream)))


def pp_objective(inst: Instance, chosen, obj, stream=None):
    """chosen [B][W][n] uint8, obj [B] int64: CUDA tensors."""
    _check(_lib.pp_objective(inst.handle, int(obj.shape[0]), _dev(chosen), _dev(obj), _stream(stream)))


@dataclass
class PlanResult:
    placement: np.ndarray
    objective: int
    best_start: int
    per_start_objective: np.ndarray
    per_start_sweeps: np.ndarray
    per_start_accepted: np.ndarray
    orders: np.ndarray
    dp_count: int
    dp_cells: int
    kernel_launches: int
    phase_ms: tuple = ()
    dp_rows_swept: int = 0
    dp_launches: int = 0
    safeguard_objective: tuple = ()     # Independent, Popularity, LocalDedup (requester-side)
    used_top2: bool = False             # source-dependent marginals from top-2 holder tables
    schedule: int = 0                   # 1 lock step, 2 per-start streams
    hw_queues: int = 0                  # hardware queues the automatic schedule assumed


def pp_plan_run(inst: Instance, n_starts: int, orders=None, max_rounds: int = 0, stream=None,
                time_phases: bool = False, safeguards: bool = True, marginals: int = 0,
                schedule: int = 0) -> PlanResult:
    """marginals (source-dependent): 0 automatic, 1 holder scan, 2 top-2 tables.
    schedule: 0 automatic, 1 lock step (one batched launch per step), 2 one
    stream per start; the results are identical."""
    S, W, n = int(n_starts), inst.W, inst.n
    placement = np.zeros((W, max(n, 1)), np.uint8)
    obj = _i64(0)
    per = np.zeros(S, np.int64)
    sw = np.zeros(S, np.int32)
    acc = np.zeros(S, np.int32)
    used = np.zeros((S, W), np.int32)
    st = PlanStats(per.ctypes.data, sw.ctypes.data, acc.ctypes.data, used.ctypes.data, 0, 0, 0, 0, 0,
                   int(bool(time_phases)))
    st.no_safeguards = int(not safeguards)
    st.marginals = int(marginals)
    st.schedule = int(schedule)
    op = None
    if orders is not None:
        orders = _np(orders, np.int32)
        if orders.shape != (S, W):
            raise ValueError("orders must be [n_starts][W]")
        op = _host(orders)
    _check(_lib.pp_plan_run(inst.handle, S, op, int(max_rounds), _host(placement), ctypes.byref(obj),
                            ctypes.byref(st), _stream(stream)))
    return PlanResult(placement[:, :n].copy(), int(obj.value), int(st.best_start), per, sw, acc, used,
                      int(st.dp_count), int(st.dp_cells), int(st.kernel_launches),
                      tuple(float(x) for x in st.phase_ms) if time_phases else (), int(st.dp_rows_swept),
                      int(st.dp_launches),
                      tuple(int(x) for x in st.safeguard_objective) if safeguards and inst.mode == 0 else (),
                      bool(st.used_top2), int(st.schedule), int(st.hw_queues))


def pp_test_inject(kind: int, value: int):
    """Testing hook: kind 1 makes chain warp `value` of later DP launches stop
    publishing its ring counter (-1 restores normal operation)."""
    _check(_lib.pp_test_inject(int(kind), int(value)))


def pp_dp_geometry(inst: Instance, batch: int, max_budget: int) -> dict:
    out = np.zeros(8, np.int32)
    _check(_lib.pp_dp_geometry(inst.handle, int(batch), int(max_budget), _host(out)))
    keys = ["wave", "cluster_ctas", "warps_per_cta", "columns_per_thread", "warps_per_dp",
            "stack_levels_smem", "smem_bytes", "kpad"]
    return {k: int(v) for k, v in zip(keys, out)}


def pp_dp_split(inst: Instance, batch: int, max_budget: int) -> dict:
    out = np.zeros(5, np.int32)
    _check(_lib.pp_dp_split(inst.handle, int(batch), int(max_budget), _host(out)))
    keys = ["wide_items", "narrow_cluster_ctas", "narrow_warps_per_cta", "narrow_stack_levels_smem",
            "wide_smem_bytes"]
    return {k: int(v) for k, v in zip(keys, out)}


def pp_tune_dp(inst: Instance, cluster_ctas: int = 0, columns_per_thread: int = 0, force_flat: bool = False,
               no_prune: bool = False):
    """Override this instance's DP launch shape (0 = automatic)."""
    _check(_lib.pp_tune_dp(inst.handle, int(cluster_ctas), int(columns_per_thread), int(bool(force_flat)),
                           int(bool(no_prune))))


def pp_dp_stack_bytes(inst: Instance) -> int:
    """Bytes of skip-row stack scratch the instance holds (0 before any spilling launch)."""
    out = ctypes.c_size_t(0)
    _check(_lib.pp_dp_stack_bytes(inst.handle, ctypes.byref(out)))
    return int(out.value)


def pp_default_orders(inst: Instance, n_starts: int, stream=None) -> np.ndarray:
    """The start orders pp_plan_run uses when given none: [n_starts][W] int32."""
    out = np.zeros((int(n_starts), inst.W), np.int32)
    _check(_lib.pp_default_orders(inst.handle, int(n_starts), _host(out), _stream(stream)))
    return out


def pp_safeguards(inst: Instance, stream=None):
    """Independent, Popularity, LocalDedup placements [3][W][n] uint8 and objectives [3] int64."""
    pl = np.zeros((3, inst.W, max(inst.n, 1)), np.uint8)
    obj = np.zeros(3, np.int64)
    _check(_lib.pp_safeguards(inst.handle, _host(pl), _host(obj), _stream(stream)))
    return pl[:, :, :inst.n].copy(), obj


class ReplanStruct(ctypes.Structure):
    _fields_ = [("incumbent_objective", _i64), ("new_objective", _i64), ("materialization_cost", _i64),
                ("break_even_requests", _i64), ("adopted", _i32)]


@dataclass
class ReplanResult:
    placement: np.ndarray
    incumbent_objective: int
    new_objective: int
    materialization_cost: int
    break_even_requests: int
    adopted: bool


def pp_replan(inst: Instance, incumbent, n_starts: int, max_rounds: int, epoch_requests: int,
              horizon_requests: int, orders=None, safeguards: bool = True, stream=None) -> ReplanResult:
    """Epoch update with the amortisation rule; incumbent [W][n] uint8 (host)."""
    inc = _np(incumbent, np.uint8)
    if inc.shape != (inst.W, inst.n):
        raise ValueError("incumbent must be [W][n]")
    pl = np.zeros((inst.W, max(inst.n, 1)), np.uint8)
    res = ReplanStruct()
    st = PlanStats()
    st.no_safeguards = int(not safeguards)
    op = None
    if orders is not None:
        orders = _np(orders, np.int32)
        if orders.shape != (int(n_starts), inst.W):
            raise ValueError("orders must be [n_starts][W]")
        op = _host(orders)
    _check(_lib.pp_replan(inst.handle, _host(inc), int(n_starts), op, int(max_rounds), int(epoch_requests),
                          int(horizon_requests), _host(pl), ctypes.byref(res), ctypes.byref(st), _stream(stream)))
    return ReplanResult(pl[:, :inst.n].copy(), int(res.incumbent_objective), int(res.new_objective),
                        int(res.materialization_cost), int(res.break_even_requests), bool(res.adopted))
