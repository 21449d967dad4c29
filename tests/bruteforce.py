"""Brute-force and first-principles checks used to pin the oracle.

Nothing here calls the oracle or the CUDA library; every function is written
from a definition in the paper that is more primitive than the one under test:
  * the materialisation rule of Section III-A (local copy 0, peer-only
    min{w, f}, none w) for the objectives,
  * "parent-closed subset within the budget" (Eq. 8) enumerated exhaustively
    for the DP and for the joint optimum.
"""
from __future__ import annotations

import itertools

import numpy as np


def materialisation_saving(inst, placement) -> int:
    """Savings over all-recompute, straight from Section III-A.

    Requester m needing chunk b pays 0 if it holds b; otherwise the cheapest of
    recomputation w_m(b) and fetching from any holder; w_m(b) with no holder.
    Source-dependent costs (mode 1) use f_{m<-h}(b) = transfer[h][m][b]."""
    W, n = inst.W, inst.n
    pl = np.asarray(placement, bool)
    total = 0
    for b in range(n):
        holders = [h for h in range(W) if pl[h, b]]
        for m in range(W):
            w = int(inst.recompute[m, b])
            if pl[m, b]:
                cost = 0
            elif holders:
                if inst.mode == 0:
                    fetch = int(inst.transfer[m, b])
                else:
                    fetch = min(int(inst.transfer[h, m, b]) for h in holders)
                cost = min(w, fetch)
            else:
                cost = w
            total += int(inst.demand[m, b]) * (w - cost)
    return total


def parent_closed_masks(parent, weight, k):
    """All parent-closed subsets of total weight <= k, as an (N, n) bool array."""
    parent = np.asarray(parent)
    n = parent.shape[0]
    masks = np.arange(1 << n, dtype=np.int64)
    bits = ((masks[:, None] >> np.arange(n)[None, :]) & 1).astype(bool)
    ok = np.ones(masks.shape[0], bool)
    for v in range(n):
        p = parent[v]
        if p >= 0:
            ok &= ~bits[:, v] | bits[:, p]
    wsum = bits.astype(np.int64) @ np.asarray(weight, np.int64)
    ok &= wsum <= k
    return bits[ok]


def preorder_positions(parent):
    """Preorder with roots then children in ascending node id (plain recursion)."""
    parent = list(int(p) for p in parent)
    n = len(parent)
    kids = {u: [] for u in range(-1, n)}
    for v in range(n):
        kids[parent[v]].append(v)
    order = []

    def visit(u):
        order.append(u)
        for c in sorted(kids[u]):
            visit(c)

    for r in sorted(kids[-1]):
        visit(r)
    return order


def best_parent_closed(parent, weight, profit, k):
    """Maximum-profit parent-closed set of weight <= k, by enumeration.

    Among optimal sets returns the lexicographically smallest 0/1 indicator
    taken in preorder (0 before 1 at the earliest differing position)."""
    sets = parent_closed_masks(parent, weight, k)
    vals = sets.astype(np.int64) @ np.asarray(profit, np.int64)
    best = vals.max()
    opt = sets[vals == best]
    order = preorder_positions(parent)
    keys = [tuple(int(row[v]) for v in order) for row in opt]
    i = min(range(len(keys)), key=lambda t: keys[t])
    return int(best), opt[i].astype(np.uint8)


def joint_optimum(inst) -> int:
    """max over all feasible joint placements (Eq. 8) of the Section III-A saving."""
    per = [parent_closed_masks(inst.parent, inst.weight, int(inst.budget[m])) for m in range(inst.W)]
    best = 0
    for combo in itertools.product(*[range(len(p)) for p in per]):
        pl = np.stack([per[m][combo[m]] for m in range(inst.W)])
        best = max(best, materialisation_saving(inst, pl))
    return best


def is_parent_closed(parent, chosen) -> bool:
    parent = np.asarray(parent)
    ch = np.asarray(chosen, bool)
    has_p = parent >= 0
    return bool(np.all(~ch[has_p] | ch[parent[has_p]]))


def requester_saving(inst, placement, m) -> int:
    """Requester m's own saving over all-recompute under the Section III-A rule
    (local copy 0, otherwise the cheapest of w_m and a fetch from any holder)."""
    pl = np.asarray(placement, bool)
    total = 0
    for b in range(inst.n):
        w = int(inst.recompute[m, b])
        holders = [h for h in range(inst.W) if pl[h, b]]
        if pl[m, b]:
            cost = 0
        elif holders:
            fetch = int(inst.transfer[m, b]) if inst.mode == 0 else min(int(inst.transfer[h, m, b]) for h in holders)
            cost = min(w, fetch)
        else:
            cost = w
        total += int(inst.demand[m, b]) * (w - cost)
    return total


def best_set_by(parent, weight, k, value):
    """Parent-closed set of weight <= k maximising value(mask); ties to the
    lexicographically smallest preorder indicator (the DP's rule)."""
    sets = parent_closed_masks(parent, weight, k)
    vals = [value(s) for s in sets]
    best = max(vals)
    order = preorder_positions(parent)
    cand = [s for s, v in zip(sets, vals) if v == best]
    return min(cand, key=lambda s: tuple(int(s[v]) for v in order)).astype(np.uint8)


def materialisation_cost(inst, old, new) -> int:
    """One-time cost of making `new` resident given `old`: for every chunk b a
    worker m holds in `new` but not in `old`, requester m's Section III-A cost
    of b under `old` (the cheaper of recomputing and fetching from an old
    holder; recomputing when nobody holds it)."""
    old = np.asarray(old, bool)
    new = np.asarray(new, bool)
    total = 0
    for m in range(inst.W):
        for b in range(inst.n):
            if not new[m, b] or old[m, b]:
                continue
            w = int(inst.recompute[m, b])
            holders = [h for h in range(inst.W) if old[h, b] and h != m]
            if holders:
                fetch = int(inst.transfer[m, b]) if inst.mode == 0 else min(int(inst.transfer[h, m, b]) for h in holders)
                w = min(w, fetch)
            total += w
    return total


def standalone_score(inst, h) -> int:
    """Worker h's best Section III-A saving when it is the only holder
    (the standalone score of Section IV-C), by enumeration."""
    best = 0
    for s in parent_closed_masks(inst.parent, inst.weight, int(inst.budget[h])):
        pl = np.zeros((inst.W, inst.n), bool)
        pl[h] = s
        best = max(best, materialisation_saving(inst, pl))
    return best


def coordinate_trajectory(inst, pi, R, sweep_order=None, stale_reference=False):
    """One start of the planner (Section IV-C) rebuilt from enumeration.

    A worker update replaces T_h by the parent-closed set within k_h that
    maximises the Section III-A saving of the whole placement with the other
    targets fixed (ties to the lexicographically smallest preorder indicator,
    the DP's rule); by Prop. 1 this is the set the DP of Eq. 9 finds on the
    worker's marginals.  Greedy pass: the workers of `pi` in turn, the later
    ones still empty.  Refinement: at most R sweeps over `pi`; a new target
    is kept only if the saving strictly exceeds the saving just before the
    update; a sweep that keeps nothing ends the start.

    `sweep_order` and `stale_reference` only exist to build deliberately
    wrong variants (another sweep order; comparing against the saving at the
    start of the sweep) and show that the pins tell them apart.
    Returns (placement [W][n] uint8, saving, sweeps, accepted)."""
    W, n = inst.W, inst.n
    T = np.zeros((W, n), np.uint8)

    def best_for(h):
        def value(s):
            X = T.copy()
            X[h] = s
            return materialisation_saving(inst, X)
        return best_set_by(inst.parent, inst.weight, int(inst.budget[h]), value)

    for h in pi:
        T[h] = best_for(h)
    sweeps = accepted = 0
    for _ in range(R):
        sweeps += 1
        kept = False
        at_sweep_start = materialisation_saving(inst, T)
        for h in (pi if sweep_order is None else sweep_order):
            before = at_sweep_start if stale_reference else materialisation_saving(inst, T)
            old = T[h].copy()
            T[h] = best_for(h)
            if materialisation_saving(inst, T) > before:
                kept = True
                accepted += 1
            else:
                T[h] = old
        if not kept:
            break
    return T, materialisation_saving(inst, T), sweeps, accepted
