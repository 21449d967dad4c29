"""Start sharding across processes (CPU ranks over gloo, no GPU).

The starts of Algorithm 1 are independent chains, so P ranks can each plan
the starts s with s % P == rank and exchange only the final choice.  These
checks run the per-rank planning with the CPU oracle and compare the sharded
result with one process planning every start: same objective, same winning
start (ties to the lowest index) and the same placement.  A rank that dies
before the exchange must make the survivors fail with an error, not hang.
"""
import json
import os
import socket
import time

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

from paper_2608_01655_gb300 import workloads as wl  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _instance(seed):
    rng = np.random.default_rng(seed)
    return wl.random_small(rng, 60, 5, seed % 2, k_max=20, w_max=2, demand_max=30)


def _worker(rank, world, port, seed, S, R, out_dir, die_rank):
    import datetime

    import oracle
    from paper_2608_01655_gb300 import shard

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world,
                            timeout=datetime.timedelta(seconds=8))
    inst = _instance(seed)
    prob = oracle.Problem.from_instance(inst)
    orders = oracle.default_orders(prob, S)

    def run_starts(sub):
        r = oracle.plan(prob, sub.shape[0], R, orders=sub, threads=1)
        return r.per_start_objective, r.best_start, r.placement

    if rank == die_rank:
        os._exit(3)                      # leaves between steps, before the exchange
    t0 = time.time()
    try:
        res = shard.plan_sharded(run_starts, orders, (inst.W, inst.n), rank, world)
        rec = {"ok": True, "objective": res.objective, "start": res.best_start,
               "placement": res.placement.astype(int).tolist()}
    except Exception as e:               # a lost peer must surface as an error
        rec = {"ok": False, "error": type(e).__name__, "seconds": time.time() - t0}
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump(rec, f)
    if rec["ok"]:
        dist.destroy_process_group()


def _run(world, seed, S, R, tmp_path, die_rank=-1):
    """Start `world` spawned ranks and wait for each (a rank that exits early
    does not take the others down)."""
    port = _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_worker, args=(r, world, port, seed, S, R, str(tmp_path), die_rank))
             for r in range(world)]
    for p in procs:
        p.start()
    deadline = time.time() + 120
    for p in procs:
        p.join(timeout=max(1.0, deadline - time.time()))
    alive = [p for p in procs if p.is_alive()]
    for p in alive:
        p.kill()
        p.join()
    assert not alive, "ranks did not finish"
    return [p.exitcode for p in procs]


@pytest.mark.parametrize("world,S,seed", [(2, 5, 1), (3, 4, 2), (3, 2, 3)])
def test_sharded_starts_match_one_process(oracle_lib, tmp_path, world, S, seed):
    codes = _run(world, seed, S, 3, tmp_path)
    assert codes == [0] * world
    inst = _instance(seed)
    prob = oracle_lib.Problem.from_instance(inst)
    full = oracle_lib.plan(prob, S, 3, orders=oracle_lib.default_orders(prob, S), threads=1)
    for r in range(world):
        rec = json.load(open(tmp_path / f"rank{r}.json"))
        assert rec["ok"], rec
        assert rec["objective"] == full.objective
        assert rec["start"] == full.best_start
        np.testing.assert_array_equal(np.array(rec["placement"], np.uint8), full.placement)


def _bench_worker(rank, world, port, seed, S, R, scaling, out_dir):
    """The benchmark's rank logic (shard.rank_orders, then shard.exchange)
    with the oracle as the planner."""
    import datetime

    import oracle
    from paper_2608_01655_gb300 import shard

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world,
                            timeout=datetime.timedelta(seconds=20))
    inst = _instance(seed)
    prob = oracle.Problem.from_instance(inst)
    orders, idx = shard.rank_orders(lambda total: oracle.default_orders(prob, total), S, rank, world, scaling)
    if len(idx):
        r = oracle.plan(prob, len(idx), R, orders=orders, threads=1)
        obj, start, placement = r.objective, int(idx[r.best_start]), r.placement
    else:
        obj, start, placement = 0, -1, np.zeros((inst.W, inst.n), np.uint8)
    won = shard.exchange(obj, start, placement)
    with open(os.path.join(out_dir, f"bench{rank}.json"), "w") as f:
        json.dump({"objective": won.objective, "start": won.best_start, "planned": idx.tolist(),
                   "placement": won.placement.astype(int).tolist()}, f)
    dist.destroy_process_group()


@pytest.mark.parametrize("world,scaling", [(2, "weak"), (3, "weak"), (2, "strong"), (3, "strong")])
def test_bench_rank_logic_weak_and_strong(oracle_lib, tmp_path, world, scaling):
    """Weak scaling: S starts per rank out of S * world default orders; strong
    scaling: the S starts of one plan split over the ranks.  Either way the
    ranks plan disjoint round-robin shares that cover every start, and the
    exchanged winner equals one process planning all of those starts."""
    S, R, seed = 4, 2, 5
    port = _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_bench_worker, args=(r, world, port, seed, S, R, scaling, str(tmp_path)))
             for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert [p.exitcode for p in procs] == [0] * world
    total = S * world if scaling == "weak" else S
    inst = _instance(seed)
    prob = oracle_lib.Problem.from_instance(inst)
    full = oracle_lib.plan(prob, total, R, orders=oracle_lib.default_orders(prob, total), threads=1)
    recs = [json.load(open(tmp_path / f"bench{r}.json")) for r in range(world)]
    assert sorted(sum((rec["planned"] for rec in recs), [])) == list(range(total))
    for rec in recs:
        assert rec["objective"] == full.objective and rec["start"] == full.best_start
        np.testing.assert_array_equal(np.array(rec["placement"], np.uint8), full.placement)


def test_lost_rank_is_reported(oracle_lib, tmp_path):
    """Rank 1 exits before the exchange; rank 0 gets an error within the
    process-group timeout instead of waiting forever."""
    codes = _run(2, 4, 4, 3, tmp_path, die_rank=1)
    assert codes[1] == 3
    rec = json.load(open(tmp_path / "rank0.json"))
    assert not rec["ok"]
    assert rec["seconds"] < 60


def test_round_robin_split():
    from paper_2608_01655_gb300 import shard
    parts = [shard.my_starts(10, r, 3).tolist() for r in range(3)]
    assert sorted(sum(parts, [])) == list(range(10))
    assert parts[1] == [1, 4, 7]
    assert shard.choose_winner([5, 7, 7, 2], [0, 3, 1, 2]) == (7, 1)
    assert shard.choose_winner([5, 9], [0, -1]) == (5, 0)
