"""Multi-rank paths on CPU ranks (gloo, world size 2, no GPU).

1. bench.py's whole-job aggregation over replicas: the slowest rank's time and the units all ranks
   processed.
2. The sample-sharded decision rule: the loss change of a candidate is a sum over samples (Eq. 2), so
   ranks holding disjoint sample shards can each evaluate every candidate of a batch on their shard,
   exchange the K partial sums (one all-gather per batch), add them in rank order and take the same
   decision (Eq. 6). The trajectory must follow the single-process oracle's, outside the tie band.
"""
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _run(fn, world, *args):
    import torch.multiprocessing as mp
    port = _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_entry, args=(fn, r, world, port, q) + args) for r in range(world)]
    for p in procs:
        p.start()
    import queue
    import time
    out = {}
    t0 = time.time()
    while len(out) < world:
        try:
            r, res = q.get(timeout=1.0)
            out[r] = res
        except queue.Empty:
            dead = [p for p in procs if p.exitcode not in (None, 0)]
            if dead or time.time() - t0 > 300:
                for p in procs:
                    if p.is_alive():
                        p.terminate()
                pytest.fail(f"rank process failed (exit codes {[p.exitcode for p in procs]})")
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return out


def _entry(fn, rank, world, port, q, *args):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        q.put((rank, fn(rank, world, *args)))
    finally:
        dist.destroy_process_group()


def _aggregate(rank, world):
    import bench
    return bench.job_totals(10.0 + 5.0 * rank, 100.0 * (rank + 1), device="cpu")


def test_replica_aggregation_gloo():
    out = _run(_aggregate, 2)
    assert out[0] == out[1] == (15.0, 300.0)


def _sharded_trajectory(rank, world, n_trials, K):
    import torch
    import torch.distributed as dist
    from oracle import mca_oracle as O
    from paper_2607_08406_gb300 import workloads as W
    wl = W.mlp_small(N=300)
    XT = wl.X.T.astype(np.float64)
    shard = np.array_split(np.arange(wl.N), world)[rank]
    XTs, ys = XT[:, shard], wl.y[shard]
    params = O.Params(wl.layers, wl.init)
    decisions = []
    tau = 0
    while tau < n_trials:
        kb = min(K, n_trials - tau)
        cache = O._Cache(params, XTs, ys, wl.loss)
        props = [O.propose(wl.seed, tau + k, params, wl.domain) for k in range(kb)]
        part = np.array([O._candidate(params, cache, XTs, ys, wl.loss, p)[0] if p.valid else 0.0
                         for p in props], dtype=np.float64)
        gathered = [torch.zeros(kb, dtype=torch.float64) for _ in range(world)]
        dist.all_gather(gathered, torch.from_numpy(part))
        dS = np.zeros(kb)
        for g in gathered:                        # rank order: the same sum on every rank
            dS = dS + g.numpy()
        kstar = next((k for k in range(kb) if props[k].valid and dS[k] <= 0.0), -1)
        last = kstar if kstar >= 0 else kb - 1
        for k in range(last + 1):
            decisions.append((tau + k, props[k].idx, k == kstar, float(dS[k])))
        if kstar >= 0:
            O.apply_proposal(params, props[kstar])
            tau += kstar + 1
        else:
            tau += kb
    return decisions, params.flat_eff32()


def test_sample_sharded_decisions_match_single_process_oracle():
    from oracle import mca_oracle as O
    from paper_2607_08406_gb300 import workloads as W
    from parity import TIE_REL
    n = 120
    out = _run(_sharded_trajectory, 2, n, 8)
    assert out[0][0] == out[1][0] and np.array_equal(out[0][1], out[1][1])
    wl = W.mlp_small(N=300)
    tr, params, S = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, n, wl.seed,
                                      wl.domain)
    dec = out[0][0]
    assert [d[0] for d in dec] == list(range(n))
    assert [d[1] for d in dec] == [int(i) for i in tr["idx"]]
    band = np.abs(tr["dS"]) < TIE_REL * np.abs(tr["S"])
    for (t, idx, acc, dS), oacc, odS, tie in zip(dec, tr["accept"], tr["dS"], band):
        if tie:
            break                                 # after a tie-band decision the runs may part
        assert acc == bool(oacc), t
        assert abs(dS - odS) <= 1e-9 * max(1.0, abs(odS)), (t, dS, odS)
    else:
        assert np.array_equal(out[0][1], params.flat_eff32())
