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


class OracleShard:
    """A shard of ShardedChain evaluated by the oracle's cached-field mode on the rank's samples
    (the CPU stand-in for a handle on one GPU); records every consumed trial."""

    def __init__(self, wl, shard_rows):
        from oracle import mca_oracle as O
        self.O = O
        self.wl = wl
        self.XT = wl.X.T.astype(np.float64)[:, shard_rows]
        self.y = wl.y[shard_rows]
        self.params = O.Params(wl.layers, wl.init)
        self.cache = O._Cache(self.params, self.XT, self.y, wl.loss)
        self.props, self.updates, self.ell, self.last_dS = [], [], [], None
        self.record = []

    def eval_trials(self, seed, tau, n):
        O = self.O
        self.props = [O.propose(seed, tau + k, self.params, self.wl.domain) for k in range(n)]
        valid = np.array([p.valid for p in self.props])
        res = [O._candidate(self.params, self.cache, self.XT, self.y, self.wl.loss, p)
               if p.valid else (0.0, None, None) for p in self.props]
        self.updates = [r[1] for r in res]
        self.ell = [r[2] for r in res]
        part = np.array([r[0] for r in res], np.float64)
        return valid, part, np.array([p.idx for p in self.props])

    def decide(self, seed, tau, valid, dS, n_samples):
        O = self.O
        self.last_dS = dS
        for k in range(len(valid)):
            if valid[k] and O._decide(float(dS[k]), self.wl.domain.strict,
                                      O._threshold(seed, tau + k, self.wl.domain, n_samples)):
                return k
        return -1

    def commit(self, seed, tau, m, kstar):
        for k in range(m):
            self.record.append((tau + k, self.props[k].idx, k == kstar))
        if kstar >= 0:
            self.O.apply_proposal(self.params, self.props[kstar])
            for lay, upd in self.updates[kstar]:
                if upd[0] == "row":
                    self.cache.Z[lay][upd[1]] = upd[2]
                else:
                    self.cache.Z[lay] = upd[1]
            self.cache.ell = self.ell[kstar]


def _chain_ranks(rank, world, n_trials, K, beta):
    import dataclasses
    from paper_2607_08406_gb300 import workloads as W
    from paper_2607_08406_gb300.sharded import ShardedChain
    wl = W.mlp_small(N=300)
    wl.domain = dataclasses.replace(wl.domain, beta=beta)
    shard = OracleShard(wl, np.array_split(np.arange(wl.N), world)[rank])
    chain = ShardedChain(shard, n_samples=wl.N, K=K)
    st = chain.run(n_trials, wl.seed)
    return shard.record, shard.params.flat_eff32(), st


@pytest.mark.parametrize("beta", [float("inf"), 400.0])
def test_sharded_chain_module_over_gloo_ranks(beta):
    """paper_2607_08406_gb300.sharded.ShardedChain over two gloo ranks (each an oracle shard on half
    of the samples) follows the single-process oracle's trajectory: greedy (Eq. 6) and Eq. 7 with
    the chain's whole sample count in the threshold."""
    import dataclasses
    from oracle import mca_oracle as O
    from paper_2607_08406_gb300 import workloads as W
    from parity import TIE_REL
    n = 150
    out = _run(_chain_ranks, 2, n, 16, beta)
    assert out[0][0] == out[1][0] and np.array_equal(out[0][1], out[1][1])
    assert out[0][2]["exchanges"] == out[0][2]["batches"] < n
    wl = W.mlp_small(N=300)
    dom = dataclasses.replace(wl.domain, beta=beta)
    tr, params, S = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, n, wl.seed, dom)
    theta = O.metropolis_threshold(wl.seed, np.arange(n, dtype=np.uint64), beta, wl.N)
    band = np.abs(tr["dS"] - theta) < TIE_REL * np.abs(tr["S"])
    rec = out[0][0]
    assert [r[0] for r in rec] == list(range(n))
    assert [r[1] for r in rec] == [int(i) for i in tr["idx"]]
    if beta != float("inf"):
        assert 0 < int(tr["accept"].sum()) and np.any(tr["accept"] & (tr["dS"] > 0))
    for (t, idx, acc), oacc, tie in zip(rec, tr["accept"], band):
        if tie:
            break                                 # after a tie-band decision the runs may part
        assert acc == bool(oacc), t
    else:
        assert np.array_equal(out[0][1], params.flat_eff32())
