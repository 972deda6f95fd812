"""The sample-sharded chain (paper_2607_08406_gb300.sharded) through the C ABI (needs a GPU).

The loss is a sum over samples (Eq. 2), so one chain can be split over ranks that each hold part
of the samples: every rank evaluates each trial of a batch on its own samples (mca_eval_trials),
the partial loss changes are all-gathered and added in rank order, every rank takes the same
decision (mca_decide_batch) and commits it on its shard. Here two ranks are two processes (gloo
for the exchange) whose handles hold the two halves of a workload's samples on the one GPU;
nothing on the device waits for another rank. The chain must follow the oracle's single-process
trajectory, and both shards must end with the same weights.
"""
import os
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))
from test_multirank_cpu import _run  # noqa: E402


def _workload(kind):
    from paper_2607_08406_gb300 import workloads as W
    if kind == "wide":
        return W.make("mlp_wide", N=4000, H=96)
    if kind == "deep":
        return W.make("mlp_deep", N=1200, width=40, depth=3)
    spec = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=2, n_head=2, d_ff=32)
    return W.char_transformer(batch=8, text_len=20000, spec=spec, n_trials=300, K=8)


def _rank(rank, world, kind, n, K, seed, forced):
    import torch
    from paper_2607_08406_gb300 import mca
    from paper_2607_08406_gb300 import workloads as W
    from paper_2607_08406_gb300.sharded import LibraryShard, ShardedChain
    torch.cuda.set_device(0)
    wl = _workload(kind)
    if kind == "tfm":                        # the loss is a sum over sequences: shard those
        rows = np.array_split(np.arange(wl.tokens.shape[0]), world)[rank]
        sub = W.TfmWorkload(wl.name, wl.spec, np.ascontiguousarray(wl.tokens[rows]), wl.init, n,
                            K, seed, wl.domain)
        h = mca.create_from_tfm_workload(sub, K=K, trace_cap=n)
        n_total, n_mine = wl.tokens.shape[0] * wl.spec.ctx, len(rows) * wl.spec.ctx
    else:
        rows = np.array_split(np.arange(wl.N), world)[rank]
        sub = W.MLPWorkload(wl.name, wl.layers, wl.loss, np.ascontiguousarray(wl.X[rows]),
                            np.ascontiguousarray(wl.y[rows]), wl.init, n, K, seed, wl.domain)
        h = mca.create_from_workload(sub, K=K, trace_cap=n)
        n_total, n_mine = wl.N, len(rows)
    chain = ShardedChain(LibraryShard(h), n_samples=n_total, K=K)
    st = chain.run(n, seed, forced=forced)
    tr = mca.mca_get_trace(h, n)
    out = (st, mca.mca_get_params(h, wl.n_params), tr["idx"].astype(np.int64),
           tr["accept"].astype(bool), mca.mca_loss(h) * n_mine)
    h.close()
    return out


@pytest.mark.parametrize("kind,n,K", [("wide", 400, 16), ("deep", 300, 8), ("tfm", 200, 8)])
def test_two_rank_sharded_chain_follows_the_single_process_trajectory(gpu_lib, kind, n, K):
    """Single hidden layer, a deep net (samples split) and a Transformer (sequences split)."""
    from oracle import mca_oracle as O
    from oracle import mca_tfm as T
    from parity import TIE_REL, tie_band
    wl = _workload(kind)
    seed = 6
    if kind == "tfm":
        tr, flat, S = T.run_full_tfm(wl.spec, wl.tokens, wl.init, n, seed, wl.domain)
    else:
        tr, params, S = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, n, seed,
                                          wl.domain)
        flat = params.flat_eff32()
    band = tie_band(tr)
    forced = {int(t): bool(a) for t, a in zip(tr["tau"][band], tr["accept"][band])}
    out = _run(_rank, 2, kind, n, K, seed, forced)
    (st0, p0, idx0, acc0, S0), (st1, p1, idx1, acc1, S1) = out[0], out[1]
    assert st0 == st1 and st0["trials"] == n
    assert st0["exchanges"] == st0["batches"] < n           # batches consumed several trials
    assert np.array_equal(idx0, tr["idx"]) and np.array_equal(idx1, tr["idx"])
    assert np.array_equal(acc0, tr["accept"]) and np.array_equal(acc1, tr["accept"])
    assert np.array_equal(p0, p1) and np.array_equal(p0, flat)
    assert S0 + S1 == pytest.approx(S, rel=TIE_REL)


def test_eval_trials_and_decide_batch_match_the_handles_own_run(gpu_lib):
    """One handle: mca_eval_trials proposes and evaluates exactly what mca_run would (index, old and
    new weights, dS of every trial before the first accept), and mca_decide_batch takes mca_run's
    decision."""
    from paper_2607_08406_gb300 import workloads as W
    from parity import TIE_REL
    for wl in (W.make("mlp_wide", N=3000, H=64), W.make("mlp_ternary", N=3000, H=64),
               W.make("mlp_deep", N=600, width=40, depth=3)):
        h = gpu_lib.create_from_workload(wl, K=16, trace_cap=64)
        h2 = gpu_lib.create_from_workload(wl, K=16, trace_cap=64)
        tau = 0
        for _ in range(6):
            rec = gpu_lib.mca_eval_trials(h, 3, tau, 16)
            k = gpu_lib.mca_decide_batch(h, 3, tau, rec["valid"], np.nan_to_num(rec["dS"]))
            m = k + 1 if k >= 0 else 16
            v = rec["valid"][:m].astype(bool)
            S = float(rec["S"][0])
            tie = bool(np.any(np.abs(rec["dS"][:m][v]) < TIE_REL * S))
            if tie:                                  # either decision is correct: take this one
                gpu_lib.mca_force_decisions(h2, np.arange(tau, tau + m, dtype=np.uint64),
                                            (np.arange(m) == k).astype(np.uint8))
            gpu_lib.mca_run(h2, m, 3)
            gpu_lib.mca_force_decisions(h2, [], [])
            g = gpu_lib.mca_get_trace(h2, m)[-m:]
            assert np.array_equal(g["idx"], rec["idx"][:m])
            assert np.array_equal(g["old_w"], rec["old_w"][:m])
            assert np.array_equal(g["new_w"], rec["new_w"][:m])
            assert np.array_equal(g["valid"], rec["valid"][:m])
            # the explicit evaluation may add a range's shares in another order than the loop
            assert np.all(np.abs(g["dS"][v] - rec["dS"][:m][v]) <= TIE_REL * S)
            assert np.array_equal(g["accept"].astype(bool), np.arange(m) == k)
            gpu_lib.mca_force_decisions(h, np.arange(tau, tau + m, dtype=np.uint64),
                                        (np.arange(m) == k).astype(np.uint8))
            gpu_lib.mca_run(h, m, 3)
            gpu_lib.mca_force_decisions(h, [], [])
            tau += m
        assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params),
                              gpu_lib.mca_get_params(h2, wl.n_params))
        h.close()
        h2.close()
