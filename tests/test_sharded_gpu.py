"""The sample-sharded chain through the C ABI on one GPU (needs a GPU).

The loss is a sum over samples (Eq. 2), so one chain can be split over shards that each hold part
of the samples: every shard evaluates each candidate of a batch on its own samples, the K partial
loss changes are exchanged and added in shard order, every shard takes the same decision (Eq. 6)
and commits the same accepted candidate. Here two handles hold the two halves of a workload's
samples on one GPU and the host does the exchange (a multi-GPU run would all-gather the K floats);
nothing on the device waits for another handle. The chain must follow the oracle's single-process
trajectory, and the two shards must end with the same weights.
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

from parity import TIE_REL, tie_band

pytestmark = pytest.mark.gpu


def test_two_shard_chain_follows_the_single_process_trajectory(gpu_lib):
    wl = W.make("mlp_wide", N=4000, H=96)
    n, K, seed = 400, 8, 6
    tr, params, S = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, n, seed, wl.domain)
    band = tie_band(tr)
    halves = (slice(0, 2000), slice(2000, 4000))
    shards = []
    for hs in halves:
        sub = W.MLPWorkload(wl.name, wl.layers, wl.loss, np.ascontiguousarray(wl.X[hs]),
                            np.ascontiguousarray(wl.y[hs]), wl.init, n, K, seed, wl.domain)
        shards.append(gpu_lib.create_from_workload(sub, K=K))
    words = O.draw_words(seed, np.arange(n, dtype=np.uint64))
    P = wl.n_params
    idx = ((words[:, 0] * np.uint64(P)) >> np.uint64(32)).astype(np.uint32)
    u = (words[:, 1] >> np.uint64(8)).astype(np.float32) * np.float32(2.0 ** -24)
    new = (np.float32(-1.0) + np.float32(2.0) * u).astype(np.float32)   # replacement values
    tau, exchanges = 0, 0
    while tau < n:
        kb = min(K, n - tau)
        part = [gpu_lib.mca_eval_candidates(h, idx[tau:tau + kb], new[tau:tau + kb])
                for h in shards]
        exchanges += 1
        dS = part[0] + part[1]                               # added in shard order
        kstar, dec = -1, []
        for k in range(kb):
            t = tau + k
            assert abs(dS[k] - tr["dS"][t]) <= TIE_REL * abs(tr["S"][t]), t
            d = bool(tr["accept"][t]) if band[t] else bool(dS[k] <= 0.0)
            if not band[t]:
                assert d == bool(tr["accept"][t]), t
            dec.append(d)
            if d:
                kstar = k
                break
        m = kstar + 1 if kstar >= 0 else kb
        for h in shards:                                     # every shard commits the same way
            gpu_lib.mca_force_decisions(h, np.arange(tau, tau + m, dtype=np.uint64),
                                        np.array(dec[:m] if kstar >= 0 else [False] * m))
            st = gpu_lib.mca_run(h, m, seed)
            assert st["tau"] == tau + m
        tau += m
    p0 = gpu_lib.mca_get_params(shards[0], P)
    assert np.array_equal(p0, gpu_lib.mca_get_params(shards[1], P))
    assert np.array_equal(p0, params.flat_eff32())
    assert exchanges < n                                     # batches consumed several trials
    L = sum(gpu_lib.mca_loss(h) * 2000 for h in shards)
    assert L == pytest.approx(S, rel=TIE_REL)
