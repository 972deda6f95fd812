"""Parity of mca_run_channels (Section 2.3's channel mutations) with the CPU oracle (needs a GPU).

Each trial changes the weight of every layer on one input-to-output channel, recomputes the cached
fields with the full forward pass and keeps the channel iff the loss does not increase. Compared
with the oracle's run_channel on the same seeds: every decision (replaying the oracle's inside the
1e-5 S tie band), every dS within that band, and the final weights bit for bit, for both schemes on
a single-hidden-layer net and on deep nets (SIMT and tensor-core forward passes).
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

from parity import TIE_REL

pytestmark = pytest.mark.gpu

CASES = {
    # name: (workload builder, trials)
    "single_hidden": (lambda: W.make("mlp_small", N=300, H=32), 150),
    "deep_w40": (lambda: W.mlp_deep(N=700, width=40, depth=3, n_trials=150, K=8), 150),
    "deep_tc_w256": (lambda: W.mlp_deep(N=1100, width=256, depth=4, n_trials=120, K=8), 120),
}


@pytest.mark.parametrize("scheme", ["he", "zero"])
@pytest.mark.parametrize("case", list(CASES))
def test_channel_trajectory(gpu_lib, case, scheme):
    build, n = CASES[case]
    wl = build()
    seed = 5
    rows, params, S = O.run_channel(wl.layers, wl.loss, wl.X, wl.y, wl.init, n, seed, scheme)
    taus = np.array([r[0] for r in rows], np.uint64)
    S_o = np.array([r[2] for r in rows])
    dS_o = np.array([r[3] for r in rows])
    acc_o = np.array([r[4] for r in rows])
    assert 3 < acc_o.sum() < n - 3
    h = gpu_lib.create_from_workload(wl)
    band = np.abs(dS_o) < TIE_REL * np.abs(S_o)
    gpu_lib.mca_force_decisions(h, taus[band], acc_o[band])
    acc, dS = gpu_lib.mca_run_channels(h, n, seed, scheme)
    bad = np.nonzero(acc != acc_o)[0]
    assert len(bad) == 0, (bad[:5], dS[bad[:5]], dS_o[bad[:5]])
    assert np.all(np.abs(dS - dS_o) <= TIE_REL * np.abs(S_o))
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())
    assert gpu_lib.mca_loss(h) == pytest.approx(S / wl.N, rel=TIE_REL)
    st = gpu_lib.mca_get_stats(h)
    assert st["tau"] == n
