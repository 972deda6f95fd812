"""Parity of the CUDA path's current-layer schedule (Section 2.1) with the CPU oracle (needs a GPU).

With mca_domain.layer_stretch = M, the trials of stretch s = tau / M all mutate one layer chosen at
random for that stretch (its own Philox counter), the index uniform inside the layer. The GPU
derives every candidate's index this way in the windowed single-hidden-layer loop (the producer
warps' slot preparation) and in the deep path (evaluation, decision and commit); proposals and final
weights are compared bit for bit, decisions exactly outside the 1e-5 S tie band, as for the
uniform draw.
"""
import dataclasses

import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

from parity import compare, forced_from_oracle, oracle_trace, TIE_REL

pytestmark = pytest.mark.gpu


def _with_stretch(wl, M):
    wl.domain = dataclasses.replace(wl.domain, layer_stretch=M)
    return wl


CASES = {
    # name: (workload builder, stretch M, trials)
    "wide_window": (lambda: W.make("mlp_wide", N=12003, H=256), 50, 1500),
    "deep_w40": (lambda: W.mlp_deep(N=700, width=40, depth=3, n_trials=600, K=16), 30, 600),
    "deep_tc_w256": (lambda: W.mlp_deep(N=1100, width=256, depth=5, n_trials=500, K=16), 40, 500),
}


@pytest.mark.parametrize("case", list(CASES))
def test_schedule_trajectory(gpu_lib, case):
    build, M, n = CASES[case]
    wl = _with_stretch(build(), M)
    tr, params, S = oracle_trace(wl, n)
    lay = O.stretch_layer(wl.seed, np.arange(n) // M, len(wl.layers))
    assert (tr["layer"] == lay).all()
    h = gpu_lib.create_from_workload(wl, trace_cap=n)
    gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr))
    st = gpu_lib.mca_run(h, n, wl.seed)
    assert st["trials"] == n and st["tau"] == n
    compare(gpu_lib.mca_get_trace(h, n), tr)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())
    assert gpu_lib.mca_loss(h) == pytest.approx(S / wl.N, rel=TIE_REL)


def test_schedule_K_invariance_deep_tensor_cores(gpu_lib):
    """Under the schedule every batch's candidates share a layer; the trajectory still does not
    depend on K."""
    wl = _with_stretch(W.mlp_deep(N=1100, width=256, depth=5, n_trials=400, K=16), 25)
    ref = None
    for K in (1, 16, 128):
        h = gpu_lib.create_from_workload(wl, K=K, trace_cap=400)
        st = gpu_lib.mca_run(h, 400, 4)
        assert st["tensor_cores"] == 1
        out = (gpu_lib.mca_get_trace(h, 400), gpu_lib.mca_get_params(h, wl.n_params))
        if ref is None:
            ref = out
        else:
            assert np.array_equal(out[0], ref[0])
            assert np.array_equal(out[1], ref[1])
        h.close()
