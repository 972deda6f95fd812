"""Parity with the oracle for the paper's other transfer functions (needs a GPU).

Section 2 trains deep nets with ReLU and with the Gaussian exp(-gamma x^2) at gamma = 0.4; the five
workloads use tanh (and gamma = 1). Here the single-hidden-layer loop (ReLU, GELU and Gaussian hidden
layers run its run-time-activation kernel) and the deep chains (the tensor-core chain with ReLU and
with the Gaussian at gamma = 0.4; the SIMT chain with sigmoid hidden layers and MSE) follow the
oracle's trajectory: proposals and final weights bit for bit, decisions exactly outside the 1e-5 S
tie band, candidate dS within it.
"""
import numpy as np
import pytest

from paper_2607_08406_gb300 import workloads as W

from parity import compare, oracle_trace, TIE_REL

pytestmark = pytest.mark.gpu


def _acts(wl, hidden, gamma=0.0, out=None, loss=None):
    for L in wl.layers[:-1]:
        L.act = hidden
        L.act_param = gamma
    if out is not None:
        wl.layers[-1].act = out
    if loss is not None:
        wl.loss = loss
    return wl


CASES = {
    # name: (workload builder, trials, expect tensor cores)
    "wide_relu_ce": (lambda: _acts(W.make("mlp_wide", N=5003, H=128), "relu"), 1500, 0),
    "wide_gelu_ce": (lambda: _acts(W.make("mlp_wide", N=5003, H=128), "gelu"), 1500, 0),
    "wide_gauss04_mse": (lambda: _acts(W.make("mlp_wide", N=5003, H=128), "gaussian", 0.4,
                                       out="sigmoid", loss="mse_onehot"), 1500, 0),
    "deep_tc_relu_ce": (lambda: _acts(W.mlp_deep(N=1100, width=256, depth=4, n_trials=400,
                                                 K=16), "relu"), 400, 1),
    "deep_tc_gauss04_ce": (lambda: _acts(W.mlp_deep(N=1100, width=256, depth=4, n_trials=400,
                                                    K=16), "gaussian", 0.4), 400, 1),
    "deep_w64_sigmoid_mse": (lambda: _acts(W.mlp_deep(N=900, width=64, depth=3, n_trials=600,
                                                      K=16), "sigmoid", out="sigmoid",
                                           loss="mse_onehot"), 600, 0),
}


@pytest.mark.parametrize("case", list(CASES))
def test_transfer_function_trajectory(gpu_lib, case):
    build, n, tc = CASES[case]
    wl = build()
    tr, params, S = oracle_trace(wl, n)
    assert tr["accept"].sum() > 20
    h = gpu_lib.create_from_workload(wl, trace_cap=n)
    # ReLU's kink: a candidate whose fp64 activations do not change at all (dS = 0 exactly in the
    # oracle) can move an fp32 activation that sits within rounding of 0, so here exact zeros are
    # replayed too (the exactness of true no-ops is tested with the tanh workloads)
    band = tr["valid"] & (np.abs(tr["dS"]) < TIE_REL * np.abs(tr["S"]))
    gpu_lib.mca_force_decisions(h, tr["tau"][band].astype(np.uint64), tr["accept"][band])
    st = gpu_lib.mca_run(h, n, wl.seed)
    assert st["trials"] == n and st["tensor_cores"] == tc
    compare(gpu_lib.mca_get_trace(h, n), tr)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())
    assert gpu_lib.mca_loss(h) == pytest.approx(S / wl.N, rel=TIE_REL)
