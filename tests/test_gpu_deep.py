"""Parity of the CUDA deep-MLP path (three or more weight layers) with the CPU oracle (needs a GPU).

Small nets with ragged tiles and widths that are not multiples of the GEMM tile check trajectories
bit for bit on proposals, decisions (tie band replayed) and final weights; the 24 x 256 workload is
checked at full size on candidates of every layer kind and on a short run.
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

from parity import compare, forced_from_oracle, oracle_trace, TIE_REL

pytestmark = pytest.mark.gpu


def _deep(N=700, width=40, depth=3, loss="softmax_ce", out_act="identity", hidden="tanh"):
    wl = W.mlp_deep(N=N, width=width, depth=depth, n_trials=1500, K=16)
    if hidden != "tanh":
        for L in wl.layers[:-1]:
            L.act = hidden
            L.act_param = 1.0 if hidden == "gaussian" else 0.0
    wl.layers[-1].act = out_act
    wl.loss = loss
    return wl


CASES = {
    "ce_w40_d3": dict(),
    "mse_sigmoid_w33_d4": dict(width=33, depth=4, loss="mse_onehot", out_act="sigmoid"),
    "gauss_w64_d2": dict(N=513, width=64, depth=2, hidden="gaussian"),
    # 256-wide inner layers: the dense chain runs on the tensor cores (3xTF32); 1100 samples leave a
    # ragged last tile of 76; Gaussian hidden layers take the kernel's run-time transfer function
    "tc_ce_w256_d5": dict(N=1100, width=256, depth=5),
    "tc_gauss_mse_w256_d4": dict(N=1100, width=256, depth=4, loss="mse_onehot", out_act="sigmoid",
                                 hidden="gaussian"),
}


@pytest.mark.parametrize("case", list(CASES))
def test_deep_initial_loss_and_trajectory(gpu_lib, case):
    wl = _deep(**CASES[case])
    n = wl.n_trials
    h = gpu_lib.create_from_workload(wl, trace_cap=n)
    S0 = O.total_loss(O.Params(wl.layers, wl.init), wl.X.T.astype(np.float64), wl.y, wl.loss)
    assert gpu_lib.mca_loss(h) == pytest.approx(S0 / wl.N, rel=1e-6)
    tr, params, S = oracle_trace(wl, n)
    gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr))
    st = gpu_lib.mca_run(h, n, wl.seed)
    assert st["trials"] == n
    assert st["tensor_cores"] == int(case.startswith("tc_"))
    compare(gpu_lib.mca_get_trace(h, n), tr)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())
    assert gpu_lib.mca_loss(h) == pytest.approx(S / wl.N, rel=TIE_REL)
    assert st["accepts"] > 20


@pytest.mark.parametrize("width", [40, 256])
def test_deep_K_invariance(gpu_lib, width):
    """Trajectories and weights do not depend on the batch width K (SIMT chain at width 40, the
    tensor-core chain at width 256, whose CTAs are ordered by chain length within each batch)."""
    wl = _deep(N=700 if width == 40 else 1100, width=width, depth=3 if width == 40 else 5)
    ref = None
    for K in (1, 5, 32, 128):
        h = gpu_lib.create_from_workload(wl, K=K, trace_cap=400)
        gpu_lib.mca_run(h, 400, 2)
        g = gpu_lib.mca_get_trace(h, 400)
        p = gpu_lib.mca_get_params(h, wl.n_params)
        if ref is None:
            ref = (g, p)
        else:
            assert np.array_equal(g, ref[0]) and np.array_equal(p, ref[1])
        h.close()


def _oracle_candidates(wl, params, idxs, news):
    XT = wl.X.T.astype(np.float64)
    cache = O._Cache(params, XT, wl.y, wl.loss)
    out = []
    for idx, v in zip(idxs, news):
        l = max(q for q in range(len(wl.layers)) if params.offsets[q] <= idx)
        row, col = divmod(int(idx) - params.offsets[l], wl.layers[l].n_in)
        old = float(params.eff32(l)[row, col])
        p = O.Proposal(0, int(idx), l, row, col, old, float(v), 0, 0, float(v), True)
        out.append(O._candidate(params, cache, XT, wl.y, wl.loss, p)[0])
    return np.array(out), float(cache.ell.sum())


def _idx_per_layer(wl, rng, per_layer):
    offs = np.cumsum([0] + [L.n_in * L.n_out for L in wl.layers])
    return np.concatenate([rng.integers(offs[l], offs[l + 1], per_layer)
                           for l in range(len(wl.layers))]).astype(np.uint32)


@pytest.mark.parametrize("width", [40, 256])
def test_deep_eval_candidates_every_layer(gpu_lib, width):
    wl = _deep(width=width, depth=4, N=700 if width == 40 else 1100)
    h = gpu_lib.create_from_workload(wl)
    gpu_lib.mca_run(h, 300, 5)
    params = O.Params(wl.layers, gpu_lib.mca_get_params(h, wl.n_params))
    rng = np.random.default_rng(3)
    idx = _idx_per_layer(wl, rng, 6)
    new = rng.uniform(-1, 1, len(idx)).astype(np.float32)
    d = gpu_lib.mca_eval_candidates(h, idx, new)
    want, S = _oracle_candidates(wl, params, idx, new)
    assert np.all(np.abs(d - want) <= TIE_REL * S)
    assert np.array_equal(gpu_lib.mca_eval_candidates(h, idx, new), d)


def test_deep_resync_keeps_loss(gpu_lib):
    wl = _deep()
    h = gpu_lib.create_from_workload(wl)
    st = gpu_lib.mca_run(h, 1200, 8)
    assert st["accepts"] > 50
    L_inc = gpu_lib.mca_loss(h)
    gpu_lib.mca_resync(h)
    assert gpu_lib.mca_loss(h) == pytest.approx(L_inc, rel=1e-6)
