"""Per-trial parity at the five workloads' full sizes, in the launch configuration the bench uses
(the workload's K, automatic grid, adaptive batch width), against the CPU oracle (needs a GB300).

Every trial of a prefix is compared with the oracle's own run on the same seeded inputs: proposals
bit for bit, decisions exactly (trials whose oracle |dS| < 1e-5 S take the oracle's decision through
the forced-decision hook: either decision is correct there), candidate dS within 1e-5 S, then the
final weights (and ternary codes / mask bits) bit for bit and the final loss. The oracle runs its
cached-field mode (Section 2.4) for the MLPs and the full-recompute definition for the
Transformer.

  784-16384-10 CE, N = 60000          3000 trials
  784-(256 x 24)-10 CE, N = 10000      200 trials   (tensor-core chain)
  784-4096-10 ternary, N = 60000      3000 trials   (codes compared with ==)
  784-4096-10 masked, N = 60000       3000 trials   (mask bits compared with ==)
  GPT vocab 65 / ctx 64 / d 128 / 2 x 4 heads / FFN 512, 256 sequences: 64 trials on the
  tensor-core kernels and on the SIMT kernels, plus candidates of every parameter stage
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from oracle import mca_tfm as T
from paper_2607_08406_gb300 import workloads as W

from parity import compare, forced_from_oracle, oracle_trace, TIE_REL

pytestmark = pytest.mark.gpu

MLP_CASES = {
    "wide": (W.mlp_wide, 3000),
    "deep": (W.mlp_deep, 200),
    "ternary": (W.mlp_ternary, 3000),
    "masked": (W.mlp_masked, 3000),
}


@pytest.fixture(scope="module")
def mlp_traces():
    cache = {}

    def get(case):
        if case not in cache:
            make, n = MLP_CASES[case]
            wl = make()
            cache.clear()                    # one config-sized oracle state at a time
            cache[case] = (wl, n) + oracle_trace(wl, n)
        return cache[case]
    return get


@pytest.mark.parametrize("case", list(MLP_CASES))
def test_config_size_trajectory(gpu_lib, mlp_traces, case):
    wl, n, tr, params, S = mlp_traces(case)
    h = gpu_lib.create_from_workload(wl, trace_cap=n)
    assert gpu_lib.mca_loss(h) * wl.N == pytest.approx(tr["S"][0], rel=1e-6)
    ft, fa = forced_from_oracle(tr)
    gpu_lib.mca_force_decisions(h, ft, fa)
    st = gpu_lib.mca_run(h, n, wl.seed)
    assert st["trials"] == n and st["accepts"] == int(tr["accept"].sum())
    if case == "deep":
        assert st["tensor_cores"] == 1
    compare(gpu_lib.mca_get_trace(h, n), tr)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())
    assert np.array_equal(gpu_lib.mca_get_codes(h, wl.n_params), params.flat_codes())
    assert gpu_lib.mca_loss(h) * wl.N == pytest.approx(S, rel=TIE_REL)
    if case == "wide":
        # sampled candidates of both layers at the final state, one by one against the oracle
        XT = wl.X.T.astype(np.float64)
        Z2 = O.output_fields_blocked(params, XT)
        rng = np.random.default_rng(1)
        P1 = wl.layers[0].n_in * wl.layers[0].n_out
        idx = np.concatenate([rng.integers(0, P1, 24), rng.integers(P1, wl.n_params, 8)])
        new = rng.uniform(-1, 1, len(idx)).astype(np.float32)
        d = gpu_lib.mca_eval_candidates(h, idx, new)
        for m in range(len(idx)):
            want = O.candidate_dS_two_layer(params, XT, wl.y, wl.loss, Z2, int(idx[m]),
                                            float(new[m]))
            assert abs(d[m] - want) <= TIE_REL * S, (m, d[m], want)
    h.close()


# ------------------------------------------------------------------------------------------------
# Transformer (Section 2.5), config size
# ------------------------------------------------------------------------------------------------

TFM_TRIALS = 64


def _stage_offsets(spec):
    offs, o = {}, 0
    for name, shape in spec.blocks():
        n = int(np.prod(shape))
        offs[name] = (o, n)
        o += n
    return offs


def every_stage_indices(spec, rng):
    """One random parameter of every named tensor of the flat layout (all 16 per block)."""
    return np.array([o + rng.integers(0, n) for o, n in _stage_offsets(spec).values()], np.uint32)


@pytest.fixture(scope="module")
def tfm_case():
    wl = W.char_transformer()
    tr, flat, S = T.run_full_tfm(wl.spec, wl.tokens, wl.init, TFM_TRIALS, wl.seed, wl.domain)
    rng = np.random.default_rng(9)
    idx = every_stage_indices(wl.spec, rng)
    new = rng.uniform(-1, 1, len(idx)).astype(np.float32)
    f64 = wl.init.astype(np.float64)
    S0 = T.tfm_seq_losses(wl.spec, f64, wl.tokens).sum()
    want = []
    for i, v in zip(idx, new):
        f2 = f64.copy()
        f2[int(i)] = float(np.float32(v))
        want.append(T.tfm_seq_losses(wl.spec, f2, wl.tokens).sum() - S0)
    return wl, tr, flat, S, idx, new, np.array(want), S0


@pytest.mark.parametrize("tensor_cores", ["1", "0"])
def test_config_size_transformer(gpu_lib, monkeypatch, tfm_case, tensor_cores):
    """vocab 65, context 64, d_model 128, 2 blocks x 4 heads, FFN 512, 256 sequences: the initial
    loss, one candidate in every parameter tensor (embeddings, both blocks' LN gains and biases,
    projections and their biases, FFN, final LN, head and its bias) against the oracle's full
    recompute, then 64 trials compared trial by trial with the oracle's run."""
    monkeypatch.setenv("MCA_TFM_TENSOR_CORES", tensor_cores)
    wl, tr, flat, S, idx, new, want, S0 = tfm_case
    BT = wl.tokens.shape[0] * wl.spec.ctx
    h = gpu_lib.create_from_tfm_workload(wl, trace_cap=TFM_TRIALS)
    assert gpu_lib.mca_get_stats(h)["tensor_cores"] == int(tensor_cores)
    assert gpu_lib.mca_loss(h) * BT == pytest.approx(S0, rel=1e-5)
    d = gpu_lib.mca_eval_candidates(h, idx, new)
    bad = np.nonzero(np.abs(d - want) > TIE_REL * S0)[0]
    names = list(_stage_offsets(wl.spec))
    assert len(bad) == 0, [(names[b], d[b], want[b]) for b in bad]
    gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr))
    st = gpu_lib.mca_run(h, TFM_TRIALS, wl.seed)
    assert st["trials"] == TFM_TRIALS
    compare(gpu_lib.mca_get_trace(h, TFM_TRIALS), tr)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), flat)
    assert gpu_lib.mca_loss(h) * BT == pytest.approx(S, rel=1e-5)
    h.close()


def test_config_size_drift_bound(gpu_lib):
    """784-16384-10 CE, N = 60000: 2 x 10^5 trials of incremental fp32 commits without a resync
    (the bench's setting) keep the cached loss within 1e-5 of a fresh full forward pass."""
    wl = W.mlp_wide()
    h = gpu_lib.create_from_workload(wl)
    st = gpu_lib.mca_run(h, 200_000, wl.seed)
    assert st["resyncs"] == 0 and st["accepts"] > 10_000
    L_inc = gpu_lib.mca_loss(h)
    gpu_lib.mca_resync(h)
    assert gpu_lib.mca_loss(h) == pytest.approx(L_inc, rel=1e-5)
    h.close()


@pytest.mark.parametrize("case", ["wide", "deep", "ternary"])
def test_forward_pass_tensor_cores_against_simt(gpu_lib, monkeypatch, case):
    """The forward pass on the tensor cores (3xTF32) and the SIMT SGEMM give the same loss to
    fp32 rounding at the full sizes, and the dyadic workload's exactly representable first layer
    gives the same loss bit for bit."""
    make = MLP_CASES[case][0]
    wl = make()
    S = {}
    for flag in ("1", "0"):
        monkeypatch.setenv("MCA_FORWARD_TENSOR_CORES", flag)
        h = gpu_lib.create_from_workload(wl)
        S[flag] = gpu_lib.mca_loss(h)
        h.close()
    assert S["1"] == pytest.approx(S["0"], rel=5e-6)
    if case == "ternary":
        assert S["1"] == S["0"]
