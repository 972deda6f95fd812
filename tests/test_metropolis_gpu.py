"""Parity of the CUDA path's Metropolis rule (Section 3.1, Eq. 7) with the CPU oracle (needs a GPU).

With a finite selection intensity beta, trial tau is kept iff its loss-sum change dS is at most
theta_tau = -(N / beta) ln u_tau, u_tau drawn from the fourth Philox word of the trial's counter
(N = samples, or predicted tokens for the Transformer). Each workload below takes a beta at which
theta is of the order of the uphill changes, so that many uphill moves are kept. As for the greedy
rule, proposals and final weights / codes are compared bit for bit, candidate dS within 1e-5 S,
and decisions exactly after replaying the oracle's decision on the trials whose |dS - theta| <
1e-5 S (either decision is correct there) through the forced-decision hook. Every decision site
is covered: the windowed loop, the other single-hidden-layer loop (one CTA, records in global
memory), the deep decide kernel after the SIMT and the tensor-core chains, and the Transformer's.
"""
import dataclasses

import numpy as np
import pytest

from oracle import mca_oracle as O
from oracle import mca_tfm as T
from paper_2607_08406_gb300 import workloads as W

from parity import compare, forced_from_oracle, oracle_trace, TIE_REL

pytestmark = pytest.mark.gpu


def _with_beta(wl, beta):
    wl.domain = dataclasses.replace(wl.domain, beta=beta)
    return wl


MLP2_CASES = {
    # name: (workload, size overrides, beta, trials, grid; 0 = automatic, the windowed loop)
    "wide_window": ("mlp_wide", dict(N=12003, H=256), 6000.0, 2000, 0),
    "wide_one_range": ("mlp_wide", dict(N=12003, H=256), 6000.0, 600, 1),
    "ternary": ("mlp_ternary", dict(N=12000, H=256), 24000.0, 2000, 0),
    "masked": ("mlp_masked", dict(N=12000, H=256), 24000.0, 2000, 0),
}


def _run_and_compare(gpu_lib, h, wl, tr, theta, n):
    gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr, theta))
    st = gpu_lib.mca_run(h, n, wl.seed)
    assert st["trials"] == n and st["tau"] == n
    compare(gpu_lib.mca_get_trace(h, n), tr)
    assert ((tr["dS"] > 0) & tr["accept"]).sum() > 20       # uphill moves were kept
    return st


@pytest.mark.parametrize("case", list(MLP2_CASES))
def test_metropolis_trajectory_single_hidden_layer(gpu_lib, case):
    name, kw, beta, n, grid = MLP2_CASES[case]
    wl = _with_beta(W.make(name, **kw), beta)
    tr, params, S = oracle_trace(wl, n)
    theta = O.metropolis_threshold(wl.seed, tr["tau"], beta, wl.N)
    h = gpu_lib.create_from_workload(wl, trace_cap=n, grid=grid)
    _run_and_compare(gpu_lib, h, wl, tr, theta, n)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())
    assert np.array_equal(gpu_lib.mca_get_codes(h, wl.n_params), params.flat_codes())
    assert gpu_lib.mca_loss(h) == pytest.approx(S / wl.N, rel=TIE_REL)


def test_metropolis_K_invariance(gpu_lib):
    """theta depends only on the trial's own counter, so the kept trajectory does not depend on the
    speculation width K under Eq. 7 either."""
    wl = _with_beta(W.make("mlp_wide", N=12003, H=256), 6000.0)
    ref = None
    for K in (1, 16, 128):
        h = gpu_lib.create_from_workload(wl, K=K, trace_cap=1200)
        gpu_lib.mca_run(h, 800, 3)
        gpu_lib.mca_run(h, 400, 3)
        out = (gpu_lib.mca_get_trace(h, 1200), gpu_lib.mca_get_params(h, wl.n_params))
        if ref is None:
            ref = out
        else:
            assert np.array_equal(out[0], ref[0])
            assert np.array_equal(out[1], ref[1])
        h.close()


DEEP_CASES = {
    # name: (sizes, beta, trials); 256-wide inner layers run the tensor-core chain
    "w40_d3": (dict(N=700, width=40, depth=3), 1750.0, 600),
    "tc_w256_d5": (dict(N=1100, width=256, depth=5), 9000.0, 500),
}


@pytest.mark.parametrize("case", list(DEEP_CASES))
def test_metropolis_trajectory_deep(gpu_lib, case):
    kw, beta, n = DEEP_CASES[case]
    wl = _with_beta(W.mlp_deep(n_trials=n, K=16, **kw), beta)
    tr, params, S = oracle_trace(wl, n)
    theta = O.metropolis_threshold(wl.seed, tr["tau"], beta, wl.N)
    h = gpu_lib.create_from_workload(wl, trace_cap=n)
    st = _run_and_compare(gpu_lib, h, wl, tr, theta, n)
    assert st["tensor_cores"] == int(case.startswith("tc_"))
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())
    assert gpu_lib.mca_loss(h) == pytest.approx(S / wl.N, rel=TIE_REL)


def test_metropolis_trajectory_transformer(gpu_lib):
    spec = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=2, n_head=2, d_ff=32)
    batch, n, beta = 6, 400, 600.0
    wl = _with_beta(W.char_transformer(seed=0, batch=batch, text_len=20000, spec=spec,
                                       n_trials=n, K=8), beta)
    tr, flat, S = T.run_full_tfm(spec, wl.tokens, wl.init, n, wl.seed, wl.domain)
    theta = O.metropolis_threshold(wl.seed, tr["tau"], beta, batch * spec.ctx)
    h = gpu_lib.create_from_tfm_workload(wl, trace_cap=n)
    _run_and_compare(gpu_lib, h, wl, tr, theta, n)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), flat)
    assert gpu_lib.mca_loss(h) * batch * spec.ctx == pytest.approx(S, rel=TIE_REL)
