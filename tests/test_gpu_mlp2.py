"""Parity of the CUDA single-hidden-layer path with the CPU oracle (needs a GB300).

Every comparison runs both sides on the same seeded inputs. Proposals and the final integer /
mask / weight state are compared bit for bit; candidate loss changes within 1e-5 of the loss sum;
decisions exactly, after replaying the oracle's decision on trials whose |dS| < 1e-5 S (either
decision is correct there) through the library's forced-decision hook.
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

from parity import compare, forced_from_oracle, oracle_trace, TIE_REL

pytestmark = pytest.mark.gpu

CASES = {
    # (workload, size overrides, trials)
    "small_full": ("mlp_small", dict(), 20000),            # 784-64-10 MSE, N=1000, the full case
    "wide_ragged": ("mlp_wide", dict(N=12003, H=256), 3000),
    "ternary": ("mlp_ternary", dict(N=12000, H=256), 3000),
    "masked": ("mlp_masked", dict(N=12000, H=256), 3000),
}


def _make(case, **over):
    name, kw, n = CASES[case]
    kw = dict(kw, **over)
    return W.make(name, **kw), n


@pytest.fixture(scope="module")
def traces():
    cache = {}

    def get(case):
        if case not in cache:
            wl, n = _make(case)
            cache[case] = (wl, n) + oracle_trace(wl, n)
        return cache[case]
    return get


@pytest.mark.parametrize("case", list(CASES))
def test_initial_loss(gpu_lib, case):
    wl, _ = _make(case)
    h = gpu_lib.create_from_workload(wl)
    L = gpu_lib.mca_loss(h)
    S = O.total_loss(O.Params(wl.layers, wl.init), wl.X.T.astype(np.float64), wl.y, wl.loss)
    assert L == pytest.approx(S / wl.N, rel=1e-6)
    got = gpu_lib.mca_get_params(h, wl.n_params)
    assert np.array_equal(got, O.Params(wl.layers, wl.init).flat_eff32())


@pytest.mark.parametrize("case", list(CASES))
def test_trajectory_parity(gpu_lib, traces, case):
    wl, n, tr, params, S = traces(case)
    h = gpu_lib.create_from_workload(wl, trace_cap=n)
    ft, fa = forced_from_oracle(tr)
    gpu_lib.mca_force_decisions(h, ft, fa)
    st = gpu_lib.mca_run(h, n, wl.seed)
    assert st["trials"] == n and st["tau"] == n
    g = gpu_lib.mca_get_trace(h, n)
    compare(g, tr)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())
    assert np.array_equal(gpu_lib.mca_get_codes(h, wl.n_params), params.flat_codes())
    assert gpu_lib.mca_loss(h) == pytest.approx(S / wl.N, rel=TIE_REL)
    assert st["accepts"] == int(tr["accept"].sum())
    assert st["forced"] <= len(ft)


def test_noop_trials_exact_zero(gpu_lib, traces):
    """Ternary proposals equal to the old code: dS is exactly 0 on the GPU and accepted (Eq. 6)."""
    wl, n, tr, _, _ = traces("ternary")
    h = gpu_lib.create_from_workload(wl, trace_cap=n)
    gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr))
    gpu_lib.mca_run(h, n, wl.seed)
    g = gpu_lib.mca_get_trace(h, n)
    noop = g["old_w"] == g["new_w"]
    assert noop.sum() > 100
    assert np.all(g["dS"][noop] == 0.0) and np.all(g["accept"][noop] == 1)
    assert np.all(tr["dS"][noop] == 0.0)


@pytest.mark.parametrize("Ks", [(1, 7, 64, 128)])
def test_K_invariance(gpu_lib, Ks):
    """The accepted trajectory and every candidate's dS do not depend on the speculation width K."""
    wl, _ = _make("wide_ragged")
    ref = None
    for K in Ks:
        h = gpu_lib.create_from_workload(wl, K=K, trace_cap=1500)
        gpu_lib.mca_run(h, 1000, 3)
        gpu_lib.mca_run(h, 500, 3)
        g = gpu_lib.mca_get_trace(h, 1500)
        p = gpu_lib.mca_get_params(h, wl.n_params)
        out = (g, p, gpu_lib.mca_loss(h))
        if ref is None:
            ref = out
        else:
            assert np.array_equal(out[0], ref[0])
            assert np.array_equal(out[1], ref[1])
            assert out[2] == ref[2]
        h.close()


def test_batches_without_live_candidates_stay_in_step(gpu_lib):
    """Ternary proposals that keep the old code change nothing; with one candidate per batch a third
    of the batches have nothing to exchange. The CTAs must still advance batch by batch (the
    per-batch exchange buffers rotate), and the trajectory must equal the adaptive-width one."""
    wl, _ = _make("ternary")
    runs = []
    for kw in (dict(K=1, fixed_K=True), dict(K=64)):
        h = gpu_lib.create_from_workload(wl, trace_cap=3000, **kw)
        gpu_lib.mca_run(h, 3000, 5)
        runs.append((gpu_lib.mca_get_trace(h, 3000), gpu_lib.mca_get_codes(h, wl.n_params)))
        h.close()
    assert np.array_equal(runs[0][0], runs[1][0])
    assert np.array_equal(runs[0][1], runs[1][1])
    noop = runs[0][0]["old_w"] == runs[0][0]["new_w"]
    assert noop.sum() > 500


@pytest.mark.parametrize("grid", [1, 5, 0])
def test_grid_choices_match_oracle(gpu_lib, traces, grid):
    """The sample ranges (one CTA each) fix the summation order of dS; every choice of their
    number follows the oracle's trajectory, and repeats itself bit for bit."""
    wl, n, tr, params, S = traces("wide_ragged")
    m = 800
    sub = {k: v[:m] for k, v in tr.items()}
    runs = []
    for _ in range(2):
        h = gpu_lib.create_from_workload(wl, grid=grid, trace_cap=m)
        gpu_lib.mca_force_decisions(h, *forced_from_oracle(sub))
        gpu_lib.mca_run(h, m, wl.seed)
        runs.append(gpu_lib.mca_get_trace(h, m))
        h.close()
    compare(runs[0], sub)
    assert np.array_equal(runs[0], runs[1])


def test_eval_candidates_vs_oracle_and_no_commit(gpu_lib):
    wl, _ = _make("wide_ragged")
    h = gpu_lib.create_from_workload(wl)
    gpu_lib.mca_run(h, 400, 0)
    params = gpu_lib.mca_get_params(h, wl.n_params)
    L0 = gpu_lib.mca_loss(h)
    rng = np.random.default_rng(0)
    P1 = 784 * 256
    idx = np.concatenate([rng.integers(0, P1, 40), rng.integers(P1, wl.n_params, 24)])
    new = rng.uniform(-1, 1, len(idx)).astype(np.float32)
    new[0] = params[idx[0]]                           # a no-op candidate
    d1 = gpu_lib.mca_eval_candidates(h, idx, new)
    d2 = gpu_lib.mca_eval_candidates(h, idx, new)
    assert np.array_equal(d1, d2)
    assert d1[0] == 0.0
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params)
    assert gpu_lib.mca_loss(h) == L0
    op = O.Params(wl.layers, params)
    XT = wl.X.T.astype(np.float64)
    Z2 = O.output_fields_blocked(op, XT)
    S = L0 * wl.N
    for m in range(len(idx)):
        want = O.candidate_dS_two_layer(op, XT, wl.y, wl.loss, Z2, int(idx[m]), float(new[m]))
        assert abs(d1[m] - want) <= TIE_REL * S, (m, d1[m], want)


def test_rejects_leave_state_bit_identical(gpu_lib):
    wl, _ = _make("wide_ragged")
    h = gpu_lib.create_from_workload(wl, trace_cap=300)
    gpu_lib.mca_run(h, 200, 5)
    p0 = gpu_lib.mca_get_params(h, wl.n_params)
    L0 = gpu_lib.mca_loss(h)
    idx = np.arange(0, wl.n_params, 997)[:100].astype(np.uint32)
    new = np.linspace(-0.9, 0.9, len(idx)).astype(np.float32)
    d0 = gpu_lib.mca_eval_candidates(h, idx, new)
    gpu_lib.mca_force_decisions(h, np.arange(200, 500), np.zeros(300, bool))
    st = gpu_lib.mca_run(h, 300, 5)
    assert st["forced"] == 300
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), p0)
    assert gpu_lib.mca_loss(h) == L0
    assert np.array_equal(gpu_lib.mca_eval_candidates(h, idx, new), d0)


def test_resync_keeps_loss(gpu_lib):
    """Incrementally maintained fields agree with a fresh full forward pass within 1e-5."""
    wl, _ = _make("wide_ragged")
    h = gpu_lib.create_from_workload(wl)
    st = gpu_lib.mca_run(h, 3000, 1)
    assert st["accepts"] > 100
    L_inc = gpu_lib.mca_loss(h)
    gpu_lib.mca_resync(h)
    L_new = gpu_lib.mca_loss(h)
    assert L_inc == pytest.approx(L_new, rel=1e-6)
    S = O.total_loss(O.Params(wl.layers, gpu_lib.mca_get_params(h, wl.n_params)),
                     wl.X.T.astype(np.float64), wl.y, wl.loss)
    assert L_new == pytest.approx(S / wl.N, rel=1e-6)


def test_periodic_resync_parity(gpu_lib, traces):
    """With a resync every 700 trials the trajectory still matches the oracle."""
    wl, n, tr, params, S = traces("small_full")
    m = 3000
    h = gpu_lib.create_from_workload(wl, trace_cap=m, resync_period=700)
    gpu_lib.mca_force_decisions(h, *forced_from_oracle({k: v[:m] for k, v in tr.items()}))
    st = gpu_lib.mca_run(h, m, wl.seed)
    assert st["resyncs"] == m // 700
    compare(gpu_lib.mca_get_trace(h, m), {k: v[:m] for k, v in tr.items()})


def test_edge_cases(gpu_lib):
    import torch
    # ragged tiny N, a feature that is zero in every sample, K=128, trials not a multiple of K
    wl = W.mlp_wide(N=37, H=9)
    wl.X[:, 5] = 0.0
    tr, params, S = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, 1000, 2, wl.domain)
    h = gpu_lib.create_from_workload(wl, K=128, trace_cap=1000)
    gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr))
    gpu_lib.mca_run(h, 0, 2)
    gpu_lib.mca_run(h, 1000, 2)
    g = gpu_lib.mca_get_trace(h, 1000)
    compare(g, tr)
    on5 = (tr["idx"] < 784 * 9) & (tr["idx"] % 784 == 5)
    assert np.all(g["dS"][on5] == 0.0)
    # N = 1
    wl1 = W.mlp_small(N=1, H=3)
    tr1, p1, _ = O.run_incremental(wl1.layers, wl1.loss, wl1.X, wl1.y, wl1.init, 300, 0,
                                   wl1.domain)
    h1 = gpu_lib.create_from_workload(wl1, K=5, trace_cap=300)
    gpu_lib.mca_force_decisions(h1, *forced_from_oracle(tr1))
    gpu_lib.mca_run(h1, 300, 0)
    compare(gpu_lib.mca_get_trace(h1, 300), tr1)
    # host (numpy) inputs, device output buffer
    h2 = gpu_lib.mca_create(wl.layers, wl.loss, wl.domain, wl.X, wl.y, wl.init, K=4)
    out = torch.empty(wl.n_params, dtype=torch.float32, device="cuda")
    gpu_lib.mca_get_params(h2, wl.n_params, out)
    assert np.array_equal(out.cpu().numpy(), O.Params(wl.layers, wl.init).flat_eff32())


def test_strict_and_perturb_domain(gpu_lib):
    wl = W.mlp_small(N=300, H=12)
    dom = W.Domain(op="perturb", delta=0.05, bound=0.1, strict=True)
    tr, params, S = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, 2000, 4, dom)
    assert (~tr["valid"]).sum() > 10
    h = gpu_lib.mca_create(wl.layers, wl.loss, dom, wl.X, wl.y, wl.init, K=16, trace_cap=2000)
    gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr))
    gpu_lib.mca_run(h, 2000, 4)
    compare(gpu_lib.mca_get_trace(h, 2000), tr)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), params.flat_eff32())


def test_bad_inputs_rejected(gpu_lib):
    wl = W.mlp_small(N=50, H=4)
    with pytest.raises(gpu_lib.MCAError) as e:
        gpu_lib.mca_create(wl.layers, wl.loss, wl.domain, wl.X, wl.y, wl.init, K=0)
    assert e.value.status == gpu_lib.MCA_ERR_INVALID
    with pytest.raises(gpu_lib.MCAError):
        gpu_lib.mca_create(wl.layers, wl.loss, wl.domain, wl.X, wl.y, wl.init, K=129)
    y = wl.y.copy()
    y[3] = 10
    with pytest.raises(gpu_lib.MCAError) as e:
        gpu_lib.mca_create(wl.layers, wl.loss, wl.domain, wl.X, y, wl.init)
    assert e.value.status == gpu_lib.MCA_ERR_INVALID
    X = wl.X.copy()
    X[2, 3] = np.nan
    with pytest.raises(gpu_lib.MCAError) as e:
        gpu_lib.mca_create(wl.layers, wl.loss, wl.domain, X, wl.y, wl.init)
    assert e.value.status == gpu_lib.MCA_ERR_NUMERIC
    init = wl.init.copy()
    init[7] = np.inf
    with pytest.raises(gpu_lib.MCAError) as e:
        gpu_lib.mca_create(wl.layers, wl.loss, wl.domain, wl.X, wl.y, init)
    assert e.value.status == gpu_lib.MCA_ERR_NUMERIC


def test_set_params_resume(gpu_lib):
    """Resume from (params, codes, tau) equals an uninterrupted run when the checkpoint is at a
    resync boundary (both sides then start from freshly computed fields)."""
    wl, _ = _make("masked")
    h = gpu_lib.create_from_workload(wl, trace_cap=2000, resync_period=1000)
    gpu_lib.mca_run(h, 2000, 9)
    full = gpu_lib.mca_get_trace(h, 2000)
    h2 = gpu_lib.create_from_workload(wl, trace_cap=1000, resync_period=1000)
    gpu_lib.mca_run(h2, 1000, 9)
    p = gpu_lib.mca_get_params(h2, wl.n_params)
    c = gpu_lib.mca_get_codes(h2, wl.n_params)
    fixed = wl.init.copy()                           # masked layers resume from fixed weights
    h3 = gpu_lib.create_from_workload(wl, trace_cap=1000, resync_period=1000)
    gpu_lib.mca_set_params(h3, fixed, c, tau=1000)
    assert np.array_equal(gpu_lib.mca_get_params(h3, wl.n_params), p)
    gpu_lib.mca_run(h3, 1000, 9)
    assert np.array_equal(gpu_lib.mca_get_trace(h3, 1000), full[1000:])
