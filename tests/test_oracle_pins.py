"""Pins of the CPU oracle against things other than itself (CPU only).

Each test ties one part of the oracle to a published vector, a library routine, a closed form,
brute-force enumeration or an invariant of the method, chosen so that a plausible mistake (a dropped
term, a wrong sign or index, a transposed operand) fails at least one of them.
"""
import itertools
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- Philox (proposal stream)

def _kat_rows():
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            v = [int(t, 16) for t in line.split()]
            rows.append((v[0:4], v[4:6], v[6:10]))
    return rows


@pytest.mark.parametrize("ctr,key,want", _kat_rows())
def test_philox_known_answers(ctr, key, want):
    got = [int(w) for w in oracle.philox4x32_10(ctr, key)]
    assert got == want


def test_philox_vectorised_equals_scalar():
    taus = np.arange(1000, dtype=np.uint64) * np.uint64(7919) + np.uint64(2 ** 33 + 5)
    many = O.draw_words(12345, taus)
    for t in (0, 17, 999):
        one = O.draw_words(12345, int(taus[t]))
        assert (one == many[t]).all()


def test_counter_high_word_matters():
    # tau and tau + 2^32 must give different words (the counter's second word is used)
    a = O.draw_words(3, 5)
    b = O.draw_words(3, 5 + 2 ** 32)
    assert not (a == b).all()


# ---------------------------------------------------------------- proposal mapping (Eq. 1)

def _net(dims, acts, wkind="fp32", scale=1.0):
    return [W.Layer(dims[l], dims[l + 1], acts[l], 1.0 if acts[l] == "gaussian" else 0.0, wkind,
                    scale) for l in range(len(dims) - 1)]


def test_proposal_touches_exactly_flat_index():
    """Applying a proposal changes the flat parameter vector at position idx only (flat order:
    layers in forward order, [out x in] row-major). A swapped row/col decode fails this."""
    layers = _net([7, 5, 3], ["tanh", "identity"])
    rng = np.random.default_rng(0)
    init = rng.uniform(-0.1, 0.1, size=7 * 5 + 5 * 3).astype(np.float32)
    params = O.Params(layers, init)
    dom = W.Domain()
    seen_layers = set()
    for tau in range(300):
        p = O.propose(7, tau, params, dom)
        before = params.flat_eff32().copy()
        O.apply_proposal(params, p)
        after = params.flat_eff32()
        diff = np.nonzero(before != after)[0]
        assert list(diff) == [p.idx]
        assert after[p.idx] == np.float32(p.new)
        assert before[p.idx] == np.float32(p.old)
        O.revert_proposal(params, p)
        assert (params.flat_eff32() == before).all()
        seen_layers.add(p.layer)
    assert seen_layers == {0, 1}


def test_index_uniform_chi2():
    """idx is uniform over the P parameters (chi-square over 2e5 draws, P = 97)."""
    P = 97
    r = O.draw_words(11, np.arange(200_000, dtype=np.uint64))
    idx = (r[:, 0].astype(object) * P) >> 32
    counts = np.bincount(np.asarray(idx, dtype=np.int64), minlength=P)
    expect = len(idx) / P
    chi2 = float(((counts - expect) ** 2 / expect).sum())
    # 96 dof: mean 96, sd ~13.9; 6 sd is far outside sampling noise
    assert chi2 < 96 + 6 * 13.9
    assert counts.min() > 0


def test_replacement_values_exact_and_in_range():
    layers = _net([4, 3], ["identity"])
    params = O.Params(layers, np.zeros(12, np.float32))
    dom = W.Domain()
    vals = np.array([O.propose(5, t, params, dom).new for t in range(5000)])
    assert vals.min() >= -1.0 and vals.max() < 1.0
    # every value is a multiple of 2^-23 (exact dyadic grid of the U[-1,1) draw)
    assert np.all(vals * 2.0 ** 23 == np.round(vals * 2.0 ** 23))
    # uniform: mean ~ 0, variance ~ 1/3
    assert abs(vals.mean()) < 0.05
    assert abs(vals.var() - 1.0 / 3.0) < 0.02


def test_replacement_end_points():
    """r1 = 0 maps to lo, r1 = 2^32-1 maps to hi - 2^-23 (for [-1, 1))."""
    f32 = np.float32
    for r1, want in ((0, -1.0), (0xFFFFFFFF, 1.0 - 2.0 ** -23), (0x80000000, 0.0)):
        u = f32(r1 >> 8) * f32(2.0 ** -24)
        v = f32(f32(-1.0) + f32(f32(2.0) * u))
        assert float(v) == want


def test_ternary_codes_uniform():
    layers = _net([5, 4], ["identity"], "ternary_i8", 0.25)
    params = O.Params(layers, np.zeros(20, np.float32))
    codes = np.array([O.propose(9, t, params, W.Domain()).new_code for t in range(6000)])
    assert set(np.unique(codes)) == {-1, 0, 1}
    frac = np.bincount(codes + 1) / len(codes)
    assert np.all(np.abs(frac - 1 / 3) < 0.03)


def test_perturb_domain_rejects():
    """Eq. 1's constraint |w| < Delta: every accepted weight stays inside the bound, and a proposal
    outside it is rejected without evaluation."""
    layers = _net([6, 3, 2], ["tanh", "sigmoid"])
    wl = W.mlp_small(N=30, H=3, D=6)
    dom = W.Domain(op="perturb", delta=0.05, bound=0.08)
    init = np.full(6 * 3 + 3 * 2, 0.07, np.float32)
    tr, params, S = O.run_full(layers, "mse_onehot", wl.X, wl.y % 2, init, 600, 1, dom)
    assert (~tr["valid"]).sum() > 0
    assert np.all(np.isnan(tr["dS"][~tr["valid"]]))
    assert not tr["accept"][~tr["valid"]].any()
    assert np.all(np.abs(params.flat_eff32()) < 0.08 + 1e-7)


# ---------------------------------------------------------------- transfer functions and losses

def test_act_closed_forms():
    z = np.array([0.0, 1.0, -2.0])
    assert np.allclose(O.act_fn("gaussian", z, 1.0), [1.0, math.exp(-1.0), math.exp(-4.0)])
    assert np.allclose(O.act_fn("gaussian", z, 0.4), [1.0, math.exp(-0.4), math.exp(-1.6)])
    assert O.act_fn("tanh", np.array([0.0]))[0] == 0.0
    assert O.act_fn("sigmoid", np.array([0.0]))[0] == 0.5
    assert np.allclose(O.act_fn("relu", z), [0.0, 1.0, 0.0])


def test_act_vs_torch():
    z = np.linspace(-6, 6, 1001)
    t = torch.from_numpy(z)
    assert np.allclose(O.act_fn("tanh", z), torch.tanh(t).numpy(), rtol=0, atol=1e-15)
    assert np.allclose(O.act_fn("sigmoid", z), torch.sigmoid(t).numpy(), rtol=1e-14, atol=1e-16)
    assert np.allclose(O.act_fn("gelu", z), torch.nn.functional.gelu(t).numpy(), rtol=1e-13,
                       atol=1e-15)


def test_loss_closed_forms():
    """All-zero weights: sigmoid outputs 0.5 -> MSE per sample = 9 * 0.25 + 0.25 = 2.5;
    identity outputs 0 -> CE per sample = ln 10."""
    wl = W.mlp_small(N=50, H=8)
    z = np.zeros(wl.n_params, np.float32)
    XT = wl.X.T.astype(np.float64)
    S = O.total_loss(O.Params(wl.layers, z), XT, wl.y, "mse_onehot")
    assert S == pytest.approx(50 * 2.5, rel=1e-15)
    layers = _net([784, 8, 10], ["tanh", "identity"])
    S = O.total_loss(O.Params(layers, z), XT, wl.y, "softmax_ce")
    assert S == pytest.approx(50 * math.log(10.0), rel=1e-14)


def test_losses_vs_torch():
    rng = np.random.default_rng(3)
    out = rng.normal(size=(10, 64)) * 3.0
    y = rng.integers(0, 10, size=64)
    ce = O.loss_per_sample("softmax_ce", out, y)
    ref = torch.nn.functional.cross_entropy(torch.from_numpy(out.T), torch.from_numpy(y),
                                            reduction="none").numpy()
    assert np.allclose(ce, ref, rtol=1e-13, atol=1e-13)
    a = 1.0 / (1.0 + np.exp(-out))
    mse = O.loss_per_sample("mse_onehot", a, y)
    oh = torch.nn.functional.one_hot(torch.from_numpy(y), 10).double()
    ref = ((torch.from_numpy(a.T) - oh) ** 2).sum(dim=1).numpy()
    assert np.allclose(mse, ref, rtol=1e-14)
    ref2 = torch.nn.functional.mse_loss(torch.from_numpy(a.T), oh, reduction="sum").item()
    assert mse.sum() == pytest.approx(ref2, rel=1e-13)


def test_ce_two_class_is_logistic():
    """Two-class softmax CE reduces to log(1 + exp(-(z_y - z_other)))."""
    rng = np.random.default_rng(5)
    out = rng.normal(size=(2, 40)) * 4
    y = rng.integers(0, 2, 40)
    m = out[y, np.arange(40)] - out[1 - y, np.arange(40)]
    assert np.allclose(O.loss_per_sample("softmax_ce", out, y), np.log1p(np.exp(-m)), rtol=1e-12)


# ---------------------------------------------------------------- forward pass vs torch.nn

def _torch_mlp(layers, params):
    mods = []
    acts = {"tanh": torch.nn.Tanh(), "sigmoid": torch.nn.Sigmoid(), "identity": torch.nn.Identity(),
            "relu": torch.nn.ReLU(), "gelu": torch.nn.GELU()}
    for l, L in enumerate(layers):
        lin = torch.nn.Linear(L.n_in, L.n_out, bias=False).double()
        with torch.no_grad():
            lin.weight.copy_(torch.from_numpy(params.eff64(l)))
        mods.append(lin)
        mods.append(acts[L.act])
    return torch.nn.Sequential(*mods)


@pytest.mark.parametrize("dims,acts", [([3, 2, 2], ["tanh", "sigmoid"]),
                                       ([4, 3, 2], ["tanh", "identity"]),
                                       ([6, 5, 4, 3], ["relu", "gelu", "identity"])])
def test_forward_vs_torch_tiny(dims, acts):
    layers = _net(dims, acts)
    rng = np.random.default_rng(sum(dims))
    n = sum(a * b for a, b in zip(dims[:-1], dims[1:]))
    params = O.Params(layers, rng.uniform(-1, 1, n).astype(np.float32))
    X = rng.random((5, dims[0]))
    _, out = O.forward(params, X.T.copy())
    ref = _torch_mlp(layers, params)(torch.from_numpy(X)).detach().numpy().T
    assert np.allclose(out, ref, rtol=1e-13, atol=1e-15)


def test_forward_gaussian_brute_force():
    """A Gaussian hidden layer written out neuron by neuron in plain Python."""
    layers = [W.Layer(3, 2, "gaussian", 0.7), W.Layer(2, 2, "sigmoid")]
    rng = np.random.default_rng(1)
    init = rng.uniform(-1, 1, 10).astype(np.float32)
    params = O.Params(layers, init)
    X = rng.random((4, 3))
    _, out = O.forward(params, X.T.copy())
    w1 = init[:6].astype(float).reshape(2, 3)
    w2 = init[6:].astype(float).reshape(2, 2)
    for n in range(4):
        h = [math.exp(-0.7 * sum(w1[j][i] * X[n][i] for i in range(3)) ** 2) for j in range(2)]
        for k in range(2):
            s = sum(w2[k][j] * h[j] for j in range(2))
            assert out[k, n] == pytest.approx(1.0 / (1.0 + math.exp(-s)), rel=1e-14)


def test_linear_net_associativity():
    """Identity transfer functions: the net is the single matrix W3 W2 W1."""
    layers = _net([6, 5, 4, 3], ["identity"] * 3)
    rng = np.random.default_rng(2)
    init = rng.uniform(-1, 1, 30 + 20 + 12).astype(np.float32)
    params = O.Params(layers, init)
    X = rng.random((7, 6))
    _, out = O.forward(params, X.T.copy())
    M = params.eff64(2) @ (params.eff64(1) @ params.eff64(0))
    assert np.allclose(out, M @ X.T, rtol=1e-13)


# ---------------------------------------------------------------- selection (Eq. 6) by enumeration

def test_greedy_trajectory_matches_enumeration():
    """A 2-2-2 ternary net has 3^8 states. The loss of every state is enumerated with torch; the
    oracle's greedy trajectory must accept exactly when S(new state) <= S(old state)."""
    layers = [W.Layer(2, 2, "tanh", 0.0, "ternary_i8", 0.5),
              W.Layer(2, 2, "sigmoid", 0.0, "ternary_i8", 0.5)]
    rng = np.random.default_rng(4)
    X = rng.random((6, 2)).astype(np.float32)
    y = np.array([0, 1, 1, 0, 1, 0], np.int32)
    Xt = torch.from_numpy(X.astype(np.float64))
    oh = torch.nn.functional.one_hot(torch.from_numpy(y).long(), 2).double()
    table = {}
    for codes in itertools.product((-1, 0, 1), repeat=8):
        w1 = torch.tensor(codes[:4], dtype=torch.float64).reshape(2, 2) * 0.5
        w2 = torch.tensor(codes[4:], dtype=torch.float64).reshape(2, 2) * 0.5
        out = torch.sigmoid(torch.tanh(Xt @ w1.T) @ w2.T)
        table[codes] = ((out - oh) ** 2).sum().item()
    init = np.array([1, -1, 0, 1, 0, 1, -1, 1], np.float32)
    for run in (O.run_full, O.run_incremental):
        tr, params, S = run(layers, "mse_onehot", X, y, init, 400, 21, W.Domain())
        state = tuple(int(c) for c in init)
        for t in range(400):
            new = list(state)
            new[int(tr["idx"][t])] = int(tr["new_code"][t])
            new = tuple(new)
            S_old, S_new = table[state], table[new]
            assert tr["S"][t] == pytest.approx(S_old, rel=1e-12, abs=1e-12)
            if abs(S_new - S_old) > 1e-12:
                assert bool(tr["accept"][t]) == (S_new <= S_old), t
            if tr["accept"][t]:
                state = new
        assert tuple(int(c) for c in params.flat_codes()) == state
        assert tr["accept"].sum() > 10


# ---------------------------------------------------------------- invariants of the trial loop

@pytest.mark.parametrize("name,kw", [
    ("mlp_small", dict(N=120, H=12)),
    ("mlp_wide", dict(N=150, H=40)),
    ("mlp_deep", dict(N=80, width=16, depth=3)),
    ("mlp_ternary", dict(N=150, H=20)),
    ("mlp_masked", dict(N=150, H=20)),
])
def test_incremental_equals_full(name, kw):
    wl = W.make(name, **kw)
    tf, pf, Sf = O.run_full(wl.layers, wl.loss, wl.X, wl.y, wl.init, 300, 0, wl.domain)
    ti, pi, Si = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, 300, 0, wl.domain,
                                   check_every=50)
    assert (tf["idx"] == ti["idx"]).all()
    scale = np.abs(tf["S"]).max()
    both = np.abs(tf["dS"]) > 1e-9 * scale
    assert (tf["accept"][both] == ti["accept"][both]).all()
    assert np.allclose(tf["dS"], ti["dS"], rtol=0, atol=1e-9 * scale)
    assert Sf == pytest.approx(Si, rel=1e-10)
    assert (pf.flat_eff32() == pi.flat_eff32()).all()
    assert tf["accept"].sum() > 0


def test_accepted_loss_monotone_and_rejects_leave_state():
    wl = W.mlp_small(N=100, H=10)
    tr, _, _ = O.run_full(wl.layers, wl.loss, wl.X, wl.y, wl.init, 200, 0, wl.domain)
    S = tr["S"]
    assert np.all(np.diff(S) <= 0.0)                       # accepted S never rises
    rej = ~tr["accept"][:-1]
    assert np.all(S[1:][rej] == S[:-1][rej])               # a reject leaves S bit-identical
    # step by step: a rejected trial leaves every parameter bit-identical
    params = O.Params(wl.layers, wl.init)
    n_rej = 0
    for tau in range(120):
        snap = [v.copy() for v in params.vals]
        tr1, params, _ = O.run_full(wl.layers, wl.loss, wl.X, wl.y, None, 1, 0, wl.domain,
                                    tau0=tau, params=params)
        assert tr1["accept"][0] == tr["accept"][tau]
        if not tr1["accept"][0]:
            n_rej += 1
            assert all((a.view(np.uint8) == b.view(np.uint8)).all()
                       for a, b in zip(snap, params.vals))
    assert n_rej > 10


def test_noop_ternary_trials_are_exact_zero():
    """A ternary proposal equal to the old code leaves every field unchanged: dS == 0 exactly in
    both modes, and it is accepted under the <= rule (Eq. 6)."""
    wl = W.mlp_ternary(N=90, H=12)
    for run in (O.run_full, O.run_incremental):
        tr, _, _ = run(wl.layers, wl.loss, wl.X, wl.y, wl.init, 300, 0, wl.domain)
        noop = tr["old"] == tr["new"]
        assert noop.sum() > 30
        assert np.all(tr["dS"][noop] == 0.0)
        assert np.all(tr["accept"][noop])


def test_strict_rule_rejects_noops():
    wl = W.mlp_ternary(N=60, H=8)
    dom = W.Domain(strict=True)
    tr, _, _ = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, 200, 0, dom)
    noop = tr["old"] == tr["new"]
    assert noop.sum() > 10 and not tr["accept"][noop].any()


def test_layer1_fields_exact_on_dyadic_grid():
    """Ternary/masked workloads: inputs k/256 and dyadic weights make every first-layer field an
    exact fp32 value (sums of at most 784 terms of a 2^-17 grid below 2^24 units)."""
    for name in ("mlp_ternary", "mlp_masked"):
        wl = W.make(name, N=64, H=32)
        params = O.Params(wl.layers, wl.init)
        Z, _ = O.forward(params, wl.X.T.astype(np.float64))
        z1 = Z[0]
        assert np.all(z1.astype(np.float32).astype(np.float64) == z1)
        assert np.all(np.abs(z1) * 2 ** 17 < 2 ** 24)


# ---------------------------------------------------------------- the pins have teeth

def test_planted_sign_error_is_caught(monkeypatch):
    """Planting a sign error in the CE loss makes the torch pin fail."""
    orig = O.loss_per_sample

    def bad(kind, out, y):
        if kind == "softmax_ce":
            m = out.max(axis=0)
            return m + np.log(np.exp(out - m).sum(axis=0)) + out[y, np.arange(out.shape[1])]
        return orig(kind, out, y)

    monkeypatch.setattr(O, "loss_per_sample", bad)
    with pytest.raises(AssertionError):
        test_losses_vs_torch()


def test_planted_transposed_decode_is_caught(monkeypatch):
    """Planting a transposed (row, col) decode in the proposal makes the flat-index pin fail."""
    orig = O.propose

    def bad(seed, tau, params, domain):
        p = orig(seed, tau, params, domain)
        L = params.layers[p.layer]
        off = p.idx - params.offsets[p.layer]
        p.col, p.row = divmod(off, L.n_out)
        if p.row >= L.n_out or p.col >= L.n_in:
            p.row, p.col = p.row % L.n_out, p.col % L.n_in
        return p

    monkeypatch.setattr(O, "propose", bad)
    with pytest.raises(AssertionError):
        test_proposal_touches_exactly_flat_index()


def test_planted_dropped_rank1_term_is_caught(monkeypatch):
    """Dropping the next-layer rank-1 term (W[:, j] times the activation change) from the
    incremental mode breaks incremental == full."""
    real_outer = np.outer
    monkeypatch.setattr(O.np, "outer", lambda a, b: np.zeros_like(real_outer(a, b)))
    with pytest.raises(AssertionError):
        test_incremental_equals_full("mlp_small", dict(N=60, H=6))


def test_blocked_single_candidate_helpers_match_full_recompute():
    """output_fields_blocked equals the full forward's output fields, and candidate_dS_two_layer
    equals S(W') - S(W) from two full forward passes, for first- and output-layer weights."""
    wl = W.mlp_wide(N=400, H=37)
    p = O.Params(wl.layers, wl.init)
    XT = wl.X.T.astype(np.float64)
    Z2 = O.output_fields_blocked(p, XT, block=8)
    Zs, _ = O.forward(p, XT)
    assert np.allclose(Z2, Zs[1], rtol=0, atol=1e-13)
    S = O.total_loss(p, XT, wl.y, wl.loss)
    P1 = 784 * 37
    for idx, v in ((5, 0.37), (P1 - 1, -0.8), (P1 + 3, 0.9), (wl.n_params - 1, -0.2)):
        q = p.copy()
        l, off = (0, idx) if idx < P1 else (1, idx - P1)
        q.vals[l].reshape(-1)[off] = np.float32(v)
        want = O.total_loss(q, XT, wl.y, wl.loss) - S
        got = O.candidate_dS_two_layer(p, XT, wl.y, wl.loss, Z2, idx, float(np.float32(v)))
        assert got == pytest.approx(want, rel=1e-9, abs=1e-10)
