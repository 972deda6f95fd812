"""Pins of the oracle's Metropolis rule (Section 3.1, Eq. 7), CPU only.

Eq. 7 keeps a mutation with probability min{1, exp(-beta dL)}. The oracle draws the trial's uniform
number from the fourth Philox word of its counter and turns it into a threshold theta_tau on the
loss-sum change (keep iff dS <= theta_tau). These tests tie that threshold to the acceptance
probability Eq. 7 prescribes (a statistical test over many counters), to the greedy rule in the
beta -> infinity limit, and to brute-force enumeration of a tiny ternary net's states.
"""
import dataclasses
import itertools
import math

import numpy as np
import pytest
import torch
from scipy import stats

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

TAUS = np.arange(200_000)


def test_threshold_gives_the_metropolis_acceptance_probability():
    """Over 2e5 counters the fraction of trials whose threshold admits a change dS equals
    min{1, exp(-beta dS / N)} within 5 binomial standard deviations, for several beta, N and dS;
    downhill and zero changes are always admitted; and exp(-beta theta / N) -- the uniform number
    the threshold was made from -- is uniform on (0, 1) (Kolmogorov-Smirnov)."""
    for beta, N in ((2.0, 10), (0.5, 1000), (40.0, 7)):
        th = O.metropolis_threshold(3, TAUS, beta, N)
        assert np.all(th > 0.0)
        for dL in (-0.5, 0.0):
            assert np.all(dL * N <= th)
        for dL in (0.01, 0.2, 1.0, 3.0):
            p = math.exp(-beta * dL)
            f = float(np.mean(dL * N <= th))
            sig = math.sqrt(p * (1.0 - p) / len(TAUS))
            assert abs(f - p) <= 5.0 * sig + 1e-6, (beta, N, dL, f, p)
        u = np.exp(-beta * th / N)
        assert stats.kstest(u, "uniform").pvalue > 1e-4


def test_infinite_and_large_beta_give_the_greedy_rule():
    """beta = inf is the greedy rule exactly; a huge finite beta (threshold ~1e-28) takes the same
    decisions as greedy on a real workload."""
    assert O.metropolis_threshold(0, 5, float("inf"), 100) == 0.0
    wl = W.mlp_small(N=100, H=10)
    g, pg, Sg = O.run_full(wl.layers, wl.loss, wl.X, wl.y, wl.init, 150, 0, wl.domain)
    big = dataclasses.replace(wl.domain, beta=1e30)
    m, pm, Sm = O.run_full(wl.layers, wl.loss, wl.X, wl.y, wl.init, 150, 0, big)
    assert (g["idx"] == m["idx"]).all() and (g["accept"] == m["accept"]).all()
    assert Sg == Sm and (pg.flat_eff32() == pm.flat_eff32()).all()


def _ternary_table():
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
    return layers, X, y, table


def test_metropolis_trajectory_matches_enumeration():
    """The 3^8 states of a 2-2-2 ternary net are enumerated with torch. Under beta = 20 both oracle
    modes accept trial tau exactly when S(new) - S(old) <= theta_tau, and some uphill mutations are
    kept (the point of the rule)."""
    layers, X, y, table = _ternary_table()
    beta, n, seed = 20.0, 600, 21
    dom = W.Domain(beta=beta)
    theta = O.metropolis_threshold(seed, np.arange(n), beta, len(y))
    init = np.array([1, -1, 0, 1, 0, 1, -1, 1], np.float32)
    for run in (O.run_full, O.run_incremental):
        tr, params, S = run(layers, "mse_onehot", X, y, init, n, seed, dom)
        state = tuple(int(c) for c in init)
        uphill = 0
        for t in range(n):
            new = list(state)
            new[int(tr["idx"][t])] = int(tr["new_code"][t])
            new = tuple(new)
            d = table[new] - table[state]
            assert tr["S"][t] == pytest.approx(table[state], rel=1e-12, abs=1e-12)
            if abs(d - theta[t]) > 1e-12:
                assert bool(tr["accept"][t]) == (d <= theta[t]), t
            if tr["accept"][t]:
                uphill += d > 1e-12
                state = new
        assert tuple(int(c) for c in params.flat_codes()) == state
        assert uphill > 5


def test_metropolis_incremental_equals_full():
    """The cached-field mode takes the full mode's Metropolis decisions on a real workload."""
    wl = W.mlp_small(N=120, H=12)
    dom = dataclasses.replace(wl.domain, beta=2000.0)
    tf, pf, Sf = O.run_full(wl.layers, wl.loss, wl.X, wl.y, wl.init, 300, 0, dom)
    ti, pi, Si = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, 300, 0, dom)
    th = O.metropolis_threshold(0, np.arange(300), 2000.0, 120)
    clear = np.abs(tf["dS"] - th) > 1e-9 * np.abs(tf["S"]).max()
    assert (tf["accept"][clear] == ti["accept"][clear]).all()
    assert (pf.flat_eff32() == pi.flat_eff32()).all()
    assert ((tf["dS"] > 0) & tf["accept"]).sum() > 0       # uphill moves were kept


def test_planted_missing_sample_count_is_caught(monkeypatch):
    """A threshold on dS instead of dL = dS / N (the sample count dropped) fails the probability
    pin."""
    orig = O.metropolis_threshold
    monkeypatch.setattr(O, "metropolis_threshold", lambda s, t, b, N: orig(s, t, b, 1))
    with pytest.raises(AssertionError):
        test_threshold_gives_the_metropolis_acceptance_probability()


def test_planted_wrong_counter_is_caught(monkeypatch):
    """Drawing trial tau's uniform number from the counter tau + 1 fails the enumeration pin."""
    orig = O._threshold
    monkeypatch.setattr(O, "_threshold", lambda s, t, d, N: orig(s, t + 1, d, N))
    with pytest.raises(AssertionError):
        test_metropolis_trajectory_matches_enumeration()


# ---- the Transformer oracle under Eq. 7 (N = predicted tokens, B sequences x T positions)

from oracle import mca_tfm as T  # noqa: E402

TFM_TINY = W.TfmSpec(vocab=11, ctx=6, d_model=8, n_layer=1, n_head=2, d_ff=16)


def _tfm_run(beta, n=400, tokens=None):
    wl = W.char_transformer(seed=1, batch=4, text_len=4000, spec=TFM_TINY, n_trials=n, K=8)
    tok = wl.tokens if tokens is None else tokens
    dom = dataclasses.replace(wl.domain, beta=beta)
    return wl, T.run_full_tfm(TFM_TINY, tok, wl.init, n, wl.seed, dom)


def test_tfm_metropolis_limits():
    """A huge beta takes the greedy trajectory (Eq. 6); a tiny beta (theta above any loss change)
    keeps every valid proposal, so the final parameters are the initial ones with every valid
    proposal applied in order."""
    wl, (tg, fg, Sg) = _tfm_run(float("inf"), n=150)
    _, (tb, fb, Sb) = _tfm_run(1e30, n=150)
    assert (tg["accept"] == tb["accept"]).all() and (fg == fb).all() and Sg == Sb
    assert 0 < tg["accept"].sum() < tg["valid"].sum()
    _, (tt, ft, St) = _tfm_run(1e-30, n=150)
    assert (tt["accept"] == tt["valid"]).all()
    want = np.array(wl.init, dtype=np.float32)
    for i, v, ok in zip(tt["idx"], tt["new"], tt["valid"]):
        if ok:
            want[int(i)] = np.float32(v)
    assert (ft == want).all()


def test_tfm_metropolis_acceptance_probability():
    """Eq. 7 on the mean loss per predicted token (L = S / (B T)): given the chain's past, trial t
    is kept with probability p_t = min{1, exp(-beta dS_t / (B T))}. The number of kept trials must
    match sum p_t within 5 standard deviations of the Poisson-binomial sum, and uphill moves must
    be among them."""
    beta = 400.0
    wl, (tr, _, _) = _tfm_run(beta)
    v = tr["valid"]
    n_tok = wl.tokens.shape[0] * TFM_TINY.ctx
    p = np.minimum(1.0, np.exp(-beta * tr["dS"][v] / n_tok))
    kept = tr["accept"][v].sum()
    sig = math.sqrt(float((p * (1.0 - p)).sum()))
    assert abs(kept - p.sum()) <= 5.0 * sig + 1.0, (kept, p.sum(), sig)
    uphill = (tr["dS"] > 0) & tr["accept"]
    assert uphill.sum() > 10
    assert ((p > 0.05) & (p < 0.95)).sum() > 50       # the test is not decided by the limits


def test_tfm_metropolis_batch_duplication_invariance():
    """Repeating every sequence doubles S, each dS and the token count B T, so Eq. 7's decisions
    do not change (trials within 1e-9 of their threshold excepted)."""
    wl, (t1, f1, S1) = _tfm_run(400.0, n=200)
    tok2 = np.concatenate([wl.tokens, wl.tokens])
    _, (t2, f2, S2) = _tfm_run(400.0, n=200, tokens=tok2)
    assert S2 == pytest.approx(2.0 * S1, rel=1e-12)
    assert (t1["accept"] == t2["accept"]).all() and (f1 == f2).all()


def test_planted_sequence_count_for_token_count_is_caught(monkeypatch):
    """Taking N = B sequences instead of B T predicted tokens fails the probability pin."""
    orig = T.metropolis_threshold
    monkeypatch.setattr(T, "metropolis_threshold",
                        lambda s, t, b, N: orig(s, t, b, N // TFM_TINY.ctx))
    with pytest.raises(AssertionError):
        test_tfm_metropolis_acceptance_probability()
