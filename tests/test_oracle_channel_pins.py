"""Pins of the oracle's multi-parameter channel mutations (Section 2.3), CPU only.

A channel is a path from one input through one node of every hidden layer to one output; a trial
changes the weight of every layer on that path (He-normalised redraws, or all set to zero) and is
kept iff the loss does not increase. These tests tie the oracle to that: the changed weights form a
path with one weight per layer, the nodes are uniform, the redrawn values are uniform within He's
amplitude, the zero scheme only removes weights, and every decision agrees with losses computed by
an independent torch forward pass.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as Fn
from scipy import stats

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W


def _net(n_in=7, widths=(5, 3), n_out=4, N=24, seed=0):
    dims = [n_in, *widths, n_out]
    layers = [W.Layer(dims[m], dims[m + 1], "tanh" if m + 1 < len(dims) - 1 else "identity")
              for m in range(len(dims) - 1)]
    rng = np.random.default_rng(seed)
    init = np.concatenate([rng.uniform(-0.5, 0.5, L.n_in * L.n_out) for L in layers]).astype(
        np.float32)
    X = rng.uniform(0, 1, (N, n_in)).astype(np.float32)
    y = rng.integers(0, n_out, N).astype(np.int32)
    return layers, init, X, y


@pytest.mark.parametrize("scheme", ["he", "zero"])
def test_channel_is_a_path_with_one_weight_per_layer(scheme):
    layers, init, X, y = _net()
    params = O.Params(layers, init)
    for tau in range(500):
        ch = O.propose_channel(3, tau, params, scheme)
        assert [c[0] for c in ch] == list(range(len(layers)))
        for (m, r, c, old, new), L in zip(ch, layers):
            assert 0 <= r < L.n_out and 0 <= c < L.n_in
            assert old == float(params.vals[m][r, c])
        for a, b in zip(ch[:-1], ch[1:]):
            assert b[2] == a[1]                    # the next layer leaves from this layer's node


def test_channel_nodes_uniform():
    layers, init, X, y = _net()
    params = O.Params(layers, init)
    n = 20_000
    nodes = np.array([[c[2] for c in O.propose_channel(8, t, params, "zero")] +
                      [O.propose_channel(8, t, params, "zero")[-1][1]] for t in range(n)])
    sizes = [layers[0].n_in] + [L.n_out for L in layers]
    for m, k in enumerate(sizes):
        assert stats.chisquare(np.bincount(nodes[:, m], minlength=k)).pvalue > 1e-4, m


def test_he_values_uniform_within_amplitude_and_zero_scheme():
    layers, init, X, y = _net(n_in=50, widths=(20,), n_out=6)
    params = O.Params(layers, init)
    vals = np.array([[c[4] for c in O.propose_channel(5, t, params, "he")] for t in range(20_000)])
    for m, L in enumerate(layers):
        a = np.sqrt(6.0 / L.n_in)
        assert np.all(np.abs(vals[:, m]) <= a * (1 + 1e-7))
        h = np.histogram(vals[:, m] / a, bins=10, range=(-1.0, 1.0))[0]
        assert stats.chisquare(h).pvalue > 1e-4
    zeros = [[c[4] for c in O.propose_channel(5, t, params, "zero")] for t in range(100)]
    assert np.all(np.array(zeros) == 0.0)


def _torch_loss(layers, flat, X, y):
    a = torch.from_numpy(X.astype(np.float64))
    o = 0
    for L in layers:
        Wm = torch.from_numpy(flat[o:o + L.n_in * L.n_out].astype(np.float64)).reshape(L.n_out,
                                                                                      L.n_in)
        o += L.n_in * L.n_out
        z = Fn.linear(a, Wm)
        a = torch.tanh(z) if L.act == "tanh" else z
    return float(Fn.cross_entropy(a, torch.from_numpy(y.astype(np.int64)), reduction="sum"))


@pytest.mark.parametrize("scheme", ["he", "zero"])
def test_channel_decisions_follow_an_independent_forward(scheme):
    """Replaying the trials on a flat copy: each kept trial's channel lowered (or kept) the loss
    computed by torch, each rejected one raised it, and the final parameters are the initial ones
    with exactly the kept channels applied."""
    layers, init, X, y = _net()
    rows, params, S = O.run_channel(layers, "softmax_ce", X, y, init, 300, 11, scheme)
    offs = np.cumsum([0] + [L.n_in * L.n_out for L in layers])
    flat = init.astype(np.float32).copy()
    kept = 0
    for tau, ch, S_before, dS, acc in rows:
        before = _torch_loss(layers, flat, X, y)
        trial = flat.copy()
        for m, r, c, old, new in ch:
            trial[offs[m] + r * layers[m].n_in + c] = np.float32(new)
        after = _torch_loss(layers, trial, X, y)
        assert S_before == pytest.approx(before, rel=1e-12)
        if abs(after - before) > 1e-9 * before:
            assert acc == (after <= before), tau
        if acc:
            flat = trial
            kept += 1
    assert 5 < kept < 295
    assert np.array_equal(params.flat_eff32(), flat)


def test_zero_scheme_only_removes_weights():
    layers, init, X, y = _net()
    rows, params, S = O.run_channel(layers, "softmax_ce", X, y, init, 300, 2, "zero")
    assert np.count_nonzero(params.flat_eff32()) < np.count_nonzero(init)
    assert all(r[3] <= 0.0 for r in rows if r[4])                   # greedy: kept changes <= 0


def test_planted_disconnected_channel_is_caught(monkeypatch):
    """Drawing every layer's input node afresh (no path) fails the path pin."""
    orig = O.propose_channel

    def bad(seed, tau, params, scheme):
        ch = orig(seed, tau, params, scheme)
        out = []
        for m, r, c, old, new in ch:
            c2 = (c + tau + m) % params.layers[m].n_in if m > 0 else c
            out.append((m, r, c2, float(params.vals[m][r, c2]), new))
        return out
    monkeypatch.setattr(O, "propose_channel", bad)
    with pytest.raises(AssertionError):
        test_channel_is_a_path_with_one_weight_per_layer("he")
