"""Pins of the oracle's current-layer schedule (Section 2.1), CPU only.

The paper trains deep nets by picking a layer at random, running many Monte Carlo mutations inside
that layer, then moving to another randomly picked layer. The oracle's reading: trials come in
stretches of M; stretch s = floor(tau / M) mutates only layer l_s, drawn uniformly from the weight
layers by its own Philox counter; inside the layer the index is uniform. These tests tie that to
what the paper fixes (one layer per stretch, a uniform layer choice, a uniform parameter inside the
layer, fresh independent choices from stretch to stretch) and to the invariant every schedule keeps
(the cached-field mode takes the full mode's decisions).
"""
import dataclasses

import numpy as np
import pytest
from scipy import stats

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

DEEP_OFFS = [0] + list(np.cumsum([784 * 256] + [256 * 256] * 23 + [256 * 10]))   # 25 layers
WIDE_OFFS = [0, 784 * 64, 784 * 64 + 64 * 10]


def _layer_of(idx, offs):
    return int(np.searchsorted(offs, idx, side="right") - 1)


@pytest.mark.parametrize("offs,M", [(DEEP_OFFS, 7), (WIDE_OFFS, 100)])
def test_one_layer_per_stretch_and_uniform_inside(offs, M):
    """Every trial of a stretch mutates the stretch's layer; inside a layer the index is uniform
    (chi-square over 16 equal bins of the layer's index range)."""
    seed, n_stretch = 5, 300
    words = O.draw_words(seed, np.arange(n_stretch * M))[:, 0]
    layers = O.stretch_layer(seed, np.arange(n_stretch), len(offs) - 1)
    rel = {}
    for tau in range(n_stretch * M):
        idx = O.proposal_index(seed, tau, int(words[tau]), offs, M)
        l = _layer_of(idx, offs)
        assert l == int(layers[tau // M])
        rel.setdefault(l, []).append((idx - offs[l]) / (offs[l + 1] - offs[l]))
    big = max(rel, key=lambda k: len(rel[k]))
    h = np.histogram(rel[big], bins=16, range=(0.0, 1.0))[0]
    assert stats.chisquare(h).pvalue > 1e-4


@pytest.mark.parametrize("n_layers", [2, 3, 25])
def test_stretch_layers_uniform_and_independent(n_layers):
    """Over 4e4 stretches the layer choice is uniform, consecutive choices are independent (chi-
    square on the L x L table of (l_s, l_s+1)), and the choice is independent of the trial words
    (it agrees with the layer a uniform draw of trial s's own first word would give in a fraction
    1/L of the stretches, within 5 binomial standard deviations)."""
    seed, n = 11, 40_000
    l = O.stretch_layer(seed, np.arange(n), n_layers).astype(np.int64)
    assert stats.chisquare(np.bincount(l, minlength=n_layers)).pvalue > 1e-4
    table = np.zeros((n_layers, n_layers))
    np.add.at(table, (l[:-1], l[1:]), 1.0)
    assert stats.chi2_contingency(table)[1] > 1e-4
    r0 = O.draw_words(seed, np.arange(n))[:, 0]
    same = (((r0 * np.uint64(n_layers)) >> np.uint64(32)).astype(np.int64) == l).mean()
    p = 1.0 / n_layers
    assert abs(same - p) <= 5.0 * np.sqrt(p * (1 - p) / n)


def test_stretch_zero_is_uniform_over_all_parameters():
    """Without the schedule the index is uniform over the whole flat parameter space: the layer
    frequencies follow the layer sizes (chi-square)."""
    seed, n = 2, 60_000
    r0 = O.draw_words(seed, np.arange(n))[:, 0]
    idx = [O.proposal_index(seed, t, int(r0[t]), WIDE_OFFS, 0) for t in range(n)]
    cnt = np.bincount([_layer_of(i, WIDE_OFFS) for i in idx], minlength=2)
    sizes = np.diff(WIDE_OFFS)
    assert stats.chisquare(cnt, sizes / sizes.sum() * n).pvalue > 1e-4


@pytest.mark.parametrize("kind", ["deep", "single_hidden"])
def test_schedule_incremental_equals_full(kind):
    """Under the schedule the cached-field mode takes the full mode's decisions and ends in the same
    state, and every accepted change lies in its stretch's layer."""
    if kind == "deep":
        wl = W.mlp_deep(N=150, width=12, depth=4, n_trials=240, K=8)
    else:
        wl = W.mlp_small(N=120, H=12)
    M = 20
    dom = dataclasses.replace(wl.domain, layer_stretch=M)
    n = 240
    tf, pf, Sf = O.run_full(wl.layers, wl.loss, wl.X, wl.y, wl.init, n, 3, dom)
    ti, pi, Si = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, n, 3, dom)
    clear = np.abs(tf["dS"]) > 1e-9 * np.abs(tf["S"]).max()
    assert (tf["accept"][clear] == ti["accept"][clear]).all()
    assert (pf.flat_eff32() == pi.flat_eff32()).all()
    lay = O.stretch_layer(3, np.arange(n) // M, len(wl.layers))
    assert (tf["layer"] == lay).all()
    assert len(set(tf["layer"][tf["accept"]].tolist())) > 1


def test_planted_remainder_for_quotient_is_caught(monkeypatch):
    """Taking the stretch as tau mod M instead of floor(tau / M) breaks the one-layer-per-stretch
    pin."""
    def bad(seed, tau, r0, offsets, stretch):
        if stretch <= 0:
            return (r0 * offsets[-1]) >> 32
        l = int(O.stretch_layer(seed, tau % stretch, len(offsets) - 1))
        return offsets[l] + ((r0 * (offsets[l + 1] - offsets[l])) >> 32)
    monkeypatch.setattr(O, "proposal_index", bad)
    with pytest.raises(AssertionError):
        test_one_layer_per_stretch_and_uniform_inside(DEEP_OFFS, 7)


def test_planted_size_weighted_layer_is_caught(monkeypatch):
    """Choosing the stretch's layer in proportion to its size (what a uniform parameter draw would
    give) instead of uniformly breaks the uniform-layer pin."""
    def bad(seed, s, n_layers):
        q = O.draw_words(seed + 99, s)[..., 0]
        cut = np.uint64(2 ** 31 + 2 ** 30)                     # 3/4 of the draws to layer 0
        return np.where(q < cut, 0, 1 + (q - cut) % np.uint64(max(n_layers - 1, 1)))
    monkeypatch.setattr(O, "stretch_layer", bad)
    with pytest.raises(AssertionError):
        test_stretch_layers_uniform_and_independent(3)
