"""Pins of the oracle's mini-batch schedule (Sections 2.2 and 2.5), CPU only.

The paper trains on batches of the training set (30,000 of 60,000 samples; a batch size that grows
during training): each trial decides on the loss summed over the current batch only, and the
weights and the trial counter carry over from batch to batch. These tests tie run_batches to that:
one batch of every sample is the full-batch loop, each stretch follows the full-forward definition
on its own samples, samples outside every batch cannot influence anything, and the order of the
samples inside a batch does not matter.
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

M = 120


def _wl():
    return W.make("mlp_small", N=360, H=12)


def test_single_batch_of_all_samples_is_the_full_batch_loop():
    wl = _wl()
    tr, p, S = O.run_batches(wl.layers, wl.loss, wl.X, wl.y, wl.init, [np.arange(wl.N)], 300, 4,
                             wl.domain)
    tr0, p0, S0 = O.run_incremental(wl.layers, wl.loss, wl.X, wl.y, wl.init, 300, 4, wl.domain)
    for k in tr0:
        assert np.array_equal(tr[k], tr0[k], equal_nan=True), k
    assert np.array_equal(p.flat_eff32(), p0.flat_eff32()) and S == S0


def test_each_stretch_follows_the_definition_on_its_batch():
    """Trials of stretch s, replayed by the full-forward definition on batch s's samples from the
    weights the previous stretch left, take the same decisions (outside 1e-9 S) and end in the
    same weights."""
    wl = _wl()
    bs = W.minibatches(wl.N, 180, 3, seed=2)
    tr, p, S = O.run_batches(wl.layers, wl.loss, wl.X, wl.y, wl.init, bs, M, 4, wl.domain)
    params = O.Params(wl.layers, wl.init)
    for s, b in enumerate(bs):
        tf, params, Sf = O.run_full(wl.layers, wl.loss, wl.X[b], wl.y[b], None, M, 4, wl.domain,
                                    tau0=s * M, params=params)
        sl = slice(s * M, (s + 1) * M)
        clear = np.abs(tf["dS"]) > 1e-9 * np.abs(tf["S"])
        assert np.array_equal(tf["accept"][clear], tr["accept"][sl][clear])
        assert np.array_equal(tf["tau"], tr["tau"][sl])
    assert np.array_equal(params.flat_eff32(), p.flat_eff32())
    assert tr["accept"].sum() > 20


def test_samples_outside_every_batch_do_not_matter():
    wl = _wl()
    bs = W.minibatches(wl.N, 150, 2, seed=5)
    used = np.zeros(wl.N, bool)
    for b in bs:
        used[b] = True
    assert (~used).sum() > 50
    tr, p, S = O.run_batches(wl.layers, wl.loss, wl.X, wl.y, wl.init, bs, M, 1, wl.domain)
    X2, y2 = wl.X.copy(), wl.y.copy()
    rng = np.random.default_rng(0)
    X2[~used] = rng.uniform(0, 1, X2[~used].shape).astype(np.float32)
    y2[~used] = rng.integers(0, 10, (~used).sum()).astype(y2.dtype)
    tr2, p2, S2 = O.run_batches(wl.layers, wl.loss, X2, y2, wl.init, bs, M, 1, wl.domain)
    assert np.array_equal(tr["accept"], tr2["accept"]) and np.array_equal(tr["dS"], tr2["dS"])
    assert np.array_equal(p.flat_eff32(), p2.flat_eff32())


def test_sample_order_inside_a_batch_does_not_matter():
    wl = _wl()
    bs = W.minibatches(wl.N, 200, 2, seed=3)
    rng = np.random.default_rng(1)
    shuffled = [rng.permutation(b) for b in bs]
    tr, p, S = O.run_batches(wl.layers, wl.loss, wl.X, wl.y, wl.init, bs, M, 2, wl.domain)
    tr2, p2, S2 = O.run_batches(wl.layers, wl.loss, wl.X, wl.y, wl.init, shuffled, M, 2,
                                wl.domain)
    clear = np.abs(tr["dS"]) > 1e-9 * np.abs(tr["S"])
    assert np.array_equal(tr["accept"][clear], tr2["accept"][clear])
    assert np.allclose(tr["dS"], tr2["dS"], rtol=1e-9, atol=1e-9 * np.abs(tr["S"]).max())


def test_planted_previous_batch_is_caught(monkeypatch):
    """Deciding stretch s on batch s - 1 fails the definition pin."""
    orig = O.run_batches

    def shifted(layers, loss, X, y, init, batches, stretch, seed, domain, params=None):
        return orig(layers, loss, X, y, init, [batches[0]] + list(batches[:-1]), stretch, seed,
                    domain, params)
    monkeypatch.setattr(O, "run_batches", shifted)
    with pytest.raises(AssertionError):
        test_each_stretch_follows_the_definition_on_its_batch()


def test_minibatch_generator_draws_without_replacement():
    """Each batch holds distinct sample indices in ascending order, every sample is equally likely
    to be drawn (chi-square over 4000 batches), and the same seed gives the same batches."""
    from scipy import stats
    bs = W.minibatches(100, 30, 4000, seed=8)
    for b in bs[:50]:
        assert len(b) == 30 and np.all(np.diff(b) > 0) and b[0] >= 0 and b[-1] < 100
    counts = np.bincount(np.concatenate(bs), minlength=100)
    assert stats.chisquare(counts).pvalue > 1e-4
    assert all(np.array_equal(a, b) for a, b in zip(bs[:5], W.minibatches(100, 30, 5, seed=8)))
