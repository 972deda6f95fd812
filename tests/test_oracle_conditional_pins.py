"""Pin of the conditional loss change of a later candidate given an earlier kept one (CPU only).

For two first-layer candidates on different hidden rows, dS(c2 | c1) -- the loss change of c2 once
c1 is kept -- equals dS(c2) plus a correction over the samples where both input features are
non-zero. This is the identity a speculative batch needs to decide a second candidate after a first
accepted one without another exchange; it is checked here against the definition, two full forward
passes (S(c1 and c2 kept) - S(c1 kept)), on several loss / transfer-function pairs.
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W


def _gaussian_mse():
    wl = W.make("mlp_small", N=2000, H=48)
    for L in wl.layers[:-1]:
        L.act, L.act_param = "gaussian", 1.0
    return wl


NETS = {
    "tanh_ce": lambda: W.make("mlp_wide", N=2000, H=48),
    "tanh_sigmoid_mse": lambda: W.make("mlp_small", N=2000, H=48),
    "gaussian_sigmoid_mse": _gaussian_mse,
}


@pytest.mark.parametrize("name", list(NETS))
def test_conditional_dS_equals_two_full_passes(name):
    wl = NETS[name]()
    XT = wl.X.T.astype(np.float64)
    params = O.Params(wl.layers, wl.init)
    props = [p for p in (O.propose(3, t, params, wl.domain) for t in range(400)) if p.layer == 0]
    S0 = O.total_loss(params, XT, wl.y, wl.loss)
    checked = 0
    for p1, p2 in zip(props[0::2], props[1::2]):
        if p1.row == p2.row:
            continue
        c, u, nb = O.conditional_dS_two_layer(params, XT, wl.y, wl.loss, p1, p2)
        q = params.copy()
        O.apply_proposal(q, p1)
        S1 = O.total_loss(q, XT, wl.y, wl.loss)
        O.apply_proposal(q, p2)
        S12 = O.total_loss(q, XT, wl.y, wl.loss)
        assert c == pytest.approx(S12 - S1, rel=1e-9, abs=1e-10 * S0)
        assert nb == int(((XT[p1.col] != 0) & (XT[p2.col] != 0)).sum())
        checked += 1
    assert checked > 50


def test_conditional_dS_refuses_the_same_hidden_row():
    wl = W.make("mlp_small", N=200, H=8)
    params = O.Params(wl.layers, wl.init)
    props = [p for p in (O.propose(1, t, params, wl.domain) for t in range(300)) if p.layer == 0]
    same = next((a, b) for a in props for b in props if a is not b and a.row == b.row)
    with pytest.raises(ValueError):
        O.conditional_dS_two_layer(params, wl.X.T.astype(np.float64), wl.y, wl.loss, *same)


def test_planted_missing_correction_is_caught(monkeypatch):
    """Dropping the correction (taking dS(c2) for dS(c2 | c1)) fails the pin."""
    orig = O.conditional_dS_two_layer

    def bad(*a):
        c, u, nb = orig(*a)
        return u, u, nb
    monkeypatch.setattr(O, "conditional_dS_two_layer", bad)
    with pytest.raises(AssertionError):
        test_conditional_dS_equals_two_full_passes("tanh_ce")
