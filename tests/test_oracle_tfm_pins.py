"""Pins of the Transformer oracle (CPU only): a torch.nn.functional implementation of the same
pre-LN GPT (library routines: layer_norm, scaled_dot_product_attention with the causal mask, GELU,
cross_entropy), closed forms, causality, and the trial-loop invariants."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import mca_tfm as T
from paper_2607_08406_gb300 import workloads as W

SPEC = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=2, n_head=2, d_ff=32)


def _wl(spec=SPEC, batch=6, seed=0):
    return W.char_transformer(seed=seed, batch=batch, text_len=3000, spec=spec, n_trials=300, K=8)


def _torch_seq_losses(spec, flat, tokens_full):
    p = {k: torch.from_numpy(np.ascontiguousarray(v)) for k, v in T.tfm_views(spec, flat).items()}
    tok = torch.from_numpy(tokens_full.astype(np.int64))
    inp, tgt = tok[:, :-1], tok[:, 1:]
    B, Tn = inp.shape
    d, H = spec.d_model, spec.n_head
    x = p["tok_emb"][inp] + p["pos_emb"][:Tn]
    for b in range(spec.n_layer):
        h = F.layer_norm(x, (d,), p[f"b{b}.ln1.g"], p[f"b{b}.ln1.b"], spec.ln_eps)
        q = F.linear(h, p[f"b{b}.wq"], p[f"b{b}.bq"]).view(B, Tn, H, d // H).transpose(1, 2)
        k = F.linear(h, p[f"b{b}.wk"], p[f"b{b}.bk"]).view(B, Tn, H, d // H).transpose(1, 2)
        v = F.linear(h, p[f"b{b}.wv"], p[f"b{b}.bv"]).view(B, Tn, H, d // H).transpose(1, 2)
        a = F.scaled_dot_product_attention(q, k, v, is_causal=True)
        x = x + F.linear(a.transpose(1, 2).reshape(B, Tn, d), p[f"b{b}.wo"], p[f"b{b}.bo"])
        h2 = F.layer_norm(x, (d,), p[f"b{b}.ln2.g"], p[f"b{b}.ln2.b"], spec.ln_eps)
        u = F.linear(h2, p[f"b{b}.w1"], p[f"b{b}.b1"])
        u = F.gelu(u) if spec.act == "gelu" else torch.exp(-spec.act_param * u * u)
        x = x + F.linear(u, p[f"b{b}.w2"], p[f"b{b}.b2"])
    h = F.layer_norm(x, (d,), p["lnf.g"], p["lnf.b"], spec.ln_eps)
    z = F.linear(h, p["w_head"], p["b_head"])
    ce = F.cross_entropy(z.reshape(-1, spec.vocab), tgt.reshape(-1), reduction="none")
    return ce.view(B, Tn).sum(dim=1).numpy()


@pytest.mark.parametrize("act", ["gelu", "gaussian"])
def test_forward_vs_torch_functional(act):
    spec = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=2, n_head=2, d_ff=32, act=act)
    wl = _wl(spec)
    rng = np.random.default_rng(1)
    flat = wl.init.astype(np.float64) + rng.normal(0, 0.3, wl.n_params)   # away from the init
    got = T.tfm_seq_losses(spec, flat, wl.tokens)
    want = _torch_seq_losses(spec, flat, wl.tokens)
    assert np.allclose(got, want, rtol=1e-11, atol=1e-11)


def test_zero_parameters_give_uniform_prediction():
    """All matrices, embeddings and biases zero, LN gains 1: every logit is 0, CE = ln V."""
    wl = _wl()
    flat = np.zeros(wl.n_params)
    views = T.tfm_views(SPEC, flat)
    for name, v in views.items():
        if name.endswith(".g"):
            v[...] = 1.0
    got = T.tfm_seq_losses(SPEC, flat, wl.tokens)
    assert np.allclose(got, SPEC.ctx * math.log(SPEC.vocab), rtol=1e-13)


def test_causal_prefix_property():
    """Changing the input at position p leaves the logits of positions < p unchanged."""
    wl = _wl()
    rng = np.random.default_rng(2)
    flat = wl.init.astype(np.float64) + rng.normal(0, 0.3, wl.n_params)
    inp = wl.tokens[:, :-1].copy()
    z0 = T.tfm_forward(SPEC, flat, inp)
    inp[:, 5] = (inp[:, 5] + 3) % SPEC.vocab
    z1 = T.tfm_forward(SPEC, flat, inp)
    assert np.array_equal(z0[:, :5], z1[:, :5])
    assert not np.allclose(z0[:, 5:], z1[:, 5:])


def test_sequence_permutation_equivariance():
    wl = _wl()
    flat = wl.init.astype(np.float64)
    perm = np.array([3, 0, 5, 1, 4, 2])
    a = T.tfm_seq_losses(SPEC, flat, wl.tokens)
    b = T.tfm_seq_losses(SPEC, flat, wl.tokens[perm])
    assert np.allclose(a[perm], b, rtol=1e-14)


def test_tfm_trial_loop_invariants():
    wl = _wl()
    tr, flat, S = T.run_full_tfm(SPEC, wl.tokens, wl.init, 300, 3, wl.domain)
    assert np.all(np.diff(tr["S"]) <= 0.0)
    rej = ~tr["accept"][:-1]
    assert np.all(tr["S"][1:][rej] == tr["S"][:-1][rej])
    assert 0 < tr["accept"].sum() < 300
    # the final parameters are the initial ones with exactly the accepted proposals applied
    want = wl.init.copy()
    for t in range(300):
        if tr["accept"][t]:
            want[tr["idx"][t]] = np.float32(tr["new"][t])
    assert np.array_equal(flat, want)
    assert S == pytest.approx(T.tfm_seq_losses(SPEC, flat.astype(np.float64), wl.tokens).sum(),
                              rel=1e-12)


def test_markov_text_statistics():
    """The order-2 chain follows its Dirichlet transition rows: empirical bigram->next frequencies
    of a long stream match the rows drawn with the same generator."""
    rng = np.random.default_rng(5)
    text = W.markov_text(np.random.default_rng(5), 5, 200_000, alpha=1.0)
    rows = rng.dirichlet(np.full(5, 1.0), size=25)
    counts = np.zeros((25, 5))
    for t in range(2, len(text)):
        counts[text[t - 2] * 5 + text[t - 1], text[t]] += 1
    freq = counts / counts.sum(axis=1, keepdims=True)
    assert np.abs(freq - rows).max() < 0.03


def test_planted_missing_causal_mask_is_caught(monkeypatch):
    orig = np.triu

    def no_mask(m, k=0):
        return np.zeros_like(orig(m, k))

    monkeypatch.setattr(T.np, "triu", no_mask)
    with pytest.raises(AssertionError):
        test_forward_vs_torch_functional("gelu")
