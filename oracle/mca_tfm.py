"""Plain fp64 oracle of MCA on a character-level Transformer (paper, Section 2.5).

TEST INFRASTRUCTURE ONLY -- imported by tests/, __graft_entry__.smoke() and bench.py's CPU legs.

The model (a reading of the paper's sparse description): token + learned position embeddings; per
block a pre-LN causal multi-head self-attention and a pre-LN feed-forward network (exact-erf GELU, or
the Gaussian exp(-gamma x^2)), both with residual connections; a final LN and an untied linear head.
The loss of a sequence is the sum of the next-character cross-entropies of its positions; the trial
loop decides on the sum S over all sequences (Eq. 2 with R = 0, Eq. 6) and reports S / (B * T).
With a finite selection intensity beta the decision is Eq. 7's Metropolis rule on the mean loss
L = S / (B * T), i.e. the threshold of metropolis_threshold with N = B * T predicted tokens.

The trial loop is the definition: a full forward pass of every sequence after every mutation.
"""
from __future__ import annotations

import numpy as np

from .mca_oracle import Trace, act_fn, draw_words, metropolis_threshold

__all__ = ["tfm_views", "tfm_forward", "tfm_seq_losses", "tfm_propose", "run_full_tfm"]


def tfm_views(spec, flat) -> dict:
    """Named views (float64) of a flat parameter vector."""
    out, o = {}, 0
    flat = np.asarray(flat, dtype=np.float64)
    for name, shape in spec.blocks():
        n = int(np.prod(shape))
        out[name] = flat[o:o + n].reshape(shape)
        o += n
    return out


def _layer_norm(x, g, b, eps):
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * g + b


def tfm_forward(spec, flat, tokens):
    """Logits [B, T, V] for input tokens [B, T]."""
    p = tfm_views(spec, flat)
    B, T = tokens.shape
    d, H = spec.d_model, spec.n_head
    dh = d // H
    x = p["tok_emb"][tokens] + p["pos_emb"][:T][None, :, :]
    causal = np.triu(np.ones((T, T), dtype=bool), k=1)
    for b in range(spec.n_layer):
        h = _layer_norm(x, p[f"b{b}.ln1.g"], p[f"b{b}.ln1.b"], spec.ln_eps)
        q = h @ p[f"b{b}.wq"].T + p[f"b{b}.bq"]
        k = h @ p[f"b{b}.wk"].T + p[f"b{b}.bk"]
        v = h @ p[f"b{b}.wv"].T + p[f"b{b}.bv"]
        q = q.reshape(B, T, H, dh).transpose(0, 2, 1, 3)
        k = k.reshape(B, T, H, dh).transpose(0, 2, 1, 3)
        v = v.reshape(B, T, H, dh).transpose(0, 2, 1, 3)
        s = q @ k.transpose(0, 1, 3, 2) / np.sqrt(dh)
        s = np.where(causal[None, None], -np.inf, s)
        s = s - s.max(axis=-1, keepdims=True)
        w = np.exp(s)
        w = w / w.sum(axis=-1, keepdims=True)
        att = (w @ v).transpose(0, 2, 1, 3).reshape(B, T, d)
        x = x + att @ p[f"b{b}.wo"].T + p[f"b{b}.bo"]
        h2 = _layer_norm(x, p[f"b{b}.ln2.g"], p[f"b{b}.ln2.b"], spec.ln_eps)
        u = act_fn(spec.act, h2 @ p[f"b{b}.w1"].T + p[f"b{b}.b1"], spec.act_param)
        x = x + u @ p[f"b{b}.w2"].T + p[f"b{b}.b2"]
    h = _layer_norm(x, p["lnf.g"], p["lnf.b"], spec.ln_eps)
    return h @ p["w_head"].T + p["b_head"]


def tfm_seq_losses(spec, flat, tokens_full):
    """Per-sequence sums of next-character CE; tokens_full [B, T+1]."""
    inp, tgt = tokens_full[:, :-1], tokens_full[:, 1:]
    z = tfm_forward(spec, flat, inp)
    m = z.max(axis=-1, keepdims=True)
    lse = (m + np.log(np.exp(z - m).sum(axis=-1, keepdims=True)))[..., 0]
    zt = np.take_along_axis(z, tgt[..., None], axis=-1)[..., 0]
    return (lse - zt).sum(axis=1)


def tfm_propose(seed, tau, flat32, domain):
    """Eq. 1 over the flat parameter vector (every parameter fp32): index by multiply-shift of r0,
    new value from r1 as for the MLPs. Returns (idx, old, new, valid)."""
    r = draw_words(seed, tau)
    r0, r1 = int(r[0]), int(r[1])
    P = flat32.shape[0]
    idx = (r0 * P) >> 32
    f32 = np.float32
    old = f32(flat32[idx])
    u = f32(r1 >> 8) * f32(2.0 ** -24)
    if domain.op == "replace":
        new = f32(f32(domain.lo) + f32(f32(f32(domain.hi) - f32(domain.lo)) * u))
    else:
        new = f32(old + f32(f32(domain.delta) * (f32(f32(2.0) * u) - f32(1.0))))
    valid = not (domain.bound > 0 and not (abs(new) < f32(domain.bound)))
    return idx, float(old), float(new), valid


class _P:
    """Minimal proposal record for Trace.add."""

    def __init__(self, tau, idx, old, new, valid):
        self.tau, self.idx, self.layer, self.row, self.col = tau, idx, 0, 0, 0
        self.old, self.new, self.new_code, self.valid = old, new, 0, valid


def run_full_tfm(spec, tokens_full, init, n_trials, seed, domain, tau0=0):
    """Returns (trace arrays, final flat fp32 parameters, final S)."""
    flat = np.array(init, dtype=np.float32)
    S = float(tfm_seq_losses(spec, flat.astype(np.float64), tokens_full).sum())
    tr = Trace()
    for t in range(n_trials):
        idx, old, new, valid = tfm_propose(seed, tau0 + t, flat, domain)
        p = _P(tau0 + t, idx, old, new, valid)
        if not valid:
            tr.add(p, S, float("nan"), False)
            continue
        flat[idx] = np.float32(new)
        S_new = float(tfm_seq_losses(spec, flat.astype(np.float64), tokens_full).sum())
        dS = S_new - S
        theta = float(metropolis_threshold(seed, tau0 + t, getattr(domain, "beta", float("inf")),
                                           tokens_full.shape[0] * spec.ctx))
        acc = dS < theta if domain.strict else dS <= theta
        tr.add(p, S, dS, acc)
        if acc:
            S = S_new
        else:
            flat[idx] = np.float32(old)
    return tr.arrays(), flat, S
