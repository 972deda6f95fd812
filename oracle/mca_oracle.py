"""Plain fp64 CPU oracle of the Monte Carlo mutation-selection (MCA) trial loop.

TEST INFRASTRUCTURE ONLY -- imported by tests/, __graft_entry__.smoke() and bench.py's CPU legs;
never by the product path, and sharing no code with it.

What it computes (paper "Beyond Backpropagation: Monte Carlo Method Can Train Deep Neural
Networks", Section 2 Eq. 1 and Section 3.1 Eq. 6):

    for tau = 0, 1, ...:
        pick one parameter uniformly at random and draw its new value   (Eq. 1, Section 2)
        reject without evaluating if the new value leaves the domain |w| < Delta   (Eq. 1)
        W' = W with that one parameter changed
        S' = sum over all N samples of the per-sample loss of f_W'   (full batch, Eq. 2 with R = 0)
        keep W' iff S' <= S, else keep W   (greedy rule, Eq. 6; or Eq. 7's Metropolis rule with
                                             a finite selection intensity beta, as a per-trial
                                             threshold S' - S <= theta_tau, metropolis_threshold)

Multi-parameter channel mutations (Section 2.3) have their own loop, ``run_channel``: every weight on
one input-to-output path changes at once and a full forward pass decides. Mini-batch schedules
(Sections 2.2 and 2.5) run the cached-field loop on one given batch of samples per stretch of
trials, ``run_batches``.

Two evaluation modes, which must agree (the invariant the incremental GPU path relies on):

* ``run_full``: a full forward pass of all N samples after every mutation -- the definition.
* ``run_incremental``: the paper's cached-field scheme (Section 2.4): only the mutated neuron's
  field row changes (rank-1 in the mutated layer l), the next layer's fields change by the
  mutated neuron's activation change times one weight column (rank-1 in l+1), and the layers from
  l+2 on are recomputed densely.

Readings of points the paper leaves open (the paper is silent on each):

* Proposal stream: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11), key = (seed_lo, seed_hi),
  counter = (tau_lo, tau_hi, 0, 0); words r0 (index) and r1 (value) are used.
* Index: idx = floor(r0 * P / 2^32) over the flat parameter space (layers in forward order,
  each weight matrix [out x in] row-major). With the current-layer schedule of Section 2.1
  (domain.layer_stretch = M > 0), stretches of M trials each mutate one layer chosen uniformly at
  random, the index uniform inside it (proposal_index, stretch_layer).
* Replacement value: u = (r1 >> 8) * 2^-24 in fp32, w' = lo + (hi - lo) * u with two fp32
  roundings (for [lo, hi) = [-1, 1) this is exact). Perturbation: r = 2u - 1 (exact),
  w' = w + delta * r in fp32.
* Ternary layers: new code floor(r1 * 3 / 2^32) - 1 (may equal the old code: a no-op trial).
  Masked layers: the mutation toggles the mask bit of the chosen fixed weight.
* MSE loss: sum over outputs of (a_k - onehot_k)^2; CE: natural-log softmax cross-entropy.
  Decisions use the loss sum S; the reported loss is S / N.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import List, Optional, Sequence

import numpy as np
from scipy.special import erf as _erf

__all__ = [
    "philox4x32_10", "draw_words", "propose", "Proposal", "Params", "act_fn", "loss_per_sample",
    "forward", "total_loss", "run_full", "run_incremental", "Trace", "output_fields_blocked",
    "candidate_dS_two_layer", "metropolis_threshold", "stretch_layer", "proposal_index",
    "channel_words", "propose_channel", "run_channel", "run_batches", "conditional_dS_two_layer",
]

# ------------------------------------------------------------------------------------------------
# Philox4x32-10 (Salmon et al., "Parallel random numbers: as easy as 1, 2, 3", SC'11, Section 3.2):
# a 10-round bijection of a 128-bit counter under a 64-bit key.
# ------------------------------------------------------------------------------------------------
_M32 = np.uint64(0xFFFFFFFF)
_PH_M0 = np.uint64(0xD2511F53)
_PH_M1 = np.uint64(0xCD9E8D57)
_PH_W0 = np.uint64(0x9E3779B9)
_PH_W1 = np.uint64(0xBB67AE85)
_S32 = np.uint64(32)


def philox4x32_10(ctr, key) -> np.ndarray:
    """ctr: (..., 4) and key: (..., 2) arrays of 32-bit words. Returns (..., 4) uint64 words."""
    c = np.asarray(ctr, dtype=np.uint64)
    k = np.asarray(key, dtype=np.uint64)
    c0, c1, c2, c3 = c[..., 0], c[..., 1], c[..., 2], c[..., 3]
    k0, k1 = k[..., 0], k[..., 1]
    for rnd in range(10):
        if rnd:
            k0 = (k0 + _PH_W0) & _M32
            k1 = (k1 + _PH_W1) & _M32
        p0 = c0 * _PH_M0          # both factors < 2^32: the product fits in 64 bits
        p1 = c2 * _PH_M1
        c0, c1, c2, c3 = ((p1 >> _S32) ^ c1 ^ k0, p1 & _M32, (p0 >> _S32) ^ c3 ^ k1, p0 & _M32)
    return np.stack([c0, c1, c2, c3], axis=-1)


def draw_words(seed: int, tau) -> np.ndarray:
    """The four Philox words of trial tau (scalar or array) under proposal key ``seed``."""
    tau = np.asarray(tau, dtype=np.uint64)
    ctr = np.stack([tau & _M32, tau >> _S32, np.zeros_like(tau), np.zeros_like(tau)], axis=-1)
    s = np.uint64(seed)
    key = np.broadcast_to(np.array([s & _M32, s >> _S32], dtype=np.uint64), ctr.shape[:-1] + (2,))
    return philox4x32_10(ctr, key)


# ------------------------------------------------------------------------------------------------
# Parameters
# ------------------------------------------------------------------------------------------------

class Params:
    """Per-layer weight state. fp32 layers: the weights; ternary layers: int8 codes in {-1,0,1}
    (effective weight scale * code); masked layers: fixed fp32 weights and a 0/1 mask (effective
    weight w * m). ``init`` is the flat fp32 vector (codes for ternary layers); masks start at 1."""

    def __init__(self, layers, init: np.ndarray):
        self.layers = layers
        self.vals: List[np.ndarray] = []
        self.mask: List[Optional[np.ndarray]] = []
        o = 0
        init = np.asarray(init, dtype=np.float32)
        for L in layers:
            n = L.n_in * L.n_out
            block = init[o:o + n].reshape(L.n_out, L.n_in)
            if L.wkind == "ternary_i8":
                self.vals.append(block.astype(np.int8).copy())
                self.mask.append(None)
            elif L.wkind == "masked_fp32":
                self.vals.append(block.astype(np.float32).copy())
                self.mask.append(np.ones((L.n_out, L.n_in), dtype=np.uint8))
            else:
                self.vals.append(block.astype(np.float32).copy())
                self.mask.append(None)
            o += n
        self.n_params = o
        self.offsets = np.cumsum([0] + [L.n_in * L.n_out for L in layers])[:-1].tolist()

    def copy(self) -> "Params":
        p = Params.__new__(Params)
        p.layers = self.layers
        p.vals = [v.copy() for v in self.vals]
        p.mask = [None if m is None else m.copy() for m in self.mask]
        p.n_params = self.n_params
        p.offsets = list(self.offsets)
        return p

    def eff32(self, l: int) -> np.ndarray:
        L = self.layers[l]
        if L.wkind == "ternary_i8":
            return np.float32(L.scale) * self.vals[l].astype(np.float32)
        if L.wkind == "masked_fp32":
            return np.where(self.mask[l] != 0, self.vals[l], np.float32(0.0)).astype(np.float32)
        return self.vals[l]

    def eff64(self, l: int) -> np.ndarray:
        return self.eff32(l).astype(np.float64)

    def flat_eff32(self) -> np.ndarray:
        return np.concatenate([self.eff32(l).ravel() for l in range(len(self.layers))])

    def flat_codes(self) -> np.ndarray:
        """int8 per parameter: ternary code, mask bit, or 0 for fp32 layers."""
        out = []
        for l, L in enumerate(self.layers):
            if L.wkind == "ternary_i8":
                out.append(self.vals[l].ravel().astype(np.int8))
            elif L.wkind == "masked_fp32":
                out.append(self.mask[l].ravel().astype(np.int8))
            else:
                out.append(np.zeros(L.n_in * L.n_out, dtype=np.int8))
        return np.concatenate(out)


# ------------------------------------------------------------------------------------------------
# Proposal (Eq. 1): one parameter, one new value
# ------------------------------------------------------------------------------------------------

@dataclass
class Proposal:
    tau: int
    idx: int
    layer: int
    row: int            # output neuron j of the layer
    col: int            # input neuron i of the layer
    old: float          # effective weights (exact fp32 values, held as Python floats)
    new: float
    old_code: int       # ternary code / mask bit (0 for fp32 layers)
    new_code: int
    new_raw: float      # the value stored in the fp32 slot (fp32 layers: == new)
    valid: bool         # False: outside the weight domain, rejected without evaluation


def stretch_layer(seed: int, s, n_layers: int):
    """Layer of stretch s under the current-layer schedule (Section 2.1): a layer chosen uniformly at
    random, l_s = floor(q * n_layers / 2^32), q the first word of Philox4x32-10 under the proposal
    key at counter (s_lo, s_hi, 1, 0) -- the third counter word keeps these draws apart from the
    trials' own words (counter (tau_lo, tau_hi, 0, 0))."""
    s = np.asarray(s, dtype=np.uint64)
    ctr = np.stack([s & _M32, s >> _S32, np.ones_like(s), np.zeros_like(s)], axis=-1)
    k = np.uint64(seed)
    key = np.broadcast_to(np.array([k & _M32, k >> _S32], dtype=np.uint64), ctr.shape[:-1] + (2,))
    q = philox4x32_10(ctr, key)[..., 0]
    return (q * np.uint64(n_layers)) >> _S32


def proposal_index(seed: int, tau: int, r0: int, offsets: Sequence[int], stretch: int) -> int:
    """Flat index of trial tau's parameter; offsets: the first index of every layer, then P.
    stretch = 0: uniform over all P parameters (Eq. 1),
    floor(r0 P / 2^32). stretch = M > 0, the current-layer schedule of Section 2.1: the trials of
    stretch s = floor(tau / M) mutate only layer l_s (stretch_layer), each trial's index uniform
    inside that layer, offsets[l_s] + floor(r0 P_l / 2^32)."""
    if stretch <= 0:
        return (r0 * offsets[-1]) >> 32
    l = int(stretch_layer(seed, tau // stretch, len(offsets) - 1))
    return offsets[l] + ((r0 * (offsets[l + 1] - offsets[l])) >> 32)


def propose(seed: int, tau: int, params: Params, domain) -> Proposal:
    r = draw_words(seed, tau)
    r0, r1 = int(r[0]), int(r[1])
    idx = proposal_index(seed, tau, r0, list(params.offsets) + [params.n_params],
                         getattr(domain, "layer_stretch", 0))
    l = 0
    while l + 1 < len(params.layers) and idx >= params.offsets[l + 1]:
        l += 1
    L = params.layers[l]
    off = idx - params.offsets[l]
    row, col = divmod(off, L.n_in)
    f32 = np.float32
    if L.wkind == "ternary_i8":
        oc = int(params.vals[l][row, col])
        nc = ((r1 * 3) >> 32) - 1
        old = float(f32(L.scale) * f32(oc))
        new = float(f32(L.scale) * f32(nc))
        return Proposal(tau, idx, l, row, col, old, new, oc, nc, new, True)
    if L.wkind == "masked_fp32":
        w = f32(params.vals[l][row, col])
        om = int(params.mask[l][row, col])
        nm = 1 - om
        old = float(w) if om else 0.0
        new = float(w) if nm else 0.0
        return Proposal(tau, idx, l, row, col, old, new, om, nm, float(w), True)
    oldv = f32(params.vals[l][row, col])
    u = f32(r1 >> 8) * f32(2.0 ** -24)                       # exact, in [0, 1)
    if domain.op == "replace":
        newv = f32(f32(domain.lo) + f32(f32(f32(domain.hi) - f32(domain.lo)) * u))
    elif domain.op == "perturb":
        rr = f32(f32(2.0) * u) - f32(1.0)                      # exact, in [-1, 1)
        newv = f32(oldv + f32(f32(domain.delta) * rr))
    else:
        raise ValueError(domain.op)
    valid = True
    if domain.bound > 0 and not (abs(newv) < f32(domain.bound)):
        valid = False
    return Proposal(tau, idx, l, row, col, float(oldv), float(newv), 0, 0, float(newv), valid)


def apply_proposal(params: Params, p: Proposal) -> None:
    L = params.layers[p.layer]
    if L.wkind == "ternary_i8":
        params.vals[p.layer][p.row, p.col] = p.new_code
    elif L.wkind == "masked_fp32":
        params.mask[p.layer][p.row, p.col] = p.new_code
    else:
        params.vals[p.layer][p.row, p.col] = np.float32(p.new_raw)


def revert_proposal(params: Params, p: Proposal) -> None:
    L = params.layers[p.layer]
    if L.wkind == "ternary_i8":
        params.vals[p.layer][p.row, p.col] = p.old_code
    elif L.wkind == "masked_fp32":
        params.mask[p.layer][p.row, p.col] = p.old_code
    else:
        params.vals[p.layer][p.row, p.col] = np.float32(p.old)


# ------------------------------------------------------------------------------------------------
# Forward pass and loss (Section 2: transfer functions; Eq. 2 with R = 0)
# ------------------------------------------------------------------------------------------------

def act_fn(name: str, z: np.ndarray, gamma: float = 0.0) -> np.ndarray:
    if name == "identity":
        return z
    if name == "tanh":
        return np.tanh(z)
    if name == "sigmoid":
        with np.errstate(over="ignore"):
            return 1.0 / (1.0 + np.exp(-z))
    if name == "relu":
        return np.maximum(z, 0.0)
    if name == "gaussian":                     # f(x) = exp(-gamma x^2), Section 2
        return np.exp(-gamma * z * z)
    if name == "gelu":                         # exact-erf GELU
        return 0.5 * z * (1.0 + _erf(z / np.sqrt(2.0)))
    raise ValueError(name)


def loss_per_sample(kind: str, out: np.ndarray, y: np.ndarray) -> np.ndarray:
    """out: [C, N] output activations; y: [N] labels. Returns [N] per-sample losses."""
    n = out.shape[1]
    if kind == "mse_onehot":
        t = np.zeros_like(out)
        t[y, np.arange(n)] = 1.0
        return ((out - t) ** 2).sum(axis=0)
    if kind == "softmax_ce":
        m = out.max(axis=0)
        lse = m + np.log(np.exp(out - m).sum(axis=0))
        return lse - out[y, np.arange(n)]
    raise ValueError(kind)


def forward(params: Params, XT: np.ndarray):
    """XT: [D, N] float64. Returns (Z list of [n_out, N] fields, final activations [C, N])."""
    a = XT
    Zs = []
    for l, L in enumerate(params.layers):
        z = params.eff64(l) @ a
        Zs.append(z)
        a = act_fn(L.act, z, L.act_param)
    return Zs, a


def total_loss(params: Params, XT: np.ndarray, y: np.ndarray, loss: str) -> float:
    _, out = forward(params, XT)
    return float(loss_per_sample(loss, out, y).sum())


# ------------------------------------------------------------------------------------------------
# Trial loops
# ------------------------------------------------------------------------------------------------

class Trace:
    """Per-trial record: tau, idx, layer, row, col, old, new (effective fp32 weights), valid,
    S_before, dS (S' - S; NaN when not evaluated), accept."""
    FIELDS = ("tau", "idx", "layer", "row", "col", "old", "new", "new_code", "valid", "S", "dS",
              "accept")

    def __init__(self):
        self.rows = []

    def add(self, p: Proposal, S: float, dS: float, accept: bool):
        self.rows.append((p.tau, p.idx, p.layer, p.row, p.col, p.old, p.new, p.new_code, p.valid,
                          S, dS, accept))

    def arrays(self):
        cols = list(zip(*self.rows)) if self.rows else [[] for _ in self.FIELDS]
        dt = {"tau": np.int64, "idx": np.int64, "layer": np.int32, "row": np.int32,
              "col": np.int32, "old": np.float64, "new": np.float64, "new_code": np.int32,
              "valid": bool, "S": np.float64, "dS": np.float64, "accept": bool}
        return {f: np.asarray(c, dtype=dt[f]) for f, c in zip(self.FIELDS, cols)}


def metropolis_threshold(seed: int, tau, beta: float, N: int):
    """Acceptance threshold of trial tau on the loss-sum change dS (Section 3.1, Eq. 7).

    Eq. 7 keeps a mutation with probability A = min{1, exp(-beta dL)}, dL the change of the mean
    loss L = S / N. The trial's uniform number is u = (r3 + 1/2) 2^-32, r3 the fourth Philox word
    of its counter (words r0, r1 draw the proposal), and the trial is kept iff u < exp(-beta dL),
    i.e. iff dS <= theta = -(N / beta) ln u (theta > 0 since u < 1). beta = inf gives theta = 0,
    the greedy rule of Eq. 6. Every trial's decision depends only on its own dS and counter, so
    evaluating several trials against the same state and keeping the lowest-index accepted one
    reproduces the sequential chain, as for the greedy rule."""
    if beta == float("inf"):
        return np.zeros(np.shape(tau)) if np.ndim(tau) else 0.0
    r3 = draw_words(seed, tau)[..., 3].astype(np.float64)
    u = (r3 + 0.5) * 2.0 ** -32
    return -(float(N) / beta) * np.log(u)


def _decide(dS: float, strict: bool, theta: float = 0.0) -> bool:
    return (dS < theta) if strict else (dS <= theta)


def _threshold(seed: int, tau: int, domain, N: int) -> float:
    return float(metropolis_threshold(seed, tau, getattr(domain, "beta", float("inf")), N))


def run_full(layers, loss: str, X: np.ndarray, y: np.ndarray, init, n_trials: int, seed: int,
             domain, tau0: int = 0, params: Optional[Params] = None):
    """The definition: a full forward pass of all samples after every mutation.
    Returns (trace arrays, final Params, final S)."""
    XT = np.ascontiguousarray(np.asarray(X, dtype=np.float64).T)
    y = np.asarray(y)
    params = Params(layers, init) if params is None else params
    S = total_loss(params, XT, y, loss)
    tr = Trace()
    for t in range(n_trials):
        p = propose(seed, tau0 + t, params, domain)
        if not p.valid:
            tr.add(p, S, float("nan"), False)
            continue
        apply_proposal(params, p)
        S_new = total_loss(params, XT, y, loss)
        dS = S_new - S
        acc = _decide(dS, domain.strict, _threshold(seed, tau0 + t, domain, XT.shape[1]))
        tr.add(p, S, dS, acc)
        if acc:
            S = S_new
        else:
            revert_proposal(params, p)
    return tr.arrays(), params, S


class _Cache:
    """Cached fields of every layer for all samples, plus the per-sample losses."""

    def __init__(self, params: Params, XT: np.ndarray, y: np.ndarray, loss: str):
        self.Z, out = forward(params, XT)
        self.ell = loss_per_sample(loss, out, y)


def _candidate(params: Params, cache: _Cache, XT, y, loss, p: Proposal):
    """Incremental evaluation of one proposal against the cached state (Section 2.4).
    Returns (dS, list of (layer, new field matrix or (row, new row)) to commit, new ell)."""
    layers = params.layers
    l, j, i = p.layer, p.row, p.col
    nl = len(layers)
    delta = p.new - p.old                                   # exact in fp64 (fp32 operands)
    if l == 0:
        a_prev_i = XT[i]
    else:
        Lp = layers[l - 1]
        a_prev_i = act_fn(Lp.act, cache.Z[l - 1][i], Lp.act_param)
    zrow = cache.Z[l][j] + delta * a_prev_i                 # rank-1 update of layer l, row j
    updates = [(l, ("row", j, zrow))]
    if l == nl - 1:
        Zout = cache.Z[l].copy()
        Zout[j] = zrow
        out = act_fn(layers[l].act, Zout, layers[l].act_param)
    else:
        L = layers[l]
        da = act_fn(L.act, zrow, L.act_param) - act_fn(L.act, cache.Z[l][j], L.act_param)
        Wn = params.eff64(l + 1)
        z = cache.Z[l + 1] + np.outer(Wn[:, j], da)         # rank-1 update of layer l+1
        updates.append((l + 1, ("full", z)))
        a = act_fn(layers[l + 1].act, z, layers[l + 1].act_param)
        for m in range(l + 2, nl):                          # dense recompute from l+2 on
            z = params.eff64(m) @ a
            updates.append((m, ("full", z)))
            a = act_fn(layers[m].act, z, layers[m].act_param)
        out = a
    ell_new = loss_per_sample(loss, out, y)
    dS = float((ell_new - cache.ell).sum())
    return dS, updates, ell_new


def run_incremental(layers, loss: str, X: np.ndarray, y: np.ndarray, init, n_trials: int,
                    seed: int, domain, tau0: int = 0, params: Optional[Params] = None,
                    check_every: int = 0):
    """The paper's cached-field scheme. ``check_every`` > 0 asserts, every that many trials, that
    the cached S equals a full recompute within 1e-9 relative. Returns (trace, Params, S)."""
    XT = np.ascontiguousarray(np.asarray(X, dtype=np.float64).T)
    y = np.asarray(y)
    params = Params(layers, init) if params is None else params
    cache = _Cache(params, XT, y, loss)
    S = float(cache.ell.sum())
    tr = Trace()
    for t in range(n_trials):
        p = propose(seed, tau0 + t, params, domain)
        if not p.valid:
            tr.add(p, S, float("nan"), False)
            continue
        dS, updates, ell_new = _candidate(params, cache, XT, y, loss, p)
        acc = _decide(dS, domain.strict, _threshold(seed, tau0 + t, domain, XT.shape[1]))
        tr.add(p, S, dS, acc)
        if acc:
            apply_proposal(params, p)
            for m, upd in updates:
                if upd[0] == "row":
                    cache.Z[m][upd[1]] = upd[2]
                else:
                    cache.Z[m] = upd[1]
            cache.ell = ell_new
            S = S + dS
        if check_every and (t + 1) % check_every == 0:
            S_full = total_loss(params, XT, y, loss)
            assert abs(S_full - S) <= 1e-9 * max(1.0, abs(S_full)), (t, S_full, S)
    return tr.arrays(), params, S


# ------------------------------------------------------------------------------------------------
# Single-candidate evaluation at large sizes (two-layer nets): the hidden layer is formed in row
# blocks so that only the output fields are held for all samples.
# ------------------------------------------------------------------------------------------------

def output_fields_blocked(params: Params, XT: np.ndarray, block: int = 1024) -> np.ndarray:
    """Output fields Z2 = W2 f(W1 X^T) of a two-layer net, [C, N], built over hidden-row blocks."""
    L1 = params.layers[0]
    W1 = params.eff64(0)
    W2 = params.eff64(1)
    Z2 = np.zeros((W2.shape[0], XT.shape[1]))
    for j0 in range(0, W1.shape[0], block):
        A = act_fn(L1.act, W1[j0:j0 + block] @ XT, L1.act_param)
        Z2 += W2[:, j0:j0 + block] @ A
    return Z2


def candidate_dS_two_layer(params: Params, XT: np.ndarray, y: np.ndarray, loss: str,
                           Z2: np.ndarray, idx: int, new_eff: float) -> float:
    """S' - S when the flat weight idx takes the effective value new_eff (Section 2.4's update:
    one hidden field row, then the output fields through one weight column)."""
    L1, L2 = params.layers
    W1 = params.eff64(0)
    W2 = params.eff64(1)
    P1 = L1.n_in * L1.n_out
    ell = loss_per_sample(loss, act_fn(L2.act, Z2, L2.act_param), y)
    if idx < P1:
        j, i = divmod(idx, L1.n_in)
        delta = float(new_eff) - W1[j, i]
        z = W1[j] @ XT
        da = act_fn(L1.act, z + delta * XT[i], L1.act_param) - act_fn(L1.act, z, L1.act_param)
        Z2n = Z2 + np.outer(W2[:, j], da)
    else:
        o, j = divmod(idx - P1, L2.n_in)
        delta = float(new_eff) - W2[o, j]
        a = act_fn(L1.act, W1[j] @ XT, L1.act_param)
        Z2n = Z2.copy()
        Z2n[o] += delta * a
    ell_new = loss_per_sample(loss, act_fn(L2.act, Z2n, L2.act_param), y)
    return float((ell_new - ell).sum())


# ------------------------------------------------------------------------------------------------
# Multi-parameter channel mutations (Section 2.3). A channel is a path from one input node through
# one node of every hidden layer to one output node; a mutation changes the one weight of every
# layer that lies on it, either redrawing each with He-normalised amplitude or setting all to zero
# (the Dropout-like scheme), and is kept iff the loss does not increase. fp32 layers only.
# ------------------------------------------------------------------------------------------------

def channel_words(seed: int, tau: int, n: int) -> np.ndarray:
    """n Philox words for trial tau's channel: counters (tau_lo, tau_hi, 2, q), q = 0, 1, ..., four
    words each -- apart from the trial's own counter (tau, 0, 0, 0) and the schedule's (s, 0, 1, 0)."""
    q = np.arange((n + 3) // 4, dtype=np.uint64)
    t = np.uint64(tau)
    ctr = np.stack([np.full_like(q, t & _M32), np.full_like(q, t >> _S32),
                    np.full_like(q, 2), q], axis=-1)
    s = np.uint64(seed)
    key = np.broadcast_to(np.array([s & _M32, s >> _S32], dtype=np.uint64), ctr.shape[:-1] + (2,))
    return philox4x32_10(ctr, key).reshape(-1)[:n]


def propose_channel(seed: int, tau: int, params: Params, scheme: str):
    """The channel of trial tau and its new weights: a list of (layer m, row, col, old, new) with
    W_m[c_{m+1}, c_m] for m = 0 .. L-1. Nodes: c_m = floor(v_m n_m / 2^32) over the L + 1 node
    counts (inputs, every hidden width, outputs), v_m the channel words. scheme "he": the new
    weight of layer m is a_m (2 u_m - 1) in fp32, u_m = (v_{L+1+m} >> 8) 2^-24 and
    a_m = fp32(sqrt(6 / fan_in_m)) (He's uniform amplitude); scheme "zero": 0."""
    layers = params.layers
    L = len(layers)
    sizes = [layers[0].n_in] + [ly.n_out for ly in layers]
    v = channel_words(seed, tau, 2 * L + 1)
    nodes = [int((int(v[m]) * sizes[m]) >> 32) for m in range(L + 1)]
    f32 = np.float32
    out = []
    for m, ly in enumerate(layers):
        if ly.wkind != "fp32":
            raise ValueError("channel mutations take fp32 layers")
        row, col = nodes[m + 1], nodes[m]
        old = f32(params.vals[m][row, col])
        if scheme == "he":
            a = f32(np.sqrt(6.0 / ly.n_in))
            u = f32(int(v[L + 1 + m]) >> 8) * f32(2.0 ** -24)
            new = f32(a * f32(f32(f32(2.0) * u) - f32(1.0)))
        elif scheme == "zero":
            new = f32(0.0)
        else:
            raise ValueError(scheme)
        out.append((m, row, col, float(old), float(new)))
    return out


def run_channel(layers, loss: str, X: np.ndarray, y: np.ndarray, init, n_trials: int, seed: int,
                scheme: str, strict: bool = False, beta: float = float("inf"), tau0: int = 0,
                params: Optional[Params] = None):
    """Channel-mutation trial loop, by definition: apply every weight of the channel, run a full
    forward pass, keep iff dS <= theta (Eq. 6; Eq. 7 for a finite beta), else restore every weight.
    Returns (list of (tau, channel, S before, dS, accepted), final Params, final S)."""
    XT = np.ascontiguousarray(np.asarray(X, dtype=np.float64).T)
    y = np.asarray(y)
    params = Params(layers, init) if params is None else params
    S = total_loss(params, XT, y, loss)
    rows = []
    for t in range(n_trials):
        tau = tau0 + t
        ch = propose_channel(seed, tau, params, scheme)
        for m, r, c, old, new in ch:
            params.vals[m][r, c] = np.float32(new)
        S_new = total_loss(params, XT, y, loss)
        dS = S_new - S
        acc = _decide(dS, strict, float(metropolis_threshold(seed, tau, beta, XT.shape[1])))
        rows.append((tau, ch, S, dS, acc))
        if acc:
            S = S_new
        else:
            for m, r, c, old, new in reversed(ch):
                params.vals[m][r, c] = np.float32(old)
    return rows, params, S


# ------------------------------------------------------------------------------------------------
# Mini-batch schedules (Sections 2.2 and 2.5: a batch of 30,000 of the 60,000 samples; a batch size
# that grows during training). The trials of stretch s = tau // stretch decide on the loss summed
# over batch s only (Eq. 2 over the batch's samples); the weights and the trial counter carry over
# from batch to batch. Which samples form each batch is an input (the paper gives no rule).
# ------------------------------------------------------------------------------------------------

def run_batches(layers, loss: str, X: np.ndarray, y: np.ndarray, init, batches, stretch: int,
                seed: int, domain, params: Optional[Params] = None):
    """Trials 0 .. len(batches) * stretch - 1; batch s (an index array into X, y) serves trials
    s * stretch .. (s + 1) * stretch - 1 through the cached-field mode on its samples. Returns
    (concatenated trace arrays, final Params, loss sum of the last batch)."""
    params = Params(layers, init) if params is None else params
    traces, S = [], 0.0
    for s, b in enumerate(batches):
        b = np.asarray(b)
        tr, params, S = run_incremental(layers, loss, X[b], y[b], None, stretch, seed, domain,
                                        tau0=s * stretch, params=params)
        traces.append(tr)
    return {k: np.concatenate([t[k] for t in traces]) for k in traces[0]}, params, S


# ------------------------------------------------------------------------------------------------
# Loss change of a later first-layer candidate given that an earlier one is kept (two-layer nets).
# A speculative batch whose decision keeps candidate c1 can decide a later candidate c2 in the same
# pass if it knows dS(c2 | c1). When both change first-layer weights of different hidden rows
# (j1 != j2), c2's output-field change is unaffected by c1, so dS(c2 | c1) differs from dS(c2) only
# on the samples where both input features are non-zero:
#   dS(c2 | c1) = dS(c2) + sum_{n: x[n,i1] != 0 != x[n,i2]}
#                 [l(z + d1 + d2) - l(z + d1) - l(z + d2) + l(z)]_n
# with z the cached output fields and d_k = W2[:, j_k] (f(z1[j_k] + D_k x[i_k]) - f(z1[j_k])).
# ------------------------------------------------------------------------------------------------

def conditional_dS_two_layer(params: Params, XT: np.ndarray, y: np.ndarray, loss: str, p1, p2):
    """dS of proposal p2 given that proposal p1 was kept, by the correction above; p1 and p2 are
    first-layer proposals (layer 0) on different hidden rows. Returns (dS(p2 | p1), dS(p2),
    number of samples in the correction)."""
    if p1.layer != 0 or p2.layer != 0 or p1.row == p2.row:
        raise ValueError("two first-layer proposals on different hidden rows")
    L1, L2 = params.layers
    W1, W2 = params.eff64(0), params.eff64(1)
    z = W2 @ act_fn(L1.act, W1 @ XT, L1.act_param)

    def change(p):
        zr = W1[p.row] @ XT
        da = act_fn(L1.act, zr + (p.new - p.old) * XT[p.col], L1.act_param) - \
            act_fn(L1.act, zr, L1.act_param)
        return np.outer(W2[:, p.row], da)

    def ell(zz):
        return loss_per_sample(loss, act_fn(L2.act, zz, L2.act_param), y)

    d1, d2 = change(p1), change(p2)
    dS2 = float((ell(z + d2) - ell(z)).sum())
    both = (XT[p1.col] != 0) & (XT[p2.col] != 0)
    zb, d1b, d2b, yb = z[:, both], d1[:, both], d2[:, both], y[both]

    def ellb(zz):
        return loss_per_sample(loss, act_fn(L2.act, zz, L2.act_param), yb)
    corr = float((ellb(zb + d1b + d2b) - ellb(zb + d1b) - ellb(zb + d2b) + ellb(zb)).sum())
    return dS2 + corr, dS2, int(both.sum())
