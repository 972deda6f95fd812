"""Seeded synthetic workloads for the Monte Carlo mutation-selection (MCA) trial loop.

This module only *draws inputs*: the data matrix X, the labels y and the initial parameters.
It holds none of the method's arithmetic (no proposal, no loss, no selection), so both the CUDA
path and the CPU oracle can take their inputs from here without sharing any code of the method.

The paper trains on MNIST (60,000 training samples, 28x28 grey images, 10 classes; Section 2) and
on Tiny Shakespeare (Section 2.5). Neither dataset is used: seeded synthetic stand-ins with the same
shapes replace them.

* Images: 784 features with values in [0, 1], each entry zeroed with probability 0.8 (MNIST's
  pixel sparsity).  ``dyadic=True`` draws the non-zero values as k/256, k in 1..255, so that they
  are exact in fp32 and in uint8 (used by the discrete-weight / pruning workload, whose first layer
  then sums exactly in any order).
* Labels: argmax of a fixed random teacher MLP 784-32-10 (tanh hidden layer, weights uniform in
  +-sqrt(3/fan_in), no biases). The teacher is data synthesis only, not part of the method.
* Initial weights: uniform in +-a (a per workload), drawn in fp32.

Every array is drawn from numpy's PCG64 with a seed sequence (workload id, seed, stream id), so the
same call gives the same bytes on every machine.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np

ACTS = ("identity", "tanh", "sigmoid", "relu", "gaussian", "gelu")
LOSSES = ("mse_onehot", "softmax_ce")
WKINDS = ("fp32", "ternary_i8", "masked_fp32")
OPS = ("replace", "perturb")

# stream ids of the seed sequence
_S_X, _S_TEACHER, _S_INIT, _S_MASKVAL = 1, 2, 3, 4


@dataclass
class Layer:
    n_in: int
    n_out: int
    act: str = "tanh"
    act_param: float = 0.0      # gamma of the Gaussian exp(-gamma x^2); unused otherwise
    wkind: str = "fp32"
    scale: float = 1.0          # ternary layers: the effective weight is scale * code


@dataclass
class Domain:
    """Mutation operator and weight domain (Eq. 1)."""
    op: str = "replace"         # replace: w <- U[lo, hi); perturb: w <- w + delta * U[-1, 1)
    lo: float = -1.0
    hi: float = 1.0
    delta: float = 0.01
    bound: float = 0.0          # > 0: a proposal with |w'| >= bound is rejected unevaluated
    strict: bool = False        # False: accept iff dS <= 0 (Eq. 1, Eq. 6); True: dS < 0
    beta: float = float("inf")  # selection intensity of the Metropolis rule (Eq. 7); inf: greedy
    layer_stretch: int = 0      # > 0: current-layer schedule (Section 2.1), stretches of this many
                                #   trials each mutating one randomly chosen layer; 0: uniform


@dataclass
class MLPWorkload:
    name: str
    layers: List[Layer]
    loss: str
    X: np.ndarray               # [N, D] float32, sample-major
    y: np.ndarray               # [N] int32
    init: np.ndarray            # [P] float32; ternary layers hold codes in {-1,0,1}
    n_trials: int
    K: int
    seed: int = 0
    domain: Domain = field(default_factory=Domain)

    @property
    def n_params(self) -> int:
        return sum(l.n_in * l.n_out for l in self.layers)

    @property
    def N(self) -> int:
        return int(self.X.shape[0])


def _rng(workload_id: int, seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([workload_id, seed, stream])))


def synth_images(rng: np.random.Generator, n: int, d: int = 784, density: float = 0.2,
                 dyadic: bool = False) -> np.ndarray:
    """[n, d] float32 in [0, 1]; each entry non-zero with probability ``density``."""
    keep = rng.random((n, d), dtype=np.float32) < np.float32(density)
    if dyadic:
        vals = (rng.integers(1, 256, size=(n, d), dtype=np.int32).astype(np.float32)
                * np.float32(1.0 / 256.0))
    else:
        vals = rng.random((n, d), dtype=np.float32)
    x = np.where(keep, vals, np.float32(0.0)).astype(np.float32)
    return np.ascontiguousarray(x)


def teacher_labels(rng: np.random.Generator, X: np.ndarray, hidden: int = 32,
                   n_classes: int = 10) -> np.ndarray:
    """Labels = argmax of a fixed random teacher MLP d-hidden-n_classes (tanh hidden layer)."""
    d = X.shape[1]
    a1 = np.sqrt(3.0 / d)
    a2 = np.sqrt(3.0 / hidden)
    W1 = rng.uniform(-a1, a1, size=(hidden, d))
    W2 = rng.uniform(-a2, a2, size=(n_classes, hidden))
    h = np.tanh(X.astype(np.float64) @ W1.T)
    return np.ascontiguousarray(np.argmax(h @ W2.T, axis=1).astype(np.int32))


def uniform_init(rng: np.random.Generator, layers: List[Layer], a) -> np.ndarray:
    parts = []
    for l, layer in enumerate(layers):
        al = a[l] if isinstance(a, (list, tuple)) else a
        parts.append(rng.uniform(-al, al, size=layer.n_in * layer.n_out).astype(np.float32))
    return np.ascontiguousarray(np.concatenate(parts).astype(np.float32))


# ------------------------------------------------------------------------------------------------
# The five workloads (sizes may be scaled down for parity cases; defaults are the full sizes)
# ------------------------------------------------------------------------------------------------

def mlp_small(seed: int = 0, N: int = 1000, H: int = 64, D: int = 784, n_trials: int = 20000,
              K: int = 16) -> MLPWorkload:
    """784-64-10, tanh hidden, sigmoid outputs, MSE vs one-hot; N=1000; init U[-0.1,0.1];
    replacement mutations U[-1,1); 20k trials."""
    wid = 1
    X = synth_images(_rng(wid, seed, _S_X), N, D)
    y = teacher_labels(_rng(wid, seed, _S_TEACHER), X)
    layers = [Layer(D, H, "tanh"), Layer(H, 10, "sigmoid")]
    init = uniform_init(_rng(wid, seed, _S_INIT), layers, 0.1)
    return MLPWorkload("mlp784-64-10_mse_n1000", layers, "mse_onehot", X, y, init, n_trials, K, seed)


def mlp_wide(seed: int = 0, N: int = 60000, H: int = 16384, D: int = 784,
             n_trials: int = 1_000_000, K: int = 64) -> MLPWorkload:
    """784-16384-10, tanh, softmax CE; N=60000; init U[-0.05,0.05]; replacement U[-1,1); K=64."""
    wid = 2
    X = synth_images(_rng(wid, seed, _S_X), N, D)
    y = teacher_labels(_rng(wid, seed, _S_TEACHER), X)
    layers = [Layer(D, H, "tanh"), Layer(H, 10, "identity")]
    init = uniform_init(_rng(wid, seed, _S_INIT), layers, 0.05)
    return MLPWorkload(f"mlp784-{H}-10_ce_n{N}", layers, "softmax_ce", X, y, init, n_trials, K, seed)


def mlp_deep(seed: int = 0, N: int = 10000, width: int = 256, depth: int = 24, D: int = 784,
             n_trials: int = 200_000, K: int = 128) -> MLPWorkload:
    """24 hidden tanh layers of width 256 (25 weight matrices), 784 in, 10 out, softmax CE, no
    normalisation, no residuals; N=10000; init U[+-sqrt(3/fan_in)]."""
    wid = 3
    X = synth_images(_rng(wid, seed, _S_X), N, D)
    y = teacher_labels(_rng(wid, seed, _S_TEACHER), X)
    dims = [D] + [width] * depth + [10]
    layers = [Layer(dims[l], dims[l + 1], "tanh" if l < depth else "identity")
              for l in range(depth + 1)]
    init = uniform_init(_rng(wid, seed, _S_INIT), layers,
                        [float(np.sqrt(3.0 / layer.n_in)) for layer in layers])
    return MLPWorkload(f"mlp784-{width}x{depth}-10_ce_n{N}", layers, "softmax_ce", X, y, init,
                       n_trials, K, seed)


def mlp_ternary(seed: int = 0, N: int = 60000, H: int = 4096, D: int = 784,
                n_trials: int = 1_000_000, K: int = 64) -> MLPWorkload:
    """784-4096-10 ternary weights {-1,0,+1} (int8 codes, fixed per-layer dyadic scales 2^-4 and
    2^-6), Gaussian exp(-x^2) hidden, sigmoid outputs, MSE; dyadic inputs k/256."""
    wid = 4
    X = synth_images(_rng(wid, seed, _S_X), N, D, dyadic=True)
    y = teacher_labels(_rng(wid, seed, _S_TEACHER), X)
    layers = [Layer(D, H, "gaussian", 1.0, "ternary_i8", 2.0 ** -4),
              Layer(H, 10, "sigmoid", 0.0, "ternary_i8", 2.0 ** -6)]
    rng = _rng(wid, seed, _S_INIT)
    init = rng.integers(-1, 2, size=D * H + H * 10).astype(np.float32)
    return MLPWorkload(f"mlp784-{H}-10_ternary_gauss_mse_n{N}", layers, "mse_onehot", X, y,
                       np.ascontiguousarray(init), n_trials, K, seed)


def mlp_masked(seed: int = 0, N: int = 60000, H: int = 4096, D: int = 784,
               n_trials: int = 1_000_000, K: int = 64) -> MLPWorkload:
    """784-4096-10 pruning net: fixed random-init fp32 weights on a dyadic grid (layer 1: q/512,
    |q| <= 64; layer 2: q/1024, |q| <= 64), a mask bit per weight toggled by each mutation;
    Gaussian exp(-x^2) hidden, sigmoid outputs, MSE; dyadic inputs k/256."""
    wid = 5
    X = synth_images(_rng(wid, seed, _S_X), N, D, dyadic=True)
    y = teacher_labels(_rng(wid, seed, _S_TEACHER), X)
    layers = [Layer(D, H, "gaussian", 1.0, "masked_fp32"),
              Layer(H, 10, "sigmoid", 0.0, "masked_fp32")]
    rng = _rng(wid, seed, _S_MASKVAL)
    w1 = rng.integers(-64, 65, size=D * H).astype(np.float32) / np.float32(512.0)
    w2 = rng.integers(-64, 65, size=H * 10).astype(np.float32) / np.float32(1024.0)
    init = np.ascontiguousarray(np.concatenate([w1, w2]).astype(np.float32))
    return MLPWorkload(f"mlp784-{H}-10_masked_gauss_mse_n{N}", layers, "mse_onehot", X, y, init,
                       n_trials, K, seed)


MLP_WORKLOADS = {
    "mlp_small": mlp_small,
    "mlp_wide": mlp_wide,
    "mlp_deep": mlp_deep,
    "mlp_ternary": mlp_ternary,
    "mlp_masked": mlp_masked,
}


def minibatches(n_samples: int, batch: int, n_batches: int, seed: int = 0) -> List[np.ndarray]:
    """Sample indices of n_batches mini-batches of ``batch`` samples each, every batch drawn without
    replacement (ascending indices) from the n_samples of a workload; consecutive batches are
    independent. Input generation only: which batch a trial uses is the caller's schedule."""
    rng = np.random.default_rng([7, seed, 9])
    return [np.sort(rng.choice(n_samples, size=batch, replace=False)).astype(np.int64)
            for _ in range(n_batches)]


def make(name: str, **kw) -> MLPWorkload:
    return MLP_WORKLOADS[name](**kw)



# ------------------------------------------------------------------------------------------------
# Character-level Transformer workload (stand-in for Tiny Shakespeare, Section 2.5)
# ------------------------------------------------------------------------------------------------

@dataclass
class TfmSpec:
    vocab: int = 65
    ctx: int = 64
    d_model: int = 128
    n_layer: int = 2
    n_head: int = 4
    d_ff: int = 512
    act: str = "gelu"           # FFN transfer function: "gelu" (exact erf) or "gaussian"
    act_param: float = 1.0      # gamma of the Gaussian
    ln_eps: float = 1e-5

    def blocks(self):
        """Flat parameter layout: (name, shape) in order. Matrices are [out x in] row-major."""
        d, f, v, t = self.d_model, self.d_ff, self.vocab, self.ctx
        out = [("tok_emb", (v, d)), ("pos_emb", (t, d))]
        for b in range(self.n_layer):
            out += [(f"b{b}.ln1.g", (d,)), (f"b{b}.ln1.b", (d,)),
                    (f"b{b}.wq", (d, d)), (f"b{b}.bq", (d,)),
                    (f"b{b}.wk", (d, d)), (f"b{b}.bk", (d,)),
                    (f"b{b}.wv", (d, d)), (f"b{b}.bv", (d,)),
                    (f"b{b}.wo", (d, d)), (f"b{b}.bo", (d,)),
                    (f"b{b}.ln2.g", (d,)), (f"b{b}.ln2.b", (d,)),
                    (f"b{b}.w1", (f, d)), (f"b{b}.b1", (f,)),
                    (f"b{b}.w2", (d, f)), (f"b{b}.b2", (d,))]
        out += [("lnf.g", (d,)), ("lnf.b", (d,)), ("w_head", (v, d)), ("b_head", (v,))]
        return out

    @property
    def n_params(self) -> int:
        return int(sum(np.prod(s) for _, s in self.blocks()))


@dataclass
class TfmWorkload:
    name: str
    spec: TfmSpec
    tokens: np.ndarray          # [B, ctx + 1] int32: inputs tokens[:, :ctx], targets tokens[:, 1:]
    init: np.ndarray            # [P] float32, flat layout of spec.blocks()
    n_trials: int
    K: int
    seed: int = 0
    domain: Domain = field(default_factory=Domain)

    @property
    def n_params(self) -> int:
        return self.spec.n_params


def markov_text(rng: np.random.Generator, vocab: int, length: int, alpha: float = 0.1):
    """A stream of `length` symbols from an order-2 Markov chain over `vocab` symbols whose
    transition rows are Dirichlet(alpha) draws; the first two symbols are uniform."""
    rows = rng.dirichlet(np.full(vocab, alpha), size=vocab * vocab)
    cdf = np.cumsum(rows, axis=1)
    cdf[:, -1] = 1.0
    u = rng.random(length)
    out = np.empty(length, dtype=np.int32)
    out[:2] = rng.integers(0, vocab, 2)
    for t in range(2, length):
        r = out[t - 2] * vocab + out[t - 1]
        out[t] = min(int(np.searchsorted(cdf[r], u[t], side="right")), vocab - 1)
    return out


def tfm_init(rng: np.random.Generator, spec: TfmSpec, std: float = 0.02) -> np.ndarray:
    """GPT-style initialisation: N(0, std) matrices and embeddings, zero biases, LN gains 1."""
    parts = []
    for name, shape in spec.blocks():
        n = int(np.prod(shape))
        if name.endswith(".g"):
            parts.append(np.ones(n, np.float32))
        elif len(shape) == 1:
            parts.append(np.zeros(n, np.float32))
        else:
            parts.append(rng.normal(0.0, std, n).astype(np.float32))
    return np.ascontiguousarray(np.concatenate(parts).astype(np.float32))


def char_transformer(seed: int = 0, batch: int = 256, text_len: int = 1_000_000,
                     spec: Optional[TfmSpec] = None, n_trials: int = 500_000,
                     K: int = 64) -> TfmWorkload:
    """Tiny char-level Transformer: vocab 65, context 64, d_model 128, 2 pre-LN blocks of 4 heads,
    FFN 512 (exact GELU), learned positions, untied head; next-char CE over a fixed batch of 256
    windows of an order-2 Markov stream (Dirichlet(0.1) rows, 1M symbols)."""
    wid = 6
    spec = spec or TfmSpec()
    rng = _rng(wid, seed, _S_X)
    text = markov_text(rng, spec.vocab, text_len)
    starts = _rng(wid, seed, _S_TEACHER).integers(0, text_len - spec.ctx - 1, batch)
    tokens = np.stack([text[s:s + spec.ctx + 1] for s in starts]).astype(np.int32)
    init = tfm_init(_rng(wid, seed, _S_INIT), spec)
    name = (f"gpt_v{spec.vocab}_t{spec.ctx}_d{spec.d_model}_l{spec.n_layer}_h{spec.n_head}"
            f"_f{spec.d_ff}_b{batch}")
    return TfmWorkload(name, spec, np.ascontiguousarray(tokens), init, n_trials, K, seed)
