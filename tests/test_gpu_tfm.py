"""Parity of the CUDA Transformer path with the CPU oracle (needs a GPU).

Small specs check trajectories (proposals bit for bit, decisions with the tie band replayed, final
parameters) on the SIMT kernels; the config-sized spec (vocab 65, context 64, d_model 128, 2 blocks
of 4 heads, FFN 512, 256 sequences) is checked on candidates of every stage and on a short run, on
the tensor-core kernels and on the SIMT kernels.
"""
import numpy as np
import pytest

from oracle import mca_tfm as T
from paper_2607_08406_gb300 import workloads as W

from parity import compare, forced_from_oracle, TIE_REL

pytestmark = pytest.mark.gpu

SMALL = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=2, n_head=2, d_ff=32)
MID = W.TfmSpec(vocab=23, ctx=20, d_model=40, n_layer=1, n_head=4, d_ff=200, act="gaussian")


def _wl(spec, batch, seed=0, trials=400):
    return W.char_transformer(seed=seed, batch=batch, text_len=20000, spec=spec,
                              n_trials=trials, K=8)


@pytest.mark.parametrize("spec,batch,trials", [(SMALL, 6, 400), (MID, 5, 150)])
def test_tfm_initial_loss_and_trajectory(gpu_lib, spec, batch, trials):
    wl = _wl(spec, batch, trials=trials)
    h = gpu_lib.create_from_tfm_workload(wl, trace_cap=trials)
    S0 = T.tfm_seq_losses(spec, wl.init.astype(np.float64), wl.tokens).sum()
    assert gpu_lib.mca_loss(h) * batch * spec.ctx == pytest.approx(S0, rel=1e-5)
    tr, flat, S = T.run_full_tfm(spec, wl.tokens, wl.init, trials, wl.seed, wl.domain)
    gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr))
    st = gpu_lib.mca_run(h, trials, wl.seed)
    assert st["trials"] == trials and st["accepts"] > 10
    compare(gpu_lib.mca_get_trace(h, trials), tr)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), flat)
    assert gpu_lib.mca_loss(h) * batch * spec.ctx == pytest.approx(S, rel=TIE_REL)


def test_tfm_K_invariance(gpu_lib):
    wl = _wl(SMALL, 6)
    ref = None
    for K in (1, 4, 32):
        h = gpu_lib.create_from_tfm_workload(wl, K=K, trace_cap=200)
        gpu_lib.mca_run(h, 200, 1)
        g = gpu_lib.mca_get_trace(h, 200)
        if ref is None:
            ref = g
        else:
            assert np.array_equal(g, ref)
        h.close()


def _stage_indices(spec, rng):
    offs, o = {}, 0
    for name, shape in spec.blocks():
        n = int(np.prod(shape))
        offs[name] = (o, n)
        o += n
    names = ["tok_emb", "pos_emb", "b0.ln1.g", "b0.wq", "b0.bv", "b0.wo", "b0.w1", "b0.b2",
             f"b{spec.n_layer - 1}.wk", f"b{spec.n_layer - 1}.w2", "lnf.g", "lnf.b", "w_head",
             "b_head"]
    return np.array([offs[nm][0] + rng.integers(0, offs[nm][1]) for nm in names], np.uint32)


def _oracle_dS(spec, flat, tokens, idx, new):
    base = T.tfm_seq_losses(spec, flat.astype(np.float64), tokens).sum()
    out = []
    for i, v in zip(idx, new):
        f2 = flat.copy()
        f2[int(i)] = np.float32(v)
        out.append(T.tfm_seq_losses(spec, f2.astype(np.float64), tokens).sum() - base)
    return np.array(out), base


@pytest.mark.parametrize("spec,batch", [(SMALL, 6), (MID, 5)])
def test_tfm_eval_candidates_every_stage(gpu_lib, spec, batch):
    wl = _wl(spec, batch)
    h = gpu_lib.create_from_tfm_workload(wl)
    gpu_lib.mca_run(h, 100, 2)
    flat = gpu_lib.mca_get_params(h, wl.n_params)
    rng = np.random.default_rng(4)
    idx = _stage_indices(spec, rng)
    new = rng.uniform(-1, 1, len(idx)).astype(np.float32)
    d = gpu_lib.mca_eval_candidates(h, idx, new)
    want, S = _oracle_dS(spec, flat, wl.tokens, idx, new)
    assert np.all(np.abs(d - want) <= TIE_REL * S), (d, want)


def test_tfm_resync_keeps_loss(gpu_lib):
    wl = _wl(MID, 5)
    h = gpu_lib.create_from_tfm_workload(wl)
    st = gpu_lib.mca_run(h, 300, 3)
    assert st["accepts"] > 20
    L = gpu_lib.mca_loss(h)
    gpu_lib.mca_resync(h)
    assert gpu_lib.mca_loss(h) == pytest.approx(L, rel=1e-5)


@pytest.mark.parametrize("tensor_cores", ["1", "0"])
def test_tfm_full_size(gpu_lib, monkeypatch, tensor_cores):
    """vocab 65, context 64, d_model 128, 2 blocks x 4 heads, FFN 512, 256 sequences, on the
    tensor-core kernels (the default at this shape) and on the SIMT kernels: the initial loss and
    candidates of every stage against the oracle, then 64 trials replayed through the oracle's
    proposal rule with the final loss."""
    monkeypatch.setenv("MCA_TFM_TENSOR_CORES", tensor_cores)
    wl = W.char_transformer()
    spec = wl.spec
    h = gpu_lib.create_from_tfm_workload(wl, trace_cap=64)
    assert gpu_lib.mca_get_stats(h)["tensor_cores"] == int(tensor_cores)
    rng = np.random.default_rng(9)
    idx = _stage_indices(spec, rng)[[0, 1, 3, 6, 9, 12]]
    new = rng.uniform(-1, 1, len(idx)).astype(np.float32)
    d = gpu_lib.mca_eval_candidates(h, idx, new)
    want, S0 = _oracle_dS(spec, wl.init, wl.tokens, idx, new)
    assert gpu_lib.mca_loss(h) * 256 * 64 == pytest.approx(S0, rel=1e-5)
    assert np.all(np.abs(d - want) <= TIE_REL * S0), (d, want)
    st = gpu_lib.mca_run(h, 64, wl.seed)
    g = gpu_lib.mca_get_trace(h, 64)
    assert st["trials"] == 64
    flat = wl.init.copy()
    for t in range(64):
        idx_t, old, newv, valid = T.tfm_propose(wl.seed, t, flat, wl.domain)
        assert idx_t == int(g["idx"][t]) and np.float32(newv) == g["new_w"][t]
        if g["accept"][t]:
            flat[idx_t] = np.float32(newv)
    assert np.array_equal(gpu_lib.mca_get_params(h, wl.n_params), flat)
    S = T.tfm_seq_losses(spec, flat.astype(np.float64), wl.tokens).sum()
    assert gpu_lib.mca_loss(h) * 256 * 64 == pytest.approx(S, rel=1e-5)
