"""Parity of the CUDA Transformer path with the CPU oracle (needs a GPU).

Small specs check trajectories (proposals bit for bit, decisions with the tie band replayed, final
parameters) on the SIMT kernels; specs of the tensor-core kernels' shape (context 64, d_model 128,
4 heads, d_ff a multiple of 128, an even number of sequences) with few sequences and narrow FFNs
check trajectories and candidates of every parameter tensor on the tensor-core kernels. The
config-sized spec is in test_gpu_config_size.py.
"""
import numpy as np
import pytest

from oracle import mca_tfm as T
from paper_2607_08406_gb300 import workloads as W

from parity import compare, forced_from_oracle, TIE_REL

pytestmark = pytest.mark.gpu

SMALL = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=2, n_head=2, d_ff=32)
MID = W.TfmSpec(vocab=23, ctx=20, d_model=40, n_layer=1, n_head=4, d_ff=200, act="gaussian")
# the tensor-core kernels' shape with one or two blocks, narrow FFNs and few sequences
TC_ONE = W.TfmSpec(vocab=65, ctx=64, d_model=128, n_layer=1, n_head=4, d_ff=128)
TC_TWO = W.TfmSpec(vocab=65, ctx=64, d_model=128, n_layer=2, n_head=4, d_ff=128, act="gaussian",
                   act_param=0.4)


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


@pytest.mark.parametrize("spec,batch,trials", [(TC_ONE, 4, 150), (TC_TWO, 2, 120)])
def test_tfm_tensor_core_trajectory(gpu_lib, monkeypatch, spec, batch, trials):
    """The tensor-core kernels (the default at the workload's shape) trial by trial against the
    oracle's full-recompute loop: proposals, decisions, dS, final parameters and loss."""
    monkeypatch.delenv("MCA_TFM_TENSOR_CORES", raising=False)
    wl = _wl(spec, batch, trials=trials)
    h = gpu_lib.create_from_tfm_workload(wl, trace_cap=trials)
    assert gpu_lib.mca_get_stats(h)["tensor_cores"] == 1
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
    # one random parameter of every named tensor (all 16 of every block)
    return np.array([o + rng.integers(0, n) for o, n in offs.values()], np.uint32)


def _oracle_dS(spec, flat, tokens, idx, new):
    base = T.tfm_seq_losses(spec, flat.astype(np.float64), tokens).sum()
    out = []
    for i, v in zip(idx, new):
        f2 = flat.copy()
        f2[int(i)] = np.float32(v)
        out.append(T.tfm_seq_losses(spec, f2.astype(np.float64), tokens).sum() - base)
    return np.array(out), base


@pytest.mark.parametrize("spec,batch", [(SMALL, 6), (MID, 5), (TC_ONE, 4), (TC_TWO, 2)])
def test_tfm_eval_candidates_every_stage(gpu_lib, monkeypatch, spec, batch):
    monkeypatch.delenv("MCA_TFM_TENSOR_CORES", raising=False)
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


def test_tfm_one_ahead_batches_match_round_trip_batches(gpu_lib, monkeypatch):
    """The tensor-core path enqueues each batch before the host reads the previous decision (the
    trial counter lives on the device) unless the handle has a resync period; with a period longer
    than the run (the round-trip loop, no resync) the trace, parameters and loss are bit-identical,
    over runs of several lengths (one trial, a few batches, and a longer one) continuing the chain."""
    monkeypatch.delenv("MCA_TFM_TENSOR_CORES", raising=False)
    wl = W.char_transformer()
    out = []
    for R in (0, 10 ** 9):
        h = gpu_lib.create_from_tfm_workload(wl, trace_cap=400, resync_period=R)
        n = 0
        for m in (1, 7, 150):
            st = gpu_lib.mca_run(h, m, 11)
            n += m
            assert st["trials"] == n and st["tau"] == n and st["tensor_cores"] == 1
        out.append((gpu_lib.mca_get_trace(h, n), gpu_lib.mca_get_params(h, wl.n_params),
                    gpu_lib.mca_loss(h)))
        assert st["resyncs"] == 0
        h.close()
    assert np.array_equal(out[0][0], out[1][0])
    assert np.array_equal(out[0][1], out[1][1])
    assert out[0][2] == out[1][2]
