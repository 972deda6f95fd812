"""A mini-batch schedule through the C ABI against the oracle's run_batches (needs a GPU).

Sections 2.2 and 2.5 train on batches of the training set (half of it; a batch size that grows).
Through the C ABI a batch is a handle created on that batch's samples: at each switch the caller
reads the weights (mca_get_params), creates a handle on the next batch with them as the initial
weights and sets the trial counter (mca_set_params, which recomputes every cached field), then
runs the stretch's trials. Decisions, dS and the final weights must follow the oracle's schedule,
as for the full-batch loop.
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

from parity import compare, forced_from_oracle, TIE_REL

pytestmark = pytest.mark.gpu

CASES = {
    # name: (workload builder, batch size, batches, trials per batch)
    "wide_half_batches": (lambda: W.make("mlp_wide", N=6000, H=128), 3000, 4, 500),
    "deep_tc_half_batches": (lambda: W.mlp_deep(N=2200, width=256, depth=4, n_trials=450, K=16),
                             1100, 3, 150),
}


@pytest.mark.parametrize("case", list(CASES))
def test_minibatch_schedule_through_the_abi(gpu_lib, case):
    build, B, nb, M = CASES[case]
    wl = build()
    batches = W.minibatches(wl.N, B, nb, seed=4)
    tr, params, S = O.run_batches(wl.layers, wl.loss, wl.X, wl.y, wl.init, batches, M, wl.seed,
                                  wl.domain)
    flat = wl.init.copy()
    for s, b in enumerate(batches):
        sub = W.MLPWorkload(wl.name, wl.layers, wl.loss, np.ascontiguousarray(wl.X[b]),
                            np.ascontiguousarray(wl.y[b]), flat, M, wl.K, wl.seed, wl.domain)
        h = gpu_lib.create_from_workload(sub, trace_cap=M)
        gpu_lib.mca_set_params(h, flat, tau=s * M)
        part = {k: v[s * M:(s + 1) * M] for k, v in tr.items()}
        gpu_lib.mca_force_decisions(h, *forced_from_oracle(part))
        st = gpu_lib.mca_run(h, M, wl.seed)
        assert st["tau"] == (s + 1) * M
        compare(gpu_lib.mca_get_trace(h, M), part)
        flat = gpu_lib.mca_get_params(h, wl.n_params)
        h.close()
    assert np.array_equal(flat, params.flat_eff32())
    assert tr["accept"].sum() > 30


def test_growing_batch_of_sequences_transformer(gpu_lib):
    """Section 2.5's adaptive batch size: the Transformer trains on 4, then 8, then 16 sequences
    (each batch a handle created with the previous batch's weights), against the oracle's
    full-recompute loop on the same batches."""
    from oracle import mca_tfm as T
    import dataclasses
    spec = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=2, n_head=2, d_ff=32)
    wl = W.char_transformer(seed=0, batch=16, text_len=20000, spec=spec, n_trials=300, K=8)
    M = 100
    flat_o = wl.init.copy()
    flat = wl.init.copy()
    for s, B in enumerate((4, 8, 16)):
        tok = np.ascontiguousarray(wl.tokens[:B])
        tr, flat_o, S = T.run_full_tfm(spec, tok, flat_o, M, wl.seed, wl.domain, tau0=s * M)
        sub = dataclasses.replace(wl, tokens=tok, init=flat)
        h = gpu_lib.create_from_tfm_workload(sub, trace_cap=M)
        gpu_lib.mca_set_params(h, flat, tau=s * M)
        gpu_lib.mca_force_decisions(h, *forced_from_oracle(tr))
        gpu_lib.mca_run(h, M, wl.seed)
        compare(gpu_lib.mca_get_trace(h, M), tr)
        flat = gpu_lib.mca_get_params(h, wl.n_params)
        assert gpu_lib.mca_loss(h) * B * spec.ctx == pytest.approx(S, rel=TIE_REL)
        h.close()
    assert np.array_equal(flat, flat_o)
