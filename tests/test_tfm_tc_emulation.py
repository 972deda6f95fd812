"""The Transformer tensor-core kernel's design, emulated on the CPU (tests/tc_emulator.py), against
the oracle: losses of every sequence after a forward pass, the loss change of candidates in every
stage and of every parameter kind (the rank-1 term of each weight matrix and the patched reads of
biases, LN parameters and embeddings), and the commit writing exactly what the evaluation computed.

This checks the kernel's offsets, descriptors, chunk schedule, swizzles and epilogue terms, not the
hardware: the kernel itself is compared with the oracle by the GPU tests.
"""
import numpy as np
import pytest

from oracle import mca_tfm as OT
from paper_2607_08406_gb300 import workloads as W

import tc_emulator as E


@pytest.fixture(scope="module")
def setup():
    spec = W.TfmSpec(d_ff=128)
    wl = W.char_transformer(batch=4, spec=spec, text_len=20000)
    a = E.Args(spec, wl.init, wl.tokens)
    a.split()
    for pair in range(a.B // 2):
        E.CTA(a, E.FORWARD, None, pair).run()
    return spec, a


def _cand(a, idx, neww):
    neww = np.float32(neww)
    row = idx // a.d if idx < a.o_pos else -1
    return (idx, neww, np.float32(neww - a.params[idx]), E.tfm_stage(a, idx), row)


def _picks(a):
    b0, b1 = a.o_blk0, a.o_blk0 + a.blk_size
    return {
        "tok_emb": int(a.tokens[0, 3]) * a.d + 5, "pos_emb": a.o_pos + 7 * a.d + 100,
        "ln1.g": b0 + a.r_ln1g + 9, "wq": b0 + a.r_wq + 37 * a.d + 101,
        "wk": b0 + a.r_wk + 70 * a.d + 3, "wv": b1 + a.r_wv + 127 * a.d + 64,
        "bq": b1 + a.r_bq + 31, "wo": b0 + a.r_wo + 12 * a.d + 99, "ln2.b": b1 + a.r_ln2b + 1,
        "w1": b0 + a.r_w1 + 77 * a.d + 18, "b1": b1 + a.r_b1 + 100,
        "w2": b1 + a.r_w2 + 40 * a.F + 90, "lnf.g": a.o_lnf_g + 60,
        "w_head": a.o_wh + 20 * a.d + 66, "b_head": a.o_bh + 64,
    }


def test_emulated_forward_and_candidates_match_oracle(setup):
    spec, a = setup
    ell = OT.tfm_seq_losses(spec, a.params.astype(np.float64), a.tokens)
    assert np.all(np.abs(a.ell - ell) <= 2e-6 * ell)
    for name, idx in _picks(a).items():
        c = _cand(a, idx, 0.37)
        q = a.params.copy()
        q[idx] = c[1]
        want = OT.tfm_seq_losses(spec, q.astype(np.float64), a.tokens) - ell
        got = np.concatenate([E.CTA(a, E.EVAL, c, p).run() for p in range(a.B // 2)])
        assert np.all(np.abs(got - want) <= 2e-6 * ell), (name, got, want)


def test_emulated_commit_writes_what_evaluation_computed(setup):
    spec, a = setup
    for name in ("wq", "w2", "tok_emb", "w_head"):
        c = _cand(a, _picks(a)[name], -0.55)
        ell0 = a.ell.copy()
        dS = np.concatenate([E.CTA(a, E.EVAL, c, p).run() for p in range(a.B // 2)])
        a.params[c[0]] = c[1]                       # the decide kernel's write
        for p in range(a.B // 2):
            E.CTA(a, E.COMMIT, c, p).run()
        np.testing.assert_array_equal(a.ell, (ell0 + dS).astype(np.float32))
        t = E.tc_target(a, c[0], c[3])              # the image refresh after the commit
        if t[0] != E.kNone:
            o = E.image_offset(t[0], c[3], t[1], t[2], a.F, a.nL)
            hi = E.tf32_rna(c[1])
            a.wimg[o] = hi
            a.wimg[o + E.lo_off(t[0])] = E.tf32_rna(c[1] - hi)
        refreshed = a.wimg.copy()
        a.split()
        np.testing.assert_array_equal(refreshed, a.wimg)
        ell = OT.tfm_seq_losses(spec, a.params.astype(np.float64), a.tokens)
        assert np.all(np.abs(a.ell - ell) <= 2e-6 * ell), name
