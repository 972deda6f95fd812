"""The Transformer tensor-core kernel's design, emulated on the CPU (tests/tc_emulator.py), against
the oracle: losses of every sequence after a forward pass, the loss change of candidates in every
stage and of every parameter kind (the rank-1 term of each weight matrix and the patched reads of
biases, LN parameters and embeddings), and the commit writing exactly what the evaluation computed.

This checks the kernel's offsets, descriptors, chunk schedule, swizzles and epilogue terms, not the
hardware: the kernel itself is compared with the oracle by the GPU tests.
"""
import copy

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
    old = np.float32(a.params[idx])
    return (idx, neww, np.float32(neww - old), E.tfm_stage(a, idx), row, old)


def _picks(a):
    b0, b1 = a.o_blk0, a.o_blk0 + a.blk_size
    return {
        "tok_emb": int(a.tokens[0, 3]) * a.d + 5, "pos_emb": a.o_pos + 7 * a.d + 100,
        "ln1.g": b0 + a.r_ln1g + 9, "wq": b0 + a.r_wq + 37 * a.d + 101,
        "wk": b0 + a.r_wk + 70 * a.d + 3, "wv": b1 + a.r_wv + 127 * a.d + 64,
        "bq": b1 + a.r_bq + 31, "wo": b0 + a.r_wo + 12 * a.d + 99, "ln2.b": b1 + a.r_ln2b + 1,
        "w1": b0 + a.r_w1 + 77 * a.d + 18, "b1": b1 + a.r_b1 + 100,
        "w2": b1 + a.r_w2 + 40 * a.F + 90, "w2.b0": b0 + a.r_w2 + 127 * a.F + 3,
        "b2": b0 + a.r_b2 + 17, "lnf.g": a.o_lnf_g + 60,
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


def test_emulated_adoption_writes_what_the_commit_writes(setup):
    """An evaluation with a scratch slot followed by the adopt kernel leaves the residual streams
    (block inputs and mid streams) and sequence losses exactly as the commit kernel would, for a
    candidate of every stage kind: token embeddings (one whose token some sequences lack: they keep
    theirs), a position embedding, a block-0 projection, LN2 of block 0 and the last block's FFN
    (both restart at their block's mid stream) and the head."""
    spec, a0 = setup
    picks = _picks(a0)
    # a token that some sequences contain and others do not
    present = np.array([[np.any(a0.tokens[s, :E.kT] == v) for s in range(a0.B)]
                        for v in range(a0.V)])
    partial = np.nonzero(present.any(axis=1) & ~present.all(axis=1))[0]
    assert len(partial) > 0
    picks["tok_emb_partial"] = int(partial[0]) * a0.d + 11
    picks["ln2.b0"] = a0.o_blk0 + a0.r_ln2b + 3
    for name in ("tok_emb", "tok_emb_partial", "pos_emb", "wq", "ln2.b0", "w2", "w_head"):
        a = copy.deepcopy(a0)
        c = _cand(a, picks[name], 0.37)
        slot = E.Slot(a)
        for p in range(a.B // 2):
            E.CTA(a, E.EVAL, c, p, slot).run()
        b = copy.deepcopy(a)
        a.params[c[0]] = c[1]                       # the decide kernel's write
        b.params[c[0]] = c[1]
        for p in range(a.B // 2):
            E.CTA(a, E.COMMIT, c, p).run()
        E.adopt(b, slot, c)
        np.testing.assert_array_equal(b.X, a.X, err_msg=name)
        np.testing.assert_array_equal(b.Xmid, a.Xmid, err_msg=name)
        np.testing.assert_array_equal(b.ell, a.ell, err_msg=name)


def test_emulated_kernel_at_the_largest_shape_it_takes():
    """Vocabulary 128, d_ff 1024 and three blocks (the largest vocabulary and hidden width the
    tensor-core kernels accept): forward losses, and candidates at the last row / column of every
    weight matrix, the last hidden chunk, the last position and the last vocabulary entry, against
    the oracle; a commit writes what the evaluation computed."""
    spec = W.TfmSpec(vocab=128, d_ff=1024, n_layer=3)
    wl = W.char_transformer(batch=2, spec=spec, text_len=20000)
    a = E.Args(spec, wl.init, wl.tokens)
    a.split()
    for pair in range(a.B // 2):
        E.CTA(a, E.FORWARD, None, pair).run()
    ell = OT.tfm_seq_losses(spec, a.params.astype(np.float64), a.tokens)
    assert np.all(np.abs(a.ell - ell) <= 2e-6 * ell)
    d, F, V, T = a.d, a.F, spec.vocab, spec.ctx
    bl = a.o_blk0 + 2 * a.blk_size                       # the last block
    last_tok = int(a.tokens[1, T - 1])
    picks = {
        "tok_emb": last_tok * d + d - 1, "pos_emb": a.o_pos + (T - 1) * d + d - 1,
        "wq": bl + a.r_wq + (d - 1) * d + d - 1, "wv": bl + a.r_wv + (d - 1) * d,
        "wo": bl + a.r_wo + d - 1, "w1": bl + a.r_w1 + (F - 1) * d + d - 1,
        "b1": bl + a.r_b1 + F - 1, "w2": bl + a.r_w2 + (d - 1) * F + F - 1,
        "b2": bl + a.r_b2 + d - 1, "lnf.b": a.o_lnf_b + d - 1,
        "w_head": a.o_wh + (V - 1) * d + d - 1, "b_head": a.o_bh + V - 1,
    }
    for name, idx in picks.items():
        c = _cand(a, idx, -0.29)
        q = a.params.copy()
        q[idx] = c[1]
        want = OT.tfm_seq_losses(spec, q.astype(np.float64), a.tokens) - ell
        got = np.concatenate([E.CTA(a, E.EVAL, c, p).run() for p in range(a.B // 2)])
        assert np.all(np.abs(got - want) <= 2e-6 * ell), (name, got, want)
    c = _cand(a, picks["w1"], 0.61)
    ell0 = a.ell.copy()
    dS = np.concatenate([E.CTA(a, E.EVAL, c, p).run() for p in range(a.B // 2)])
    a.params[c[0]] = c[1]
    for p in range(a.B // 2):
        E.CTA(a, E.COMMIT, c, p).run()
    np.testing.assert_array_equal(a.ell, (ell0 + dS).astype(np.float32))


def test_emulated_kernel_with_an_odd_number_of_hidden_pairs():
    """d_ff 384 (three pairs of 64-wide hidden chunks per W1 product) in one Gaussian block: the
    forward losses, and candidates at the first and last hidden unit of every pair (W1 rows, b1,
    W2 columns: the rank-1 steps), LN2 (the mid-stream restart) and b2, against the oracle; an
    evaluation with a scratch slot plus adoption equals the commit."""
    spec = W.TfmSpec(d_ff=384, n_layer=1, act="gaussian", act_param=0.4)
    wl = W.char_transformer(batch=2, spec=spec, text_len=20000)
    a = E.Args(spec, wl.init, wl.tokens)
    a.split()
    for pair in range(a.B // 2):
        E.CTA(a, E.FORWARD, None, pair).run()
    ell = OT.tfm_seq_losses(spec, a.params.astype(np.float64), a.tokens)
    assert np.all(np.abs(a.ell - ell) <= 2e-6 * ell)
    d, F = a.d, a.F
    b0 = a.o_blk0
    picks = {"ln2.g": b0 + a.r_ln2g + 17, "b2": b0 + a.r_b2 + 100}
    for u in (0, 127, 128, 255, 256, 383):
        picks[f"w1[{u}]"] = b0 + a.r_w1 + u * d + (u * 7) % d
        picks[f"b1[{u}]"] = b0 + a.r_b1 + u
        picks[f"w2[:,{u}]"] = b0 + a.r_w2 + ((u * 5) % d) * F + u
    for name, idx in picks.items():
        c = _cand(a, idx, 0.43)
        q = a.params.copy()
        q[idx] = c[1]
        want = OT.tfm_seq_losses(spec, q.astype(np.float64), a.tokens) - ell
        got = np.concatenate([E.CTA(a, E.EVAL, c, p).run() for p in range(a.B // 2)])
        assert np.all(np.abs(got - want) <= 2e-6 * ell), (name, got, want)
    for name in ("w1[255]", "ln2.g"):
        b = copy.deepcopy(a)
        c = _cand(b, picks[name], -0.71)
        slot = E.Slot(b)
        for p in range(b.B // 2):
            E.CTA(b, E.EVAL, c, p, slot).run()
        r = copy.deepcopy(b)
        b.params[c[0]] = c[1]
        r.params[c[0]] = c[1]
        for p in range(b.B // 2):
            E.CTA(b, E.COMMIT, c, p).run()
        E.adopt(r, slot, c)
        np.testing.assert_array_equal(r.X, b.X, err_msg=name)
        np.testing.assert_array_equal(r.Xmid, b.Xmid, err_msg=name)
        np.testing.assert_array_equal(r.ell, b.ell, err_msg=name)
