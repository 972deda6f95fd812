"""The CUDA path's proposal-stream and decision helpers, compiled for the host, against the oracle.

csrc/mca_device.cuh and csrc/mca_deep.cuh mark the helpers that turn a trial counter into a
proposal or a decision (Philox4x32-10, the Metropolis threshold of Eq. 7, the acceptance rule, the
current-layer schedule's layer choice, the flat index of a trial, and the channel draws of
Section 2.3's multi-parameter mutations) as host-and-device functions.
tests/device_math_host.cu is a host program around them; this test builds it with nvcc (no GPU
needed) and compares its answers with the oracle's independent implementation: Philox words and
indices bit for bit, thresholds to fp32 rounding. The GPU tests then cover the same functions
running inside the kernels.
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

from oracle import mca_oracle as O

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


@pytest.fixture(scope="module")
def harness(tmp_path_factory):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not available")
    exe = str(tmp_path_factory.mktemp("dmh") / "device_math_host")
    subprocess.run([nvcc, "-std=c++17", "-O2", "-I", os.path.join(ROOT, "include"), "-I",
                    os.path.join(ROOT, "paper_2607_08406_gb300", "csrc"), "-o", exe,
                    os.path.join(HERE, "device_math_host.cu")], check=True, capture_output=True)

    def ask(lines):
        r = subprocess.run([exe], input="\n".join(lines) + "\n", capture_output=True, text=True,
                           check=True)
        return r.stdout.split("\n")[:len(lines)]
    return ask


SEEDS = [0, 1, 0xDEADBEEF, 0x1234_5678_9ABC_DEF0]


def test_philox_words_bit_exact(harness):
    rng = np.random.default_rng(0)
    taus = np.concatenate([np.arange(50), rng.integers(0, 2 ** 63, 150, dtype=np.int64)])
    cmds = [f"words {s} {int(t)}" for s in SEEDS for t in taus]
    got = np.array([[int(v) for v in l.split()] for l in harness(cmds)], dtype=np.uint64)
    want = np.concatenate([O.draw_words(s, taus.astype(np.uint64)) for s in SEEDS])
    assert np.array_equal(got, want)


def test_metropolis_threshold_and_acceptance(harness):
    """theta = -(N / beta) ln u from the trial's fourth word (host fp64, rounded to fp32) equals the
    oracle's threshold to fp32 rounding; accept_change compares with it (and with 0 when the rule
    is greedy), strict or not."""
    taus = np.arange(300)
    for seed, N, beta in ((7, 1000, 250.0), (0xABCDEF, 60000, 6000.0), (3, 48, 600.0)):
        got = np.array([float(l) for l in harness([f"theta {seed} {t} {N / beta!r}"
                                                   for t in taus])])
        want = O.metropolis_threshold(seed, taus, beta, N)
        assert np.all(np.abs(got - want) <= 2e-7 * np.abs(want) + 1e-30)
        th = got[:40]
        cmds = []
        for t in range(40):
            for d in (float(np.float32(th[t]) * np.float32(0.999)), float(np.float32(th[t])),
                      float(np.float32(th[t]) * np.float32(1.001))):
                for strict in (0, 1):
                    cmds.append(f"accept {d!r} {strict} 1 {seed} {t} {N / beta!r}")
        acc = np.array([int(l) for l in harness(cmds)]).reshape(40, 3, 2)
        assert (acc[:, 0, :] == 1).all()                 # below theta: kept
        assert (acc[:, 1, 0] == 1).all() and (acc[:, 1, 1] == 0).all()   # at theta: <= vs <
        assert (acc[:, 2, :] == 0).all()                 # above theta: rejected
    greedy = harness([f"accept {d} {s} 0 5 9 0.0" for d in (-1e-30, 0.0, 1e-30) for s in (0, 1)])
    assert [int(v) for v in greedy] == [1, 1, 1, 0, 0, 0]


def test_stretch_layer_and_trial_indices(harness):
    """The schedule's layer choice and both index helpers equal the oracle's proposal_index, with
    and without the schedule."""
    for seed in SEEDS[:3]:
        for nl in (2, 3, 25):
            got = [int(v) for v in harness([f"stretch {seed} {s} {nl}" for s in range(200)])]
            assert got == O.stretch_layer(seed, np.arange(200), nl).astype(int).tolist()
    offs2 = [0, 784 * 16384, 784 * 16384 + 16384 * 10]
    deep = [0] + np.cumsum([784 * 256] + [256 * 256] * 23 + [256 * 10]).tolist()
    for seed in (0, 77):
        words = O.draw_words(seed, np.arange(400))[:, 0]
        for M in (0, 1, 13, 100):
            c2 = [f"idx2 {offs2[2]} {offs2[1]} {seed} {t} {int(words[t])} {M}" for t in range(400)]
            cd = [f"idxd {seed} {t} {int(words[t])} {M} {len(deep) - 1} " + " ".join(map(str, deep))
                  for t in range(400)]
            want2 = [O.proposal_index(seed, t, int(words[t]), offs2, M) for t in range(400)]
            wantd = [O.proposal_index(seed, t, int(words[t]), deep, M) for t in range(400)]
            assert [int(v) for v in harness(c2)] == want2
            assert [int(v) for v in harness(cd)] == wantd


def test_channel_draws(harness):
    """The channel of mca_run_channels (nodes of every layer, He redraws) equals the oracle's
    propose_channel bit for bit."""
    from paper_2607_08406_gb300 import workloads as W
    dims = [784, 256, 256, 40, 10]
    layers = [W.Layer(dims[m], dims[m + 1]) for m in range(len(dims) - 1)]
    params = O.Params(layers, np.zeros(sum(a * b for a, b in zip(dims[:-1], dims[1:])),
                                       np.float32))
    L = len(layers)
    for seed in (0, 0xFEED_F00D_1234):
        cmds = [f"chan {seed} {t} {L} " + " ".join(map(str, dims)) + " " +
                " ".join(str(d) for d in dims[:-1]) for t in range(200)]
        for t, line in enumerate(harness(cmds)):
            vals = line.split()
            ch = O.propose_channel(seed, t, params, "he")
            nodes = [c[2] for c in ch] + [ch[-1][1]]
            assert [int(v) for v in vals[:L + 1]] == nodes
            assert [np.float32(float(v)) for v in vals[L + 1:]] == [np.float32(c[4]) for c in ch]


def test_batch_width_cost_model(harness):
    """The width of the host-driven batches (deep nets, the Transformer) is the K in 1 .. Kmax that
    maximises the expected trials a batch consumes, (1 - (1-p)^K) / p with p = (A + 1/2) / (T + 1),
    per unit of its cost r + K: checked against a brute-force argmax in double precision, and
    against its limits (a certain accept takes one candidate; a rarely accepting chain with a costly
    batch takes many, capped at Kmax)."""
    rng = np.random.default_rng(5)
    cases = [(float(a), float(a + t), float(r), int(k))
             for a, t, r, k in zip(rng.uniform(0, 30, 200), rng.uniform(0, 200, 200),
                                   rng.choice([0.0, 0.38, 0.5, 1.9, 8.0], 200),
                                   rng.integers(1, 129, 200))]
    cases += [(1000.0, 1000.0, 1.9, 64), (0.0, 10000.0, 50.0, 64), (0.0, 10000.0, 50.0, 7)]
    got = [int(v) for v in harness([f"width {a!r} {t!r} {r!r} {k}" for a, t, r, k in cases])]
    for (a, t, r, k), w in zip(cases, got):
        p = (np.float32(a) + 0.5) / (np.float32(t) + 1.0)
        v = [(1.0 - (1.0 - p) ** K) / (r + K) for K in range(1, k + 1)]
        assert w == int(np.argmax(v)) + 1, (a, t, r, k, w)
    assert got[-3] == 1 and got[-2] > 40 and got[-1] == 7
