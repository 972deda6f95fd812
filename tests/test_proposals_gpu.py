"""The device proposal stream against the oracle's Philox4x32-10 over 10^6 trials (needs a GPU).

Every trial's parameter index (the first Philox word, Eq. 1's uniform choice) and replacement value
(the second word, U[-1, 1) on the exact 2^-23 grid) do not depend on the state, so the trace of a
long run must reproduce them bit for bit from the oracle's own Philox words, whatever was accepted.
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def test_proposal_stream_matches_oracle_over_a_million_trials(gpu_lib):
    wl = W.mlp_small()
    n, seed = 1_000_000, 0x1234_5678_9ABC
    h = gpu_lib.create_from_workload(wl, trace_cap=n)
    st = gpu_lib.mca_run(h, n, seed)
    assert st["trials"] == n
    g = gpu_lib.mca_get_trace(h, n)
    taus = np.arange(n, dtype=np.uint64)
    assert np.array_equal(g["tau"], taus)
    r = O.draw_words(seed, taus)
    idx = (r[:, 0] * np.uint64(wl.n_params)) >> np.uint64(32)
    assert np.array_equal(g["idx"].astype(np.uint64), idx)
    u = (r[:, 1] >> np.uint64(8)).astype(np.float32) * np.float32(2.0 ** -24)
    new = np.float32(-1.0) + np.float32(2.0) * u
    assert new.dtype == np.float32
    assert np.array_equal(g["new_w"], new)
    assert g["valid"].all()
