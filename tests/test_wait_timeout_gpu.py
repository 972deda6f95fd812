"""Failure detection without a GPU fault (needs a GPU).

Every device-side wait of the library is bounded: when a peer never arrives, the waiting CTA gives
up after its limit, records MCA_ERR_TIMEOUT and returns, and the host reads that status. Here the
trial loop's grid barrier waits, in one CTA, for a second CTA that is never launched. Nothing
faults, traps or hangs: the wait must end by itself after about 2 s, and the context must stay
usable for a normal run afterwards.
"""
import numpy as np
import pytest

from oracle import mca_oracle as O
from paper_2607_08406_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def test_bounded_wait_gives_up_and_the_context_stays_usable(gpu_lib):
    status, ms = gpu_lib.mca_selftest_wait_timeout()
    assert status == gpu_lib.MCA_ERR_TIMEOUT
    assert 1900.0 <= ms <= 20000.0, ms
    wl = W.mlp_small(N=200, H=16)
    h = gpu_lib.create_from_workload(wl, trace_cap=300)
    st = gpu_lib.mca_run(h, 300, 0)
    assert st["trials"] == 300
    S = O.total_loss(O.Params(wl.layers, wl.init), wl.X.T.astype(np.float64), wl.y, wl.loss)
    assert gpu_lib.mca_get_trace(h, 300)["S"][0] == pytest.approx(S, rel=1e-6)
