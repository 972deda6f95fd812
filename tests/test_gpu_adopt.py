"""Adoption of accepted candidates from the scratch slots their evaluation wrote (the deep and the
Transformer tensor-core paths) against the commit kernels' recomputation (needs a GPU).

With MCA_ADOPT=0 a handle has no slots and every accepted candidate is recomputed by the commit
kernel. The same trials must then give a bit-identical trace (decisions, loss changes, loss), final
parameters and cached loss. Fixed batches of 32 candidates against 16 slots also accept candidates
beyond the slots, which the commit kernel recomputes in the adopting handle too.
"""
import numpy as np
import pytest

from paper_2607_08406_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _outcome(gpu_lib, h, n, seed, n_params):
    st = gpu_lib.mca_run(h, n, seed)
    out = (gpu_lib.mca_get_trace(h, n), gpu_lib.mca_get_params(h, n_params), gpu_lib.mca_loss(h), st)
    h.close()
    return out


def _same(a, b):
    assert np.array_equal(a[0], b[0])
    assert np.array_equal(a[1], b[1])
    assert a[2] == b[2]
    for key in ("trials", "accepts", "candidates"):
        assert a[3][key] == b[3][key], key


@pytest.mark.parametrize("fixed_K", [0, 32])
def test_tfm_adoption_matches_commit(gpu_lib, monkeypatch, fixed_K):
    monkeypatch.delenv("MCA_TFM_TENSOR_CORES", raising=False)
    wl = W.char_transformer()
    n = 240
    kw = dict(K=fixed_K, fixed_K=True) if fixed_K else {}
    monkeypatch.delenv("MCA_ADOPT", raising=False)
    h = gpu_lib.create_from_tfm_workload(wl, trace_cap=n, **kw)
    adopted = _outcome(gpu_lib, h, n, 3, wl.n_params)
    assert adopted[3]["tensor_cores"] == 1 and adopted[3]["accepts"] > 20
    monkeypatch.setenv("MCA_ADOPT", "0")
    h = gpu_lib.create_from_tfm_workload(wl, trace_cap=n, **kw)
    recomputed = _outcome(gpu_lib, h, n, 3, wl.n_params)
    _same(adopted, recomputed)


@pytest.mark.parametrize("fixed_K", [0, 32])
def test_deep_adoption_matches_commit(gpu_lib, monkeypatch, fixed_K):
    wl = W.mlp_deep(N=1100, width=256, depth=5, n_trials=600, K=16)
    n = 600
    kw = dict(K=fixed_K, fixed_K=True) if fixed_K else {}
    monkeypatch.delenv("MCA_ADOPT", raising=False)
    h = gpu_lib.create_from_workload(wl, trace_cap=n, **kw)
    adopted = _outcome(gpu_lib, h, n, 4, wl.n_params)
    assert adopted[3]["tensor_cores"] == 1 and adopted[3]["accepts"] > 20
    monkeypatch.setenv("MCA_ADOPT", "0")
    h = gpu_lib.create_from_workload(wl, trace_cap=n, **kw)
    recomputed = _outcome(gpu_lib, h, n, 4, wl.n_params)
    _same(adopted, recomputed)
