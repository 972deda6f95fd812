"""The config-sized Transformer on the tensor-core kernels: K-invariance and resync (needs a GPU).

vocab 65, context 64, d_model 128, 2 blocks x 4 heads, FFN 512, 256 sequences -- the shape the
tensor-core kernels run by default. Parity with the oracle at this shape is in test_gpu_tfm.py.
"""
import numpy as np
import pytest

from paper_2607_08406_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def test_tfm_tensor_cores_K_invariance_and_resync(gpu_lib):
    """Config-sized Transformer on the tensor-core kernels: 300 trials give a bit-identical trace and
    parameters for K = 1, 8 and 64 (each batch ranks its candidates by recomputation length, so
    the CTA that evaluates a (candidate, sequence pair) depends on K), and a resync (a fresh
    forward pass) reproduces the incrementally kept loss."""
    wl = W.char_transformer()
    ref = None
    for K in (1, 8, 64):
        h = gpu_lib.create_from_tfm_workload(wl, K=K, trace_cap=300)
        st = gpu_lib.mca_run(h, 300, 5)
        assert st["tensor_cores"] == 1 and st["trials"] == 300 and st["accepts"] > 30
        out = (gpu_lib.mca_get_trace(h, 300), gpu_lib.mca_get_params(h, wl.n_params))
        if ref is None:
            ref = out
        else:
            assert np.array_equal(out[0], ref[0])
            assert np.array_equal(out[1], ref[1])
        L = gpu_lib.mca_loss(h)
        gpu_lib.mca_resync(h)
        assert gpu_lib.mca_loss(h) == pytest.approx(L, rel=1e-5)
        h.close()
