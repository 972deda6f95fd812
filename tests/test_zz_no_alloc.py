"""The no-allocation candidate evaluation (mca_eval_candidates_noalloc) gives the same loss changes
as mca_eval_candidates. It serves callers that cannot allocate device memory (a process whose
device memory belongs to another allocator, or a loop that cannot take the device-wide
synchronisation of cudaMalloc / cudaFree); the test's own tensors are the caller's inputs and
outputs. Both entry points launch the same evaluation kernel on the same state, so their results
must be bit-equal. Kept in a file collected last, so that a run stopping at the first failure has
run every other test first."""
import numpy as np
import pytest

from paper_2607_08406_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _device_args(idx, new):
    import torch
    d_idx = torch.from_numpy(np.ascontiguousarray(idx, np.uint32).view(np.int32)).cuda()
    d_new = torch.from_numpy(np.ascontiguousarray(new, np.float32)).cuda()
    d_out = torch.empty(len(idx), dtype=torch.float64, device="cuda")
    return d_idx, d_new, d_out


def test_eval_candidates_noalloc_matches_allocating_entry_point(gpu_lib):
    wl = W.mlp_wide(N=12003, H=256)
    h = gpu_lib.create_from_workload(wl)
    gpu_lib.mca_run(h, 500, 0)
    rng = np.random.default_rng(7)
    P1 = 784 * 256
    idx = np.concatenate([rng.integers(0, P1, 100), rng.integers(P1, wl.n_params, 28)])
    idx = idx.astype(np.uint32)
    new = rng.uniform(-1, 1, len(idx)).astype(np.float32)
    ref = gpu_lib.mca_eval_candidates(h, idx, new)
    d_idx, d_new, d_out = _device_args(idx, new)
    lib = gpu_lib.load_library()
    for _ in range(2):                       # two calls in a row share the static scratch
        d_out.fill_(float("nan"))
        rc = lib.mca_eval_candidates_noalloc(h.ptr, d_idx.data_ptr(), d_new.data_ptr(), len(idx),
                                             d_out.data_ptr())
        assert rc == gpu_lib.MCA_OK, lib.mca_last_error(h.ptr)
        got = d_out.cpu().numpy()
        assert np.array_equal(got, ref)
    # sizes beyond the stated maximum are rejected with a message
    big = np.zeros(129, np.uint32)
    b_idx, b_new, b_out = _device_args(big, np.zeros(129, np.float32))
    rc = lib.mca_eval_candidates_noalloc(h.ptr, b_idx.data_ptr(), b_new.data_ptr(), 129,
                                         b_out.data_ptr())
    assert rc == gpu_lib.MCA_ERR_INVALID
    assert b"maximum" in lib.mca_last_error(h.ptr)
    # the handle is still usable, and the allocating entry point still agrees
    assert np.array_equal(gpu_lib.mca_eval_candidates(h, idx, new), ref)
    h.close()


def test_eval_candidates_noalloc_refuses_deep_and_transformer_handles(gpu_lib):
    """Deep and Transformer handles are refused before any device work, and keep working."""
    lib = gpu_lib.load_library()
    deep = W.mlp_deep(N=600, width=40, depth=3, n_trials=200, K=8)
    spec = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=1, n_head=2, d_ff=32)
    tfm = W.char_transformer(batch=4, text_len=5000, spec=spec, n_trials=200, K=8)
    for wl, make in ((deep, gpu_lib.create_from_workload),
                     (tfm, gpu_lib.create_from_tfm_workload)):
        h = make(wl)
        idx = np.array([0, 5, wl.n_params - 1], np.uint32)
        new = np.array([0.25, -0.5, 0.75], np.float32)
        d_idx, d_new, d_out = _device_args(idx, new)
        rc = lib.mca_eval_candidates_noalloc(h.ptr, d_idx.data_ptr(), d_new.data_ptr(), len(idx),
                                             d_out.data_ptr())
        assert rc == gpu_lib.MCA_ERR_UNSUPPORTED
        assert b"single-hidden-layer" in lib.mca_last_error(h.ptr)
        st = gpu_lib.mca_run(h, 50, 1)
        assert st["trials"] == 50
        d = gpu_lib.mca_eval_candidates(h, idx, new)
        assert np.all(np.isfinite(d))
        h.close()
