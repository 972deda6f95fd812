"""The no-allocation candidate evaluation (mca_eval_candidates_noalloc) gives the same loss changes
as mca_eval_candidates. It serves callers that cannot allocate device memory; the test's own
tensors are the caller's inputs and outputs. Kept in a file collected last, so that a run stopping
at the first failure has run every other test first."""
import ctypes

import numpy as np
import pytest

from paper_2607_08406_gb300 import workloads as W

from parity import TIE_REL

pytestmark = pytest.mark.gpu


def test_eval_candidates_noalloc_matches_allocating_entry_point(gpu_lib):
    import torch
    wl = W.mlp_wide(N=12003, H=256)
    h = gpu_lib.create_from_workload(wl)
    gpu_lib.mca_run(h, 500, 0)
    S = gpu_lib.mca_loss(h) * wl.N
    rng = np.random.default_rng(7)
    P1 = 784 * 256
    idx = np.concatenate([rng.integers(0, P1, 100), rng.integers(P1, wl.n_params, 28)])
    idx = idx.astype(np.uint32)
    new = rng.uniform(-1, 1, len(idx)).astype(np.float32)
    ref = gpu_lib.mca_eval_candidates(h, idx, new)
    d_idx = torch.from_numpy(idx.view(np.int32)).cuda()
    d_new = torch.from_numpy(new).cuda()
    d_out = torch.empty(len(idx), dtype=torch.float64, device="cuda")
    lib = gpu_lib.load_library()
    for _ in range(2):                       # two calls in a row share the static scratch
        d_out.fill_(float("nan"))
        rc = lib.mca_eval_candidates_noalloc(h.ptr, d_idx.data_ptr(), d_new.data_ptr(), len(idx),
                                             d_out.data_ptr())
        assert rc == gpu_lib.MCA_OK, lib.mca_last_error(h.ptr)
        got = d_out.cpu().numpy()
        assert np.all(np.isfinite(got))
        assert np.all(np.abs(got - ref) <= TIE_REL * S)
    # sizes beyond the stated maximum are rejected with a message
    big = torch.zeros(129, dtype=torch.int32, device="cuda")
    bnew = torch.zeros(129, dtype=torch.float32, device="cuda")
    bout = torch.zeros(129, dtype=torch.float64, device="cuda")
    rc = lib.mca_eval_candidates_noalloc(h.ptr, big.data_ptr(), bnew.data_ptr(), 129,
                                         bout.data_ptr())
    assert rc == gpu_lib.MCA_ERR_INVALID
    assert b"maximum" in lib.mca_last_error(h.ptr)
    h.close()
