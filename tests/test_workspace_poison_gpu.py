"""No result depends on the prior contents of device memory (needs a GPU).

Every handle below is created twice, once on a workspace whose bytes are all 0xFF (NaN as fp32, -1
as integers, saturated counters and flags) and once on a zero-filled one; 300 trials from each must
give the same trace, parameters and loss bit for bit. A buffer read before the library wrote it
would carry the poison into a result.
"""
import numpy as np
import pytest

from paper_2607_08406_gb300 import workloads as W

pytestmark = pytest.mark.gpu

TFM_SMALL = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=2, n_head=2, d_ff=32)

CASES = {
    # name: (workload builder, Transformer?, create options)
    "wide_window": (lambda: W.make("mlp_wide", N=12003, H=256), False, {}),
    "wide_one_range": (lambda: W.make("mlp_wide", N=12003, H=256), False, dict(grid=1)),
    "ternary": (lambda: W.make("mlp_ternary", N=12000, H=256), False, {}),
    "deep_w40": (lambda: W.mlp_deep(N=700, width=40, depth=3, n_trials=300, K=16), False, {}),
    "deep_tc_w256": (lambda: W.mlp_deep(N=1100, width=256, depth=5, n_trials=300, K=16), False,
                     {}),
    "tfm_small": (lambda: W.char_transformer(seed=0, batch=6, text_len=20000, spec=TFM_SMALL,
                                             n_trials=300, K=8), True, {}),
    "tfm_config_tensor_cores": (lambda: W.char_transformer(), True, {}),
}


def _run(gpu_lib, monkeypatch, wl, tfm, fill, kw):
    import torch
    real = torch.empty

    def filled(*a, **k):
        return real(*a, **k).fill_(fill)
    with monkeypatch.context() as m:
        m.setattr(torch, "empty", filled)
        create = gpu_lib.create_from_tfm_workload if tfm else gpu_lib.create_from_workload
        h = create(wl, trace_cap=300, **kw)
    gpu_lib.mca_run(h, 300, 2)
    out = (gpu_lib.mca_get_trace(h, 300), gpu_lib.mca_get_params(h, wl.n_params),
           gpu_lib.mca_loss(h))
    h.close()
    return out


@pytest.mark.parametrize("case", list(CASES))
def test_poisoned_workspace_gives_the_same_run(gpu_lib, monkeypatch, case):
    build, tfm, kw = CASES[case]
    wl = build()
    a = _run(gpu_lib, monkeypatch, wl, tfm, 0xFF, kw)
    b = _run(gpu_lib, monkeypatch, wl, tfm, 0x00, kw)
    assert np.array_equal(a[0], b[0])
    assert np.array_equal(a[1], b[1])
    assert a[2] == b[2] and np.isfinite(a[2])
