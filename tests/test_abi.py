"""The C-ABI library loads, exports every entry point include/mca.h declares, and its structs match
the Python binding's layout (CPU only: no compute calls)."""
import ctypes
import os
import re
import subprocess
import tempfile

import numpy as np
import pytest

from paper_2607_08406_gb300 import mca, build as B
from paper_2607_08406_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mca.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return mca.load_library()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(mca_[a-z_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("mca_create", "mca_run", "mca_loss", "mca_get_params", "mca_destroy"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    names = declared_functions()
    out = subprocess.run(["nm", "-D", "--defined-only", mca.LIB_PATH], capture_output=True,
                         text=True).stdout
    exported = set(re.findall(r"\sT\s(mca_\w+)", out))
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    for n in names:
        assert hasattr(lib, n)
    assert set(mca.SIGNATURES) == set(names)


def test_struct_layouts_match_header(tmp_path):
    """Compile a probe against include/mca.h with gcc and compare sizes/offsets with ctypes."""
    structs = {"mca_layer": mca.mca_layer, "mca_domain": mca.mca_domain,
               "mca_dataset": mca.mca_dataset, "mca_options": mca.mca_options,
               "mca_run_stats": mca.mca_run_stats, "mca_trace_rec": mca.mca_trace_rec}
    lines = ['#include <stdio.h>', '#include <stddef.h>', f'#include "{HEADER}"', "int main(){"]
    for s, cls in structs.items():
        lines.append(f'printf("{s} %zu\\n", sizeof({s}));')
        for f, _ in cls._fields_:
            lines.append(f'printf("{s}.{f} %zu\\n", offsetof({s}, {f}));')
    lines.append("return 0;}")
    c = tmp_path / "probe.c"
    c.write_text("\n".join(lines))
    exe = tmp_path / "probe"
    subprocess.run(["gcc", "-O0", str(c), "-o", str(exe)], check=True)
    got = dict(l.split() for l in subprocess.run([str(exe)], capture_output=True, text=True,
                                                 check=True).stdout.splitlines())
    for s, cls in structs.items():
        assert int(got[s]) == ctypes.sizeof(cls), s
        for f, _ in cls._fields_:
            assert int(got[f"{s}.{f}"]) == getattr(cls, f).offset, (s, f)


def _spec(n_layers=2):
    wl = W.mlp_small(N=8, H=4)
    layers = wl.layers if n_layers == 2 else wl.layers[:1]
    return wl, mca._layers(layers), len(layers)


def test_invalid_specs_rejected_without_gpu(lib):
    """Argument checks run on the host before any CUDA call."""
    wl, L, n = _spec()
    ds = mca.mca_dataset(wl.X.ctypes.data, wl.y.ctypes.data, wl.N, 784)
    h = ctypes.c_void_p(None)
    # one layer
    rc = lib.mca_create(L, 1, 0, None, ctypes.byref(ds), wl.init.ctypes.data, None,
                        ctypes.byref(h))
    assert rc == mca.MCA_ERR_INVALID and h.value is None
    assert b"n_layers" in lib.mca_last_error(None)
    # mismatched input width
    bad = mca.mca_dataset(wl.X.ctypes.data, wl.y.ctypes.data, wl.N, 783)
    rc = lib.mca_create(L, n, 0, None, ctypes.byref(bad), wl.init.ctypes.data, None,
                        ctypes.byref(h))
    assert rc == mca.MCA_ERR_INVALID
    # unknown loss
    rc = lib.mca_create(L, n, 7, None, ctypes.byref(ds), wl.init.ctypes.data, None,
                        ctypes.byref(h))
    assert rc == mca.MCA_ERR_INVALID
    # empty dataset
    empty = mca.mca_dataset(wl.X.ctypes.data, wl.y.ctypes.data, 0, 784)
    rc = lib.mca_create(L, n, 0, None, ctypes.byref(empty), wl.init.ctypes.data, None,
                        ctypes.byref(h))
    assert rc == mca.MCA_ERR_INVALID
    # too many classes for the sample record
    big = (mca.mca_layer * 2)(mca.mca_layer(784, 4, 1, 0.0, 0, 1.0),
                              mca.mca_layer(4, 40, 2, 0.0, 0, 1.0))
    rc = lib.mca_create(big, 2, 0, None, ctypes.byref(ds), wl.init.ctypes.data, None,
                        ctypes.byref(h))
    assert rc == mca.MCA_ERR_UNSUPPORTED
    # Metropolis temperature (1 / beta, Eq. 7) must be finite and >= 0
    for t in (-1.0, float("nan"), float("inf")):
        d = mca.mca_domain(0, -1.0, 1.0, 0.01, 0.0, 0, t)
        rc = lib.mca_create(L, n, 0, ctypes.byref(d), ctypes.byref(ds), wl.init.ctypes.data,
                            None, ctypes.byref(h))
        assert rc == mca.MCA_ERR_INVALID and b"temperature" in lib.mca_last_error(None)
    # a negative current-layer stretch
    d = mca.mca_domain(0, -1.0, 1.0, 0.01, 0.0, 0, 0.0, -1)
    rc = lib.mca_create(L, n, 0, ctypes.byref(d), ctypes.byref(ds), wl.init.ctypes.data, None,
                        ctypes.byref(h))
    assert rc == mca.MCA_ERR_INVALID and b"layer_stretch" in lib.mca_last_error(None)
    # the current-layer schedule is for MLPs: a Transformer handle refuses it
    sp = W.TfmSpec(vocab=17, ctx=8, d_model=16, n_layer=1, n_head=2, d_ff=32)
    tok = np.zeros((4, 9), np.int32)
    init = np.zeros(sp.n_params, np.float32)
    d = mca.mca_domain(0, -1.0, 1.0, 0.01, 0.0, 0, 0.0, 10)
    rc = lib.mca_create_transformer(ctypes.byref(mca._tfm_spec(sp)), ctypes.byref(d),
                                    tok.ctypes.data, 4, init.ctypes.data, None, ctypes.byref(h))
    assert rc == mca.MCA_ERR_UNSUPPORTED and h.value is None
    # NULL handle calls
    assert lib.mca_run(None, 1, 0, None) == mca.MCA_ERR_INVALID
    assert lib.mca_run_channels(None, 1, 0, 0, None, None) == mca.MCA_ERR_INVALID
    lib.mca_destroy(None)


def test_binding_names_match_c_abi():
    """The Python binding exposes each C entry point under the same name."""
    for n in declared_functions():
        if n == "mca_last_error":
            continue
        assert callable(getattr(mca, n)), n


def test_binding_maps_beta_to_temperature():
    """The binding passes Eq. 7's beta as temperature = 1 / beta (0 for the greedy rule, beta = inf)
    and refuses beta <= 0."""
    assert mca._domain(W.Domain()).temperature == 0.0
    d = mca._domain(W.Domain(beta=250.0, strict=True))
    assert d.temperature == pytest.approx(1.0 / 250.0) and d.strict == 1
    for bad in (0.0, -3.0, float("nan")):
        with pytest.raises(ValueError):
            mca._domain(W.Domain(beta=bad))


def test_transformer_scratch_slots_in_the_workspace(lib, monkeypatch):
    """Workspace of the tensor-core Transformer (sized on the host, no GPU): each of the
    min(K, 16) scratch slots holds the streams a candidate's evaluation recomputes (the 2 nL + 1
    block input and mid streams of every sequence) and its sequence losses; MCA_ADOPT=0 leaves the
    slots out."""
    wl = W.char_transformer()
    sp = wl.spec
    B = 256
    stream = B * sp.ctx * sp.d_model * 4
    slot = (2 * sp.n_layer + 1) * stream + B * 4          # both parts are multiples of 256 bytes
    monkeypatch.delenv("MCA_TFM_TENSOR_CORES", raising=False)
    monkeypatch.setenv("MCA_ADOPT", "0")
    base = mca.mca_tfm_workspace_size(sp, B, 16)
    assert mca.mca_tfm_workspace_size(sp, B, 1) == base
    monkeypatch.delenv("MCA_ADOPT")
    for K, nscr in ((1, 1), (5, 5), (16, 16), (64, 16)):
        assert mca.mca_tfm_workspace_size(sp, B, K) == base + nscr * slot, K


def test_deep_scratch_slots_in_the_workspace(monkeypatch):
    """Workspace of a deep net on the tensor-core chain (sized on the host, no GPU): each of the
    min(K, 16) scratch slots holds every layer's fields and the per-sample losses (the arrays an
    accepted candidate's adoption exchanges), plus one row of the slots' pointer table; MCA_ADOPT=0
    leaves them out."""
    wl = W.mlp_deep(N=1100, width=256, depth=5, n_trials=10, K=16)
    Np = (wl.N + 127) // 128 * 128
    L = len(wl.layers)
    slot = sum(ly.n_out for ly in wl.layers) * Np * 4 + Np * 4   # each array a multiple of 256 B
    monkeypatch.setenv("MCA_ADOPT", "0")
    base = mca.mca_workspace_size(wl.layers, wl.loss, wl.X, wl.y, 16)
    monkeypatch.delenv("MCA_ADOPT")
    for K, nscr in ((1, 1), (16, 16), (64, 16)):
        table = -(-nscr * (L + 1) * 8 // 256) * 256
        assert mca.mca_workspace_size(wl.layers, wl.loss, wl.X, wl.y, K) == \
            base + nscr * slot + table, K
