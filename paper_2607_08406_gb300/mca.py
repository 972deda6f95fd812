"""Python binding of the C ABI in include/mca.h (ctypes; argument marshalling only).

Every step of the trial loop runs in libmca.so's CUDA kernels. PyTorch provides device memory
(the library's workspace is a torch tensor) and the stream. There is no CPU fallback: if the
library is missing or no GPU is present, the calls raise.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import (POINTER, Structure, c_char_p, c_double, c_float, c_int8, c_int32, c_int64,
                    c_size_t, c_uint8, c_uint32, c_uint64, c_void_p)
from typing import Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libmca.so")

MCA_OK, MCA_ERR_INVALID, MCA_ERR_CUDA, MCA_ERR_OOM, MCA_ERR_TIMEOUT, MCA_ERR_NUMERIC, \
    MCA_ERR_UNSUPPORTED = range(7)
ACT = {"identity": 0, "tanh": 1, "sigmoid": 2, "relu": 3, "gaussian": 4, "gelu": 5}
LOSS = {"mse_onehot": 0, "softmax_ce": 1}
WKIND = {"fp32": 0, "ternary_i8": 1, "masked_fp32": 2}
OP = {"replace": 0, "perturb": 1}


class mca_layer(Structure):
    _fields_ = [("n_in", c_int32), ("n_out", c_int32), ("act", c_int32), ("act_param", c_float),
                ("wkind", c_int32), ("scale", c_float)]


class mca_domain(Structure):
    _fields_ = [("op", c_int32), ("lo", c_float), ("hi", c_float), ("delta", c_float),
                ("bound", c_float), ("strict", c_int32), ("temperature", c_float),
                ("layer_stretch", c_int32)]


class mca_dataset(Structure):
    _fields_ = [("x", c_void_p), ("y", c_void_p), ("n", c_int64), ("d", c_int32)]


class mca_options(Structure):
    _fields_ = [("K", c_int32), ("resync_period", c_int32), ("stream", c_void_p),
                ("trace_cap", c_int32), ("grid", c_int32), ("workspace", c_void_p),
                ("workspace_bytes", c_size_t), ("fixed_K", c_int32)]


class mca_tfm_spec(Structure):
    _fields_ = [("vocab", c_int32), ("ctx", c_int32), ("d_model", c_int32), ("n_layer", c_int32),
                ("n_head", c_int32), ("d_ff", c_int32), ("act", c_int32), ("act_param", c_float),
                ("ln_eps", c_float)]


class mca_run_stats(Structure):
    _fields_ = [("trials", c_uint64), ("accepts", c_uint64), ("candidates", c_uint64),
                ("batches", c_uint64), ("wasted", c_uint64), ("forced", c_uint64),
                ("resyncs", c_uint64), ("launches", c_uint64), ("tau", c_uint64), ("S", c_double),
                ("alg_bytes", c_uint64), ("phase_ns", c_uint64 * 8), ("alg_flops", c_uint64),
                ("tensor_cores", c_uint32), ("reserved", c_uint32)]

    def asdict(self):
        d = {f: getattr(self, f) for f, _ in self._fields_ if f != "phase_ns"}
        d["phase_ns"] = list(self.phase_ns)
        return d


class mca_trace_rec(Structure):
    _fields_ = [("tau", c_uint64), ("idx", c_uint32), ("accept", c_int32), ("old_w", c_float),
                ("new_w", c_float), ("valid", c_int32), ("forced", c_int32), ("dS", c_double),
                ("S", c_double)]


TRACE_DTYPE = np.dtype([("tau", np.uint64), ("idx", np.uint32), ("accept", np.int32),
                        ("old_w", np.float32), ("new_w", np.float32), ("valid", np.int32),
                        ("forced", np.int32), ("dS", np.float64), ("S", np.float64)])
assert TRACE_DTYPE.itemsize == ctypes.sizeof(mca_trace_rec)

# Every function the header declares, with its ctypes signature.
SIGNATURES = {
    "mca_workspace_size": (c_int32, [POINTER(mca_layer), c_int32, c_int32, POINTER(mca_dataset),
                                     POINTER(mca_options), POINTER(c_size_t)]),
    "mca_create": (c_int32, [POINTER(mca_layer), c_int32, c_int32, POINTER(mca_domain),
                             POINTER(mca_dataset), c_void_p, POINTER(mca_options),
                             POINTER(c_void_p)]),
    "mca_tfm_workspace_size": (c_int32, [POINTER(mca_tfm_spec), c_int64, POINTER(mca_options),
                                         POINTER(c_size_t)]),
    "mca_create_transformer": (c_int32, [POINTER(mca_tfm_spec), POINTER(mca_domain), c_void_p,
                                         c_int64, c_void_p, POINTER(mca_options),
                                         POINTER(c_void_p)]),
    "mca_run": (c_int32, [c_void_p, c_uint64, c_uint64, POINTER(mca_run_stats)]),
    "mca_loss": (c_int32, [c_void_p, POINTER(c_double)]),
    "mca_get_params": (c_int32, [c_void_p, c_void_p, c_size_t]),
    "mca_get_codes": (c_int32, [c_void_p, c_void_p, c_size_t]),
    "mca_set_params": (c_int32, [c_void_p, c_void_p, c_void_p, c_size_t, c_uint64]),
    "mca_resync": (c_int32, [c_void_p]),
    "mca_get_trace": (c_int32, [c_void_p, c_void_p, c_size_t, POINTER(c_size_t)]),
    "mca_force_decisions": (c_int32, [c_void_p, c_void_p, c_void_p, c_size_t]),
    "mca_get_stats": (c_int32, [c_void_p, POINTER(mca_run_stats)]),
    "mca_eval_candidates": (c_int32, [c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "mca_eval_candidates_noalloc": (c_int32, [c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "mca_eval_trials": (c_int32, [c_void_p, c_uint64, c_uint64, c_size_t, c_void_p]),
    "mca_decide_batch": (c_int32, [c_void_p, c_uint64, c_uint64, c_size_t, c_void_p, c_void_p,
                                   c_int64, POINTER(c_int32)]),
    "mca_run_channels": (c_int32, [c_void_p, c_uint64, c_uint64, c_int32, c_void_p, c_void_p]),
    "mca_selftest_wait_timeout": (c_int32, [POINTER(c_int32), POINTER(c_double)]),
    "mca_destroy": (None, [c_void_p]),
    "mca_last_error": (c_char_p, [c_void_p]),
}

_lib = None


def load_library(path: str = LIB_PATH):
    """Load libmca.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        lib = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


class MCAError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"mca status {status}: {msg}")
        self.status = status


def _check(status: int, handle=None):
    if status != MCA_OK:
        msg = load_library().mca_last_error(handle)
        raise MCAError(status, msg.decode() if msg else "")


def _ptr(a):
    """Address of a torch tensor or numpy array (host or device), keeping it contiguous."""
    import torch
    if isinstance(a, torch.Tensor):
        assert a.is_contiguous()
        return a.data_ptr()
    assert isinstance(a, np.ndarray) and a.flags.c_contiguous
    return a.ctypes.data


def _layers(layers) -> "ctypes.Array":
    arr = (mca_layer * len(layers))()
    for k, L in enumerate(layers):
        arr[k] = mca_layer(L.n_in, L.n_out, ACT[L.act], float(L.act_param), WKIND[L.wkind],
                           float(L.scale))
    return arr


def _domain(d) -> mca_domain:
    beta = float(getattr(d, "beta", float("inf")))
    if not beta > 0.0:
        raise ValueError(f"beta = {beta}: the selection intensity must be > 0 (inf: greedy rule)")
    return mca_domain(OP[d.op], d.lo, d.hi, d.delta, d.bound, int(bool(d.strict)),
                      0.0 if beta == float("inf") else 1.0 / beta,
                      int(getattr(d, "layer_stretch", 0)))


class Handle:
    """Owns one mca_handle plus the torch tensors the library borrows (workspace, dataset)."""

    def __init__(self, ptr, keep):
        self.ptr = ptr
        self._keep = keep

    def close(self):
        if self.ptr:
            load_library().mca_destroy(self.ptr)
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def mca_workspace_size(layers, loss: str, X, y, K: int = 32, trace_cap: int = 0,
                       stream=None) -> int:
    lib = load_library()
    L = _layers(layers)
    ds = mca_dataset(_ptr(X), _ptr(y), int(X.shape[0]), int(X.shape[1]))
    opt = mca_options(K, 0, stream, trace_cap, 0, None, 0, 0)
    out = c_size_t(0)
    _check(lib.mca_workspace_size(L, len(layers), LOSS[loss], ctypes.byref(ds), ctypes.byref(opt),
                                  ctypes.byref(out)))
    return out.value


def mca_create(layers, loss: str, domain, X, y, init, K: int = 32, resync_period: int = 0,
               trace_cap: int = 0, grid: int = 0, stream=None, torch_workspace: bool = True,
               fixed_K: bool = False):
    """X: [N, D] float32, y: [N] int32, init: [P] float32 -- torch tensors (CUDA or CPU) or numpy
    arrays. The workspace is a torch CUDA tensor the handle keeps alive."""
    import torch
    lib = load_library()
    if stream is None:
        stream = torch.cuda.current_stream().cuda_stream
    L = _layers(layers)
    dom = _domain(domain)
    ds = mca_dataset(_ptr(X), _ptr(y), int(X.shape[0]), int(X.shape[1]))
    keep = [X, y, init]
    ws_ptr, ws_bytes = None, 0
    if torch_workspace:
        nbytes = mca_workspace_size(layers, loss, X, y, K, trace_cap, stream)
        ws = torch.empty(nbytes + 256, dtype=torch.uint8, device="cuda")
        base = ws.data_ptr()
        ws_ptr = (base + 255) // 256 * 256
        ws_bytes = nbytes
        keep.append(ws)
    opt = mca_options(K, resync_period, stream, trace_cap, grid, ws_ptr, ws_bytes, int(fixed_K))
    h = c_void_p(None)
    _check(lib.mca_create(L, len(layers), LOSS[loss], ctypes.byref(dom), ctypes.byref(ds),
                          _ptr(init), ctypes.byref(opt), ctypes.byref(h)))
    return Handle(h, keep)


def _tfm_spec(sp) -> mca_tfm_spec:
    return mca_tfm_spec(sp.vocab, sp.ctx, sp.d_model, sp.n_layer, sp.n_head, sp.d_ff, ACT[sp.act],
                        float(sp.act_param), float(sp.ln_eps))


def mca_tfm_workspace_size(spec, n_seq: int, K: int = 32, trace_cap: int = 0) -> int:
    opt = mca_options(K, 0, None, trace_cap, 0, None, 0, 0)
    out = c_size_t(0)
    sp = _tfm_spec(spec)
    _check(load_library().mca_tfm_workspace_size(ctypes.byref(sp), n_seq, ctypes.byref(opt),
                                                 ctypes.byref(out)))
    return out.value


def mca_create_transformer(spec, domain, tokens, init, K: int = 32, resync_period: int = 0,
                           trace_cap: int = 0, stream=None, fixed_K: bool = False):
    """tokens: [B, ctx + 1] int32, init: [P] float32 (torch tensors or numpy arrays, host or
    device). The workspace is a torch CUDA tensor the handle keeps alive."""
    import torch
    lib = load_library()
    if stream is None:
        stream = torch.cuda.current_stream().cuda_stream
    n_seq = int(tokens.shape[0])
    nbytes = mca_tfm_workspace_size(spec, n_seq, K, trace_cap)
    ws = torch.empty(nbytes + 256, dtype=torch.uint8, device="cuda")
    ws_ptr = (ws.data_ptr() + 255) // 256 * 256
    opt = mca_options(K, resync_period, stream, trace_cap, 0, ws_ptr, nbytes, int(fixed_K))
    sp = _tfm_spec(spec)
    dom = _domain(domain)
    h = c_void_p(None)
    _check(lib.mca_create_transformer(ctypes.byref(sp), ctypes.byref(dom), _ptr(tokens), n_seq,
                                      _ptr(init), ctypes.byref(opt), ctypes.byref(h)))
    return Handle(h, [tokens, init, ws])


def create_from_tfm_workload(wl, device: bool = True, **kw) -> Handle:
    import torch
    tokens, init = wl.tokens, wl.init
    if device:
        tokens = torch.from_numpy(tokens).cuda()
        init = torch.from_numpy(init).cuda()
    kw.setdefault("K", wl.K)
    return mca_create_transformer(wl.spec, wl.domain, tokens, init, **kw)


def mca_run(h: Handle, n_trials: int, seed: int) -> dict:
    st = mca_run_stats()
    _check(load_library().mca_run(h.ptr, n_trials, seed, ctypes.byref(st)), h.ptr)
    return st.asdict()


def mca_loss(h: Handle) -> float:
    v = c_double(0.0)
    _check(load_library().mca_loss(h.ptr, ctypes.byref(v)), h.ptr)
    return v.value


def mca_get_params(h: Handle, P: int, out=None):
    """Effective weights [P] float32 into `out` (numpy or torch, host or device) or a new array."""
    dst = np.empty(P, np.float32) if out is None else out
    _check(load_library().mca_get_params(h.ptr, _ptr(dst), P), h.ptr)
    return dst


def mca_get_codes(h: Handle, P: int) -> np.ndarray:
    dst = np.empty(P, np.int8)
    _check(load_library().mca_get_codes(h.ptr, dst.ctypes.data, P), h.ptr)
    return dst


def mca_set_params(h: Handle, params, codes=None, tau: int = 0):
    P = int(params.shape[0])
    _check(load_library().mca_set_params(h.ptr, _ptr(params),
                                         None if codes is None else _ptr(codes), P, tau), h.ptr)


def mca_resync(h: Handle):
    _check(load_library().mca_resync(h.ptr), h.ptr)


def mca_get_trace(h: Handle, cap: int) -> np.ndarray:
    buf = np.zeros(cap, TRACE_DTYPE)
    n = c_size_t(0)
    _check(load_library().mca_get_trace(h.ptr, buf.ctypes.data, cap, ctypes.byref(n)), h.ptr)
    return buf[:n.value]


def mca_force_decisions(h: Handle, taus: Sequence[int], accepts: Sequence[bool]):
    t = np.ascontiguousarray(np.asarray(taus, dtype=np.uint64))
    a = np.ascontiguousarray(np.asarray(accepts, dtype=np.uint8))
    _check(load_library().mca_force_decisions(h.ptr, t.ctypes.data if len(t) else None,
                                              a.ctypes.data if len(a) else None, len(t)), h.ptr)


def mca_get_stats(h: Handle) -> dict:
    st = mca_run_stats()
    _check(load_library().mca_get_stats(h.ptr, ctypes.byref(st)), h.ptr)
    return st.asdict()


def mca_eval_candidates(h: Handle, flat_idx, new_w) -> np.ndarray:
    idx = np.ascontiguousarray(np.asarray(flat_idx, dtype=np.uint32))
    nw = np.ascontiguousarray(np.asarray(new_w, dtype=np.float32))
    out = np.zeros(len(idx), np.float64)
    _check(load_library().mca_eval_candidates(h.ptr, idx.ctypes.data, nw.ctypes.data, len(idx),
                                              out.ctypes.data), h.ptr)
    return out


def mca_eval_candidates_noalloc(h: Handle, flat_idx, new_w, dS):
    """flat_idx (int32/uint32 bits), new_w (float32) and dS (float64): CUDA tensors of equal length
    owned by the caller; the library allocates nothing for this call."""
    n = int(flat_idx.numel())
    _check(load_library().mca_eval_candidates_noalloc(h.ptr, flat_idx.data_ptr(), new_w.data_ptr(),
                                                      n, dS.data_ptr()), h.ptr)
    return dS


def mca_eval_trials(h: Handle, seed: int, tau: int, n: int) -> np.ndarray:
    """Proposals of trials tau .. tau+n-1 and their loss changes on this handle's samples (no
    commit): a structured array of TRACE_DTYPE records."""
    buf = np.zeros(n, TRACE_DTYPE)
    _check(load_library().mca_eval_trials(h.ptr, seed, tau, n, buf.ctypes.data), h.ptr)
    return buf


def mca_decide_batch(h: Handle, seed: int, tau: int, valid, dS, n_samples: int = 0) -> int:
    """Index of the accepted trial of a batch under the handle's rule (Eq. 6 / Eq. 7), -1 if none."""
    v = np.ascontiguousarray(np.asarray(valid, dtype=np.uint8))
    d = np.ascontiguousarray(np.asarray(dS, dtype=np.float64))
    k = c_int32(-1)
    _check(load_library().mca_decide_batch(h.ptr, seed, tau, len(v), v.ctypes.data, d.ctypes.data,
                                           n_samples, ctypes.byref(k)), h.ptr)
    return k.value


CHANNEL = {"he": 0, "zero": 1}


def mca_run_channels(h: Handle, n_trials: int, seed: int, scheme: str):
    """Channel-mutation trials (Section 2.3); returns (accepted [n] bool, dS [n] float64)."""
    acc = np.zeros(n_trials, np.uint8)
    dS = np.zeros(n_trials, np.float64)
    _check(load_library().mca_run_channels(h.ptr, n_trials, seed, CHANNEL[scheme],
                                           acc.ctypes.data, dS.ctypes.data), h.ptr)
    return acc.astype(bool), dS


def mca_selftest_wait_timeout():
    """(status recorded by the kernel, host milliseconds): the trial loop's bounded grid barrier
    waiting for a peer CTA that never arrives must give up with MCA_ERR_TIMEOUT."""
    st, ms = ctypes.c_int32(-1), ctypes.c_double(0.0)
    _check(load_library().mca_selftest_wait_timeout(ctypes.byref(st), ctypes.byref(ms)))
    return st.value, ms.value


def mca_destroy(h: Handle):
    h.close()


def create_from_workload(wl, device: bool = True, **kw) -> Handle:
    """mca_create for a workloads.MLPWorkload, with its arrays moved to the GPU by torch."""
    import torch
    X, y, init = wl.X, wl.y, wl.init
    if device:
        X = torch.from_numpy(X).cuda()
        y = torch.from_numpy(y).cuda()
        init = torch.from_numpy(init).cuda()
    kw.setdefault("K", wl.K)
    return mca_create(wl.layers, wl.loss, wl.domain, X, y, init, **kw)
