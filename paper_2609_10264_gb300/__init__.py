"""Python binding of libpvmvmd (include/pvmvmd.h): argument marshalling only.

Every function has the name of the C entry point it calls.  Device buffers are
torch CUDA tensors (uint32 field data may be held as torch.int32 or
torch.uint32; both are passed as raw 32-bit words).  Streams default to
torch's current stream.  Errors raise PvmvmdError with the library's message.

The library must be built (``python -m paper_2609_10264_gb300.build`` or
``__graft_entry__.build()``).  It is opened on the first call (or by
``load_library()``), which fails loudly when it is missing: there is no
fallback path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libpvmvmd.so")

PVMVMD_Q = 2013265921
PVMVMD_MAX_K = 131071
PVMVMD_MAX_T = 4096
PVMVMD_NOALLOC_SCRATCH_BYTES = 16 << 20
PVMVMD_OK = 0
PVMVMD_E_ARG = -1
PVMVMD_E_SHAPE = -2
PVMVMD_E_PARAM = -3
PVMVMD_E_CUDA = -4
PVMVMD_E_NOMEM = -5
PVMVMD_E_DEVICE_TIMEOUT = -6
PVMVMD_E_NODEVICE = -7


class PvmvmdError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {pvmvmd_strerror(status)} (status {status})")


class pvmvmd_key(ctypes.Structure):
    _fields_ = [("k", ctypes.c_uint32 * 8)]


class pvmvmd_params(ctypes.Structure):
    _fields_ = [("lambda_", ctypes.c_int), ("kappa", ctypes.c_int), ("rate", ctypes.c_int),
                ("delta", ctypes.c_double), ("t_x", ctypes.c_int), ("t_y", ctypes.c_int),
                ("ell", ctypes.c_int), ("scratch_batch", ctypes.c_int)]


_cu32p = ctypes.POINTER(ctypes.c_uint32)


class pvmvmd_ctx_view(ctypes.Structure):
    _fields_ = [("m", ctypes.c_int), ("K", ctypes.c_int), ("rate", ctypes.c_int),
                ("N_x", ctypes.c_int), ("N_y", ctypes.c_int), ("t_x", ctypes.c_int),
                ("t_y", ctypes.c_int), ("ell", ctypes.c_int),
                ("gx_pi1", ctypes.c_void_p), ("gx_pi2", ctypes.c_void_p), ("gx_v1", ctypes.c_void_p),
                ("gx_v2", ctypes.c_void_p), ("gy_pi1", ctypes.c_void_p), ("gy_pi2", ctypes.c_void_p),
                ("gy_v1", ctypes.c_void_p), ("gy_v2", ctypes.c_void_p),
                ("PT", ctypes.c_void_p), ("Q", ctypes.c_void_p)]


class pvmvmd_bv_params(ctypes.Structure):
    _fields_ = [("rate", ctypes.c_int), ("t", ctypes.c_int), ("ell", ctypes.c_int), ("t2", ctypes.c_int),
                ("ell2", ctypes.c_int)]


class pvmvmd_bv_view(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int) for f in ("B", "m", "n", "rate", "N", "N2", "t", "ell", "t2", "ell2")] + \
               [("Qs", ctypes.c_void_p), ("QauxT", ctypes.c_void_p), ("chal2", ctypes.c_void_p)]


class pvmvmd_mvm_batch_job(ctypes.Structure):
    _fields_ = [("W_dev", ctypes.c_void_p), ("Xhat_dev", ctypes.c_void_p), ("Yhat_dev", ctypes.c_void_p),
                ("m", ctypes.c_int), ("K", ctypes.c_int), ("B", ctypes.c_int)]


class pvmvmd_mvm_job(ctypes.Structure):
    _fields_ = [("W_dev", ctypes.c_void_p), ("xhat_dev", ctypes.c_void_p), ("yhat_dev", ctypes.c_void_p),
                ("m", ctypes.c_int), ("K", ctypes.c_int)]


# Exported symbols and their ctypes signatures (mirrors include/pvmvmd.h).
_vp, _i, _sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
SIGNATURES = {
    "pvmvmd_params_resolve": (_i, [ctypes.POINTER(pvmvmd_params), _i, _i, ctypes.POINTER(pvmvmd_params)]),
    "pvmvmd_preprocess": (_i, [_vp, _i, _i, ctypes.POINTER(pvmvmd_params), ctypes.POINTER(pvmvmd_key), _vp,
                               ctypes.POINTER(_vp)]),
    "pvmvmd_state_size": (_i, [_vp, _i, ctypes.POINTER(_sz)]),
    "pvmvmd_encode": (_i, [_vp, _vp, _i, ctypes.POINTER(pvmvmd_key), _vp, _vp, _vp]),
    "pvmvmd_server_mvm": (_i, [_vp, _i, _i, _vp, _i, _vp, _vp]),
    "pvmvmd_server_mvm_multi": (_i, [ctypes.POINTER(pvmvmd_mvm_job), _i, _vp]),
    "pvmvmd_server_mvm_noalloc": (_i, [_vp, _i, _i, _vp, _i, _vp, _vp]),
    "pvmvmd_server_mvm_grouped": (_i, [ctypes.POINTER(pvmvmd_mvm_batch_job), _i, _vp]),
    "pvmvmd_decode_verify": (_i, [_vp, _vp, _vp, _vp, _i, ctypes.POINTER(pvmvmd_key), _vp, _vp, _vp]),
    "pvmvmd_boost_prepare": (_i, [_vp, _i, ctypes.POINTER(pvmvmd_key), _vp, _vp, _vp, _vp]),
    "pvmvmd_boost_encode": (_i, [_vp, _vp, _i, _i, _vp, _vp]),
    "pvmvmd_boost_decode_verify": (_i, [_vp, _vp, _vp, _vp, _i, ctypes.POINTER(pvmvmd_key), _vp, _vp,
                                        _vp]),
    "pvmvmd_bv_preprocess": (_i, [_vp, _i, _i, _i, ctypes.POINTER(pvmvmd_bv_params), ctypes.POINTER(pvmvmd_key),
                                  _vp, ctypes.POINTER(_vp)]),
    "pvmvmd_bv_challenge": (_i, [_vp, ctypes.POINTER(pvmvmd_key), _vp, _vp]),
    "pvmvmd_bv_server_project": (_i, [_vp, _vp, _vp, _vp]),
    "pvmvmd_bv_check": (_i, [_vp, _vp, _vp, _vp, _vp, ctypes.POINTER(pvmvmd_key), _vp, _vp]),
    "pvmvmd_bv_info": (_i, [_vp, ctypes.POINTER(pvmvmd_bv_view)]),
    "pvmvmd_bv_destroy": (None, [_vp]),
    "pvmvmd_weights_split_i16": (_i, [_vp, _i, _i, _vp, _vp, _vp]),
    "pvmvmd_server_mvm_i16": (_i, [_vp, _vp, _i, _i, _vp, _i, _vp, _vp, _vp]),
    "pvmvmd_preprocess_i16": (_i, [_vp, _i, _i, ctypes.POINTER(pvmvmd_params), ctypes.POINTER(pvmvmd_key), _vp,
                                   ctypes.POINTER(_vp)]),
    "pvmvmd_code_encode_scratch": (_i, [_vp, _i, _i, ctypes.POINTER(_sz)]),
    "pvmvmd_code_encode_lanes": (_i, [_vp, _i, _vp, _i, _vp, _vp, _vp]),
    "pvmvmd_device_status": (_i, [_vp]),
    "pvmvmd_kernel_launches": (ctypes.c_ulonglong, []),
    "pvmvmd_debug_expire_wait": (_i, [_i, ctypes.c_uint32, ctypes.c_uint64]),
    "pvmvmd_ctx_info": (_i, [_vp, ctypes.POINTER(pvmvmd_ctx_view)]),
    "pvmvmd_destroy": (None, [_vp]),
    "pvmvmd_strerror": (ctypes.c_char_p, [_i]),
    "pvmvmd_code_sample_host": (_i, [ctypes.POINTER(pvmvmd_key), _i, ctypes.c_uint32, _cu32p, _cu32p,
                                     _cu32p, _cu32p]),
}


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"{LIB_PATH} is not built: run `python -c 'import __graft_entry__ as g; g.build()'` "
            "(needs nvcc); this package has no fallback path")
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


class _Library:
    """libpvmvmd.so, opened on first use.  Importing the package (for example
    only its input generators) maps no CUDA library; the first call of any
    entry point opens it and raises ImportError if it is not built."""
    _handle = None

    def __getattr__(self, name):
        if _Library._handle is None:
            _Library._handle = _load()
        return getattr(_Library._handle, name)


_lib = _Library()


def load_library():
    """Open libpvmvmd.so now (ImportError if it is missing) and return it."""
    if _Library._handle is None:
        _Library._handle = _load()
    return _Library._handle


def _check(status: int, where: str) -> None:
    if status != PVMVMD_OK:
        raise PvmvmdError(status, where)


def pvmvmd_strerror(status: int) -> str:
    return _lib.pvmvmd_strerror(int(status)).decode()


# --------------------------------------------------------------------------- marshalling

def make_key(seed) -> pvmvmd_key:
    """A pvmvmd_key from an integer < 2^256 (little-endian 32-bit words), from 32
    bytes, or from 8 words."""
    k = pvmvmd_key()
    if isinstance(seed, pvmvmd_key):
        return seed
    if isinstance(seed, (bytes, bytearray)):
        if len(seed) != 32:
            raise ValueError("a key is 32 bytes")
        words = np.frombuffer(bytes(seed), dtype="<u4")
    elif isinstance(seed, (int, np.integer)):
        s = int(seed)
        if s < 0 or s >= 1 << 256:
            raise ValueError("integer key must be in [0, 2^256)")
        words = [(s >> (32 * i)) & 0xFFFFFFFF for i in range(8)]
    else:
        words = [int(w) for w in seed]
        if len(words) != 8:
            raise ValueError("a key is 8 words")
    for i in range(8):
        k.k[i] = int(words[i])
    return k


def _stream_ptr(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _dev_ptr(t, name: str, dtypes, numel=None):
    import torch
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype not in dtypes:
        raise TypeError(f"{name} must have dtype in {dtypes}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name} has {t.numel()} elements, expected {numel}")
    return ctypes.c_void_p(t.data_ptr())


def _u32_types():
    import torch
    types = [torch.int32]
    if hasattr(torch, "uint32"):
        types.append(torch.uint32)
    return tuple(types)


def _new_u32(shape, like=None):
    import torch
    dev = like.device if like is not None else "cuda"
    return torch.empty(shape, dtype=torch.int32, device=dev)


# --------------------------------------------------------------------------- API

def pvmvmd_params_resolve(m: int, K: int, params: pvmvmd_params | None = None) -> pvmvmd_params:
    out = pvmvmd_params()
    _check(_lib.pvmvmd_params_resolve(ctypes.byref(params) if params is not None else None, m, K,
                                      ctypes.byref(out)), "pvmvmd_params_resolve")
    return out


class Ctx:
    """Owner of a pvmvmd_ctx handle (public parameters pp on the device)."""

    def __init__(self, handle: int, m: int, K: int):
        self.handle = ctypes.c_void_p(handle)
        self.m, self.K = m, K
        v = pvmvmd_ctx_info(self)
        self.t_x, self.t_y, self.ell = v.t_x, v.t_y, v.ell
        self.N_x, self.N_y, self.rate = v.N_x, v.N_y, v.rate

    def destroy(self) -> None:
        if self.handle is not None and self.handle.value:
            _lib.pvmvmd_destroy(self.handle)
        self.handle = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def pvmvmd_preprocess(W, key, params: pvmvmd_params | None = None, stream=None) -> Ctx:
    import torch
    if W.dim() != 2:
        raise ValueError("W must be m x K")
    m, K = W.shape
    ptr = _dev_ptr(W, "W", (torch.int8,))
    out = ctypes.c_void_p()
    k = make_key(key)
    _check(_lib.pvmvmd_preprocess(ptr, m, K, ctypes.byref(params) if params is not None else None,
                                  ctypes.byref(k), _stream_ptr(stream), ctypes.byref(out)),
           "pvmvmd_preprocess")
    return Ctx(out.value, m, K)


def pvmvmd_preprocess_i16(W, key, params: pvmvmd_params | None = None, stream=None) -> Ctx:
    """As pvmvmd_preprocess for a 16-bit M (int16 m x K, entries in [-32768, 32639])."""
    import torch
    if W.dim() != 2:
        raise ValueError("W must be m x K")
    m, K = W.shape
    out = ctypes.c_void_p()
    _check(_lib.pvmvmd_preprocess_i16(_dev_ptr(W, "W", (torch.int16,)), m, K,
                                      ctypes.byref(params) if params is not None else None,
                                      ctypes.byref(make_key(key)), _stream_ptr(stream), ctypes.byref(out)),
           "pvmvmd_preprocess_i16")
    return Ctx(out.value, m, K)


def pvmvmd_weights_split_i16(W, stream=None):
    """16-bit M -> (M_hi, M_lo) int8 planes with M = 256 M_hi + M_lo."""
    import torch
    m, K = W.shape
    hi = torch.empty((m, K), dtype=torch.int8, device=W.device)
    lo = torch.empty((m, K), dtype=torch.int8, device=W.device)
    _check(_lib.pvmvmd_weights_split_i16(_dev_ptr(W, "W", (torch.int16,)), m, K, _dev_ptr(hi, "hi", (torch.int8,)),
                                         _dev_ptr(lo, "lo", (torch.int8,)), _stream_ptr(stream)),
           "pvmvmd_weights_split_i16")
    return hi, lo


def pvmvmd_server_mvm_i16(Whi, Wlo, Xhat, Yhat=None, Ytmp=None, stream=None):
    """Y_hat = (256 M_hi + M_lo) X_hat over F_q from the two int8 planes."""
    import torch
    m, K = Whi.shape
    B = _batch(Xhat, K, "Xhat")
    shape = (m,) if Xhat.dim() == 1 else (B, m)
    if Yhat is None:
        Yhat = _new_u32(shape, Xhat)
    if Ytmp is None:
        Ytmp = _new_u32(shape, Xhat)
    _check(_lib.pvmvmd_server_mvm_i16(_dev_ptr(Whi, "Whi", (torch.int8,)), _dev_ptr(Wlo, "Wlo", (torch.int8,)), m, K,
                                      _dev_ptr(Xhat, "Xhat", _u32_types()), B,
                                      _dev_ptr(Yhat, "Yhat", _u32_types(), B * m),
                                      _dev_ptr(Ytmp, "Ytmp", _u32_types(), B * m), _stream_ptr(stream)),
           "pvmvmd_server_mvm_i16")
    return Yhat


def pvmvmd_ctx_info(ctx: Ctx) -> pvmvmd_ctx_view:
    v = pvmvmd_ctx_view()
    _check(_lib.pvmvmd_ctx_info(ctx.handle, ctypes.byref(v)), "pvmvmd_ctx_info")
    return v


def pvmvmd_state_size(ctx: Ctx, B: int) -> int:
    n = ctypes.c_size_t()
    _check(_lib.pvmvmd_state_size(ctx.handle, B, ctypes.byref(n)), "pvmvmd_state_size")
    return n.value


def _batch(X, L: int, name: str) -> int:
    if X.dim() == 1:
        if X.numel() != L:
            raise ValueError(f"{name} must have {L} entries")
        return 1
    if X.dim() != 2 or X.shape[1] != L:
        raise ValueError(f"{name} must be B x {L}")
    return X.shape[0]


def pvmvmd_encode(ctx: Ctx, X, key, Xhat=None, st=None, stream=None):
    """Encrypt B vectors: returns (Xhat, st)."""
    B = _batch(X, ctx.K, "X")
    xp = _dev_ptr(X, "X", _u32_types())
    if Xhat is None:
        Xhat = _new_u32(X.shape, X)
    if st is None:
        st = _new_u32((B, 2 * ctx.t_x), X)
    _check(_lib.pvmvmd_encode(ctx.handle, xp, B, ctypes.byref(make_key(key)),
                              _dev_ptr(Xhat, "Xhat", _u32_types(), X.numel()),
                              _dev_ptr(st, "st", _u32_types(), B * 2 * ctx.t_x), _stream_ptr(stream)),
           "pvmvmd_encode")
    return Xhat, st


def pvmvmd_code_encode_scratch(ctx: Ctx, which: int, L: int) -> int:
    """Bytes of scratch pvmvmd_code_encode_lanes needs for L lanes."""
    n = _sz()
    _check(_lib.pvmvmd_code_encode_scratch(ctx.handle, which, L, ctypes.byref(n)), "pvmvmd_code_encode_scratch")
    return n.value


def pvmvmd_code_encode_lanes(ctx: Ctx, which: int, X, Y=None, scratch=None, stream=None):
    """Y = G^T X for the context's code G_x (which = 0) or G_y (which = 1):
    X is n x L (row i holds entry i of every lane), Y is N x L."""
    import torch
    n = ctx.K if which == 0 else ctx.m
    N = n * ctx.rate
    if X.dim() != 2 or X.shape[0] != n:
        raise ValueError(f"X must be {n} x L")
    L = X.shape[1]
    if Y is None:
        Y = _new_u32((N, L), X)
    if scratch is None:
        scratch = torch.empty(pvmvmd_code_encode_scratch(ctx, which, L), dtype=torch.uint8, device=X.device)
    _check(_lib.pvmvmd_code_encode_lanes(ctx.handle, which, _dev_ptr(X, "X", _u32_types()), L,
                                         _dev_ptr(Y, "Y", _u32_types(), N * L),
                                         _dev_ptr(scratch, "scratch", (torch.uint8,)), _stream_ptr(stream)),
           "pvmvmd_code_encode_lanes")
    return Y


def pvmvmd_server_mvm(W, Xhat, Yhat=None, stream=None):
    """Y_hat = M X_hat over F_q for Xhat of shape (K,) or (B, K)."""
    import torch
    m, K = W.shape
    B = _batch(Xhat, K, "Xhat")
    if Yhat is None:
        Yhat = _new_u32((m,) if Xhat.dim() == 1 else (B, m), Xhat)
    _check(_lib.pvmvmd_server_mvm(_dev_ptr(W, "W", (torch.int8,)), m, K, _dev_ptr(Xhat, "Xhat", _u32_types()),
                                  B, _dev_ptr(Yhat, "Yhat", _u32_types(), B * m), _stream_ptr(stream)),
           "pvmvmd_server_mvm")
    return Yhat


def pvmvmd_server_mvm_noalloc(W, Xhat, Yhat, stream=None) -> None:
    """Y_hat = M X_hat like pvmvmd_server_mvm, for callers that cannot let the
    library allocate device memory: the call allocates nothing (the caller
    passes the output) and uses the library's fixed 16 MiB device buffer,
    shared by all such calls (order them on one stream)."""
    import torch
    m, K = W.shape
    B = _batch(Xhat, K, "Xhat")
    _check(_lib.pvmvmd_server_mvm_noalloc(_dev_ptr(W, "W", (torch.int8,)), m, K,
                                          _dev_ptr(Xhat, "Xhat", _u32_types()), B,
                                          _dev_ptr(Yhat, "Yhat", _u32_types(), B * m), _stream_ptr(stream)),
           "pvmvmd_server_mvm_noalloc")


def batch_jobs(triples):
    """A ctypes job array for pvmvmd_server_mvm_grouped from (W, Xhat, Yhat)
    tensors (Xhat B x K, Yhat B x m); reusable across calls while the tensors
    live."""
    import torch
    arr = (pvmvmd_mvm_batch_job * len(triples))()
    for i, (W, Xh, Yh) in enumerate(triples):
        m, K = W.shape
        B = _batch(Xh, K, "Xhat")
        arr[i].W_dev = _dev_ptr(W, "W", (torch.int8,)).value
        arr[i].Xhat_dev = _dev_ptr(Xh, "Xhat", _u32_types()).value
        arr[i].Yhat_dev = _dev_ptr(Yh, "Yhat", _u32_types(), B * m).value
        arr[i].m, arr[i].K, arr[i].B = m, K, B
    return arr


def pvmvmd_server_mvm_grouped(jobs, stream=None) -> None:
    """Several independent server products in as few launches as possible:
    `jobs` is a list of (W, Xhat, Yhat) tensors or an array from batch_jobs."""
    if not isinstance(jobs, ctypes.Array):
        jobs = batch_jobs(jobs)
    _check(_lib.pvmvmd_server_mvm_grouped(jobs, len(jobs), _stream_ptr(stream)), "pvmvmd_server_mvm_grouped")


def mvm_jobs(triples):
    """A ctypes job array for pvmvmd_server_mvm_multi from (W, xhat, yhat)
    tensors; reusable across calls while the tensors live."""
    import torch
    arr = (pvmvmd_mvm_job * len(triples))()
    for i, (W, xh, yh) in enumerate(triples):
        m, K = W.shape
        arr[i].W_dev = _dev_ptr(W, "W", (torch.int8,)).value
        arr[i].xhat_dev = _dev_ptr(xh, "xhat", _u32_types(), K).value
        arr[i].yhat_dev = _dev_ptr(yh, "yhat", _u32_types(), m).value
        arr[i].m, arr[i].K = m, K
    return arr


def pvmvmd_server_mvm_multi(jobs, stream=None) -> None:
    """Independent batch-1 products: `jobs` is a list of (W, xhat, yhat)
    tensors or an array from mvm_jobs()."""
    if not isinstance(jobs, ctypes.Array):
        jobs = mvm_jobs(jobs)
    _check(_lib.pvmvmd_server_mvm_multi(jobs, len(jobs), _stream_ptr(stream)), "pvmvmd_server_mvm_multi")


def pvmvmd_decode_verify(ctx: Ctx, st, Xhat, Yhat, challenge_key, Y=None, accept=None, stream=None):
    """Verify and decrypt: returns (Y, accept) with accept an int32 tensor of 0/1."""
    import torch
    B = _batch(Xhat, ctx.K, "Xhat")
    if Y is None:
        Y = _new_u32(Yhat.shape, Yhat)
    if accept is None:
        accept = torch.empty(B, dtype=torch.int32, device=Yhat.device)
    _check(_lib.pvmvmd_decode_verify(ctx.handle, _dev_ptr(st, "st", _u32_types(), B * 2 * ctx.t_x),
                                     _dev_ptr(Xhat, "Xhat", _u32_types()),
                                     _dev_ptr(Yhat, "Yhat", _u32_types(), B * ctx.m), B,
                                     ctypes.byref(make_key(challenge_key)),
                                     _dev_ptr(Y, "Y", _u32_types(), B * ctx.m),
                                     _dev_ptr(accept, "accept", (torch.int32,), B), _stream_ptr(stream)),
           "pvmvmd_decode_verify")
    return Y, accept


def pvmvmd_boost_prepare(ctx: Ctx, B: int, key, mask_in=None, mask_out=None, st=None, device=None,
                         stream=None):
    """Boost mode, offline: the masks of vectors 0 .. B-1 under `key`.
    Returns (mask_in [B x K] = G_x e_x, mask_out [B x m] = P e_x, st)."""
    like = None
    for t in (mask_in, mask_out, st):
        if t is not None:
            like = t
            break
    dev = like.device if like is not None else (device or "cuda")
    import torch
    if mask_in is None:
        mask_in = torch.empty((B, ctx.K), dtype=torch.int32, device=dev)
    if mask_out is None:
        mask_out = torch.empty((B, ctx.m), dtype=torch.int32, device=dev)
    if st is None:
        st = torch.empty((B, 2 * ctx.t_x), dtype=torch.int32, device=dev)
    _check(_lib.pvmvmd_boost_prepare(ctx.handle, B, ctypes.byref(make_key(key)),
                                     _dev_ptr(mask_in, "mask_in", _u32_types(), B * ctx.K),
                                     _dev_ptr(mask_out, "mask_out", _u32_types(), B * ctx.m),
                                     _dev_ptr(st, "st", _u32_types(), B * 2 * ctx.t_x), _stream_ptr(stream)),
           "pvmvmd_boost_prepare")
    return mask_in, mask_out, st


def pvmvmd_boost_encode(X, mask_in, Xhat=None, stream=None):
    """Boost mode, online: Xhat = X + mask_in over F_q (X and mask_in B x K)."""
    if X.shape != mask_in.shape:
        raise ValueError("X and mask_in must have the same shape")
    K = X.shape[-1]
    B = X.numel() // K
    if Xhat is None:
        Xhat = _new_u32(X.shape, X)
    _check(_lib.pvmvmd_boost_encode(_dev_ptr(X, "X", _u32_types()), _dev_ptr(mask_in, "mask_in", _u32_types()),
                                    B, K, _dev_ptr(Xhat, "Xhat", _u32_types(), X.numel()), _stream_ptr(stream)),
           "pvmvmd_boost_encode")
    return Xhat


def pvmvmd_boost_decode_verify(ctx: Ctx, mask_out, Xhat, Yhat, challenge_key, Y=None, accept=None,
                               stream=None):
    """Boost mode, online: verify and Y = Yhat - mask_out; returns (Y, accept)."""
    import torch
    B = _batch(Xhat, ctx.K, "Xhat")
    if Y is None:
        Y = _new_u32(Yhat.shape, Yhat)
    if accept is None:
        accept = torch.empty(B, dtype=torch.int32, device=Yhat.device)
    _check(_lib.pvmvmd_boost_decode_verify(ctx.handle, _dev_ptr(mask_out, "mask_out", _u32_types(), B * ctx.m),
                                           _dev_ptr(Xhat, "Xhat", _u32_types()),
                                           _dev_ptr(Yhat, "Yhat", _u32_types(), B * ctx.m), B,
                                           ctypes.byref(make_key(challenge_key)),
                                           _dev_ptr(Y, "Y", _u32_types(), B * ctx.m),
                                           _dev_ptr(accept, "accept", (torch.int32,), B), _stream_ptr(stream)),
           "pvmvmd_boost_decode_verify")
    return Y, accept


class BvCtx:
    """A batch-verification (Protocol 2) context; released by destroy() or
    garbage collection."""

    def __init__(self, handle, view):
        self.handle = handle
        for f, _ in pvmvmd_bv_view._fields_:
            setattr(self, f, getattr(view, f))

    def destroy(self):
        if self.handle:
            _lib.pvmvmd_bv_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def pvmvmd_bv_preprocess(Ws, key, params: pvmvmd_bv_params | None = None, stream=None) -> BvCtx:
    """Ws: B x m x n int8 device tensor (the B matrices)."""
    import torch
    if Ws.dim() != 3:
        raise ValueError("Ws must be B x m x n")
    B, m, n = Ws.shape
    h = ctypes.c_void_p()
    _check(_lib.pvmvmd_bv_preprocess(_dev_ptr(Ws, "Ws", (torch.int8,)), B, m, n,
                                     ctypes.byref(params) if params is not None else None,
                                     ctypes.byref(make_key(key)), _stream_ptr(stream), ctypes.byref(h)),
           "pvmvmd_bv_preprocess")
    v = pvmvmd_bv_view()
    _check(_lib.pvmvmd_bv_info(h, ctypes.byref(v)), "pvmvmd_bv_info")
    return BvCtx(h, v)


def pvmvmd_bv_challenge(ctx: BvCtx, key, chal=None, device=None, stream=None):
    import torch
    if chal is None:
        chal = torch.empty((ctx.ell, 2 * ctx.t), dtype=torch.int32, device=device or "cuda")
    _check(_lib.pvmvmd_bv_challenge(ctx.handle, ctypes.byref(make_key(key)),
                                    _dev_ptr(chal, "chal", _u32_types(), ctx.ell * 2 * ctx.t), _stream_ptr(stream)),
           "pvmvmd_bv_challenge")
    return chal


def pvmvmd_bv_server_project(ctx: BvCtx, chal, u=None, stream=None):
    import torch
    if u is None:
        u = torch.empty((ctx.ell, ctx.B * ctx.n), dtype=torch.int32, device=chal.device)
    _check(_lib.pvmvmd_bv_server_project(ctx.handle, _dev_ptr(chal, "chal", _u32_types(), ctx.ell * 2 * ctx.t),
                                         _dev_ptr(u, "u", _u32_types(), ctx.ell * ctx.B * ctx.n), _stream_ptr(stream)),
           "pvmvmd_bv_server_project")
    return u


def pvmvmd_bv_check(ctx: BvCtx, X, Y, chal, u, key2, accept=None, stream=None):
    """-> int32 tensor of one element: 1 accept, 0 reject."""
    import torch
    if accept is None:
        accept = torch.empty(1, dtype=torch.int32, device=X.device)
    _check(_lib.pvmvmd_bv_check(ctx.handle, _dev_ptr(X, "X", _u32_types(), ctx.B * ctx.n),
                                _dev_ptr(Y, "Y", _u32_types(), ctx.B * ctx.m),
                                _dev_ptr(chal, "chal", _u32_types(), ctx.ell * 2 * ctx.t),
                                _dev_ptr(u, "u", _u32_types(), ctx.ell * ctx.B * ctx.n),
                                ctypes.byref(make_key(key2)), _dev_ptr(accept, "accept", (torch.int32,), 1),
                                _stream_ptr(stream)),
           "pvmvmd_bv_check")
    return accept


PVMVMD_DEBUG_WAIT_OFF = 0
PVMVMD_DEBUG_WAIT_SCAN = 1
PVMVMD_DEBUG_WAIT_PRODUCT = 2


def pvmvmd_debug_expire_wait(site: int, index: int = 0, limit: int = 0) -> None:
    """Test hook: make one bounded device wait expire (see the header)."""
    _check(_lib.pvmvmd_debug_expire_wait(int(site), int(index), int(limit)), "pvmvmd_debug_expire_wait")


def pvmvmd_device_status(stream=None) -> int:
    """Synchronise and return the device status (raises on a timeout)."""
    s = _lib.pvmvmd_device_status(_stream_ptr(stream))
    _check(s, "pvmvmd_device_status")
    return s


def pvmvmd_kernel_launches() -> int:
    """Kernels the library has enqueued in this process so far (launches
    captured into a CUDA graph count once, at capture)."""
    return int(_lib.pvmvmd_kernel_launches())


def pvmvmd_destroy(ctx: Ctx) -> None:
    ctx.destroy()


def pvmvmd_code_sample_host(key, which: int, N: int):
    """Host sampling of one RAA generator: (pi1, pi2, v1, v2) numpy uint32 arrays."""
    arrs = [np.zeros(N, np.uint32) for _ in range(4)]
    ptrs = [a.ctypes.data_as(_cu32p) for a in arrs]
    _check(_lib.pvmvmd_code_sample_host(ctypes.byref(make_key(key)), which, N, *ptrs),
           "pvmvmd_code_sample_host")
    return tuple(arrs)


def as_u32(t) -> np.ndarray:
    """Device or host 32-bit tensor -> numpy uint32 (for checks and printing)."""
    import torch
    t = t.detach()
    if t.dtype != torch.int32:
        t = t.view(torch.int32)
    return t.cpu().contiguous().numpy().view(np.uint32).reshape(tuple(t.shape))


class _CudaArray:
    def __init__(self, ptr: int, count: int):
        self.__cuda_array_interface__ = {"shape": (count,), "typestr": "<i4", "data": (int(ptr), False),
                                         "version": 2, "strides": None}


def device_view(ptr, count: int):
    """A torch.int32 CUDA tensor aliasing `count` 32-bit words at device
    pointer `ptr` (e.g. a table of pvmvmd_ctx_info); valid while its owner
    lives."""
    import torch
    p = ptr.value if isinstance(ptr, ctypes.c_void_p) else ptr
    return torch.as_tensor(_CudaArray(p, count), device="cuda")
