"""Python binding of the JARQ C ABI (``include/jarq.h``).

Argument marshalling only: every step of the refinement runs in the CUDA
library ``libjarq.so``.  Tensors are passed as raw pointers on torch's
current CUDA stream; NumPy arrays are passed as host pointers and staged by
the library.  There is no CPU fallback: importing this module raises if the
library has not been built.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libjarq.so")

JARQ_OK = 0
JARQ_ERR_ARG = 1
JARQ_ERR_NOT_SPD = 2
JARQ_ERR_NUMERICAL = 3
JARQ_ERR_CUDA = 4
JARQ_ERR_TIMEOUT = 5
JARQ_ERR_NOMEM = 6

# Names declared in include/jarq.h (checked by the test-suite).
EXPORTS = ("jarq_default_options", "jarq_prepare_hessian", "jarq_refine_layer",
           "jarq_objective", "jarq_hessian_din", "jarq_hessian_group_size",
           "jarq_hessian_destroy", "jarq_status_string", "jarq_profile_enable",
           "jarq_profile_reset", "jarq_profile_read", "jarq_launch_count",
           "jarq_objective_noalloc", "jarq_residual_product", "jarq_canonicalize",
           "jarq_dequantize", "jarq_pack_codes", "jarq_accumulate_hessian",
           "jarq_refine_layer_mu", "jarq_fit_scales", "jarq_multicode_probe",
           "jarq_selftest_wait_timeout")


class JarqError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


class Options(ctypes.Structure):
    _fields_ = [("max_iters", ctypes.c_int), ("early_stop", ctypes.c_int),
                ("tau_rel", ctypes.c_float), ("tau_abs", ctypes.c_float),
                ("ridge", ctypes.c_float), ("rcond", ctypes.c_float),
                ("eps", ctypes.c_float), ("ridge_accept", ctypes.c_int),
                ("fixed_grid", ctypes.c_int)]


class Stats(ctypes.Structure):
    _fields_ = [("L_host", ctypes.c_void_p), ("L_final", ctypes.c_void_p),
                ("iters", ctypes.c_void_p), ("accepted", ctypes.c_void_p),
                ("ridge_hits", ctypes.c_void_p), ("row_status", ctypes.c_void_p)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"JARQ CUDA library not built: {LIB_PATH} is missing "
                          "(run __graft_entry__.build())")
    lib = ctypes.CDLL(LIB_PATH)
    vp, ci, cf = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    lib.jarq_default_options.restype = Options
    lib.jarq_default_options.argtypes = []
    lib.jarq_prepare_hessian.restype = ci
    lib.jarq_prepare_hessian.argtypes = [vp, ci, ci, cf, ctypes.POINTER(vp), vp]
    lib.jarq_refine_layer.restype = ci
    lib.jarq_refine_layer.argtypes = [vp, vp, vp, vp, vp, ci, ci, ctypes.POINTER(Options),
                                      ctypes.POINTER(Stats), vp]
    lib.jarq_refine_layer_mu.restype = ci
    lib.jarq_refine_layer_mu.argtypes = [vp, vp, vp, vp, vp, ci, ci, vp, vp, cf, cf,
                                         ctypes.POINTER(Options), ctypes.POINTER(Stats), vp]
    lib.jarq_fit_scales.restype = ci
    lib.jarq_fit_scales.argtypes = [vp, vp, vp, vp, vp, ci, ci, ci, ci, vp, vp, vp]
    lib.jarq_multicode_probe.restype = ci
    lib.jarq_multicode_probe.argtypes = [vp, vp, vp, vp, vp, ci, ci, ci, vp, vp, vp, vp, vp, vp]
    lib.jarq_objective.restype = ci
    lib.jarq_objective.argtypes = [vp, vp, vp, vp, vp, ci, ci, vp, vp]
    lib.jarq_objective_noalloc.restype = ci
    lib.jarq_objective_noalloc.argtypes = [vp, vp, vp, vp, vp, ci, ci, vp, vp]
    lib.jarq_residual_product.restype = ci
    lib.jarq_residual_product.argtypes = [vp, vp, vp, vp, vp, ci, ci, vp, vp]
    lib.jarq_canonicalize.restype = ci
    lib.jarq_canonicalize.argtypes = [vp, vp, vp, ci, ci, ci, ci, vp]
    lib.jarq_dequantize.restype = ci
    lib.jarq_dequantize.argtypes = [vp, vp, vp, ci, ci, ci, ci, ci, vp, vp]
    lib.jarq_pack_codes.restype = ci
    lib.jarq_pack_codes.argtypes = [vp, ci, ci, ci, vp, vp]
    lib.jarq_accumulate_hessian.restype = ci
    lib.jarq_accumulate_hessian.argtypes = [vp, ci, ci, cf, vp, vp]
    lib.jarq_hessian_din.restype = ci
    lib.jarq_hessian_din.argtypes = [vp]
    lib.jarq_hessian_group_size.restype = ci
    lib.jarq_hessian_group_size.argtypes = [vp]
    lib.jarq_hessian_destroy.restype = None
    lib.jarq_hessian_destroy.argtypes = [vp]
    lib.jarq_status_string.restype = ctypes.c_char_p
    lib.jarq_status_string.argtypes = [ci]
    lib.jarq_profile_enable.restype = None
    lib.jarq_profile_enable.argtypes = [ci]
    lib.jarq_profile_reset.restype = None
    lib.jarq_profile_reset.argtypes = []
    lib.jarq_profile_read.restype = ci
    lib.jarq_profile_read.argtypes = [ctypes.c_char_p, ctypes.POINTER(ctypes.c_longlong),
                                      ctypes.POINTER(ctypes.c_double)]
    lib.jarq_launch_count.restype = ctypes.c_longlong
    lib.jarq_launch_count.argtypes = []
    lib.jarq_selftest_wait_timeout.restype = ci
    lib.jarq_selftest_wait_timeout.argtypes = [vp]
    return lib


_lib = _load()


def library():
    """The loaded ctypes library (for tests that call the C ABI directly)."""
    return _lib


KERNELS = ("validate", "residual", "init_rows", "hr_full", "grad", "gram", "scale_solve",
           "phase_hr", "babai", "symmetrize", "group_factor", "slices", "slice_rows", "proj",
           "whw", "rhs", "htilde", "ptilde", "target", "syrk", "mu_combine", "own_rhs", "scale_fit", "probe")


def profile_enable(on: bool = True):
    """Record CUDA events around each library kernel launch (instrumentation)."""
    _lib.jarq_profile_enable(1 if on else 0)


def profile_reset():
    _lib.jarq_profile_reset()


def profile_read(kernel: str):
    """(launches, total device ms) accumulated for one kernel name."""
    n = ctypes.c_longlong()
    ms = ctypes.c_double()
    if _lib.jarq_profile_read(kernel.encode(), ctypes.byref(n), ctypes.byref(ms)) != 0:
        raise KeyError(kernel)
    return int(n.value), float(ms.value)


def launch_count() -> int:
    """Kernels launched by the library since it was loaded."""
    return int(_lib.jarq_launch_count())


def selftest_wait_timeout() -> int:
    """Status of a device wait that nothing completes (JARQ_ERR_TIMEOUT when
    the bounded-wait path works), on the current torch stream."""
    import torch
    return int(_lib.jarq_selftest_wait_timeout(ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)))


def status_string(status: int) -> str:
    return _lib.jarq_status_string(int(status)).decode()


def default_options(**overrides) -> Options:
    o = _lib.jarq_default_options()
    for k, v in overrides.items():
        if not hasattr(o, k):
            raise KeyError(f"unknown option {k}")
        setattr(o, k, type(getattr(o, k))(v))
    return o


def _is_torch(x):
    return type(x).__module__.startswith("torch")


def _ptr(x, dtype_np):
    """Raw pointer of a contiguous torch tensor or NumPy array of the given dtype."""
    if x is None:
        return None
    if _is_torch(x):
        import torch
        want = {np.float32: torch.float32, np.uint8: torch.uint8, np.int32: torch.int32,
                np.float64: torch.float64}[dtype_np]
        if x.dtype != want or not x.is_contiguous():
            raise TypeError(f"expected a contiguous {want} tensor, got {x.dtype}")
        return x.data_ptr()
    if not isinstance(x, np.ndarray) or x.dtype != dtype_np or not x.flags.c_contiguous:
        raise TypeError(f"expected a C-contiguous {np.dtype(dtype_np)} array")
    return x.ctypes.data


def _stream(*tensors):
    for t in tensors:
        if _is_torch(t) and t.is_cuda:
            import torch
            return ctypes.c_void_p(torch.cuda.current_stream(t.device).cuda_stream)
    return ctypes.c_void_p(None)


class Hessian:
    """A prepared Hessian (``jarq_prepare_hessian``); freed on ``close``."""

    def __init__(self, H, group_size: int, nu2: float = 0.0):
        d = int(H.shape[0])
        if tuple(H.shape) != (d, d):
            raise ValueError("H must be square")
        handle = ctypes.c_void_p()
        st = _lib.jarq_prepare_hessian(_ptr(H, np.float32), d, int(group_size), float(nu2),
                                       ctypes.byref(handle), _stream(H))
        if st != JARQ_OK:
            raise JarqError(st, "jarq_prepare_hessian")
        self._h = handle
        self.din = d
        self.group_size = int(group_size)

    @property
    def handle(self):
        return self._h

    def close(self):
        if self._h is not None and self._h.value:
            _lib.jarq_hessian_destroy(self._h)
        self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def prepare(H, group_size: int, nu2: float = 0.0) -> Hessian:
    return Hessian(H, group_size, nu2)


@dataclass
class RefineStats:
    L_host: object
    L_final: object
    iters: object
    accepted: object
    ridge_hits: object
    row_status: object
    status: int


def _alloc_like(ref, n, dtype_np):
    if _is_torch(ref):
        import torch
        tdt = {np.float64: torch.float64, np.int32: torch.int32}[dtype_np]
        return torch.empty(n, dtype=tdt, device=ref.device)
    return np.empty(n, dtype=dtype_np)


def refine(hess: Hessian, W, S, Q, Z, bits: int, options: Options = None,
           collect_stats: bool = True, raise_on_error: bool = True, **opt):
    """``jarq_refine_layer``: refine S and Q in place; returns RefineStats."""
    o = options if options is not None else default_options(**opt)
    dout = int(W.shape[0])
    st = None
    stats = None
    if collect_stats:
        st = RefineStats(*(_alloc_like(W, dout, t) for t in
                           (np.float64, np.float64, np.int32, np.int32, np.int32, np.int32)),
                         status=0)
        stats = Stats(*(_ptr(x, t) for x, t in zip(
            (st.L_host, st.L_final, st.iters, st.accepted, st.ridge_hits, st.row_status),
            (np.float64, np.float64, np.int32, np.int32, np.int32, np.int32))))
    status = _lib.jarq_refine_layer(hess.handle, _ptr(W, np.float32), _ptr(S, np.float32),
                                    _ptr(Q, np.uint8), _ptr(Z, np.int32), dout, int(bits),
                                    ctypes.byref(o), ctypes.byref(stats) if stats else None,
                                    _stream(W, S, Q, Z))
    if st is not None:
        st.status = status
    if raise_on_error and status not in (JARQ_OK,):
        raise JarqError(status, "jarq_refine_layer")
    return st if st is not None else status


def refine_mu(hess: Hessian, W, S, Q, Z, bits: int, K, XX, mu: float, nu2: float,
              options: Options = None, collect_stats: bool = True, raise_on_error: bool = True,
              **opt):
    """``jarq_refine_layer_mu``: refinement on the propagation-corrected target
    (K = X~^T X, XX = X^T X, normalised like the prepared H = X~^T X~ + nu2 I);
    S and Q in place; returns RefineStats with the mu-objective."""
    o = options if options is not None else default_options(**opt)
    dout = int(W.shape[0])
    st = None
    stats = None
    if collect_stats:
        st = RefineStats(*(_alloc_like(W, dout, t) for t in
                           (np.float64, np.float64, np.int32, np.int32, np.int32, np.int32)),
                         status=0)
        stats = Stats(*(_ptr(x, t) for x, t in zip(
            (st.L_host, st.L_final, st.iters, st.accepted, st.ridge_hits, st.row_status),
            (np.float64, np.float64, np.int32, np.int32, np.int32, np.int32))))
    status = _lib.jarq_refine_layer_mu(hess.handle, _ptr(W, np.float32), _ptr(S, np.float32),
                                       _ptr(Q, np.uint8), _ptr(Z, np.int32), dout, int(bits),
                                       _ptr(K, np.float32), _ptr(XX, np.float32), float(mu),
                                       float(nu2), ctypes.byref(o),
                                       ctypes.byref(stats) if stats else None,
                                       _stream(W, S, Q, Z))
    if st is not None:
        st.status = status
    if raise_on_error and status not in (JARQ_OK,):
        raise JarqError(status, "jarq_refine_layer_mu")
    return st if st is not None else status


JARQ_FIT_JOINT, JARQ_FIT_INDEPENDENT, JARQ_FIT_COORDINATE = 0, 1, 2


def fit_scales(hess: Hessian, W, S, Q, Z, bits: int, method: str = "joint", passes: int = 3):
    """``jarq_fit_scales``: refit S in place for the codes Q with the joint,
    independent or coordinate-descent fit; returns (F_before, F_after)."""
    code = {"joint": JARQ_FIT_JOINT, "independent": JARQ_FIT_INDEPENDENT,
            "coordinate": JARQ_FIT_COORDINATE}[method]
    dout = int(W.shape[0])
    Fb, Fa = _alloc_like(W, dout, np.float64), _alloc_like(W, dout, np.float64)
    status = _lib.jarq_fit_scales(hess.handle, _ptr(W, np.float32), _ptr(S, np.float32),
                                  _ptr(Q, np.uint8), _ptr(Z, np.int32), dout, int(bits), code,
                                  int(passes), _ptr(Fb, np.float64), _ptr(Fa, np.float64),
                                  _stream(W, S, Q, Z))
    if status != JARQ_OK:
        raise JarqError(status, "jarq_fit_scales")
    return Fb, Fa


def multicode_probe(hess: Hessian, W, S, Q, Z, bits: int, group: int):
    """``jarq_multicode_probe``: dict of q_search [dout][g] (uint8), moves,
    accepted, changed (int32) and dF (float64) for one group of every row."""
    dout = int(W.shape[0])
    g = hess.group_size
    if _is_torch(W):
        import torch
        qs = torch.empty(dout, g, dtype=torch.uint8, device=W.device)
    else:
        qs = np.empty((dout, g), dtype=np.uint8)
    out = {"q_search": qs, "moves": _alloc_like(W, dout, np.int32),
           "accepted": _alloc_like(W, dout, np.int32), "changed": _alloc_like(W, dout, np.int32),
           "dF": _alloc_like(W, dout, np.float64)}
    status = _lib.jarq_multicode_probe(
        hess.handle, _ptr(W, np.float32), _ptr(S, np.float32), _ptr(Q, np.uint8),
        _ptr(Z, np.int32), dout, int(bits), int(group), _ptr(qs, np.uint8),
        _ptr(out["moves"], np.int32), _ptr(out["accepted"], np.int32),
        _ptr(out["changed"], np.int32), _ptr(out["dF"], np.float64), _stream(W, S, Q, Z))
    if status != JARQ_OK:
        raise JarqError(status, "jarq_multicode_probe")
    return out


def residual_product(hess: Hessian, W, S, Q, Z, bits: int, out=None):
    """``jarq_residual_product``: H r of every row (float32, dout x din), from
    the split-precision tensor-core kernel behind ``jarq_objective``."""
    dout, din = int(W.shape[0]), int(W.shape[1])
    if out is None:
        if _is_torch(W):
            import torch
            out = torch.empty(dout, din, dtype=torch.float32, device=W.device)
        else:
            out = np.empty((dout, din), dtype=np.float32)
    status = _lib.jarq_residual_product(hess.handle, _ptr(W, np.float32), _ptr(S, np.float32),
                                        _ptr(Q, np.uint8), _ptr(Z, np.int32), dout, int(bits),
                                        _ptr(out, np.float32), _stream(W, S, Q, Z))
    if status != JARQ_OK:
        raise JarqError(status, "jarq_residual_product")
    return out


JARQ_F32, JARQ_F16, JARQ_BF16 = 0, 1, 2


def _dev_stream(*ts):
    import torch
    return ctypes.c_void_p(torch.cuda.current_stream(ts[0].device).cuda_stream)


def canonicalize(S, Q, Z, group_size: int, bits: int):
    """``jarq_canonicalize``: negative scales to the equivalent positive form,
    in place on device tensors (S float32, Q uint8, Z int32)."""
    dout, din = int(Q.shape[0]), int(Q.shape[1])
    status = _lib.jarq_canonicalize(_ptr(S, np.float32), _ptr(Q, np.uint8), _ptr(Z, np.int32),
                                    dout, din, int(group_size), int(bits), _dev_stream(S))
    if status != JARQ_OK:
        raise JarqError(status, "jarq_canonicalize")


def dequantize(S, Q, Z, group_size: int, bits: int, dtype: str = "float16"):
    """``jarq_dequantize``: s (q - z) in float32, float16 or bfloat16 (device tensors)."""
    import torch
    code = {"float32": JARQ_F32, "float16": JARQ_F16, "bfloat16": JARQ_BF16}[dtype]
    tdt = {"float32": torch.float32, "float16": torch.float16, "bfloat16": torch.bfloat16}[dtype]
    dout, din = int(Q.shape[0]), int(Q.shape[1])
    out = torch.empty(dout, din, dtype=tdt, device=Q.device)
    status = _lib.jarq_dequantize(_ptr(S, np.float32), _ptr(Q, np.uint8), _ptr(Z, np.int32), dout,
                                  din, int(group_size), int(bits), code,
                                  ctypes.c_void_p(out.data_ptr()), _dev_stream(S))
    if status != JARQ_OK:
        raise JarqError(status, "jarq_dequantize")
    return out


def pack_codes(Q, bits: int):
    """``jarq_pack_codes``: b-bit codes packed per row (int32 storage of the
    uint32 words, [dout][ceil(din b / 32)])."""
    import torch
    dout, din = int(Q.shape[0]), int(Q.shape[1])
    nw = (din * int(bits) + 31) // 32
    out = torch.empty(dout, nw, dtype=torch.int32, device=Q.device)
    status = _lib.jarq_pack_codes(_ptr(Q, np.uint8), dout, din, int(bits),
                                  ctypes.c_void_p(out.data_ptr()), _dev_stream(Q))
    if status != JARQ_OK:
        raise JarqError(status, "jarq_pack_codes")
    return out


def accumulate_hessian(X, H=None, scale: float = 1.0):
    """``jarq_accumulate_hessian``: ``H + scale * X^T X`` for a float16 device
    tensor X [tokens][din]; H (float32 [din][din], device) is updated in place
    and returned (a zero matrix when H is None)."""
    import torch
    if not (_is_torch(X) and X.is_cuda and X.dtype == torch.float16 and X.is_contiguous()):
        raise TypeError("X must be a contiguous float16 CUDA tensor [tokens][din]")
    n, d = int(X.shape[0]), int(X.shape[1])
    if H is None:
        H = torch.zeros(d, d, dtype=torch.float32, device=X.device)
    status = _lib.jarq_accumulate_hessian(ctypes.c_void_p(X.data_ptr()), n, d, float(scale),
                                          _ptr(H, np.float32), _dev_stream(X))
    if status != JARQ_OK:
        raise JarqError(status, "jarq_accumulate_hessian")
    return H


def objective(hess: Hessian, W, S, Q, Z, bits: int, out=None):
    """``jarq_objective``: per-row F_j as float64."""
    dout = int(W.shape[0])
    F = out if out is not None else _alloc_like(W, dout, np.float64)
    status = _lib.jarq_objective(hess.handle, _ptr(W, np.float32), _ptr(S, np.float32),
                                 _ptr(Q, np.uint8), _ptr(Z, np.int32), dout, int(bits),
                                 _ptr(F, np.float64), _stream(W, S, Q, Z))
    if status != JARQ_OK:
        raise JarqError(status, "jarq_objective")
    return F
