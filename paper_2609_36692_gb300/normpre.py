"""Thin ctypes binding of the NormPre C ABI (``include/normpre.h``).

Every function here only marshals arguments to the entry point of the same
name in ``libnormpre.so``; all arithmetic of the optimizer step runs in the
library's CUDA kernels.  There is no fallback: if the library is missing or
cannot be loaded, importing the functions raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libnormpre.so")

# enums (mirror include/normpre.h)
NORMPRE_G, NORMPRE_L, NORMPRE_MUON, NORMPRE_L_EXACT = 0, 1, 2, 3
NORMPRE_F32, NORMPRE_BF16 = 0, 1
NORMPRE_PREC_BF16, NORMPRE_PREC_F32 = 0, 1
(NORMPRE_OK, NORMPRE_ERR_ARG, NORMPRE_ERR_SHAPE, NORMPRE_ERR_DTYPE, NORMPRE_ERR_ALIGN,
 NORMPRE_ERR_CUDA, NORMPRE_ERR_NONFINITE, NORMPRE_ERR_NUMERIC, NORMPRE_ERR_TIMEOUT,
 NORMPRE_ERR_UNAVAILABLE) = range(10)
(NORMPRE_BUF_PSI, NORMPRE_BUF_T, NORMPRE_BUF_Q, NORMPRE_BUF_RITZ, NORMPRE_BUF_Z,
 NORMPRE_BUF_OMEGA, NORMPRE_BUF_STATS, NORMPRE_BUF_EIGS, NORMPRE_BUF_DIAG) = range(9)

STATUS_NAMES = {0: "OK", 1: "ERR_ARG", 2: "ERR_SHAPE", 3: "ERR_DTYPE", 4: "ERR_ALIGN",
                5: "ERR_CUDA", 6: "ERR_NONFINITE", 7: "ERR_NUMERIC", 8: "ERR_TIMEOUT",
                9: "ERR_UNAVAILABLE"}


class normpre_config(ctypes.Structure):
    _fields_ = [
        ("variant", ctypes.c_int),
        ("momentum", ctypes.c_float),
        ("weight_decay", ctypes.c_float),
        ("target_rms", ctypes.c_float),
        ("ns_steps", ctypes.c_int),
        ("ns_coef", ctypes.c_float * 3),
        ("ns_eps", ctypes.c_float),
        ("rank", ctypes.c_int),
        ("oversample", ctypes.c_int),
        ("power_iters", ctypes.c_int),
        ("seed", ctypes.c_uint64),
        ("precision", ctypes.c_int),
        ("orientation", ctypes.c_int),
        ("tangent", ctypes.c_int),
        ("diagnostics", ctypes.c_int),
        ("jacobi_max_sweeps", ctypes.c_int),
        ("test_stall", ctypes.c_int),
    ]


class NormPreError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__("%s: %s" % (STATUS_NAMES.get(status, status), message))
        self.status = status


_lib: Optional[ctypes.CDLL] = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libnormpre.so (raises if it is absent: there is no fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError("libnormpre.so not found at %s; build it with "
                           "paper_2609_36692_gb300.build.build()" % path)
    lib = ctypes.CDLL(path)
    P = ctypes.c_void_p
    i64 = ctypes.c_int64
    lib.normpre_default_config.argtypes = [ctypes.POINTER(normpre_config)]
    lib.normpre_default_config.restype = None
    lib.normpre_init.argtypes = [ctypes.POINTER(normpre_config), ctypes.c_int, ctypes.POINTER(i64),
                                 ctypes.POINTER(i64), ctypes.POINTER(ctypes.c_int),
                                 ctypes.POINTER(ctypes.c_int), ctypes.POINTER(P)]
    lib.normpre_init.restype = ctypes.c_int
    for name in ("normpre_step", "normpre_step_host"):
        f = getattr(lib, name)
        f.argtypes = [P, i64, ctypes.c_float, ctypes.POINTER(P), ctypes.POINTER(P), ctypes.POINTER(P), P]
        f.restype = ctypes.c_int
    lib.normpre_sync_status.argtypes = [P, P]
    lib.normpre_sync_status.restype = ctypes.c_int
    lib.normpre_buffer_info.argtypes = [P, ctypes.c_int, ctypes.c_int, ctypes.POINTER(i64),
                                        ctypes.POINTER(i64), ctypes.POINTER(ctypes.c_int)]
    lib.normpre_buffer_info.restype = ctypes.c_int
    lib.normpre_read.argtypes = [P, ctypes.c_int, ctypes.c_int, P, i64]
    lib.normpre_read.restype = ctypes.c_int
    lib.normpre_newton_schulz.argtypes = [ctypes.POINTER(normpre_config), ctypes.c_int, i64, i64, P, P, P]
    lib.normpre_newton_schulz.restype = ctypes.c_int
    lib.normpre_profile.argtypes = [P, ctypes.c_int]
    lib.normpre_profile.restype = ctypes.c_int
    lib.normpre_profile_read.argtypes = [P, ctypes.c_int, ctypes.POINTER(ctypes.c_double),
                                         ctypes.POINTER(i64)]
    lib.normpre_profile_read.restype = ctypes.c_int
    lib.normpre_normalize_cols_noalloc.argtypes = [i64, i64, ctypes.c_float, P, ctypes.c_int, P, P,
                                                   ctypes.c_int, P, P]
    lib.normpre_normalize_cols_noalloc.restype = ctypes.c_int
    lib.normpre_sketch_omega.argtypes = [ctypes.c_uint64, ctypes.c_int, i64, i64, ctypes.c_int, P, P, P, P]
    lib.normpre_sketch_omega.restype = ctypes.c_int
    lib.normpre_free.argtypes = [P]
    lib.normpre_free.restype = None
    lib.normpre_last_error.argtypes = [P]
    lib.normpre_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(rc: int, handle=None):
    if rc != NORMPRE_OK:
        msg = load_library().normpre_last_error(handle)
        raise NormPreError(rc, msg.decode() if msg else "")
    return rc


def _ptrs(xs: Sequence[int]):
    arr = (ctypes.c_void_p * len(xs))()
    for i, p in enumerate(xs):
        arr[i] = p
    return arr


# --------------------------------------------------------------------------
# entry points (same names as the C ABI)
# --------------------------------------------------------------------------
def normpre_default_config(**overrides) -> normpre_config:
    cfg = normpre_config()
    load_library().normpre_default_config(ctypes.byref(cfg))
    for k, v in overrides.items():
        if k == "ns_coef":
            for i in range(3):
                cfg.ns_coef[i] = float(v[i])
        else:
            setattr(cfg, k, v)
    return cfg


def normpre_init(cfg: normpre_config, shapes: Sequence, w_dtypes: Sequence[int],
                 g_dtypes: Sequence[int]) -> int:
    n = len(shapes)
    rows = (ctypes.c_int64 * n)(*[int(s[0]) for s in shapes])
    cols = (ctypes.c_int64 * n)(*[int(s[1]) for s in shapes])
    wd = (ctypes.c_int * n)(*[int(d) for d in w_dtypes])
    gd = (ctypes.c_int * n)(*[int(d) for d in g_dtypes])
    h = ctypes.c_void_p()
    _check(load_library().normpre_init(ctypes.byref(cfg), n, rows, cols, wd, gd, ctypes.byref(h)))
    return h.value


def normpre_step(handle: int, t: int, lr: float, W: Sequence[int], G: Sequence[int],
                 M: Sequence[int], stream: int = 0) -> int:
    return _check(load_library().normpre_step(handle, int(t), float(lr), _ptrs(W), _ptrs(G), _ptrs(M),
                                              stream), handle)


def normpre_step_host(handle: int, t: int, lr: float, W: Sequence[int], G: Sequence[int],
                      M: Sequence[int], stream: int = 0) -> int:
    return _check(load_library().normpre_step_host(handle, int(t), float(lr), _ptrs(W), _ptrs(G),
                                                   _ptrs(M), stream), handle)


def normpre_sync_status(handle: int, stream: int = 0, raise_on_error: bool = True) -> int:
    rc = load_library().normpre_sync_status(handle, stream)
    return _check(rc, handle) if raise_on_error else rc


def normpre_buffer_info(handle: int, mat: int, what: int):
    r, c, d = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int()
    _check(load_library().normpre_buffer_info(handle, mat, what, ctypes.byref(r), ctypes.byref(c),
                                              ctypes.byref(d)), handle)
    return r.value, c.value, d.value


def normpre_read(handle: int, mat: int, what: int, dst_ptr: int, capacity_bytes: int) -> int:
    return _check(load_library().normpre_read(handle, mat, what, dst_ptr, int(capacity_bytes)), handle)


def normpre_newton_schulz(cfg: normpre_config, batch: int, rows: int, cols: int, X_ptr: int,
                          T_ptr: int, stream: int = 0) -> int:
    return _check(load_library().normpre_newton_schulz(ctypes.byref(cfg), int(batch), int(rows),
                                                       int(cols), X_ptr, T_ptr, stream))


PROFILE_CLASSES = ["normalize", "ns_gram", "ns_poly", "ns_update", "apply_g", "omega", "contract",
                   "qr", "eig", "apply_l", "prescale", "exact_sweeps", "exact_select"]


def normpre_profile(handle: int, enable: bool) -> int:
    return _check(load_library().normpre_profile(handle, 1 if enable else 0), handle)


def normpre_profile_read(handle: int):
    n = len(PROFILE_CLASSES)
    ms = (ctypes.c_double * n)()
    cnt = (ctypes.c_int64 * n)()
    _check(load_library().normpre_profile_read(handle, n, ms, cnt), handle)
    return {name: (ms[i], cnt[i]) for i, name in enumerate(PROFILE_CLASSES)}


def normpre_normalize_cols_noalloc(rows: int, cols: int, mu: float, G_ptr: int, g_dtype: int,
                                   M_ptr: int, W_ptr: int, w_dtype: int, Psi_ptr: int,
                                   stream: int = 0) -> int:
    return _check(load_library().normpre_normalize_cols_noalloc(
        int(rows), int(cols), float(mu), G_ptr, int(g_dtype), M_ptr, W_ptr, int(w_dtype), Psi_ptr,
        stream))


def normpre_sketch_omega(seed: int, matrix_id: int, t: int, n_a: int, l: int, omega_ptr: int,
                         words_ptr: int = 0, uniforms_ptr: int = 0, stream: int = 0) -> int:
    return _check(load_library().normpre_sketch_omega(int(seed), int(matrix_id), int(t), int(n_a), int(l),
                                                      omega_ptr, words_ptr or None, uniforms_ptr or None,
                                                      stream))


def normpre_free(handle: int) -> None:
    if handle:
        load_library().normpre_free(handle)


def normpre_last_error(handle=None) -> str:
    m = load_library().normpre_last_error(handle)
    return m.decode() if m else ""
