"""Tensor-level convenience wrapper over the C ABI.

``NormPre`` keeps one library handle for a fixed list of matrices and turns
lists of torch tensors into the pointer arrays the ABI takes (and the current
CUDA stream into its ``stream`` argument).  It does no arithmetic of its own.
"""
from __future__ import annotations

from typing import List, Optional, Sequence

import numpy as np

from . import normpre as C

_DT = {"f32": C.NORMPRE_F32, "bf16": C.NORMPRE_BF16}


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.float32:
        return C.NORMPRE_F32
    if t.dtype == torch.bfloat16:
        return C.NORMPRE_BF16
    raise TypeError("unsupported dtype %s (float32 or bfloat16)" % t.dtype)


def _ptr_check(t):
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return t.data_ptr()


class NormPre:
    """One optimizer-step plan for a fixed list of 2-D matrices."""

    def __init__(self, shapes: Sequence, w_dtypes: Sequence, g_dtypes: Sequence, **config):
        self.cfg = C.normpre_default_config(**config)
        self.shapes = [(int(r), int(c)) for r, c in shapes]
        wd = [_DT[d] if isinstance(d, str) else int(d) for d in w_dtypes]
        gd = [_DT[d] if isinstance(d, str) else int(d) for d in g_dtypes]
        self.handle = C.normpre_init(self.cfg, self.shapes, wd, gd)

    @classmethod
    def for_tensors(cls, W: Sequence, G: Sequence, **config) -> "NormPre":
        return cls([tuple(w.shape) for w in W], [_dtype_code(w) for w in W],
                   [_dtype_code(g) for g in G], **config)

    def step(self, t: int, lr: float, W: Sequence, G: Sequence, M: Sequence, stream=None) -> None:
        import torch
        s = stream if stream is not None else torch.cuda.current_stream()
        C.normpre_step(self.handle, t, lr, [_ptr_check(x) for x in W], [_ptr_check(x) for x in G],
                       [_ptr_check(x) for x in M], s.cuda_stream)

    def step_host(self, t: int, lr: float, W: Sequence, G: Sequence, M: Sequence, stream=None) -> None:
        """Host tensors in, host tensors out (copies are part of the call)."""
        import torch
        s = stream if stream is not None else torch.cuda.current_stream()
        C.normpre_step_host(self.handle, t, lr, [_ptr_check(x) for x in W], [_ptr_check(x) for x in G],
                            [_ptr_check(x) for x in M], s.cuda_stream)

    def status(self, stream=None, raise_on_error: bool = True) -> int:
        import torch
        s = stream if stream is not None else torch.cuda.current_stream()
        return C.normpre_sync_status(self.handle, s.cuda_stream, raise_on_error)

    def read(self, mat: int, what: int) -> np.ndarray:
        """Copy a buffer of the last step to host memory as float32."""
        r, c, d = C.normpre_buffer_info(self.handle, mat, what)
        if d == C.NORMPRE_BF16:
            raw = np.empty((r, c), dtype=np.uint16)
            C.normpre_read(self.handle, mat, what, raw.ctypes.data, raw.nbytes)
            return (raw.astype(np.uint32) << 16).view(np.float32)
        out = np.empty((r, c), dtype=np.float32)
        C.normpre_read(self.handle, mat, what, out.ctypes.data, out.nbytes)
        return out

    def close(self) -> None:
        if self.handle:
            C.normpre_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def newton_schulz(X, **config):
    """Stand-alone Newton-Schulz on a [batch, rows, cols] (or [rows, cols]) CUDA tensor."""
    import torch
    cfg = C.normpre_default_config(**config)
    x = X if X.dim() == 3 else X.unsqueeze(0)
    x = x.contiguous()
    want = torch.bfloat16 if cfg.precision == C.NORMPRE_PREC_BF16 else torch.float32
    if x.dtype != want:
        raise TypeError("precision %d needs %s input" % (cfg.precision, want))
    T = torch.empty_like(x)
    C.normpre_newton_schulz(cfg, x.shape[0], x.shape[1], x.shape[2], x.data_ptr(), T.data_ptr(),
                            torch.cuda.current_stream().cuda_stream)
    return T if X.dim() == 3 else T[0]
