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


def _torch_optimizer_base():
    import torch
    return torch.optim.Optimizer


class NormPreOptimizer(_torch_optimizer_base()):
    """``torch.optim`` interface: NormPre (or Muon) on a set of 2-D CUDA matrices.

    The paper applies the matrix optimizer to the hidden attention and MLP
    weight matrices and leaves embeddings, norms and biases to AdamW; give
    those parameters to another optimizer.  Each parameter group gets one
    library plan for its matrices (fp32 or bf16 weights and gradients,
    contiguous); the momentum M is kept in fp32 in the optimizer state and the
    step counter t (number of completed steps) in the group.  ``lr`` is read
    from the group at every step, so learning-rate schedulers work as usual;
    the other hyperparameters are fixed per plan (a change rebuilds it).

    Hyperparameters (defaults are the paper's): lr, momentum=0.95,
    weight_decay=0.1 (decoupled, multiplied by lr), target_rms=0.2,
    variant="G" | "L" | "L_exact" | "muon", plus any other field of
    ``normpre_config`` (rank, oversample, power_iters, ns_steps, precision,
    orientation, tangent, seed, diagnostics).  ``check_status=True``
    synchronizes after every step to raise on device-detected errors.
    """

    _VARIANTS = {"G": C.NORMPRE_G, "L": C.NORMPRE_L, "muon": C.NORMPRE_MUON, "L_exact": C.NORMPRE_L_EXACT}
    _FIXED = ("momentum", "weight_decay", "target_rms", "variant", "config")

    def __init__(self, params, lr: float = 0.02, momentum: float = 0.95, weight_decay: float = 0.1,
                 target_rms: float = 0.2, variant: str = "G", check_status: bool = False, **config):
        if variant not in self._VARIANTS:
            raise ValueError("variant must be one of %s" % sorted(self._VARIANTS))
        defaults = dict(lr=lr, momentum=momentum, weight_decay=weight_decay, target_rms=target_rms,
                        variant=variant, config=dict(config))
        super().__init__(params, defaults)
        for group in self.param_groups:
            if len({p.device for p in group["params"]}) > 1:
                raise ValueError("the matrices of a parameter group must share one CUDA device")
            for p in group["params"]:
                if p.dim() != 2:
                    raise ValueError("NormPreOptimizer takes 2-D matrices only (got shape %s); give "
                                     "other parameters to another optimizer" % (tuple(p.shape),))
                if not p.is_cuda:
                    raise ValueError("NormPreOptimizer takes CUDA tensors")
                _dtype_code(p)
                if not p.is_contiguous():
                    raise ValueError("parameters must be contiguous")
            group.setdefault("t", 0)
        self.check_status = check_status
        self._plans = {}

    def _plan(self, gi: int, group, params):
        # a plan is fixed to its matrices, their weight and gradient dtypes and
        # the group's hyperparameters other than lr
        key = (tuple(id(p) for p in params), tuple((_dtype_code(p), _dtype_code(p.grad)) for p in params),
               tuple(repr(group[k]) for k in self._FIXED))
        plan = self._plans.get(gi)
        if plan is None or plan[0] != key:
            cfg = dict(group["config"])
            cfg.update(variant=self._VARIANTS[group["variant"]], momentum=group["momentum"],
                       weight_decay=group["weight_decay"], target_rms=group["target_rms"])
            if plan is not None:
                plan[1].close()
            plan = (key, NormPre.for_tensors(params, [p.grad for p in params], **cfg), params)
            self._plans[gi] = plan
        return plan[1]

    def step(self, closure=None):
        import torch
        loss = None
        if closure is not None:
            with torch.enable_grad():
                loss = closure()
        with torch.no_grad():
            for gi, group in enumerate(self.param_groups):
                params = [p for p in group["params"] if p.grad is not None]
                if not params:
                    continue
                for p in params:
                    if not p.grad.is_contiguous():
                        raise ValueError("gradients must be contiguous")
                    st = self.state[p]
                    if "momentum_buffer" not in st:
                        st["momentum_buffer"] = torch.zeros(p.shape, dtype=torch.float32, device=p.device)
                # the library works on the current device: make it the matrices'
                with torch.cuda.device(params[0].device):
                    plan = self._plan(gi, group, params)
                    plan.step(group["t"], float(group["lr"]), params, [p.grad for p in params],
                              [self.state[p]["momentum_buffer"] for p in params])
                    group["t"] += 1
                    if self.check_status:
                        plan.status()
        return loss

    def diagnostics(self):
        """Per matrix of the last step: NORMPRE_BUF_DIAG as a dict (spectral
        energies with variant "L_exact", descent alignment with
        diagnostics=1), plus the mean alignment over the matrices (App. E)."""
        import torch
        out, cos = {}, []
        for gi, (key, plan, params) in self._plans.items():
            with torch.cuda.device(params[0].device):
                plan.status()
            for i, p in enumerate(params):
                d = plan.read(i, C.NORMPRE_BUF_DIAG)[0]
                rec = dict(zip(("E_top", "E_remain", "E_sub", "E_global", "align", "grad_norm",
                                "update_norm", "grad_dot_update"), (float(x) for x in d)))
                out[p] = rec
                if np.isfinite(rec["align"]):
                    cos.append(rec["align"])
        return out, (float(np.mean(cos)) if cos else float("nan"))

    def __del__(self):
        for _, plan, _ in getattr(self, "_plans", {}).values():
            try:
                plan.close()
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
