"""Shared helpers of the parity tests: upload seeded inputs, run the CUDA step
through the C ABI, run the oracle on the same inputs, and compare."""
from __future__ import annotations

import numpy as np

import oracle as O
from synth import inputs as S

F32 = np.float32


def f32(x) -> float:
    """The value a float argument of the C ABI actually carries."""
    return float(np.float32(x))


def oracle_config(variant: str, **kw) -> O.OracleConfig:
    """Oracle settings equal to what the library receives (fp32-rounded floats)."""
    base = dict(momentum=f32(0.95), weight_decay=f32(0.1), target_rms=f32(0.2),
                ns_coef=(f32(3.4445), f32(-4.7750), f32(2.0315)), ns_eps=f32(1e-7))
    base.update(kw)
    for k in ("momentum", "weight_decay", "target_rms", "ns_eps"):
        base[k] = f32(base[k])
    base["ns_coef"] = tuple(f32(c) for c in base["ns_coef"])
    return O.OracleConfig(variant=variant, **base)


def to_device(mats, g_dtype: str, w_dtype: str):
    import torch
    W, G, M = [], [], []
    for m in mats:
        w = torch.from_numpy(np.ascontiguousarray(m["W"])).cuda()
        g = torch.from_numpy(np.ascontiguousarray(m["G"])).cuda()
        W.append(w.to(torch.bfloat16) if w_dtype == "bf16" else w)
        G.append(g.to(torch.bfloat16) if g_dtype == "bf16" else g)
        M.append(torch.from_numpy(np.ascontiguousarray(m["M"])).cuda())
    return W, G, M


def to_host(t) -> np.ndarray:
    import torch
    return t.float().cpu().numpy() if t.dtype == torch.bfloat16 else t.cpu().numpy()


def rel_fro(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (nb if nb > 0 else 1.0))


def max_row_rel(psi_gpu, psi_ref) -> float:
    """max_ij |dPsi_ij| / ||psi_ref,i|| over nonzero reference rows (rows have unit norm)."""
    d = np.abs(np.asarray(psi_gpu, np.float64) - psi_ref)
    nrm = np.linalg.norm(psi_ref, axis=1)
    nz = nrm > 0
    out = float((d[nz].max(axis=1) / nrm[nz]).max()) if nz.any() else 0.0
    if (~nz).any():
        out = max(out, float(d[~nz].max()))
    return out


def principal_sine(U1, U2) -> float:
    """Largest principal-angle sine between span(U1) and span(U2)."""
    if U1.shape[1] == 0 and U2.shape[1] == 0:
        return 0.0
    if U1.shape[1] != U2.shape[1]:
        return 1.0
    Q1, _ = np.linalg.qr(np.asarray(U1, np.float64))
    Q2, _ = np.linalg.qr(np.asarray(U2, np.float64))
    s = np.linalg.svd(Q1.T @ Q2, compute_uv=False)
    return float(np.sqrt(max(0.0, 1.0 - min(s.min(), 1.0) ** 2)))


def ritz_gaps_ok(ritz, rank, tol=1e-3) -> bool:
    """True when the selection C is well separated: every Ritz value among the
    top min(r, l) is at least `tol` away from 1, and the r-th and (r+1)-th
    values differ by at least `tol`."""
    r = min(rank, len(ritz))
    top = np.asarray(ritz[:r], np.float64)
    if np.any(np.abs(top - 1.0) < tol):
        return False
    if r < len(ritz) and top[-1] > 1.0 and abs(ritz[r - 1] - ritz[r]) < tol:
        return False
    return True
