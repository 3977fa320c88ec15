"""Plain, slow, fp64 reference of the NormPre per-matrix update step.

TEST INFRASTRUCTURE: this module exists to check the CUDA library.  It is
imported only by the tests, by ``__graft_entry__.smoke()`` and by the CPU
baseline legs of ``bench.py``.  It shares no code with the CUDA path and
imports nothing from it.

Everything here follows "Normalize-Then-Precondition" (NormPre) in the order
and notation of the paper, in float64, on the exact stored input values
(bf16 / fp32 inputs are widened to fp64 first):

    Algorithm 1       the optimizer step (momentum, orientation, relaxed
                      tangent momentum, diagonal-Gram normalization, spectral
                      preconditioning, consistent update RMS, weight decay)
    Eq. 3 (Sec. 2.2)  Psi = D(X)^{-1} X
    Sec. 2.3          global (msign) and localized spectral preconditioning
    Sec. 3.2          NormPre-G via the Newton-Schulz iteration of Muon,
                      NormPre-L via exact or sketched eigenspace extraction
    Algorithm 2       randomized interaction sketch (App. B)
    Prop. 1, Prop. 2  regularized / rank-constrained refinement (App. D.1)

Library primitives serve as single steps where the paper names the operation
(matrix products, ``qr``, a symmetric eigendecomposition); nothing is blocked,
fused or reordered beyond what the paper writes.

Readings taken where the paper is silent:

* Newton-Schulz polynomial: the paper defers to Muon's Newton-Schulz iteration
  with 5 steps and prints no coefficients.  We take Muon's published
  quintic X <- a X + b (X X^T) X + c (X X^T)^2 X with
  (a, b, c) = (3.4445, -4.7750, 2.0315), the input divided by
  (||X||_F + 1e-7), and the input transposed when rows > cols so that the
  Gram matrix is s x s (App. C).  The constants are parity-unpinned by the
  paper; the iteration structure is pinned by the singular-value map.
* ``t`` is the number of completed steps before this call; k_t = t mod 2.
* A zero active row (undefined in Eq. 3) gives a zero row of Psi.
* A zero preconditioned update gives a zero RMS-matched update (weight decay
  still applies).
* Sketch: Omega is drawn from Philox4x32-10 (Salmon et al., SC'11) keyed by the
  seed, with counter (element // 4, matrix id, t lo, t hi); uniforms
  ((x >> 9) + 0.5) 2^-23 (24 significant bits, so the same value in fp32 and
  fp64); normals by Box-Muller on word pairs (0,1), (2,3).
* Top-r selection: Ritz values sorted in descending order with a stable sort
  (ties keep the lower index), r' = min(r, l), then C = {i <= r' : lam_i > 1}.
* Spectral energies (App. E): "nonzero" eigenvalues are those above 1e-6 of
  the largest.
* "Row+Column/Step" (Table 5b): rows of the row-active tangent momentum
  normalized, then the columns of the result; preconditioning and the update
  in the row orientation.
* Pure-bf16 storage (App. A: the Qwen3 runs train in pure BF16): with
  ``psi_storage="bf16"`` the normalized Psi is rounded to bf16 (round to
  nearest, ties to even) once, before the spectral stage, and both the
  spectral stage and the update use the rounded Psi.  The default keeps Psi
  exact.
* Muon baseline (the comparison optimizer of Sec. 4 and App. A): the same
  momentum, the Newton-Schulz iteration applied to the momentum itself (no
  orientation, tangent or normalization step, Sec. 2.1), and the update
  RMS matched to the same target as NormPre (the Muon convention the paper
  follows in Sec. 3.1).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, Optional, Tuple

import numpy as np

# --------------------------------------------------------------------------
# Configuration (defaults from the paper's Table 4 / App. A)
# --------------------------------------------------------------------------
MUON_QUINTIC = (3.4445, -4.7750, 2.0315)


@dataclass
class OracleConfig:
    variant: str = "G"              # "G" (Newton-Schulz) or "L" (sketch) or "L_exact"
    momentum: float = 0.95          # mu
    weight_decay: float = 0.1       # lambda_wd
    target_rms: float = 0.2         # consistent update RMS
    ns_steps: int = 5               # q
    ns_coef: Tuple[float, float, float] = MUON_QUINTIC
    ns_eps: float = 1e-7
    rank: int = 32                  # r
    oversample: int = 8             # o
    power_iters: int = 1            # p
    seed: int = 0                   # Philox key for Omega
    orientation: int = 0            # 0 alternate (paper), 1 row only, 2 column only,
                                    # 3 rows then columns every step (Table 5b "Row+Column/Step")
    tangent: str = "relaxed"        # "relaxed" (paper), "strict" or "none" (Table 5a ablations)
    psi_storage: str = "exact"      # "exact", or "bf16": Psi rounded to bf16 (pure-bf16 training, App. A)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """x rounded to the nearest bf16 value (8 significant bits, the fp32
    exponent range with its subnormals), ties to even, returned as float64.
    The spacing of bf16 numbers at |x| in [2^e, 2^(e+1)) is 2^(e-7), and
    2^-133 below the smallest normal 2^-126; dividing by it is exact, so
    numpy's half-to-even rounding of the quotient is the rounding itself."""
    x = np.asarray(x, dtype=np.float64)
    ax = np.abs(x)
    e = np.floor(np.log2(np.where(ax > 0, ax, 1.0)))
    spacing = np.exp2(np.maximum(e, -126.0) - 7.0)
    return np.where(ax > 0, np.round(x / spacing) * spacing, x)


# --------------------------------------------------------------------------
# Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
# as 1, 2, 3", SC'11), written from the published round definition.
# --------------------------------------------------------------------------
_PHILOX_M0 = np.uint64(0xD2511F53)
_PHILOX_M1 = np.uint64(0xCD9E8D57)
_PHILOX_W0 = 0x9E3779B9
_PHILOX_W1 = 0xBB67AE85
_MASK32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(ctr, key):
    """Apply the 10-round Philox4x32 bijection.

    ctr: tuple of four uint32 arrays (broadcastable), key: tuple of two ints.
    Each round: (hi0, lo0) = M0 * c0, (hi1, lo1) = M1 * c2 (64-bit products),
    new state = (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0); the key is bumped by
    the Weyl constants (W0, W1) between rounds.
    """
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & _MASK32 for c in ctr)
    k0 = int(key[0]) & 0xFFFFFFFF
    k1 = int(key[1]) & 0xFFFFFFFF
    for rnd in range(10):
        p0 = _PHILOX_M0 * c0
        p1 = _PHILOX_M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = (hi1 ^ c1 ^ np.uint64(k0), lo1, hi0 ^ c3 ^ np.uint64(k1), lo0)
        k0 = (k0 + _PHILOX_W0) & 0xFFFFFFFF
        k1 = (k1 + _PHILOX_W1) & 0xFFFFFFFF
    return tuple(c.astype(np.uint32) for c in (c0, c1, c2, c3))


def philox_uniform(x: np.ndarray) -> np.ndarray:
    """uint32 -> uniform in (0, 1): ((x >> 9) + 0.5) * 2^-23.

    The result is an odd multiple of 2^-24 below 1, so it has at most 24
    significant bits and is exact in fp32 as well as fp64."""
    return ((x.astype(np.uint64) >> np.uint64(9)).astype(np.float64) + 0.5) * (2.0 ** -23)


def sketch_omega(seed: int, matrix_id: int, t: int, rows: int, ell: int) -> np.ndarray:
    """Gaussian test matrix Omega in R^{rows x ell}, Omega_ij ~ N(0,1) (Alg. 2).

    Element e = i*ell + j of the row-major matrix uses Philox counter
    (e // 4, matrix_id, t lo32, t hi32), key (seed lo32, seed hi32), word e % 4.
    Box-Muller on the word pair (2q, 2q+1) of the same block: the even word of
    the pair takes the cosine branch, the odd word the sine branch.
    """
    n = rows * ell
    nblk = (n + 3) // 4
    blk = np.arange(nblk, dtype=np.uint64)
    t = int(t) & 0xFFFFFFFFFFFFFFFF
    ctr = (blk, np.full(nblk, matrix_id & 0xFFFFFFFF, dtype=np.uint64),
           np.full(nblk, t & 0xFFFFFFFF, dtype=np.uint64),
           np.full(nblk, (t >> 32) & 0xFFFFFFFF, dtype=np.uint64))
    key = (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    x = philox4x32_10(ctr, key)
    u = [philox_uniform(w) for w in x]
    z = np.empty((nblk, 4), dtype=np.float64)
    for pair in range(2):
        ua, ub = u[2 * pair], u[2 * pair + 1]
        rad = np.sqrt(-2.0 * np.log(ua))
        z[:, 2 * pair] = rad * np.cos(2.0 * np.pi * ub)
        z[:, 2 * pair + 1] = rad * np.sin(2.0 * np.pi * ub)
    return z.reshape(-1)[:n].reshape(rows, ell)


# --------------------------------------------------------------------------
# Algorithm 1, step by step
# --------------------------------------------------------------------------
def momentum_update(M_prev: np.ndarray, G: np.ndarray, mu: float) -> np.ndarray:
    """M_t = mu M_{t-1} + G_t (Sec. 3.1, Algorithm 1)."""
    return mu * np.asarray(M_prev, dtype=np.float64) + np.asarray(G, dtype=np.float64)


def orientation_of(t: int, mode: int = 0) -> int:
    """k_t = t mod 2 (Sec. 3.1, alternating row/column orientation).

    mode 1 / 2 fix the orientation to rows / columns (the paper's row-only
    ablation and its column counterpart); mode 3 (both axes every step) works
    in the row orientation."""
    if mode in (1, 3):
        return 0
    if mode == 2:
        return 1
    return int(t) % 2


def orient(A: np.ndarray, k: int) -> np.ndarray:
    """O_0(A) = A, O_1(A) = A^T (Sec. 3.1)."""
    return A if k == 0 else A.T


def relaxed_tangent(Mbar: np.ndarray, Wbar: np.ndarray) -> np.ndarray:
    """x_i = m_i - <m_i, w_i> w_i for every active row (Sec. 3.1, relaxed tangent
    momentum; w_i is NOT normalized)."""
    a = np.einsum("ij,ij->i", Mbar, Wbar)
    return Mbar - a[:, None] * Wbar


def strict_tangent(Mbar: np.ndarray, Wbar: np.ndarray) -> np.ndarray:
    """x_i = m_i - <m_i, w_i> w_i / ||w_i||^2: the exact projection onto the
    tangent space of the row direction, which Sec. 3.1 says the relaxed form
    recovers when ||w_i|| = 1 (the "strict tangent" ablation of Table 5a).
    A zero weight row has no direction: x_i = m_i.
    A momentum row parallel to its weight row has no tangent component, and
    the fp64 subtraction leaves only rounding of it (about n * 2^-53 of
    ||m_i|| at most); a result at most 1e-12 of the momentum row's norm is
    taken as that exact zero (reading: only exact parallelism zeroes a row)."""
    a = np.einsum("ij,ij->i", Mbar, Wbar)
    ww = np.einsum("ij,ij->i", Wbar, Wbar)
    coef = np.divide(a, ww, out=np.zeros_like(a), where=ww > 0)
    X = Mbar - coef[:, None] * Wbar
    tiny = np.linalg.norm(X, axis=1) <= 1e-12 * np.linalg.norm(Mbar, axis=1)
    X[tiny] = 0.0
    return X


def tangent_step(Mbar: np.ndarray, Wbar: np.ndarray, mode: str = "relaxed") -> np.ndarray:
    """The momentum treatment before normalization: the paper's relaxed tangent,
    or the "strict tangent" / "no tangent" ablations (Table 5a)."""
    if mode == "relaxed":
        return relaxed_tangent(Mbar, Wbar)
    if mode == "strict":
        return strict_tangent(Mbar, Wbar)
    if mode == "none":
        return np.array(Mbar, dtype=np.float64, copy=True)
    raise ValueError(mode)


def diag_gram_normalize(X: np.ndarray):
    """Psi = D(X)^{-1} X with D(X) = Diag(||x_1||, ..., ||x_m||) (Eq. 3).

    Zero rows (where Eq. 3 is undefined) give zero rows.  Returns (Psi, d)."""
    d = np.sqrt(np.einsum("ij,ij->i", X, X))
    inv = np.zeros_like(d)
    nz = d > 0
    inv[nz] = 1.0 / d[nz]
    return X * inv[:, None], d


def both_axes_normalize(X: np.ndarray):
    """The "Row+Column/Step" ablation of Table 5b, read as: the rows of the
    (row-active) tangent momentum normalized as in Eq. 3, then the columns of
    the result normalized the same way (zero columns stay zero).  Returns
    (Psi, row norms)."""
    Psi, d = diag_gram_normalize(X)
    PsiT, _ = diag_gram_normalize(Psi.T)
    return PsiT.T, d


def newton_schulz(Psi: np.ndarray, steps: int = 5, coef=MUON_QUINTIC, eps: float = 1e-7) -> np.ndarray:
    """Approximate msign(Psi) by the Muon Newton-Schulz iteration (Sec. 3.2, App. B/C).

    The input is transposed when it has more rows than columns so that the
    Gram matrix is s x s with s = min(m, n); it is scaled to unit Frobenius
    norm (plus eps); then q times:  A = X X^T,  B = b A + c A A,  X = a X + B X.
    """
    a, b, c = (float(v) for v in coef)
    tall = Psi.shape[0] > Psi.shape[1]
    X = Psi.T if tall else Psi
    X = X / (np.linalg.norm(X) + eps)
    for _ in range(steps):
        A = X @ X.T
        B = b * A + c * (A @ A)
        X = a * X + B @ X
    return X.T if tall else X


def _descending(lam: np.ndarray, vecs: np.ndarray):
    order = np.argsort(-lam, kind="stable")
    return lam[order], vecs[:, order]


def interaction_sketch(Psi: np.ndarray, r: int, o: int, p: int, Omega: np.ndarray) -> Dict[str, np.ndarray]:
    """Randomized interaction sketch, Algorithm 2 (App. B).

    l = min(m, r + o); Y = Psi Omega; p times Y <- Psi (Psi^T Y); Q = qr(Y);
    Gamma_Q = (Q^T Psi)(Q^T Psi)^T; (Z, Lam) = top-r eigenpairs of Gamma_Q;
    U = Q Z; C = {i : lam_i > 1}.  Returns the selected (U_C, lam_C) plus the
    intermediates.
    """
    m, n = Psi.shape
    ell = min(m, r + o)
    assert Omega.shape == (n, ell), (Omega.shape, (n, ell))
    Y = Psi @ Omega
    for _ in range(p):
        Y = Psi @ (Psi.T @ Y)
    Q, _ = np.linalg.qr(Y, mode="reduced")
    B = Q.T @ Psi
    GammaQ = B @ B.T
    lam, Z = np.linalg.eigh(GammaQ)
    lam, Z = _descending(lam, Z)
    rr = min(r, ell)
    lam_r, Z_r = lam[:rr], Z[:, :rr]
    U = Q @ Z_r
    sel = lam_r > 1.0
    return {"ell": ell, "Y": Y, "Q": Q, "B": B, "GammaQ": GammaQ, "ritz": lam,
            "Z": Z_r, "U": U, "U_C": U[:, sel], "lam_C": lam_r[sel], "n_active": int(sel.sum())}


def exact_interaction_eigs(Psi: np.ndarray, r: int) -> Dict[str, np.ndarray]:
    """Exact eigenspace extraction (Sec. 3.2, App. B): Gamma = Psi Psi^T, full
    symmetric eigendecomposition, A = {i : lam_i > 1}, C = the min(r, |A|)
    largest active eigenvalues."""
    Gamma = Psi @ Psi.T
    lam, U = np.linalg.eigh(Gamma)
    lam, U = _descending(lam, U)
    active = lam > 1.0
    n_act = int(active.sum())
    nc = min(r, n_act)
    return {"Gamma": Gamma, "lam": lam, "U": U, "U_C": U[:, :nc], "lam_C": lam[:nc],
            "n_active_all": n_act, "n_active": nc}


def localized_apply(Psi: np.ndarray, U_C: np.ndarray, lam_C: np.ndarray) -> np.ndarray:
    """T = P^L Psi = Psi + U_C (Lam_C^{-1/2} - I) U_C^T Psi (Sec. 2.3, Algorithm 1)."""
    if U_C.shape[1] == 0:
        return Psi.copy()
    scale = lam_C ** -0.5 - 1.0
    return Psi + U_C @ (scale[:, None] * (U_C.T @ Psi))


def rms_matched(T_active: np.ndarray, k: int, target_rms: float) -> np.ndarray:
    """R_k(T) = target * O_k^{-1}(T) / RMS(T), RMS(T) = ||T||_F / sqrt(mn) (Sec. 3.1).

    A zero T gives a zero update."""
    Ts = orient(T_active, k)           # O_k^{-1} = O_k (transpose is an involution)
    m, n = Ts.shape
    nrm = np.linalg.norm(Ts)
    if nrm == 0.0:
        return np.zeros_like(Ts)
    return target_rms * Ts * (np.sqrt(m * n) / nrm)


def weight_update(W: np.ndarray, R: np.ndarray, lr: float, wd: float) -> np.ndarray:
    """W_{t+1} = W_t - eta_t (R_k(T_t) + lambda_wd W_t) (Algorithm 1)."""
    W = np.asarray(W, dtype=np.float64)
    return W - lr * (R + wd * W)


def normpre_step(W: np.ndarray, G: np.ndarray, M_prev: np.ndarray, t: int, lr: float,
                 cfg: OracleConfig, matrix_id: int = 0,
                 Omega: Optional[np.ndarray] = None) -> Dict[str, np.ndarray]:
    """One NormPre step for one matrix (Algorithm 1), returning every intermediate."""
    W = np.asarray(W, dtype=np.float64)
    M = momentum_update(M_prev, G, cfg.momentum)
    k = orientation_of(t, cfg.orientation)
    Wbar, Mbar = orient(W, k), orient(M, k)
    X = tangent_step(Mbar, Wbar, cfg.tangent)
    if cfg.orientation == 3:
        Psi, d = both_axes_normalize(X)
    else:
        Psi, d = diag_gram_normalize(X)
    if cfg.psi_storage == "bf16":
        Psi = round_to_bf16(Psi)
    elif cfg.psi_storage != "exact":
        raise ValueError(cfg.psi_storage)
    out = {"M": M, "k": k, "X": X, "Psi": Psi, "d": d}
    if cfg.variant == "G":
        T = newton_schulz(Psi, cfg.ns_steps, cfg.ns_coef, cfg.ns_eps)
    elif cfg.variant == "L":
        m_a, n_a = Psi.shape
        ell = min(m_a, cfg.rank + cfg.oversample)
        if Omega is None:
            Omega = sketch_omega(cfg.seed, matrix_id, t, n_a, ell)
        sk = interaction_sketch(Psi, cfg.rank, cfg.oversample, cfg.power_iters, Omega)
        T = localized_apply(Psi, sk["U_C"], sk["lam_C"])
        out.update({"Omega": Omega, "sketch": sk})
    elif cfg.variant == "L_exact":
        ex = exact_interaction_eigs(Psi, cfg.rank)
        T = localized_apply(Psi, ex["U_C"], ex["lam_C"])
        out.update({"exact": ex})
    else:
        raise ValueError(cfg.variant)
    R = rms_matched(T, k, cfg.target_rms)
    out.update({"T": T, "R": R, "W": weight_update(W, R, lr, cfg.weight_decay)})
    return out


def muon_step(W: np.ndarray, G: np.ndarray, M_prev: np.ndarray, lr: float,
              cfg: OracleConfig) -> Dict[str, np.ndarray]:
    """One step of the Muon baseline for one matrix: M = mu M_prev + G; the
    update orthogonalizes M itself by the Newton-Schulz iteration (Sec. 2.1:
    Muon replaces the momentum by its nearest semi-orthogonal matrix); the
    update RMS is matched to the target (Sec. 3.1); decoupled weight decay as
    in Algorithm 1."""
    W = np.asarray(W, dtype=np.float64)
    M = momentum_update(M_prev, G, cfg.momentum)
    T = newton_schulz(M, cfg.ns_steps, cfg.ns_coef, cfg.ns_eps)
    R = rms_matched(T, 0, cfg.target_rms)
    return {"M": M, "T": T, "R": R, "W": weight_update(W, R, lr, cfg.weight_decay)}


# --------------------------------------------------------------------------
# Diagnostics (App. E: spectral dynamics and training dynamics)
# --------------------------------------------------------------------------
def spectral_energies(lam: np.ndarray, r: int, nonzero_rel: float = 1e-6) -> Dict[str, float]:
    """Spectral transformation energies of App. E: with the eigenvalues lam of
    Gamma = Psi Psi^T, each mode's energy is the squared change of its singular
    value under global preconditioning, e_i = (sqrt(lam_i) - 1)^2.  E_top sums
    over C (the at most r largest eigenvalues above one), E_remain over the
    other eigenvalues above one, E_sub over the nonzero ones below one;
    E_global is their sum.  "Nonzero" is read as lam_i > nonzero_rel * lam_max
    (the paper's exact zeros are rounding-level values in floating point)."""
    lam = np.sort(np.asarray(lam, dtype=np.float64))[::-1]
    e = (np.sqrt(np.maximum(lam, 0.0)) - 1.0) ** 2
    lmax = lam[0] if lam.size else 0.0
    above = lam > 1.0
    n_c = min(int(r), int(above.sum()))
    top = float(e[:n_c].sum())
    remain = float(e[n_c:][above[n_c:]].sum())
    sub_mask = (lam > nonzero_rel * lmax) & (lam < 1.0)
    sub = float(e[sub_mask].sum())
    return {"E_top": top, "E_remain": remain, "E_sub": sub, "E_global": top + remain + sub}


def descent_alignment(G: np.ndarray, Phi: np.ndarray) -> float:
    """Per-matrix descent alignment of App. E: the cosine similarity
    <G, Phi>_F / (||G||_F ||Phi||_F) of the gradient and the update direction
    before learning-rate scaling and without weight decay (the paper averages
    it over the matrices)."""
    G = np.asarray(G, dtype=np.float64)
    Phi = np.asarray(Phi, dtype=np.float64)
    den = np.linalg.norm(G) * np.linalg.norm(Phi)
    return float(np.sum(G * Phi) / den) if den > 0 else 0.0


__all__ = [
    "MUON_QUINTIC", "OracleConfig", "round_to_bf16", "philox4x32_10", "philox_uniform", "sketch_omega",
    "momentum_update", "orientation_of", "orient", "relaxed_tangent", "strict_tangent", "tangent_step",
    "diag_gram_normalize", "both_axes_normalize",
    "newton_schulz", "interaction_sketch", "exact_interaction_eigs",
    "localized_apply", "rms_matched", "weight_update", "normpre_step", "muon_step",
    "spectral_energies", "descent_alignment",
]
