"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these tests compares the oracle with itself: each checks a closed
form, an invariant, a special case that reduces to a textbook routine (SVD,
symmetric eigendecomposition), a published known-answer value, or brute force
on tiny inputs.  CPU only.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle as O

GOLD = os.path.join(os.path.dirname(__file__), "golden")

# Muon's published quintic, typed here independently of the oracle's constant.
A_COEF, B_COEF, C_COEF = 3.4445, -4.7750, 2.0315


def _rng(s):
    return np.random.default_rng(s)


# ---------------------------------------------------------------------------
# Philox4x32-10 and the Gaussian sketch matrix (Algorithm 2, Omega sample)
# ---------------------------------------------------------------------------
def test_philox_known_answers():
    kat = json.load(open(os.path.join(GOLD, "philox4x32_10_kat.json")))
    for v in kat["vectors"]:
        ctr = tuple(np.array([int(x, 16)], dtype=np.uint64) for x in v["ctr"])
        key = tuple(int(x, 16) for x in v["key"])
        out = O.philox4x32_10(ctr, key)
        assert ["%08x" % int(w[0]) for w in out] == v["out"]


def test_philox_uniform_is_open_interval_and_exact():
    x = np.array([0, 511, 512, 0xFFFFFFFF], dtype=np.uint32)
    u = O.philox_uniform(x)
    assert u[0] == 2.0 ** -24 and u[1] == u[0]
    assert u[2] == 3.0 * 2.0 ** -24
    assert u[3] == 1.0 - 2.0 ** -24
    assert np.all((u > 0) & (u < 1))
    # odd multiples of 2^-24 below 1 have <= 24 significant bits: exact in fp32
    xs = np.random.default_rng(0).integers(0, 2 ** 32, 100000, dtype=np.uint64).astype(np.uint32)
    us = O.philox_uniform(xs)
    assert np.all(us.astype(np.float32).astype(np.float64) == us)


def test_omega_counter_layout():
    """Element e of Omega uses block e // 4 with counter (block, id, t_lo, t_hi)."""
    seed, mid, t = 0x1234_5678_9ABC_DEF0, 5, (3 << 32) + 7
    om = O.sketch_omega(seed, mid, t, 6, 10)          # 60 elements, 15 blocks
    blk = 9
    ctr = tuple(np.array([c], dtype=np.uint64) for c in (blk, mid, 7, 3))
    words = O.philox4x32_10(ctr, (0x9ABCDEF0, 0x12345678))
    u = [O.philox_uniform(w)[0] for w in words]
    z = [math.sqrt(-2 * math.log(u[0])) * math.cos(2 * math.pi * u[1]),
         math.sqrt(-2 * math.log(u[0])) * math.sin(2 * math.pi * u[1]),
         math.sqrt(-2 * math.log(u[2])) * math.cos(2 * math.pi * u[3]),
         math.sqrt(-2 * math.log(u[2])) * math.sin(2 * math.pi * u[3])]
    flat = om.reshape(-1)
    np.testing.assert_allclose(flat[36:40], z, rtol=0, atol=1e-15)
    # a different step or matrix gives an independent stream
    assert not np.allclose(om, O.sketch_omega(seed, mid, t + 1, 6, 10))
    assert not np.allclose(om, O.sketch_omega(seed, mid + 1, t, 6, 10))


def test_omega_is_standard_normal():
    from scipy import stats
    z = O.sketch_omega(42, 0, 0, 20000, 10).reshape(-1)
    assert abs(z.mean()) < 0.01
    assert abs(z.var() - 1) < 0.01
    assert abs(stats.skew(z)) < 0.03
    assert abs(stats.kurtosis(z)) < 0.06
    assert stats.kstest(z, "norm").pvalue > 1e-3


# ---------------------------------------------------------------------------
# Momentum, relaxed tangent momentum, diagonal-Gram normalization (Alg. 1, Eq. 3)
# ---------------------------------------------------------------------------
def test_hand_worked_2x3_both_orientations():
    """A 2x3 example worked by hand from Algorithm 1 with mu = 1/2."""
    W = np.array([[1.0, 0, 0], [0, 2.0, 0]])
    Mp = np.array([[2.0, 0, 0], [0, 0, 2.0]])
    G = np.array([[0, 3.0, 0], [1.0, 0, 0]])
    M = O.momentum_update(Mp, G, 0.5)
    np.testing.assert_array_equal(M, [[1, 3, 0], [1, 0, 1]])
    # row-active: row0 m=(1,3,0), w=(1,0,0): <m,w>=1, x=(0,3,0);
    #             row1 m=(1,0,1), w=(0,2,0): <m,w>=0, x=(1,0,1)
    X = O.relaxed_tangent(O.orient(M, 0), O.orient(W, 0))
    np.testing.assert_array_equal(X, [[0, 3, 0], [1, 0, 1]])
    Psi, d = O.diag_gram_normalize(X)
    np.testing.assert_allclose(d, [3, math.sqrt(2)], rtol=1e-15)
    r = 1 / math.sqrt(2)
    np.testing.assert_allclose(Psi, [[0, 1, 0], [r, 0, r]], rtol=0, atol=1e-16)
    # column-active: columns of M (1,1),(3,0),(0,1); of W (1,0),(0,2),(0,0)
    #   c0: a=1 -> x=(0,1); c1: a=0 -> x=(3,0); c2: w=0 -> x=(0,1)
    X1 = O.relaxed_tangent(O.orient(M, 1), O.orient(W, 1))
    np.testing.assert_array_equal(X1, [[0, 1], [3, 0], [0, 1]])
    Psi1, _ = O.diag_gram_normalize(X1)
    np.testing.assert_array_equal(Psi1, [[0, 1], [1, 0], [0, 1]])


def test_orientation_parity():
    assert [O.orientation_of(t) for t in range(5)] == [0, 1, 0, 1, 0]
    assert O.orientation_of(3, mode=1) == 0 and O.orientation_of(2, mode=2) == 1


def test_tangent_decomposition_identity():
    """x = g_tan + (1 - ||w||^2) g_rad and ||x||^2 = ||g||^2 [sin^2 + (1-||w||^2)^2 cos^2]
    (App. D.2, relaxed tangent gradient and Lemma 1)."""
    rng = _rng(1)
    g = rng.standard_normal((7, 40))
    w = rng.standard_normal((7, 40)) * rng.uniform(0.1, 2.0, (7, 1)) / math.sqrt(40)
    x = O.relaxed_tangent(g, w)
    wn2 = (w * w).sum(1, keepdims=True)
    g_rad = (g * w).sum(1, keepdims=True) / wn2 * w
    g_tan = g - g_rad
    np.testing.assert_allclose(x, g_tan + (1 - wn2) * g_rad, rtol=1e-12, atol=1e-12)
    cos2 = (g * w).sum(1) ** 2 / ((g * g).sum(1) * wn2[:, 0])
    lhs = (x * x).sum(1)
    rhs = (g * g).sum(1) * ((1 - cos2) + (1 - wn2[:, 0]) ** 2 * cos2)
    np.testing.assert_allclose(lhs, rhs, rtol=1e-11)


def test_tangent_special_cases():
    rng = _rng(2)
    g = rng.standard_normal((5, 30))
    # W = 0: x = m
    np.testing.assert_array_equal(O.relaxed_tangent(g, np.zeros_like(g)), g)
    # unit-norm rows: strict tangent projection, x orthogonal to w
    w = rng.standard_normal((5, 30))
    w /= np.linalg.norm(w, axis=1, keepdims=True)
    x = O.relaxed_tangent(g, w)
    np.testing.assert_allclose((x * w).sum(1), 0, atol=1e-13)


def test_normalize_unit_rows_and_inner_product():
    """Gamma_ii = 1 (Sec. 2.2) and <X, Psi>_F = sum_i ||x_i|| (Lemma 1)."""
    X = _rng(3).standard_normal((9, 33)) * np.exp(_rng(4).standard_normal((9, 1)))
    Psi, d = O.diag_gram_normalize(X)
    np.testing.assert_allclose(np.diag(Psi @ Psi.T), 1, rtol=1e-14)
    np.testing.assert_allclose((X * Psi).sum(), np.linalg.norm(X, axis=1).sum(), rtol=1e-13)
    # D(X) is the square root of the Gram diagonal
    np.testing.assert_allclose(d ** 2, np.diag(X @ X.T), rtol=1e-13)


def test_normalize_zero_row_reading():
    X = _rng(5).standard_normal((4, 8))
    X[2] = 0
    Psi, d = O.diag_gram_normalize(X)
    assert d[2] == 0 and np.all(Psi[2] == 0)
    np.testing.assert_allclose(np.linalg.norm(Psi, axis=1)[[0, 1, 3]], 1, rtol=1e-14)


def test_extreme_scale_example():
    """Sec. 1: one row norm 1e4, the rest 1e-3, fixed directions.  The raw Gram's
    leading eigenvector is the big row's axis; Psi is scale-free."""
    g = json.load(open(os.path.join(GOLD, "extreme_scale.json")))
    rng = _rng(g["direction_seed"])
    base = rng.standard_normal(g["cols"])
    dirs = g["correlation"] * base + (1 - g["correlation"]) * rng.standard_normal((g["rows"], g["cols"]))
    dirs /= np.linalg.norm(dirs, axis=1, keepdims=True)
    norms = np.full(g["rows"], g["small_norm"])
    norms[g["big_row"]] = g["big_norm"]
    X = dirs * norms[:, None]
    lam, U = np.linalg.eigh(X @ X.T)
    lead = U[:, -1]
    assert abs(lead[g["big_row"]]) > 1 - 1e-9
    Psi, _ = O.diag_gram_normalize(X)
    Psi_eq, _ = O.diag_gram_normalize(dirs)
    np.testing.assert_allclose(Psi, Psi_eq, rtol=0, atol=1e-14)
    # after normalization the correlated rows dominate the leading mode
    lamG, UG = np.linalg.eigh(Psi @ Psi.T)
    assert abs(UG[g["big_row"], -1]) < 0.6


def test_step_invariant_to_row_rescaling():
    """With M_{t-1} = 0 and a row-active step, positive per-row rescaling of G
    leaves Psi, T and the weight update unchanged (A3 is linear per row, Eq. 3
    divides the scale out).  Column rescaling plays the same role for k = 1."""
    rng = _rng(6)
    m, n = 12, 40
    W = rng.standard_normal((m, n)) * 0.05
    G = rng.standard_normal((m, n))
    Z = np.zeros((m, n))
    s_row = np.exp(2 * rng.standard_normal((m, 1)))
    s_col = np.exp(2 * rng.standard_normal((1, n)))
    for variant in ("G", "L"):
        cfg = O.OracleConfig(variant=variant, rank=4, oversample=3)
        a = O.normpre_step(W, G, Z, 0, 1e-2, cfg)
        b = O.normpre_step(W, G * s_row, Z, 0, 1e-2, cfg)
        np.testing.assert_allclose(b["Psi"], a["Psi"], atol=1e-13)
        np.testing.assert_allclose(b["W"], a["W"], atol=1e-12)
        a1 = O.normpre_step(W, G, Z, 1, 1e-2, cfg)
        b1 = O.normpre_step(W, G * s_col, Z, 1, 1e-2, cfg)
        np.testing.assert_allclose(b1["W"], a1["W"], atol=1e-12)
    # and the overall momentum scale has no effect
    cfgG = O.OracleConfig(variant="G")
    Mp = rng.standard_normal((m, n))
    a = O.normpre_step(W, G, Mp, 0, 1e-2, cfgG)
    b = O.normpre_step(W, 3.0 * G, 3.0 * Mp, 0, 1e-2, cfgG)
    np.testing.assert_allclose(b["W"], a["W"], atol=1e-12)


def test_orientation_is_transpose_symmetric():
    """A column-active step on W is the row-active step on W^T, transposed."""
    rng = _rng(7)
    W = rng.standard_normal((10, 24)) * 0.05
    G = rng.standard_normal((10, 24))
    Mp = rng.standard_normal((10, 24))
    for variant in ("G", "L_exact"):
        cfg = O.OracleConfig(variant=variant, rank=5)
        col = O.normpre_step(W, G, Mp, 1, 1e-2, cfg)
        row_t = O.normpre_step(W.T, G.T, Mp.T, 0, 1e-2, cfg)
        np.testing.assert_allclose(col["W"], row_t["W"].T, atol=1e-13)
        np.testing.assert_allclose(col["Psi"], row_t["Psi"], atol=1e-14)


# ---------------------------------------------------------------------------
# NormPre-G: Newton-Schulz (Sec. 3.2, App. B/C)
# ---------------------------------------------------------------------------
def _scalar_quintic(x, steps):
    for _ in range(steps):
        x = A_COEF * x + B_COEF * x ** 3 + C_COEF * x ** 5
    return x


@pytest.mark.parametrize("shape", [(16, 48), (48, 16), (20, 20), (1, 9)])
def test_ns_singular_value_map(shape):
    """NS acts on each singular value alone: svd(NS_q(Psi)) = p^q(sigma/||Psi||_F)
    with the singular vectors of Psi (checked with an independent SVD)."""
    rng = _rng(8)
    X = rng.standard_normal(shape) * np.exp(rng.standard_normal((shape[0], 1)))
    Psi, _ = O.diag_gram_normalize(X)
    T = O.newton_schulz(Psi, 5, eps=0.0)
    U, s, Vt = np.linalg.svd(Psi, full_matrices=False)
    expect = U @ np.diag(_scalar_quintic(s / np.linalg.norm(Psi), 5)) @ Vt
    np.testing.assert_allclose(T, expect, atol=1e-12)


def test_ns_band_of_the_polynomial():
    """After 5 quintic steps every singular value from [sigma_min/||Psi||, 1] lands in
    the band the scalar map implies (Muon's quintic oscillates around ~0.7-1.2)."""
    rng = _rng(9)
    Psi, _ = O.diag_gram_normalize(rng.standard_normal((64, 256)))
    s_in = np.linalg.svd(Psi, compute_uv=False) / np.linalg.norm(Psi)
    grid = np.linspace(s_in.min(), 1.0, 20001)
    band = _scalar_quintic(grid, 5)
    s_out = np.linalg.svd(O.newton_schulz(Psi, 5, eps=0.0), compute_uv=False)
    assert s_out.min() >= band.min() - 1e-9 and s_out.max() <= band.max() + 1e-9
    assert 0.6 < s_out.min() and s_out.max() < 1.25


def test_cubic_ns_converges_to_polar_factor():
    """With the classical cubic (1.5, -0.5, 0) iterated to convergence, NS gives
    msign(Psi) = U V^T (Sec. 2.1), which has ||T||_F^2 = min(m, n)."""
    rng = _rng(10)
    Psi, _ = O.diag_gram_normalize(rng.standard_normal((12, 30)))
    T = O.newton_schulz(Psi, 80, coef=(1.5, -0.5, 0.0), eps=0.0)
    U, s, Vt = np.linalg.svd(Psi, full_matrices=False)
    np.testing.assert_allclose(T, U @ Vt, atol=1e-10)
    assert abs((T * T).sum() - 12) < 1e-9


def test_ns_transpose_rule():
    rng = _rng(11)
    Psi = rng.standard_normal((40, 12))
    np.testing.assert_allclose(O.newton_schulz(Psi), O.newton_schulz(Psi.T).T, atol=1e-13)


def test_orthogonal_rows_are_fixed_points():
    """App. A.3: orthogonal rows normalize to Gamma = I; msign(Psi) = Psi and the
    localized preconditioner selects nothing (T = Psi)."""
    g = json.load(open(os.path.join(GOLD, "orthogonal_rows.json")))
    Qm, _ = np.linalg.qr(_rng(12).standard_normal((g["cols"], g["rows"])))
    X = Qm.T * np.array(g["row_norms"])[:, None]
    Psi, _ = O.diag_gram_normalize(X)
    np.testing.assert_allclose(Psi @ Psi.T, np.eye(g["rows"]), atol=1e-14)
    ex = O.exact_interaction_eigs(Psi, r=32)
    # every eigenvalue is one (up to rounding, which may put some a few ulps above
    # the strict lam > 1 cut; such a mode is scaled by lam^{-1/2} - 1 ~ 1e-16)
    np.testing.assert_allclose(ex["lam"], 1.0, atol=1e-14)
    np.testing.assert_allclose(O.localized_apply(Psi, ex["U_C"], ex["lam_C"]), Psi, atol=1e-14)
    T = O.newton_schulz(Psi, 80, coef=(1.5, -0.5, 0.0), eps=0.0)
    np.testing.assert_allclose(T, Psi, atol=1e-12)


# ---------------------------------------------------------------------------
# NormPre-L: Props. 1-2, Algorithm 2 (App. B, App. D.1)
# ---------------------------------------------------------------------------
def _psi(m, n, seed, corr=0.0):
    rng = _rng(seed)
    X = rng.standard_normal((m, n)) + corr * rng.standard_normal((1, n))
    X *= np.exp(rng.standard_normal((m, 1)))
    return O.diag_gram_normalize(X)[0]


def test_prop1_clipped_singular_values():
    """r >= |A|: sigma_i(T) = min(sigma_i(Psi), 1) with Psi's singular vectors (Prop. 1)."""
    Psi = _psi(10, 30, 13, corr=0.6)
    ex = O.exact_interaction_eigs(Psi, r=10)
    T = O.localized_apply(Psi, ex["U_C"], ex["lam_C"])
    U, s, Vt = np.linalg.svd(Psi, full_matrices=False)
    np.testing.assert_allclose(T, U @ np.diag(np.minimum(s, 1.0)) @ Vt, atol=1e-12)
    # and T_+ is the projection of Psi onto the unit spectral ball: nearest
    # feasible point beats random feasible perturbations
    base = np.linalg.norm(T - Psi)
    rng = _rng(14)
    for _ in range(20):
        D = rng.standard_normal(T.shape) * 1e-3
        Tp = T + D
        Tp /= max(1.0, np.linalg.norm(Tp, 2))
        assert np.linalg.norm(Tp - Psi) >= base - 1e-12


def test_prop2_rank_budget_and_trace_identity():
    """r < |A|: singular values are 1 on the r largest active modes and unchanged
    elsewhere (Prop. 2); ||T||_F^2 = m - sum_C (lam_i - 1) and eig(P) in (0, 1]
    (Lemma 2)."""
    Psi = _psi(30, 40, 15, corr=0.0)
    U, s, Vt = np.linalg.svd(Psi, full_matrices=False)
    n_act = int((s ** 2 > 1).sum())
    assert n_act >= 3
    r = n_act - 1
    ex = O.exact_interaction_eigs(Psi, r=r)
    assert ex["n_active"] == r
    T = O.localized_apply(Psi, ex["U_C"], ex["lam_C"])
    s_exp = s.copy()
    s_exp[:r] = 1.0
    np.testing.assert_allclose(T, U @ np.diag(s_exp) @ Vt, atol=1e-12)
    m = Psi.shape[0]
    assert abs((T * T).sum() - (m - (ex["lam_C"] - 1).sum())) < 1e-11
    P = np.eye(m) + ex["U_C"] @ np.diag(ex["lam_C"] ** -0.5 - 1) @ ex["U_C"].T
    ev = np.linalg.eigvalsh(P)
    assert ev.min() > 0 and ev.max() <= 1 + 1e-12


def test_sketch_full_width_equals_exact():
    """l = m: the sketch spans the whole row space, Rayleigh-Ritz is exact."""
    Psi = _psi(10, 50, 16, corr=0.7)
    om = O.sketch_omega(3, 0, 0, 50, 10)
    sk = O.interaction_sketch(Psi, r=6, o=8, p=1, Omega=om)
    assert sk["ell"] == 10
    ex = O.exact_interaction_eigs(Psi, r=6)
    assert sk["n_active"] == ex["n_active"]
    np.testing.assert_allclose(sk["lam_C"], ex["lam_C"], rtol=1e-12)
    P1 = sk["U_C"] @ sk["U_C"].T
    P2 = ex["U_C"] @ ex["U_C"].T
    np.testing.assert_allclose(P1, P2, atol=1e-10)


def test_sketch_recovers_exact_low_rank():
    """Rank-rho Psi with rho <= l: the Gaussian sketch captures range(Psi) and the
    Ritz pairs are the exact eigenpairs (Halko et al. 2011)."""
    rng = _rng(17)
    m, n, rho = 60, 200, 5
    X = rng.standard_normal((m, rho)) @ rng.standard_normal((rho, n))
    Psi, _ = O.diag_gram_normalize(X)
    sk = O.interaction_sketch(Psi, r=8, o=4, p=1, Omega=O.sketch_omega(1, 0, 0, n, 12))
    lam = np.linalg.eigvalsh(Psi @ Psi.T)[::-1]
    np.testing.assert_allclose(sk["ritz"][:rho], lam[:rho], rtol=1e-10)
    ex = O.exact_interaction_eigs(Psi, r=8)
    assert sk["n_active"] == ex["n_active"]
    np.testing.assert_allclose(sk["U_C"] @ sk["U_C"].T, ex["U_C"] @ ex["U_C"].T, atol=1e-9)


def test_sketch_ritz_values_interlace():
    """Rayleigh-Ritz values satisfy lam_hat_i <= lam_i (Cauchy interlacing), so the
    sketch never selects more modes than the exact preconditioner."""
    Psi = _psi(64, 128, 18, corr=0.5)
    lam = np.linalg.eigvalsh(Psi @ Psi.T)[::-1]
    for seed in range(4):
        sk = O.interaction_sketch(Psi, r=8, o=4, p=1, Omega=O.sketch_omega(seed, 0, 0, 128, 12))
        assert np.all(sk["ritz"] <= lam[:12] + 1e-12)
        assert sk["n_active"] <= O.exact_interaction_eigs(Psi, 8)["n_active"]


def test_sketch_basis_orthonormal_and_selection_order():
    Psi = _psi(40, 90, 19, corr=0.8)
    sk = O.interaction_sketch(Psi, r=5, o=6, p=1, Omega=O.sketch_omega(9, 2, 4, 90, 11))
    np.testing.assert_allclose(sk["Q"].T @ sk["Q"], np.eye(11), atol=1e-13)
    lam = sk["ritz"]
    assert np.all(np.diff(lam) <= 0)
    # top-r then lam > 1 equals active-then-top-r (App. B)
    active_then_top = lam[lam > 1][:5]
    np.testing.assert_array_equal(sk["lam_C"], active_then_top)


# ---------------------------------------------------------------------------
# Consistent update RMS and the weight update (Sec. 3.1, Algorithm 1)
# ---------------------------------------------------------------------------
def test_rms_matching_and_weight_update():
    rng = _rng(20)
    T = rng.standard_normal((8, 20))
    for k in (0, 1):
        Ta = T if k == 0 else T.T
        R = O.rms_matched(Ta, k, 0.2)
        assert R.shape == (8, 20)
        assert abs(np.sqrt((R * R).mean()) - 0.2) < 1e-15
        np.testing.assert_allclose(R / np.linalg.norm(R), T / np.linalg.norm(T), atol=1e-15)
    W = rng.standard_normal((8, 20))
    R = O.rms_matched(T, 0, 0.2)
    np.testing.assert_array_equal(O.weight_update(W, R, 0.0, 0.1), W)
    np.testing.assert_allclose(O.weight_update(W, R, 0.5, 0.1), W - 0.5 * R - 0.05 * W, rtol=1e-13, atol=1e-15)
    # zero update reading: only weight decay acts
    Z = O.rms_matched(np.zeros((8, 20)), 0, 0.2)
    assert np.all(Z == 0)


def test_full_step_shapes_and_rms():
    rng = _rng(21)
    for variant in ("G", "L", "L_exact"):
        cfg = O.OracleConfig(variant=variant, rank=4, oversample=4)
        for t in (0, 1):
            W = rng.standard_normal((16, 28)) * 0.02
            out = O.normpre_step(W, rng.standard_normal((16, 28)), np.zeros((16, 28)), t, 0.1, cfg)
            dW = (W - out["W"]) / 0.1 - 0.1 * W
            assert dW.shape == W.shape
            assert abs(np.sqrt((dW * dW).mean()) - 0.2) < 1e-12


# ---------------------------------------------------------------------------
# Muon baseline (the comparison optimizer of Sec. 4): momentum, Newton-Schulz
# on the momentum itself, RMS-matched update
# ---------------------------------------------------------------------------
def test_muon_reduces_to_normpre_g_on_unit_rows_and_zero_weight():
    # With W = 0 the relaxed tangent is the momentum itself, and when the
    # momentum already has unit rows the diagonal-Gram normalization is the
    # identity, so at a row-active step NormPre-G and Muon coincide.
    rng = _rng(30)
    G = rng.standard_normal((12, 40))
    G /= np.linalg.norm(G, axis=1, keepdims=True)
    W = np.zeros((12, 40))
    cfg = O.OracleConfig(variant="G")
    mu_out = O.muon_step(W, G, np.zeros_like(G), 0.05, cfg)
    np_out = O.normpre_step(W, G, np.zeros_like(G), 0, 0.05, cfg)
    np.testing.assert_allclose(mu_out["T"], np_out["T"], rtol=0, atol=1e-13)
    np.testing.assert_allclose(mu_out["W"], np_out["W"], rtol=0, atol=1e-15)


def test_muon_singular_values_follow_the_quintic_map():
    # T = U p^5(Sigma / ||M||_F) V^T for the momentum's own SVD (no
    # normalization in between), and the update RMS is the target.
    rng = _rng(31)
    G = rng.standard_normal((10, 30)) * np.exp(rng.standard_normal((10, 1)))
    Mp = rng.standard_normal((10, 30))
    cfg = O.OracleConfig(variant="G", momentum=0.9)
    out = O.muon_step(np.zeros((10, 30)), G, Mp, 0.1, cfg)
    M = 0.9 * Mp + G
    U, s, Vt = np.linalg.svd(M, full_matrices=False)
    x = s / (np.linalg.norm(M) + 1e-7)
    for _ in range(5):
        x = A_COEF * x + B_COEF * x ** 3 + C_COEF * x ** 5
    np.testing.assert_allclose(out["T"], (U * x) @ Vt, rtol=0, atol=1e-12)
    R = out["R"]
    assert abs(np.sqrt((R * R).mean()) - 0.2) < 1e-15
    # a tall momentum gives the transpose of its transpose's result
    out_t = O.muon_step(np.zeros((30, 10)), G.T, Mp.T, 0.1, cfg)
    np.testing.assert_allclose(out_t["T"], out["T"].T, rtol=0, atol=1e-13)


# ---------------------------------------------------------------------------
# Tangent ablations (Table 5a): strict projection and no tangent step
# ---------------------------------------------------------------------------
def test_strict_tangent_rows_are_orthogonal_to_the_weights():
    rng = _rng(40)
    M = rng.standard_normal((9, 25))
    W = rng.standard_normal((9, 25)) * np.exp(rng.standard_normal((9, 1)))
    W[3] = 0.0
    X = O.strict_tangent(M, W)
    # orthogonal to every nonzero weight row, equal to m on the zero row
    ip = np.einsum("ij,ij->i", X, W) / np.maximum(np.linalg.norm(W, axis=1), 1e-300)
    assert np.max(np.abs(np.delete(ip, 3))) < 1e-13
    np.testing.assert_array_equal(X[3], M[3])
    # m = x + (component along w), Pythagoras
    for i in (0, 5):
        u = W[i] / np.linalg.norm(W[i])
        np.testing.assert_allclose(M[i], X[i] + (M[i] @ u) * u, atol=1e-13)
        assert abs(M[i] @ M[i] - X[i] @ X[i] - (M[i] @ u) ** 2) < 1e-12


def test_tangent_modes_special_cases():
    rng = _rng(41)
    M = rng.standard_normal((6, 12))
    W = rng.standard_normal((6, 12))
    Wn = W / np.linalg.norm(W, axis=1, keepdims=True)
    # unit weight rows: strict == relaxed (Sec. 3.1)
    np.testing.assert_allclose(O.tangent_step(M, Wn, "strict"), O.tangent_step(M, Wn, "relaxed"), atol=1e-14)
    # no tangent step: the momentum itself
    np.testing.assert_array_equal(O.tangent_step(M, W, "none"), M)
    # strict is invariant to rescaling a weight row, relaxed is not
    S = W * np.arange(1, 7)[:, None]
    np.testing.assert_allclose(O.tangent_step(M, S, "strict"), O.tangent_step(M, W, "strict"), atol=1e-13)
    assert np.max(np.abs(O.tangent_step(M, S, "relaxed") - O.tangent_step(M, W, "relaxed"))) > 1e-3


def test_strict_tangent_of_a_parallel_row_is_zero():
    # a momentum row parallel to its weight row has no tangent component
    rng = _rng(42)
    W = rng.standard_normal((4, 7))
    M = W * np.array([[2.0], [-0.5], [0.0], [3.0]])
    X = O.strict_tangent(M, W)
    assert np.all(X == 0.0)
    # one-element rows are always parallel
    X1 = O.strict_tangent(rng.standard_normal((5, 1)), rng.standard_normal((5, 1)))
    assert np.all(X1 == 0.0)


def test_strict_tangent_keeps_a_small_tangent_part():
    """Only exact parallelism zeroes a row: a momentum row whose tangent part is
    1e-6 or 1e-9 of its norm keeps exactly that part (the projection of Sec. 3.1
    is linear), and normalizes to the unit tangent direction (Eq. 3)."""
    rng = _rng(43)
    w = rng.standard_normal(300)
    v = rng.standard_normal(300)
    v -= (v @ w) / (w @ w) * w                 # tangent direction, orthogonal to w
    v /= np.linalg.norm(v)
    for eps in (1e-6, 1e-9):
        m = 2.5 * w / np.linalg.norm(w) + eps * 2.5 * v
        X = O.strict_tangent(m[None, :], w[None, :])
        np.testing.assert_allclose(X[0], eps * 2.5 * v, atol=1e-14, rtol=0)
        Psi, d = O.diag_gram_normalize(X)
        np.testing.assert_allclose(Psi[0], v, atol=1e-5 if eps == 1e-9 else 1e-8)
        assert d[0] > 0


# --------------------------------------------------------------------------
# Diagnostics (App. E)
# --------------------------------------------------------------------------
def test_spectral_energies_hand_worked():
    """lam = (4, 2.25, 1, 0.25, 0) with r = 1: C = {4} gives (2 - 1)^2 = 1;
    2.25 remains (0.5^2); lam = 1 contributes nothing; 0.25 gives (0.5 - 1)^2;
    the zero eigenvalue is not a mode."""
    e = O.spectral_energies(np.array([0.25, 4.0, 0.0, 1.0, 2.25]), r=1)
    assert e["E_top"] == 1.0 and e["E_remain"] == 0.25 and e["E_sub"] == 0.25
    assert e["E_global"] == 1.5
    # r larger than the modes above one: everything above one is in C
    e = O.spectral_energies(np.array([4.0, 2.25, 0.25]), r=8)
    assert e["E_top"] == 1.25 and e["E_remain"] == 0.0


def test_spectral_energies_match_singular_values():
    """E_global = sum over the nonzero singular values of (sigma - 1)^2
    = ||Psi||_F^2 - 2 ||Psi||_* + rank(Psi), taken here from an SVD of Psi
    (the energies come from the eigenvalues of Psi Psi^T)."""
    rng = np.random.default_rng(5)
    Psi, _ = O.diag_gram_normalize(rng.standard_normal((24, 7)) @ rng.standard_normal((7, 40)))
    sv = np.linalg.svd(Psi, compute_uv=False)
    sv = sv[sv > 1e-8]
    want = np.sum(Psi ** 2) - 2 * sv.sum() + sv.size
    ex = O.exact_interaction_eigs(Psi, r=3)
    e = O.spectral_energies(ex["lam"], r=3)
    assert abs(e["E_global"] - want) < 1e-9 * max(1.0, want)
    assert abs(e["E_global"] - np.sum((sv - 1.0) ** 2)) < 1e-9 * max(1.0, want)
    # C holds the three largest singular values' modes (all above one here)
    assert np.all(sv[:3] > 1.0)
    assert abs(e["E_top"] - np.sum((sv[:3] - 1.0) ** 2)) < 1e-9


def test_descent_alignment_identities():
    rng = np.random.default_rng(6)
    G = rng.standard_normal((9, 13))
    assert abs(O.descent_alignment(G, G) - 1.0) < 1e-15
    assert abs(O.descent_alignment(G, -3.0 * G) + 1.0) < 1e-15
    H = rng.standard_normal((9, 13))
    H -= np.sum(G * H) / np.sum(G * G) * G          # orthogonal to G
    assert abs(O.descent_alignment(G, H)) < 1e-12
    # the RMS matching of Sec. 3.1 is a positive scale: it leaves the cosine
    T = rng.standard_normal((13, 9))
    R = O.rms_matched(T, 1, 0.2)
    assert abs(O.descent_alignment(G, R) - O.descent_alignment(G, T.T)) < 1e-12
    assert O.descent_alignment(G, np.zeros_like(G)) == 0.0


# --------------------------------------------------------------------------
# "Row+Column/Step" orientation ablation (Table 5b), the reading: rows, then columns
# --------------------------------------------------------------------------
def test_both_axes_normalize_rank_one_closed_form():
    """X = a b^T: the rows become sign(a_i) b / ||b||, then every column j is
    sign(a) sign(b_j) / sqrt(m)."""
    a = np.array([2.0, -0.5, 3.0, -1.0])
    b = np.array([0.3, -4.0, 1.5])
    Psi, _ = O.both_axes_normalize(np.outer(a, b))
    want = np.outer(np.sign(a), np.sign(b)) / np.sqrt(a.size)
    assert np.max(np.abs(Psi - want)) < 1e-15


def test_both_axes_normalize_fixed_point_and_zero_lines():
    rng = np.random.default_rng(7)
    P = np.eye(5)[rng.permutation(5)]
    D = np.diag(rng.uniform(0.5, 3.0, 5))
    Psi, _ = O.both_axes_normalize(D @ P)      # rows and columns already one-hot
    assert np.array_equal(Psi, P)
    X = rng.standard_normal((6, 9))
    X[2] = 0.0
    X[:, 4] = 0.0
    Psi, _ = O.both_axes_normalize(X)
    nc = np.linalg.norm(Psi, axis=0)
    assert np.all(Psi[2] == 0.0) and np.all(Psi[:, 4] == 0.0)
    assert np.allclose(np.delete(nc, 4), 1.0, atol=1e-14)
    # ||Psi||_F^2 = number of nonzero columns
    assert abs(np.sum(Psi ** 2) - 8) < 1e-12


def test_orientation_3_step_uses_rows():
    rng = np.random.default_rng(8)
    W = rng.standard_normal((5, 7)) * 0.1
    G = rng.standard_normal((5, 7))
    M = rng.standard_normal((5, 7))
    for t in (0, 1, 2):
        out = O.normpre_step(W, G, M, t, 0.01, O.OracleConfig(variant="G", orientation=3))
        assert out["k"] == 0
        assert np.allclose(np.linalg.norm(out["Psi"], axis=0), 1.0)


# ---------------------------------------------------------------------------
# Pure-bf16 storage of Psi (App. A: the Qwen3 runs train in pure BF16)
# ---------------------------------------------------------------------------
def test_round_to_bf16_hand_values():
    """Round to nearest, ties to even, on 8 significant bits (bf16 spacing
    2^-7 in [1, 2)), the fp32 exponent range with subnormals of 2^-133."""
    x = np.array([1.0, 1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, -(1 + 2.0 ** -8 + 2.0 ** -20), 1 + 2.0 ** -7 - 2.0 ** -30,
                  0.0, -0.0, 2.0 ** -130, 3 * 2.0 ** -134, 255.5 * 2.0 ** -7, 0.1])
    want = np.array([1.0, 1.0, 1 + 2.0 ** -6, -(1 + 2.0 ** -7), 1 + 2.0 ** -7,
                     0.0, -0.0, 2.0 ** -130, 2.0 ** -132, 2.0, 0.10009765625])
    got = O.round_to_bf16(x)
    assert np.array_equal(got, want)
    assert np.signbit(got[6])


def test_round_to_bf16_matches_the_library_conversion():
    """On fp32 inputs the rounding is torch's float32 -> bfloat16 conversion
    (round to nearest even), ties included."""
    torch = pytest.importorskip("torch")
    rng = _rng(77)
    bits = rng.integers(0, 2 ** 32, size=20000, dtype=np.uint64).astype(np.uint32)
    bits[:5000] = (bits[:5000] & np.uint32(0xFFFF0000)) | np.uint32(0x8000)   # exact ties
    bits[5000:6000] &= np.uint32(0x807FFFFF)                                   # subnormals
    x = bits.view(np.float32)
    x = x[np.isfinite(x) & (np.abs(x) < 3.0e38)]
    want = torch.from_numpy(x.copy()).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(O.round_to_bf16(x.astype(np.float64)), want)


def test_bf16_psi_storage_step():
    """With Psi stored in bf16 every Psi entry is a bf16 value within half a
    bf16 spacing of the exact Psi, and the update keeps its RMS of 0.2."""
    rng = _rng(31)
    for variant in ("G", "L"):
        for t in (0, 1):
            W = rng.standard_normal((24, 40)) * 0.02
            G = rng.standard_normal((24, 40))
            ex = O.normpre_step(W, G, np.zeros_like(W), t, 0.1, O.OracleConfig(variant=variant, rank=4, oversample=4))
            bf = O.normpre_step(W, G, np.zeros_like(W), t, 0.1,
                                O.OracleConfig(variant=variant, rank=4, oversample=4, psi_storage="bf16"))
            assert np.array_equal(O.round_to_bf16(bf["Psi"]), bf["Psi"])
            half = np.exp2(np.floor(np.log2(np.maximum(np.abs(ex["Psi"]), 2.0 ** -126))) - 8)
            assert np.all(np.abs(bf["Psi"] - ex["Psi"]) <= half)
            dW = (W - bf["W"]) / 0.1 - 0.1 * W
            assert abs(np.sqrt((dW * dW).mean()) - 0.2) < 1e-12
