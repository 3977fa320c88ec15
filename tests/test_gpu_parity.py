"""CUDA path vs the fp64 oracle, element by element, on the same seeded inputs.

Tolerances (stated by the workload and derived where it is silent):
  * momentum M_t: fp32 fma, one rounding: |dM| <= 2.5e-7 |M|.
  * normalization (fp32 Psi): max |dPsi_ij| / ||psi_i|| <= 1e-5.
  * Newton-Schulz T: relative Frobenius <= 2e-2 (bf16 operands, fp32
    accumulation) and <= 1e-4 in the fp32 parity mode.
  * NormPre-L: largest principal-angle sine between the selected Ritz
    subspaces <= 1e-3 (fp32), equal |C| whenever the Ritz values are >= 1e-3
    away from 1 and from the r-th/(r+1)-th cut.
  * weight update: the change W_{t+1} - W_t has relative Frobenius error within
    the tolerance of T (fp32 weights); bf16 weights are compared element by
    element with the oracle's W_{t+1}: within one bf16 ulp plus the update
    tolerance times (the element's own update + six times the update's
    root-mean-square); in aggregate, within the update tolerance plus half an
    ulp per element.
"""
import os

import numpy as np
import pytest

import oracle as O
from synth import inputs as S

from helpers import (f32, max_row_rel, oracle_config, principal_sine, rel_fro, ritz_gaps_ok,
                     to_device, to_host)

pytestmark = pytest.mark.gpu

LR = 0.02


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_36692_gb300 import build
    build.build()


def _normpre(shapes, w_dtypes, g_dtypes, **cfg):
    from paper_2609_36692_gb300.optim import NormPre
    return NormPre(shapes, w_dtypes, g_dtypes, **cfg)


def _run(cfgset: S.ParamSetConfig, t: int, variant: str, precision: int, indices=None,
         zero_weight=False, extra=None, lr=LR):
    """Run one library step on the whole set; return (opt, inputs, W_new, M_new)."""
    import torch
    from paper_2609_36692_gb300 import normpre as C
    if zero_weight:
        mats = [S.make_matrix(cfgset, i, zero_weight=True) for i in range(cfgset.n_mats)]
    else:
        mats = S.make_param_set(cfgset, workers=min(16, os.cpu_count() or 1))
    W, G, M = to_device(mats, cfgset.g_dtype, cfgset.w_dtype)
    kw = dict(variant={"G": C.NORMPRE_G, "L": C.NORMPRE_L, "muon": C.NORMPRE_MUON,
                       "L_exact": C.NORMPRE_L_EXACT}[variant], precision=precision,
              rank=cfgset.rank, oversample=cfgset.oversample, power_iters=cfgset.power_iters,
              seed=1234)
    kw.update(extra or {})
    opt = _normpre([(m.rows, m.cols) for m in cfgset.matrices], [cfgset.w_dtype] * cfgset.n_mats,
                   [cfgset.g_dtype] * cfgset.n_mats, **kw)
    opt.step(t, lr, W, G, M)
    torch.cuda.synchronize()
    opt.status()
    return opt, mats, [to_host(w) for w in W], [to_host(m) for m in M]


def _oracle(mats, i, t, variant, cfgset, lr=LR, **kw):
    oc = oracle_config(variant, rank=cfgset.rank, oversample=cfgset.oversample,
                       power_iters=cfgset.power_iters, seed=1234, **kw)
    m = mats[i]
    return O.normpre_step(m["W"], m["G"], m["M"], t, f32(lr), oc, matrix_id=i)


def bf16_ulp(x):
    """Spacing of bf16 numbers at |x| (8 significant bits)."""
    e = np.floor(np.log2(np.maximum(np.abs(x), 1e-38)))
    return 2.0 ** (e - 7)


def _stored(x, k):
    return x if k == 0 else x.T


SMALL = S.custom_config("small_mixed", [(128, 384), (128, 128), (128, 512), (512, 128)],
                        g_dtype="bf16", w_dtype="f32", row_sigma=1.0, col_sigma=1.0,
                        rank=8, oversample=8)
RAGGED = S.custom_config("ragged", [(50, 203), (203, 50), (1, 77), (77, 1), (33, 33)],
                         g_dtype="f32", w_dtype="f32", row_sigma=1.0, rank=4, oversample=4)
SINGLE = S.CONFIGS["single_256x1024"]
# odd sketch widths (l = 19 and 11): the Jacobi pads a zero row and column,
# the CholeskyQR rows are not float4-aligned
ODD = S.custom_config("odd_width", [(96, 160), (160, 96), (19, 300), (250, 11), (45, 45)],
                      g_dtype="f32", w_dtype="f32", row_sigma=1.0, col_sigma=1.0, rank=13, oversample=6)
# bf16 weights of even and odd widths and ragged row counts in the bf16 mode
RAGGED_BF16W = S.custom_config("ragged_bf16w", [(50, 202), (203, 50), (131, 130), (64, 77), (300, 256)],
                               g_dtype="bf16", w_dtype="bf16", row_sigma=1.0, col_sigma=1.0,
                               rank=4, oversample=4)
# tall column-active strips: clusters of 4, 8 and 12 CTAs (the last with a
# partial row block) and one matrix whose column count is not a multiple of 32
TALL = S.custom_config("tall_cols", [(1000, 40), (4100, 64), (6144, 32), (2056, 24)],
                       g_dtype="bf16", w_dtype="f32", row_sigma=1.0, col_sigma=1.0,
                       rank=4, oversample=4)


# ---------------------------------------------------------------------------
# momentum + relaxed tangent + normalization
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("cfgset", [SINGLE, SMALL, RAGGED, TALL], ids=lambda c: c.name)
@pytest.mark.parametrize("t", [0, 1])
@pytest.mark.parametrize("w_dtype", ["f32", "bf16"])
def test_normalize_and_momentum(cfgset, t, w_dtype):
    import dataclasses
    cs = dataclasses.replace(cfgset, w_dtype=w_dtype)
    opt, mats, W1, M1 = _run(cs, t, "L", precision=1)
    for i in range(cs.n_mats):
        ref = _oracle(mats, i, t, "L", cs)
        k = ref["k"]
        psi = opt.read(i, 0)   # NORMPRE_BUF_PSI
        assert max_row_rel(psi, _stored(ref["Psi"], k)) <= 1e-5, (cs.name, i)
        dm = np.abs(M1[i].astype(np.float64) - ref["M"])
        assert np.all(dm <= 2.5e-7 * np.abs(ref["M"]) + 1e-30), (cs.name, i, dm.max())
        st = opt.read(i, 6)[0]
        assert int(st[0]) == k and int(st[1]) == int((ref["d"] > 0).sum())


def _check_bf16_w(w_gpu, w_ref, dw_ref, tol, where, elem_tol=None):
    """bf16 weights: the device stores the bf16 rounding (RNE) of its fp32
    update.  Element by element, the stored value is within one bf16 ulp of the
    oracle's exact W_{t+1} plus that element's share of the update tolerance:
    the tolerance relative to the element's own update (the operand and output
    roundings of a bf16 product scale with the entry) plus 6 times the
    root-mean-square share (the error spread over the matrix).  In aggregate,
    the Frobenius error is within the update tolerance plus the half-ulp
    rounding of every element.  `elem_tol` (default `tol`) replaces the
    tolerance in the element-wise share."""
    w_gpu = np.asarray(w_gpu, np.float64)
    err = np.abs(w_gpu - w_ref)
    et = tol if elem_tol is None else elem_tol
    share = et * (np.abs(dw_ref) + 6.0 * np.sqrt(np.mean(dw_ref ** 2)))
    bound = bf16_ulp(w_ref) + share
    worst = int(np.argmax(err - bound))
    assert np.all(err <= bound), (where, worst, float(err.flat[worst]), float(bound.flat[worst]))
    assert np.linalg.norm(w_gpu - w_ref) <= tol * np.linalg.norm(dw_ref) + \
        np.linalg.norm(0.5 * bf16_ulp(w_ref)), where


# ---------------------------------------------------------------------------
# NormPre-G
# ---------------------------------------------------------------------------
def _check_g(cs, t, precision, tol_t, indices=None):
    from paper_2609_36692_gb300 import normpre as C
    opt, mats, W1, _ = _run(cs, t, "G", precision)
    idx = range(cs.n_mats) if indices is None else indices
    for i in idx:
        ref = _oracle(mats, i, t, "G", cs)
        T = opt.read(i, C.NORMPRE_BUF_T)
        err = rel_fro(T, _stored(ref["T"], ref["k"]))
        assert err <= tol_t, (cs.name, i, err)
        dW = W1[i].astype(np.float64) - mats[i]["W"]
        dW_ref = ref["W"] - mats[i]["W"]
        if cs.w_dtype == "f32":
            assert rel_fro(dW, dW_ref) <= tol_t, (cs.name, i)
        else:
            _check_bf16_w(W1[i], ref["W"], dW_ref, tol_t, (cs.name, i))
        st = opt.read(i, C.NORMPRE_BUF_STATS)[0]
        assert abs(st[2] - (ref["T"] ** 2).sum()) <= 4 * tol_t * (ref["T"] ** 2).sum()


@pytest.mark.parametrize("cfgset", [SINGLE, SMALL, RAGGED], ids=lambda c: c.name)
@pytest.mark.parametrize("t", [0, 1])
def test_g_fp32_mode(cfgset, t):
    _check_g(cfgset, t, precision=1, tol_t=1e-4)


@pytest.mark.parametrize("cfgset", [SINGLE, SMALL, RAGGED], ids=lambda c: c.name)
@pytest.mark.parametrize("t", [0, 1])
def test_g_bf16_tensor_cores(cfgset, t):
    _check_g(cfgset, t, precision=0, tol_t=2e-2)


@pytest.mark.parametrize("t", [0, 1])
def test_g_bf16_gpt2_full_size_sampled(t):
    """The full GPT-2 Small set in the launch configuration the bench times;
    one matrix of each shape is checked against the oracle."""
    cs = S.CONFIGS["gpt2_small_G"]
    _check_g(cs, t, precision=0, tol_t=2e-2, indices=[0, 1, 2, 3, 45, 46, 47])


@pytest.mark.slow
@pytest.mark.parametrize("t", [0, 1])
@pytest.mark.parametrize("name,indices", [("llama_1b", [0, 4, 6, 111]), ("qwen3_1p7b", [0, 1, 4, 6, 195])])
def test_g_bf16_large_sets_sampled(name, indices, t):
    """LLaMA ~1B (112 matrices) and Qwen3 ~1.7B (196 matrices, bf16 weights),
    full set on the GPU in the launch configuration the bench times, one matrix
    of each shape against the oracle, at both orientations."""
    _check_g(S.CONFIGS[name], t, precision=0, tol_t=2e-2, indices=indices)


# ---------------------------------------------------------------------------
# stand-alone Newton-Schulz: every GEMM phase in isolation
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("shape", [(2, 256, 1024), (3, 384, 128), (1, 128, 128), (2, 100, 300), (1, 300, 100)])
@pytest.mark.parametrize("coef,steps", [((0.0, 1.0, 0.0), 1), ((0.0, 0.0, 1.0), 1), ((1.0, 0.0, 0.0), 1),
                                        ((3.4445, -4.7750, 2.0315), 5)])
@pytest.mark.parametrize("precision", [0, 1])
def test_newton_schulz_phases(shape, coef, steps, precision):
    import torch
    from paper_2609_36692_gb300.optim import newton_schulz
    rng = np.random.default_rng(sum(shape) + steps)
    X = rng.standard_normal(shape).astype(np.float32)
    if precision == 0:
        X = S.round_to_bf16(X)
        xt = torch.from_numpy(X).cuda().to(torch.bfloat16)
    else:
        xt = torch.from_numpy(X).cuda()
    T = to_host(newton_schulz(xt, ns_steps=steps, ns_coef=coef, precision=precision))
    tol = 2e-2 if precision == 0 else 1e-4
    for b in range(shape[0]):
        ref = O.newton_schulz(X[b].astype(np.float64), steps, tuple(f32(c) for c in coef), f32(1e-7))
        assert rel_fro(T[b], ref) <= tol, (shape, coef, b, rel_fro(T[b], ref))


# ---------------------------------------------------------------------------
# NormPre-L
# ---------------------------------------------------------------------------
def _check_l(cs, t, indices=None, w_tol=2e-3):
    from paper_2609_36692_gb300 import normpre as C
    opt, mats, W1, _ = _run(cs, t, "L", precision=1)
    idx = range(cs.n_mats) if indices is None else indices
    n_checked = 0
    for i in idx:
        ref = _oracle(mats, i, t, "L", cs)
        sk = ref["sketch"]
        om = opt.read(i, C.NORMPRE_BUF_OMEGA)
        assert np.max(np.abs(om - ref["Omega"])) <= 1e-5 * (1 + np.abs(ref["Omega"]).max()), (cs.name, i)
        ritz = opt.read(i, C.NORMPRE_BUF_RITZ)[0]
        lam = sk["ritz"]
        assert np.max(np.abs(ritz - lam)) <= 1e-4 * max(1.0, lam[0]), (cs.name, i)
        st = opt.read(i, C.NORMPRE_BUF_STATS)[0]
        if ritz_gaps_ok(lam, cs.rank):
            nc = int(st[3])
            assert nc == sk["n_active"], (cs.name, i, nc, sk["n_active"])
            Q = opt.read(i, C.NORMPRE_BUF_Q)
            Z = opt.read(i, C.NORMPRE_BUF_Z)
            U = Q.astype(np.float64) @ Z[:, :nc].astype(np.float64)
            assert principal_sine(U, sk["U_C"]) <= 1e-3, (cs.name, i)
            n_checked += 1
        dW = W1[i].astype(np.float64) - mats[i]["W"]
        dW_ref = ref["W"] - mats[i]["W"]
        if cs.w_dtype == "f32":
            assert rel_fro(dW, dW_ref) <= w_tol, (cs.name, i, rel_fro(dW, dW_ref))
        else:
            _check_bf16_w(W1[i], ref["W"], dW_ref, w_tol, (cs.name, i))
    return n_checked


def _oracle_words(seed, mid, t, n):
    """The oracle's Philox words of elements 0..n-1 in the counter layout of the
    sketch (Alg. 2 "sample Omega"): element e takes word e mod 4 of block e / 4."""
    nblk = (n + 3) // 4
    blk = np.arange(nblk, dtype=np.uint64)
    full = lambda v: np.full(nblk, v & 0xFFFFFFFF, dtype=np.uint64)  # noqa: E731
    x = O.philox4x32_10((blk, full(mid), full(t), full(t >> 32)), (seed & 0xFFFFFFFF, seed >> 32))
    return np.stack(x, axis=1).reshape(-1)[:n]


@pytest.mark.parametrize("seed,mid,t,n_a,l", [(1234, 0, 0, 1024, 24), (0xDEADBEEFCAFE, 7, (1 << 33) + 5, 777, 40),
                                              (1, 195, 1, 6144, 40), (2 ** 64 - 1, 3, 12, 5, 3)])
def test_philox_stream_bit_exact(seed, mid, t, n_a, l):
    """The sketch's random stream on the GPU is the oracle's, bit for bit: the
    Philox4x32-10 words and their uniforms are compared exactly, the Box-Muller
    normals within libm rounding."""
    import torch
    from paper_2609_36692_gb300 import normpre as C
    om = torch.empty((n_a, l), dtype=torch.float32, device="cuda")
    words = torch.empty((n_a, l), dtype=torch.int32, device="cuda")
    uni = torch.empty((n_a, l), dtype=torch.float32, device="cuda")
    C.normpre_sketch_omega(seed, mid, t, n_a, l, om.data_ptr(), words.data_ptr(), uni.data_ptr(),
                           torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    w_gpu = words.cpu().numpy().view(np.uint32).reshape(-1)
    w_ref = _oracle_words(seed, mid, t, n_a * l)
    assert np.array_equal(w_gpu, w_ref)
    u_ref = O.philox_uniform(w_ref).astype(np.float32)
    assert np.array_equal(uni.cpu().numpy().reshape(-1).view(np.uint32), u_ref.view(np.uint32))
    ref = O.sketch_omega(seed, mid, t, n_a, l)
    assert np.max(np.abs(om.cpu().numpy() - ref)) <= 1e-5 * (1 + np.abs(ref).max())


@pytest.mark.parametrize("t", [0, 1])
def test_step_omega_is_the_stand_alone_stream(t):
    """The Omega a NormPre-L step draws for matrix i is, bit for bit, the
    stand-alone sketch matrix for (seed, i, t)."""
    import torch
    from paper_2609_36692_gb300 import normpre as C
    opt, mats, _, _ = _run(SMALL, t, "L", precision=1)
    for i in range(SMALL.n_mats):
        got = opt.read(i, C.NORMPRE_BUF_OMEGA)
        n_a, l = got.shape
        om = torch.empty((n_a, l), dtype=torch.float32, device="cuda")
        C.normpre_sketch_omega(1234, i, t, n_a, l, om.data_ptr(), 0, 0, torch.cuda.current_stream().cuda_stream)
        torch.cuda.synchronize()
        assert np.array_equal(got.view(np.uint32), om.cpu().numpy().view(np.uint32)), i
    opt.close()


@pytest.mark.parametrize("cfgset", [SINGLE, SMALL, RAGGED, ODD], ids=lambda c: c.name)
@pytest.mark.parametrize("t", [0, 1])
def test_l_sketch(cfgset, t):
    _check_l(cfgset, t)


@pytest.mark.parametrize("rank,oversample", [(26, 6), (44, 6), (52, 8)], ids=["l32", "l50", "l60"])
def test_l_sketch_widths(rank, oversample):
    """Sketch widths between the ones above: l = 32 and 60 take the tensor-core
    contraction (60: the widest panel, 64 + 64 columns per MMA), l = 50 the
    SIMT one; the CholeskyQR register widths 32, 56 and 64."""
    import dataclasses
    cs = dataclasses.replace(SMALL, rank=rank, oversample=oversample)
    _check_l(cs, 0)


@pytest.mark.parametrize("t", [0, 1])
def test_l_rank_deficient_sketch(t):
    """A rank-2 update with l = 8 (no tangent correction, no prior momentum):
    the sketch Y has rank 2, so the unshifted Cholesky pivots of its Gram
    matrix fall below 1e-6 tr and the first CholeskyQR pass takes its shifted
    retry.  The two selected Ritz directions, their values and the weight
    update still match the oracle (Householder QR), with no status raised."""
    import torch
    from paper_2609_36692_gb300 import normpre as C
    shapes = [(64, 96), (96, 64)]
    cs = S.custom_config("rank2", shapes, g_dtype="f32", w_dtype="f32", rank=4, oversample=4,
                         prior_momentum=False)
    mats = [S.make_matrix(cs, i) for i in range(len(shapes))]
    rng = np.random.default_rng(7)
    for m in mats:
        r, c = m["G"].shape
        m["G"][:] = (rng.standard_normal((r, 2)) @ rng.standard_normal((2, c))).astype(np.float32)
    W, G, M = to_device(mats, "f32", "f32")
    opt = _normpre(shapes, ["f32"] * 2, ["f32"] * 2, variant=C.NORMPRE_L, precision=1, rank=4,
                   oversample=4, seed=1234, tangent=_TANGENT["none"])
    opt.step(t, LR, W, G, M)
    torch.cuda.synchronize()
    assert opt.status() == C.NORMPRE_OK
    for i in range(len(shapes)):
        ref = _oracle(mats, i, t, "L", cs, tangent="none")
        sk = ref["sketch"]
        st = opt.read(i, C.NORMPRE_BUF_STATS)[0]
        assert int(st[3]) == sk["n_active"] == 2, (i, st[3], sk["n_active"])
        ritz = opt.read(i, C.NORMPRE_BUF_RITZ)[0]
        assert np.max(np.abs(ritz[:2] - sk["ritz"][:2])) <= 1e-4 * sk["ritz"][0], (i, ritz, sk["ritz"])
        Q = opt.read(i, C.NORMPRE_BUF_Q)
        Z = opt.read(i, C.NORMPRE_BUF_Z)
        U = Q.astype(np.float64) @ Z[:, :2].astype(np.float64)
        assert principal_sine(U, sk["U_C"]) <= 1e-3, i
        dW = to_host(W[i]).astype(np.float64) - mats[i]["W"]
        assert rel_fro(dW, ref["W"] - mats[i]["W"]) <= 2e-3, (i, rel_fro(dW, ref["W"] - mats[i]["W"]))


@pytest.mark.parametrize("t", [0, 1])
def test_l_gpt2_full_size_sampled(t):
    cs = S.CONFIGS["gpt2_small_L"]
    _check_l(cs, t, indices=[0, 1, 2, 3, 47])


@pytest.mark.slow
@pytest.mark.parametrize("t", [0, 1])
@pytest.mark.parametrize("name,indices", [("llama_1b", [0, 4, 6]), ("qwen3_1p7b", [0, 1, 4, 6])])
def test_l_large_sets_sampled(name, indices, t):
    """The full LLaMA ~1B and Qwen3 ~1.7B sets under NormPre-L (r = 32, o = 8,
    p = 1), one matrix of each shape against the oracle at both orientations;
    Qwen3's bf16 weights are compared element by element."""
    import dataclasses
    cs = dataclasses.replace(S.CONFIGS[name], rank=32, oversample=8)
    _check_l(cs, t, indices=indices)


# ---------------------------------------------------------------------------
# NormPre-L with Psi stored in bf16 (NORMPRE_PREC_BF16: the pure-bf16 setting
# of the paper's Qwen3 runs, App. A), against the oracle that rounds its exact
# Psi to bf16 once.  The library rounds its fp32 normalization (within 1e-5 of
# the line norm) once, so the two bf16 Psi agree except where the fp32 value
# fell across a rounding boundary: there they are one bf16 spacing apart.
# Those few one-spacing differences (~1% of the entries) perturb Psi by
# ~1e-4 of its norm, hence the looser sketch tolerances: Ritz values within
# 1e-3 of max(1, lam_1), subspaces within a principal-angle sine of 1e-2 where
# the selection is separated by 1e-2, the update within 3e-3 in aggregate.
# Element by element, a Psi entry one spacing off moves its entry of T by up to
# 2^-7 of itself, so bf16 weights take 2^-7 + 3e-3 as their element-wise share.
# ---------------------------------------------------------------------------
def _check_l_bf16(cs, t, indices=None, w_tol=3e-3):
    from paper_2609_36692_gb300 import normpre as C
    opt, mats, W1, _ = _run(cs, t, "L", precision=0)
    idx = range(cs.n_mats) if indices is None else indices
    for i in idx:
        ref = _oracle(mats, i, t, "L", cs, psi_storage="bf16")
        k = ref["k"]
        assert C.normpre_buffer_info(opt.handle, i, C.NORMPRE_BUF_PSI)[2] == C.NORMPRE_BF16
        psi = opt.read(i, C.NORMPRE_BUF_PSI).astype(np.float64)
        ref_psi = _stored(ref["Psi"], k)
        line = np.linalg.norm(ref_psi, axis=1 - k, keepdims=True)
        diff = np.abs(psi - ref_psi)
        assert np.all(diff <= bf16_ulp(ref_psi) + 1e-5 * line), (cs.name, i)
        assert np.mean(diff > 0) <= 0.05, (cs.name, i, np.mean(diff > 0))
        sk = ref["sketch"]
        ritz = opt.read(i, C.NORMPRE_BUF_RITZ)[0]
        lam = sk["ritz"]
        assert np.max(np.abs(ritz - lam)) <= 1e-3 * max(1.0, lam[0]), (cs.name, i)
        st = opt.read(i, C.NORMPRE_BUF_STATS)[0]
        if ritz_gaps_ok(lam, cs.rank, tol=1e-2 * max(1.0, lam[0])):
            nc = int(st[3])
            assert nc == sk["n_active"], (cs.name, i, nc, sk["n_active"])
            Q = opt.read(i, C.NORMPRE_BUF_Q)
            Z = opt.read(i, C.NORMPRE_BUF_Z)
            U = Q.astype(np.float64) @ Z[:, :nc].astype(np.float64)
            assert principal_sine(U, sk["U_C"]) <= 1e-2, (cs.name, i)
        dW = W1[i].astype(np.float64) - mats[i]["W"]
        dW_ref = ref["W"] - mats[i]["W"]
        if cs.w_dtype == "f32":
            assert rel_fro(dW, dW_ref) <= w_tol, (cs.name, i, rel_fro(dW, dW_ref))
        else:
            _check_bf16_w(W1[i], ref["W"], dW_ref, w_tol, (cs.name, i), elem_tol=2.0 ** -7 + w_tol)


@pytest.mark.parametrize("cfgset", [SINGLE, SMALL, RAGGED, ODD, TALL, RAGGED_BF16W], ids=lambda c: c.name)
@pytest.mark.parametrize("t", [0, 1])
def test_l_bf16_psi(cfgset, t):
    """Both contraction orientations of the bf16 kernel, ragged tiles and K
    blocks, odd sketch widths (l = 19, 11), tall strips, 1-wide matrices and
    bf16 weights of even and odd widths."""
    _check_l_bf16(cfgset, t)


@pytest.mark.parametrize("t", [0, 1])
@pytest.mark.parametrize("name,indices", [("gpt2_small_L", [0, 1, 2, 3, 47]), ("qwen3_1p7b", [0, 1, 4, 6])])
def test_l_bf16_psi_full_size_sampled(name, indices, t):
    """The GPT-2 and Qwen3 sets at full size in the bf16 mode (the Qwen3
    configuration the benchmark runs), one matrix of each shape checked."""
    import dataclasses
    cs = dataclasses.replace(S.CONFIGS[name], rank=32, oversample=8)
    _check_l_bf16(cs, t, indices=indices)


# ---------------------------------------------------------------------------
# ablation settings (Table 5): tangent treatment, fixed orientation, p >= 2
# ---------------------------------------------------------------------------
_TANGENT = {"relaxed": 0, "none": 1, "strict": 2}


@pytest.mark.parametrize("cfgset", [SMALL, RAGGED, TALL], ids=lambda c: c.name)
@pytest.mark.parametrize("t", [0, 1])
@pytest.mark.parametrize("mode", ["none", "strict"])
def test_tangent_ablation_normalization(cfgset, t, mode):
    opt, mats, W1, M1 = _run(cfgset, t, "L", precision=1, extra={"tangent": _TANGENT[mode]})
    for i in range(cfgset.n_mats):
        ref = _oracle(mats, i, t, "L", cfgset, tangent=mode)
        psi = opt.read(i, 0)   # NORMPRE_BUF_PSI, stored layout
        active = psi if ref["k"] == 0 else psi.T
        if mode == "strict":
            # every active row is either exactly parallel to its weight row (the
            # oracle's x_i vanishes to fp64 rounding; the kernels zero it at
            # their fp32 resolution, 1e-3 of ||m_i||) or keeps a tangent part
            # far above that resolution, so the comparison is well posed
            ratio = np.linalg.norm(ref["X"], axis=1) / np.maximum(
                np.linalg.norm(O.orient(ref["M"], ref["k"]), axis=1), 1e-300)
            assert np.all((ratio == 0.0) | (ratio > 1e-2)), (cfgset.name, i)
        # per normalized active row psi_i (Eq. 3): the strict projection cancels
        # part of m, so single small entries carry ~u ||m|| absolute error
        assert max_row_rel(active, ref["Psi"]) <= 1e-5, (cfgset.name, i, mode)


@pytest.mark.parametrize("t", [0, 1])
def test_strict_tangent_planted_parallel_rows(t):
    """Momentum rows (t = 0) or columns (t = 1) exactly parallel to their weight
    rows, over 384 / 1536 entries: the strict projection leaves no tangent part
    (Sec. 3.1, Table 5a), so those rows of Psi are zero and m' drops by their
    number; the other rows match the oracle per normalized row."""
    import torch
    from paper_2609_36692_gb300 import normpre as C
    rows, cols = 1536, 384
    cs = S.custom_config("planted_parallel", [(rows, cols)], g_dtype="f32", w_dtype="f32",
                         row_sigma=1.0, col_sigma=1.0, prior_momentum=False, rank=4, oversample=4)
    m = S.make_matrix(cs, 0)
    G, W = m["G"].copy(), m["W"].copy()
    picks = [3, 77, 200] if t == 0 else [5, 131, 383]
    for p in picks:
        # w = 2^-6 g (exact in fp32), and M_{t-1} = 0 there: m = g is exactly parallel to w
        if t == 0:
            W[p, :] = G[p, :] * np.float32(2.0 ** -6)
        else:
            W[:, p] = G[:, p] * np.float32(2.0 ** -6)
    mats = [{"G": G, "W": W, "M": m["M"]}]
    Wd, Gd, Md = to_device(mats, "f32", "f32")
    opt = _normpre([(rows, cols)], ["f32"], ["f32"], variant=C.NORMPRE_L, precision=1, rank=4,
                   oversample=4, seed=1234, tangent=_TANGENT["strict"])
    opt.step(t, LR, Wd, Gd, Md)
    torch.cuda.synchronize()
    opt.status()
    ref = _oracle(mats, 0, t, "L", cs, tangent="strict")
    assert np.all(ref["d"][picks] == 0.0)
    psi = opt.read(0, C.NORMPRE_BUF_PSI)
    active = psi if t == 0 else psi.T
    assert np.all(active[picks] == 0.0)
    assert max_row_rel(active, ref["Psi"]) <= 1e-5
    st = opt.read(0, C.NORMPRE_BUF_STATS)[0]
    assert int(st[1]) == int((ref["d"] > 0).sum()) == active.shape[0] - len(picks)
    opt.close()


@pytest.mark.parametrize("mode", ["none", "strict"])
@pytest.mark.parametrize("t", [0, 1])
def test_tangent_ablation_g_step(mode, t):
    from paper_2609_36692_gb300 import normpre as C
    opt, mats, W1, _ = _run(SMALL, t, "G", precision=1, extra={"tangent": _TANGENT[mode]})
    for i in range(SMALL.n_mats):
        ref = _oracle(mats, i, t, "G", SMALL, tangent=mode)
        assert rel_fro(opt.read(i, C.NORMPRE_BUF_T), _stored(ref["T"], ref["k"])) <= 1e-4, (i, mode)
        assert rel_fro(W1[i].astype(np.float64) - mats[i]["W"], ref["W"] - mats[i]["W"]) <= 1e-4, (i, mode)


@pytest.mark.parametrize("orientation", [1, 2, 3], ids=["rows_only", "columns_only", "rows_then_columns"])
@pytest.mark.parametrize("variant", ["G", "L"])
def test_fixed_orientation(orientation, variant):
    # t = 1 would be column-active under the alternating default
    from paper_2609_36692_gb300 import normpre as C
    opt, mats, W1, _ = _run(SMALL, 1, variant, precision=1, extra={"orientation": orientation})
    for i in range(SMALL.n_mats):
        ref = _oracle(mats, i, 1, variant, SMALL, orientation=orientation)
        assert ref["k"] == (1 if orientation == 2 else 0)
        st = opt.read(i, C.NORMPRE_BUF_STATS)[0]
        assert int(st[0]) == ref["k"]
        if orientation == 3:
            # Psi has unit columns; ||Psi||_F^2 (stats m') = number of nonzero columns
            psi = opt.read(i, C.NORMPRE_BUF_PSI).astype(np.float64)
            assert np.max(np.abs(psi - ref["Psi"])) <= 1e-5, (i, variant)
            assert int(st[1]) == int(np.sum(np.linalg.norm(ref["Psi"], axis=0) > 0))
        dW = W1[i].astype(np.float64) - mats[i]["W"]
        dW_ref = ref["W"] - mats[i]["W"]
        assert rel_fro(dW, dW_ref) <= (1e-4 if variant == "G" else 2e-3), (i, variant)


@pytest.mark.parametrize("t", [0, 1])
def test_rank_64(t):
    """Table 6's largest rank budget: r = 64 with o = 8 (l = 72, beyond the
    tensor-core contraction's l <= 64: the SIMT kernel takes it)."""
    import dataclasses
    cs = dataclasses.replace(SMALL, rank=64, oversample=8)
    _check_l(cs, t)


def test_rank_64_exact():
    import dataclasses
    from paper_2609_36692_gb300 import normpre as C
    cs = dataclasses.replace(SMALL, rank=64, oversample=0)
    opt, mats, W1, _ = _run(cs, 0, "L_exact", precision=1)
    for i in range(cs.n_mats):
        ref = _oracle(mats, i, 0, "L_exact", cs)
        st = opt.read(i, C.NORMPRE_BUF_STATS)[0]
        if ritz_gaps_ok(ref["exact"]["lam"], cs.rank):
            assert int(st[3]) == ref["exact"]["n_active"]
        dW = W1[i].astype(np.float64) - mats[i]["W"]
        assert rel_fro(dW, ref["W"] - mats[i]["W"]) <= 2e-3, i


def test_two_power_iterations():
    import dataclasses
    cs = dataclasses.replace(SMALL, power_iters=2)
    _check_l(cs, 0)
    _check_l(cs, 1)


# ---------------------------------------------------------------------------
# Muon baseline (the paper's comparison optimizer) on the same kernels
# ---------------------------------------------------------------------------
def _check_muon(cs, t, precision, tol, indices=None):
    from paper_2609_36692_gb300 import normpre as C
    opt, mats, W1, M1 = _run(cs, t, "muon", precision)
    idx = range(cs.n_mats) if indices is None else indices
    for i in idx:
        m = mats[i]
        ref = O.muon_step(m["W"], m["G"], m["M"], f32(LR), oracle_config("G"))
        dm = np.abs(M1[i].astype(np.float64) - ref["M"])
        assert np.all(dm <= 2.5e-7 * np.abs(ref["M"]) + 1e-30), (cs.name, i, dm.max())
        T = opt.read(i, C.NORMPRE_BUF_T)
        assert rel_fro(T, ref["T"]) <= tol, (cs.name, i, rel_fro(T, ref["T"]))
        dW = W1[i].astype(np.float64) - m["W"]
        dW_ref = ref["W"] - m["W"]
        if cs.w_dtype == "f32":
            assert rel_fro(dW, dW_ref) <= tol, (cs.name, i)
        else:
            half_ulp = 0.5 * bf16_ulp(ref["W"])
            err = np.linalg.norm(W1[i].astype(np.float64) - ref["W"])
            assert err <= tol * np.linalg.norm(dW_ref) + np.linalg.norm(half_ulp), (cs.name, i)
        st = opt.read(i, C.NORMPRE_BUF_STATS)[0]
        assert abs(st[2] - (ref["T"] ** 2).sum()) <= 4 * tol * (ref["T"] ** 2).sum()


@pytest.mark.parametrize("cfgset", [SINGLE, SMALL, RAGGED], ids=lambda c: c.name)
@pytest.mark.parametrize("t", [0, 1])
@pytest.mark.parametrize("precision,tol", [(1, 1e-4), (0, 2e-2)], ids=["fp32", "bf16"])
def test_muon_baseline(cfgset, t, precision, tol):
    _check_muon(cfgset, t, precision, tol)


def test_muon_gpt2_full_size_sampled():
    _check_muon(S.CONFIGS["gpt2_small_G"], 0, 0, 2e-2, indices=[0, 1, 2, 3, 47])


# ---------------------------------------------------------------------------
# edge cases and device status
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("variant", ["G", "L"])
def test_zero_rows_and_zero_matrix(variant):
    import torch
    from paper_2609_36692_gb300 import normpre as C
    cs = S.custom_config("zeros", [(64, 96), (64, 96)], g_dtype="f32", w_dtype="f32", rank=4,
                         oversample=4, prior_momentum=False)
    mats = [S.make_matrix(cs, i) for i in range(2)]
    mats[0]["G"][5] = 0.0
    mats[0]["G"][17] = 0.0
    mats[1]["G"][:] = 0.0
    W, G, M = to_device(mats, "f32", "f32")
    opt = _normpre([(64, 96)] * 2, ["f32"] * 2, ["f32"] * 2,
                   variant=C.NORMPRE_G if variant == "G" else C.NORMPRE_L, precision=1, rank=4,
                   oversample=4, seed=1234)
    opt.step(0, LR, W, G, M)
    torch.cuda.synchronize()
    assert opt.status() == C.NORMPRE_OK
    psi = opt.read(0, C.NORMPRE_BUF_PSI)
    assert np.all(psi[5] == 0) and np.all(psi[17] == 0)
    assert int(opt.read(0, C.NORMPRE_BUF_STATS)[0][1]) == 62
    ref = _oracle(mats, 0, 0, variant, cs)
    assert rel_fro(to_host(W[0]) - mats[0]["W"], ref["W"] - mats[0]["W"]) <= 1e-3
    # an all-zero gradient: only weight decay acts
    np.testing.assert_allclose(to_host(W[1]), mats[1]["W"] * (1 - f32(LR) * f32(0.1)), rtol=1e-6)


def test_nonfinite_momentum_is_reported():
    import torch
    from paper_2609_36692_gb300 import normpre as C
    cs = S.custom_config("nan", [(32, 64)], g_dtype="f32", w_dtype="f32")
    mats = [S.make_matrix(cs, 0)]
    mats[0]["G"][3, 7] = np.nan
    W, G, M = to_device(mats, "f32", "f32")
    opt = _normpre([(32, 64)], ["f32"], ["f32"], precision=1)
    opt.step(0, LR, W, G, M)
    assert opt.status(raise_on_error=False) == C.NORMPRE_ERR_NONFINITE
    # the flag is cleared once reported
    assert opt.status(raise_on_error=False) == C.NORMPRE_OK


@pytest.mark.parametrize("variant", ["G", "L"])
def test_deterministic(variant):
    import torch
    from paper_2609_36692_gb300 import normpre as C
    cs = SMALL
    outs = []
    for _ in range(2):
        opt, mats, W1, M1 = _run(cs, 1, variant, precision=0 if variant == "G" else 1)
        outs.append(W1)
    for a, b in zip(*outs):
        assert np.array_equal(a, b)


_HOST_VARIANTS = ["G", "L", "L_bf16", "muon", "L_exact"]


def _host_variant(variant):
    """(variant code, precision) of a host-step test case: L_bf16 is NormPre-L
    with the bf16 Psi (NORMPRE_PREC_BF16), whose sketch runs on group slices
    with their own tensor maps in the host step."""
    from paper_2609_36692_gb300 import normpre as C
    code = {"G": C.NORMPRE_G, "L": C.NORMPRE_L, "L_bf16": C.NORMPRE_L, "muon": C.NORMPRE_MUON,
            "L_exact": C.NORMPRE_L_EXACT}[variant]
    return code, 0 if variant in ("G", "muon", "L_bf16") else 1


@pytest.mark.parametrize("variant", _HOST_VARIANTS)
def test_host_entry_point_matches_device_step(variant):
    """Two consecutive host-buffer steps (row- then column-active) equal the
    device-buffer steps bit for bit: the copies overlapped with the step move
    each group's inputs in before its normalization and its results out after."""
    import torch
    cs = SMALL
    mats = S.make_param_set(cs, workers=min(16, os.cpu_count() or 1))
    code, prec = _host_variant(variant)
    kw = dict(variant=code,
              precision=prec, rank=cs.rank, oversample=cs.oversample,
              power_iters=cs.power_iters, seed=1234, diagnostics=1)
    shapes = [(m.rows, m.cols) for m in cs.matrices]
    opt = _normpre(shapes, ["f32"] * cs.n_mats, ["bf16"] * cs.n_mats, **kw)
    opt2 = _normpre(shapes, ["f32"] * cs.n_mats, ["bf16"] * cs.n_mats, **kw)
    W, G, M = to_device(mats, cs.g_dtype, cs.w_dtype)
    Wh = [torch.from_numpy(m["W"].copy()).pin_memory() for m in mats]
    Gh = [torch.from_numpy(m["G"]).to(torch.bfloat16).pin_memory() for m in mats]
    Mh = [torch.from_numpy(m["M"].copy()).pin_memory() for m in mats]
    for t in (0, 1):
        opt.step(t, LR, W, G, M)
        torch.cuda.synchronize()
        opt.status()
        opt2.step_host(t, LR, Wh, Gh, Mh)
        for i in range(cs.n_mats):
            assert np.array_equal(Wh[i].numpy(), to_host(W[i])), (t, i)
            assert np.array_equal(Mh[i].numpy(), to_host(M[i])), (t, i)


@pytest.mark.parametrize("variant", _HOST_VARIANTS)
def test_host_entry_point_in_units(variant):
    """A group larger than one host-copy unit (8 x 4096^2 fp32/bf16: about
    1.3 GB of input) is preconditioned in pieces of matrices between its copies;
    the result equals the device-buffer step (whole groups) bit for bit."""
    import torch
    shapes = [(4096, 4096)] * 8 + [(1024, 4096)] * 3
    gen = torch.Generator().manual_seed(7)
    Wc = [torch.randn(r, c, generator=gen) * 0.02 for r, c in shapes]
    Gc = [torch.randn(r, c, generator=gen).to(torch.bfloat16) for r, c in shapes]
    Mc = [torch.randn(r, c, generator=gen) * 0.1 for r, c in shapes]
    code, prec = _host_variant(variant)
    kw = dict(variant=code, precision=prec, seed=1234)
    opt = _normpre(shapes, ["f32"] * len(shapes), ["bf16"] * len(shapes), **kw)
    opt2 = _normpre(shapes, ["f32"] * len(shapes), ["bf16"] * len(shapes), **kw)
    W = [w.cuda() for w in Wc]
    G = [g.cuda() for g in Gc]
    M = [m.cuda() for m in Mc]
    Wh = [w.pin_memory() for w in Wc]
    Gh = [g.pin_memory() for g in Gc]
    Mh = [m.pin_memory() for m in Mc]
    for t in (0, 1):
        opt.step(t, LR, W, G, M)
        torch.cuda.synchronize()
        opt.status()
        opt2.step_host(t, LR, Wh, Gh, Mh)
        for i in range(len(shapes)):
            assert torch.equal(Wh[i], W[i].cpu()), (t, i)
            assert torch.equal(Mh[i], M[i].cpu()), (t, i)



# --------------------------------------------------------------------------
# NormPre-L with exact eigenspace extraction (Sec. 3.2, App. B)
# --------------------------------------------------------------------------
# --------------------------------------------------------------------------
# device-detected conditions reported through the status word
# --------------------------------------------------------------------------
def test_jacobi_sweep_cap_reports_numeric():
    """With a cap of one Jacobi sweep, the 16 x 16 Ritz problems stop before
    their off-diagonal mass reaches the fp32 floor: the kernel records one
    sweep, raises the NUMERIC flag and returns (no trap, no hang), and
    normpre_sync_status reports NORMPRE_ERR_NUMERIC.  The status word is
    cleared by that read, so a following step with the default cap is clean."""
    import torch
    from paper_2609_36692_gb300 import normpre as C
    cs = SMALL
    mats = S.make_param_set(cs)
    W, G, M = to_device(mats, cs.g_dtype, cs.w_dtype)
    shapes = [(m.rows, m.cols) for m in cs.matrices]
    opt = _normpre(shapes, [cs.w_dtype] * cs.n_mats, [cs.g_dtype] * cs.n_mats, variant=C.NORMPRE_L,
                   precision=1, rank=cs.rank, oversample=cs.oversample, seed=1234, jacobi_max_sweeps=1)
    opt.step(0, LR, W, G, M)
    torch.cuda.synchronize()
    assert opt.status(raise_on_error=False) == C.NORMPRE_ERR_NUMERIC
    assert "Jacobi" in C.normpre_last_error(opt.handle)
    for i in range(cs.n_mats):
        assert int(opt.read(i, C.NORMPRE_BUF_STATS)[0][7]) == 1
    opt.close()
    opt = _normpre(shapes, [cs.w_dtype] * cs.n_mats, [cs.g_dtype] * cs.n_mats, variant=C.NORMPRE_L,
                   precision=1, rank=cs.rank, oversample=cs.oversample, seed=1234)
    opt.step(1, LR, W, G, M)
    torch.cuda.synchronize()
    assert opt.status(raise_on_error=False) == C.NORMPRE_OK
    assert all(int(opt.read(i, C.NORMPRE_BUF_STATS)[0][7]) > 1 for i in range(cs.n_mats))
    opt.close()


@pytest.mark.parametrize("precision", [1, 0], ids=["fp32", "bf16_psi"])
def test_bounded_wait_timeout_reports_and_recovers(precision):
    """The device-side timeout path of the tensor-core kernels (the fp32
    contraction, and the bf16-Psi one): with test_stall, one CTA of each
    group's first sketch contraction never gets its first copy; the warp
    waiting for it gives up after the bounded wait (about two seconds) and set
    the CTA's abort flag, every other role of that CTA leaves its loop at its
    next wait, thread 0 waits for the copies the CTA did issue, the tensor
    memory is freed and the kernel exits; the step reports
    NORMPRE_ERR_TIMEOUT.  No trap and no hang: the context stays usable, and a
    following step on a new handle matches the oracle."""
    import time

    import torch
    from paper_2609_36692_gb300 import normpre as C
    cs = SMALL
    mats = S.make_param_set(cs)
    W, G, M = to_device(mats, cs.g_dtype, cs.w_dtype)
    shapes = [(m.rows, m.cols) for m in cs.matrices]
    opt = _normpre(shapes, [cs.w_dtype] * cs.n_mats, [cs.g_dtype] * cs.n_mats, variant=C.NORMPRE_L,
                   precision=precision, rank=cs.rank, oversample=cs.oversample, seed=1234, test_stall=1)
    t0 = time.perf_counter()
    opt.step(0, LR, W, G, M)
    torch.cuda.synchronize()
    waited = time.perf_counter() - t0
    assert opt.status(raise_on_error=False) == C.NORMPRE_ERR_TIMEOUT
    assert "gave up" in C.normpre_last_error(opt.handle)
    assert 1.0 < waited < 60.0, waited
    opt.close()
    if precision == 1:
        _check_l(cs, 1)
    else:
        _check_l_bf16(cs, 1)


# one GPT-2 Small attention qkv matrix (768 x 2304): Gamma is 768 x 768 at
# t = 0 and 2304 x 2304 at t = 1
GPT2_QKV = S.custom_config("gpt2_qkv", [(768, 2304)], g_dtype="bf16", w_dtype="f32",
                           row_sigma=1.0, col_sigma=1.0, rank=32, oversample=8)


@pytest.mark.parametrize("cfgset", [SMALL, RAGGED, GPT2_QKV], ids=lambda c: c.name)
@pytest.mark.parametrize("t", [0, 1])
def test_l_exact(cfgset, t):
    """Gamma = Psi_a Psi_a^T, all its eigenvalues, the selected eigenvectors,
    the updated weights and the spectral energies, against the oracle."""
    from paper_2609_36692_gb300 import normpre as C
    opt, mats, W1, _ = _run(cfgset, t, "L_exact", precision=1)
    n_sel = 0
    for i in range(cfgset.n_mats):
        ref = _oracle(mats, i, t, "L_exact", cfgset)
        ex = ref["exact"]
        lam = ex["lam"]
        eig = opt.read(i, C.NORMPRE_BUF_EIGS)[0].astype(np.float64)
        assert eig.shape == lam.shape, (cfgset.name, i)
        # fp32 Gamma and a backward-stable fp32 eigensolver: errors of order
        # m_a u ||Gamma||_2 (u = 2^-24), a few ulp of lambda_max for small m_a
        tol = max(2e-5, lam.size * 2.0 ** -24)
        assert np.max(np.abs(eig - lam)) <= tol * max(1.0, lam[0]), (cfgset.name, i)
        st = opt.read(i, C.NORMPRE_BUF_STATS)[0]
        if ritz_gaps_ok(lam, cfgset.rank):
            nc = int(st[3])
            assert nc == ex["n_active"], (cfgset.name, i, nc, ex["n_active"])
            Q = opt.read(i, C.NORMPRE_BUF_Q)
            assert principal_sine(Q[:, :nc], ex["U_C"]) <= 1e-3, (cfgset.name, i)
            n_sel += nc
        dW = W1[i].astype(np.float64) - mats[i]["W"]
        assert rel_fro(dW, ref["W"] - mats[i]["W"]) <= 2e-3, (cfgset.name, i)
        d = opt.read(i, C.NORMPRE_BUF_DIAG)[0].astype(np.float64)
        e = O.spectral_energies(lam, cfgset.rank)
        scale = max(1.0, e["E_global"])
        for j, key in enumerate(("E_top", "E_remain", "E_sub", "E_global")):
            assert abs(d[j] - e[key]) <= 1e-3 * scale, (cfgset.name, i, key, d[j], e[key])
        assert np.all(np.isnan(d[4:])), "alignment is off without cfg.diagnostics"
    assert n_sel > 0 or cfgset is RAGGED


# --------------------------------------------------------------------------
# Diagnostics: descent alignment (App. E)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("variant", ["G", "L", "muon"])
@pytest.mark.parametrize("t", [0, 1])
def test_descent_alignment(variant, t):
    from paper_2609_36692_gb300 import normpre as C
    cs = SMALL
    opt, mats, W1, _ = _run(cs, t, variant, precision=1, extra={"diagnostics": 1})
    for i in range(cs.n_mats):
        m = mats[i]
        if variant == "muon":
            T_stored = O.muon_step(m["W"], m["G"], m["M"], f32(LR), oracle_config("G"))["T"]
        else:
            ref = _oracle(mats, i, t, variant, cs)
            T_stored = _stored(ref["T"], ref["k"])
        want = O.descent_alignment(m["G"], T_stored)
        d = opt.read(i, C.NORMPRE_BUF_DIAG)[0].astype(np.float64)
        assert abs(d[4] - want) <= 2e-3, (variant, i, d[4], want)
        assert abs(d[5] - np.linalg.norm(m["G"])) <= 1e-5 * np.linalg.norm(m["G"]), (variant, i)
        assert abs(d[6] - np.linalg.norm(T_stored)) <= 2e-3 * np.linalg.norm(T_stored), (variant, i)
        assert np.all(np.isnan(d[:4])), "spectral energies exist only for NORMPRE_L_EXACT"
        assert -1.0 <= d[4] <= 1.0
