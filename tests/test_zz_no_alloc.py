"""normpre_normalize_cols_noalloc: the column-active normalization for callers
that cannot allocate device memory when they need it (code inside an
allocator or memory-pool callback, frameworks whose allocator must not be
re-entered, processes whose device memory is reserved in advance).  Its
scratch is a fixed array inside the library, so these tests check that it
gives what the handle-based step gives, call after call, and that it refuses
shapes whose scratch would not fit.  Each call is also checked against the
fp64 oracle's column-active step (k = 1) on the same inputs.

This file is named to be collected last: a failure here leaves every other
test already run.
"""
import numpy as np
import pytest

import oracle as O
from synth import inputs as S

from helpers import max_row_rel, oracle_config, to_device, to_host


def _lib():
    from paper_2609_36692_gb300 import build
    build.build()
    from paper_2609_36692_gb300 import normpre as C
    return C


def test_noalloc_rejects_oversized_and_bad_arguments():
    C = _lib()
    with pytest.raises(C.NormPreError) as e:
        C.normpre_normalize_cols_noalloc(16384, 16384, 0.95, 16, C.NORMPRE_F32, 16, 16, C.NORMPRE_F32, 16)
    assert e.value.status == C.NORMPRE_ERR_SHAPE
    assert "scratch" in C.normpre_last_error()
    with pytest.raises(C.NormPreError) as e:
        C.normpre_normalize_cols_noalloc(16, 16, 0.95, 0, C.NORMPRE_F32, 16, 16, C.NORMPRE_F32, 16)
    assert e.value.status == C.NORMPRE_ERR_ARG
    with pytest.raises(C.NormPreError) as e:
        C.normpre_normalize_cols_noalloc(16, 16, 0.95, 24, C.NORMPRE_F32, 16, 16, C.NORMPRE_F32, 16)
    assert e.value.status == C.NORMPRE_ERR_ALIGN


def _handle_reference(C, rows, cols, g_dtype, w_dtype, mats):
    """Psi and M_t from the existing entry point (normpre_init / normpre_step,
    column-active, fp32 Psi)."""
    import torch
    from paper_2609_36692_gb300.optim import NormPre
    W, G, M = to_device(mats, g_dtype, w_dtype)
    opt = NormPre([(rows, cols)], [w_dtype], [g_dtype], variant=C.NORMPRE_L,
                  precision=C.NORMPRE_PREC_F32, orientation=2, rank=4, oversample=4)
    opt.step(0, 0.02, W, G, M)
    torch.cuda.synchronize()
    opt.status()
    psi = opt.read(0, C.NORMPRE_BUF_PSI)
    m = to_host(M[0])
    opt.close()
    return psi, m


@pytest.mark.gpu
def test_noalloc_matches_handle_step_on_two_calls_in_a_row():
    import torch
    C = _lib()
    cases = [(1024, 768, "bf16", "f32"), (333, 200, "f32", "bf16")]   # the second reuses dirty scratch
    for rows, cols, gdt, wdt in cases:
        cs = S.custom_config("noalloc_%dx%d" % (rows, cols), [(rows, cols)], g_dtype=gdt, w_dtype=wdt,
                             row_sigma=1.0, col_sigma=1.0)
        mats = [S.make_matrix(cs, 0)]
        psi_ref, m_ref = _handle_reference(C, rows, cols, gdt, wdt, mats)
        W, G, M = to_device(mats, gdt, wdt)
        psi = torch.empty((rows, cols), dtype=torch.float32, device="cuda")
        C.normpre_normalize_cols_noalloc(rows, cols, 0.95, G[0].data_ptr(), C.NORMPRE_BF16 if gdt == "bf16" else C.NORMPRE_F32,
                                         M[0].data_ptr(), W[0].data_ptr(),
                                         C.NORMPRE_BF16 if wdt == "bf16" else C.NORMPRE_F32,
                                         psi.data_ptr(), torch.cuda.current_stream().cuda_stream)
        torch.cuda.synchronize()
        out = psi.cpu().numpy()
        # columns are the active rows: compare per column against its norm
        assert max_row_rel(out.T, psi_ref.T.astype(np.float64)) <= 1e-5, (rows, cols)
        m = to_host(M[0])
        assert np.all(np.abs(m.astype(np.float64) - m_ref) <= 2.5e-7 * np.abs(m_ref) + 1e-30), (rows, cols)
        # the oracle's column-active step (t = 1): momentum, relaxed tangent and
        # normalization of every column (Alg. 1, Eq. 3)
        ref = O.normpre_step(mats[0]["W"], mats[0]["G"], mats[0]["M"], 1, 0.02,
                             oracle_config("L", rank=4, oversample=4), matrix_id=0)
        assert ref["k"] == 1
        assert max_row_rel(out.T, ref["Psi"]) <= 1e-5, (rows, cols)
        assert np.all(np.abs(m.astype(np.float64) - ref["M"]) <= 2.5e-7 * np.abs(ref["M"]) + 1e-30), (rows, cols)
