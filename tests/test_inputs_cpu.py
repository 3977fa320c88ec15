"""The seeded synthetic parameter sets that stand in for the paper's workloads.

No corpus, model or trained gradient is available, so the parameter sets are
drawn: GPT-2 Small, LLaMA ~1B and Qwen3 ~1.7B hidden-matrix shapes (the
models of the paper's efficiency comparison, Table 2) with the value
distributions the workloads name (N(0, 1) or Student-t(3) entries,
log-normal row / column scales, bf16 storage).  These tests pin what the
generators draw: the shapes and element counts of each set, the storage
rounding, the distributions (checked against scipy's), and that every matrix
has its own reproducible streams.
"""
import numpy as np
import pytest

from synth import inputs as S

scipy_stats = pytest.importorskip("scipy.stats")


def _per_layer(cfg, layers):
    shapes = [(m.rows, m.cols) for m in cfg.matrices]
    per = len(shapes) // layers
    assert per * layers == len(shapes)
    for l in range(layers):
        assert shapes[l * per:(l + 1) * per] == shapes[:per]
    return shapes[:per]


def test_gpt2_small_shapes():
    for name in ("gpt2_small_G", "gpt2_small_L"):
        cfg = S.CONFIGS[name]
        assert _per_layer(cfg, 12) == [(768, 2304), (768, 768), (768, 3072), (3072, 768)]
        assert cfg.n_mats == 48 and cfg.elements == 84_934_656
        assert (cfg.g_dtype, cfg.w_dtype) == (S.BF16, S.F32)
    assert (S.CONFIGS["gpt2_small_L"].rank, S.CONFIGS["gpt2_small_L"].oversample) == (32, 8)


def test_llama_1b_shapes():
    cfg = S.CONFIGS["llama_1b"]
    assert _per_layer(cfg, 16) == [(2048, 2048)] * 4 + [(2048, 5504)] * 2 + [(5504, 2048)]
    assert cfg.n_mats == 112 and cfg.elements == 809_500_672
    assert cfg.grad_dist == "student_t3"


def test_qwen3_shapes():
    cfg = S.CONFIGS["qwen3_1p7b"]
    assert _per_layer(cfg, 28) == [(2048, 2048), (2048, 1024), (2048, 1024), (2048, 2048),
                                   (2048, 6144), (2048, 6144), (6144, 2048)]
    assert cfg.n_mats == 196 and cfg.elements == 1_409_286_144
    assert (cfg.g_dtype, cfg.w_dtype) == (S.BF16, S.BF16)
    # the profiling case: the first two layers, same shapes and distributions
    two = S.CONFIGS["qwen3_2layers"]
    assert [(m.rows, m.cols) for m in two.matrices] == [(m.rows, m.cols) for m in cfg.matrices[:14]]
    assert (two.row_sigma, two.col_sigma, two.g_dtype, two.w_dtype) == \
        (cfg.row_sigma, cfg.col_sigma, cfg.g_dtype, cfg.w_dtype)


def test_single_matrix_case():
    cfg = S.CONFIGS["single_256x1024"]
    assert [(m.rows, m.cols) for m in cfg.matrices] == [(256, 1024)]
    mat = S.make_matrix(cfg, 0)
    assert not mat["M"].any()                       # zero initial momentum
    assert (cfg.rank, cfg.oversample) == (16, 8)


def test_storage_rounding():
    """bf16 tensors hold bf16 values exactly (one round-to-nearest-even);
    fp32 weights are not rounded."""
    mat = S.make_matrix(S.CONFIGS["qwen3_2layers"], 1)
    for key in ("G", "M", "W"):
        assert mat[key].dtype == np.float32
        assert np.array_equal(S.round_to_bf16(mat[key]), mat[key]), key
    w32 = S.make_matrix(S.CONFIGS["gpt2_small_G"], 1)["W"]
    assert not np.array_equal(S.round_to_bf16(w32), w32)
    # round to nearest even on hand values: 1 + 2^-8 is a tie (to 1), 1 + 3 * 2^-8 goes up
    x = np.array([1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, -(1 + 2.0 ** -8 + 2.0 ** -20)], dtype=np.float32)
    assert S.round_to_bf16(x).tolist() == [1.0, 1 + 2.0 ** -6, -(1 + 2.0 ** -7)]


def _ks_pvalue(x, dist, args=()):
    return scipy_stats.kstest(x.ravel().astype(np.float64), dist, args=args).pvalue


def test_entry_distributions_against_scipy():
    """With the scales switched off, the entries are N(0, 1) or Student-t(3)."""
    n = S.custom_config("n", [(256, 512)], grad_dist="normal", row_sigma=0.0, col_sigma=0.0)
    t = S.custom_config("t", [(256, 512)], grad_dist="student_t3", row_sigma=0.0, col_sigma=0.0)
    zn = S.make_matrix(n, 0)["G"]
    zt = S.make_matrix(t, 0)["G"]
    assert _ks_pvalue(zn, "norm") > 1e-3
    assert _ks_pvalue(zt, "t", (3,)) > 1e-3
    # and each is told apart from the other
    assert _ks_pvalue(zt, "norm") < 1e-6
    assert _ks_pvalue(zn, "t", (3,)) < 1e-6


@pytest.mark.parametrize("name,sig_r,sig_c", [("qwen3_2layers", 1.5, 1.5), ("gpt2_small_G", 1.0, 1.0),
                                              ("llama_1b", 1.0, 0.0)])
def test_log_normal_line_scales(name, sig_r, sig_c):
    """log of the row (column) RMS spreads with the configured sigma: the
    entries of a line share one factor exp(sigma xi), the other factor
    averages out over the long line."""
    cfg = S.CONFIGS[name]
    assert (cfg.row_sigma, cfg.col_sigma) == (sig_r, sig_c)
    idx = [i for i, m in enumerate(cfg.matrices) if m.rows >= 768 and m.cols >= 768][0]
    g = S.make_matrix(cfg, idx)["G"].astype(np.float64)
    # robust line scale (median |g|): also defined for Student-t(3) entries
    row = np.log(np.median(np.abs(g), axis=1))
    col = np.log(np.median(np.abs(g), axis=0))
    assert abs(np.std(row) - sig_r) < 0.1, np.std(row)
    if sig_c > 0:
        assert abs(np.std(col) - sig_c) < 0.1, np.std(col)
    else:
        assert np.std(col) < 0.1, np.std(col)


def test_prior_momentum_and_weights():
    """M_{t-1} is an independent draw of the gradient's distribution (the
    momentum after one step from zero); W is N(0, 0.02^2)."""
    cfg = S.CONFIGS["gpt2_small_G"]
    mat = S.make_matrix(cfg, 1)   # 768 x 768
    g, m, w = (mat[k].astype(np.float64) for k in ("G", "M", "W"))
    assert abs(np.corrcoef(g.ravel(), m.ravel())[0, 1]) < 0.01
    lg = np.log(np.median(np.abs(g), axis=1))
    lm = np.log(np.median(np.abs(m), axis=1))
    assert abs(np.std(lg) - np.std(lm)) < 0.15
    assert abs(np.std(w) - 0.02) < 0.0005 and abs(np.mean(w)) < 0.0005


def test_streams_are_per_matrix_and_reproducible():
    cfg = S.CONFIGS["gpt2_small_G"]
    a = S.make_matrix(cfg, 5)
    b = S.make_matrix(cfg, 5)
    for k in a:
        assert np.array_equal(a[k], b[k])
    # matrix 5 and matrix 1 share a shape (attn-proj) but not their streams
    c = S.make_matrix(cfg, 1)
    assert a["G"].shape == c["G"].shape and not np.array_equal(a["G"], c["G"])
    # another base seed, other values
    d = S.make_matrix(cfg, 5, seed=1)
    assert not np.array_equal(a["G"], d["G"])
    # threaded drawing gives the serial values
    idx = [0, 1, 5]
    ser = S.make_param_set(cfg, indices=idx)
    par = S.make_param_set(cfg, indices=idx, workers=3)
    for x, y in zip(ser, par):
        for k in x:
            assert np.array_equal(x[k], y[k])
