"""The C ABI library without a GPU: it builds, loads, exports every symbol the
header declares, and rejects bad arguments on the host before any CUDA call."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "normpre.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_36692_gb300 import build
    build.build()
    from paper_2609_36692_gb300 import normpre as C
    return C


def _declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(normpre_[a-z_]+)\s*\(", src)))


def test_header_declares_the_abi():
    names = _declared_functions()
    for n in ("normpre_init", "normpre_step", "normpre_free", "normpre_last_error",
              "normpre_newton_schulz", "normpre_step_host", "normpre_read"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    so = ctypes.CDLL(lib.LIB_PATH)
    missing = [n for n in _declared_functions() if not hasattr(so, n)]
    assert not missing, missing


def test_default_config_is_the_papers(lib):
    cfg = lib.normpre_default_config()
    assert cfg.variant == lib.NORMPRE_G
    assert abs(cfg.momentum - 0.95) < 1e-7
    assert abs(cfg.weight_decay - 0.1) < 1e-7
    assert abs(cfg.target_rms - 0.2) < 1e-7
    assert cfg.ns_steps == 5
    assert [round(x, 4) for x in cfg.ns_coef] == [3.4445, -4.775, 2.0315]
    assert (cfg.rank, cfg.oversample, cfg.power_iters) == (32, 8, 1)
    assert cfg.precision == lib.NORMPRE_PREC_BF16 and cfg.orientation == 0
    assert cfg.tangent == 0      # the paper's relaxed tangent
    assert cfg.diagnostics == 0


def test_host_side_argument_errors(lib):
    C = lib
    cfg = C.normpre_default_config()
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(cfg, [], [], [])
    assert e.value.status == C.NORMPRE_ERR_ARG
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(cfg, [(0, 5)], [0], [0])
    assert e.value.status == C.NORMPRE_ERR_SHAPE
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(cfg, [(4, 5)], [7], [0])
    assert e.value.status == C.NORMPRE_ERR_DTYPE
    bad = C.normpre_default_config(ns_steps=0)
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(bad, [(4, 5)], [0], [0])
    assert e.value.status == C.NORMPRE_ERR_ARG
    bad = C.normpre_default_config(variant=C.NORMPRE_L, rank=66, oversample=8)
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(bad, [(4, 5)], [0], [0])
    assert e.value.status == C.NORMPRE_ERR_ARG
    assert "rank" in C.normpre_last_error()
    bad = C.normpre_default_config(orientation=5)
    with pytest.raises(C.NormPreError):
        C.normpre_init(bad, [(4, 5)], [0], [0])
    bad = C.normpre_default_config(tangent=3)
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(bad, [(4, 5)], [0], [0])
    assert "tangent" in C.normpre_last_error()
    bad = C.normpre_default_config(variant=4)
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(bad, [(4, 5)], [0], [0])
    assert e.value.status == C.NORMPRE_ERR_ARG
    bad = C.normpre_default_config(diagnostics=2)
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(bad, [(4, 5)], [0], [0])
    assert "diagnostics" in C.normpre_last_error()
    for sweeps in (-1, 1001):
        bad = C.normpre_default_config(variant=C.NORMPRE_L, jacobi_max_sweeps=sweeps)
        with pytest.raises(C.NormPreError) as e:
            C.normpre_init(bad, [(4, 5)], [0], [0])
        assert e.value.status == C.NORMPRE_ERR_ARG and "jacobi_max_sweeps" in C.normpre_last_error()
    assert C.normpre_default_config().jacobi_max_sweeps == 0
    bad = C.normpre_default_config(test_stall=2)
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(bad, [(4, 5)], [0], [0])
    assert e.value.status == C.NORMPRE_ERR_ARG and "test_stall" in C.normpre_last_error()
    assert C.normpre_default_config().test_stall == 0
    # exact eigenspace extraction: rank budget and the Gamma workspace limit
    bad = C.normpre_default_config(variant=C.NORMPRE_L_EXACT, rank=73)
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(bad, [(4, 5)], [0], [0])
    assert e.value.status == C.NORMPRE_ERR_ARG
    ex = C.normpre_default_config(variant=C.NORMPRE_L_EXACT)
    with pytest.raises(C.NormPreError) as e:
        C.normpre_init(ex, [(16, 20000)], [0], [0])
    assert e.value.status == C.NORMPRE_ERR_SHAPE
    # stand-alone Newton-Schulz: argument checks come before any device work
    with pytest.raises(C.NormPreError) as e:
        C.normpre_newton_schulz(cfg, 1, 4, 4, 0, 0)
    assert e.value.status == C.NORMPRE_ERR_ARG
    with pytest.raises(C.NormPreError) as e:
        C.normpre_newton_schulz(cfg, 1, 0, 4, 16, 16)
    assert e.value.status == C.NORMPRE_ERR_SHAPE
    with pytest.raises(C.NormPreError) as e:
        C.normpre_newton_schulz(cfg, 1, 4, 4, 17, 32)
    assert e.value.status == C.NORMPRE_ERR_ALIGN


def test_null_handle_calls(lib):
    C = lib
    so = C.load_library()
    assert so.normpre_step(None, 0, 0.1, None, None, None, None) == C.NORMPRE_ERR_ARG
    assert so.normpre_sync_status(None, None) == C.NORMPRE_ERR_ARG
    so.normpre_free(None)


def test_torch_optimizer_validates_parameters():
    """NormPreOptimizer takes 2-D CUDA matrices only; the checks run on the
    host before any device work."""
    torch = pytest.importorskip("torch")
    from paper_2609_36692_gb300.optim import NormPreOptimizer
    with pytest.raises(ValueError, match="2-D"):
        NormPreOptimizer([torch.nn.Parameter(torch.zeros(3))])
    with pytest.raises(ValueError, match="CUDA"):
        NormPreOptimizer([torch.nn.Parameter(torch.zeros(3, 4))])
    with pytest.raises(ValueError, match="variant"):
        NormPreOptimizer([torch.nn.Parameter(torch.zeros(3, 4))], variant="X")
    # one plan serves a group on one device
    with pytest.raises(ValueError, match="one CUDA device"):
        NormPreOptimizer([torch.nn.Parameter(torch.zeros(3, 4)),
                          torch.nn.Parameter(torch.zeros(3, 4, device="meta"))])


def _header_without_comments():
    return re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)


def test_binding_enums_mirror_the_header(lib):
    """Every enumerator the header defines has the same value in the binding."""
    src = _header_without_comments()
    values = {}
    for body in re.findall(r"\benum\s+\w+\s*\{(.*?)\}", src, flags=re.S):
        for name, val in re.findall(r"\b(NORMPRE_\w+)\s*=\s*(\d+)", body):
            values[name] = int(val)
    assert len(values) >= 30
    mirrored = {n: v for n, v in values.items() if not n.startswith("NORMPRE_PROF_")}
    for name, val in mirrored.items():
        assert getattr(lib, name) == val, name
    assert lib.STATUS_NAMES == {v: n[len("NORMPRE_"):] for n, v in values.items()
                                if n == "NORMPRE_OK" or n.startswith("NORMPRE_ERR_")}


def test_binding_config_struct_mirrors_the_header(lib):
    """normpre_config: the binding's ctypes fields in the header's order and
    types, so that the library reads every hyperparameter where it was put."""
    src = _header_without_comments()
    body = re.search(r"typedef\s+struct\s+normpre_config\s*\{(.*?)\}\s*normpre_config\s*;", src, flags=re.S).group(1)
    fields = re.findall(r"(\w+)\s+(\w+)(\[\d+\])?\s*;", body)
    c_types = {"int": ctypes.c_int, "float": ctypes.c_float, "uint64_t": ctypes.c_uint64}
    want = [(name, c_types[ty] * int(arr[1:-1]) if arr else c_types[ty]) for ty, name, arr in fields]
    got = lib.normpre_config._fields_
    assert [n for n, _ in got] == [n for n, _ in want]
    for (n, t_got), (_, t_want) in zip(got, want):
        if hasattr(t_want, "_length_"):      # a fixed-size array field
            assert t_got._length_ == t_want._length_ and t_got._type_ is t_want._type_, n
        else:
            assert t_got is t_want, n
