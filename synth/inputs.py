"""Seeded synthetic parameter sets for the NormPre step.

Each parameter set is a list of 2-D weight matrices stored row-major as
``rows x cols``.  For every matrix three tensors are drawn:

* ``G``  the gradient of this step,
* ``M``  the momentum carried in from the previous step (``M_{t-1}``),
* ``W``  the current weight.

Distributions (the paper trains on OpenWebText, C4 and the Pile; those
corpora, the models and their gradients are not available, so synthetic
tensors with the same shapes and the scale / tail structure named for each
workload stand in for them):

* gradient entries are i.i.d. N(0, 1) (or Student-t with 3 degrees of freedom)
  multiplied by a log-normal scale per row ``exp(sigma_r * xi_i)`` and, where
  the workload asks for it, per column ``exp(sigma_c * zeta_j)``;
* the prior momentum is "the momentum after one step from zero", i.e. an
  independent gradient draw from the same distribution (or exactly zero);
* weights are N(0, 0.02^2) (GPT-2 / nanoGPT style initialisation).

Values are rounded once to their storage dtype (bf16 round-to-nearest-even)
and returned as float32 arrays that hold those exact values, so that the
device (which receives the identical bits) and the fp64 oracle (which widens
them) see the same numbers.

Random streams: matrix ``i`` of a set with base seed ``s`` draws its gradient
from ``numpy.random.default_rng([s, i, 0])``, its prior momentum from
``[s, i, 1]`` and its weight from ``[s, i, 2]`` (numpy's PCG64 seeded through
SeedSequence).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np

F32 = "f32"
BF16 = "bf16"


# ----------------------------------------------------------------------------
# storage-dtype helpers
# ----------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest, ties to even."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    bias = ((u >> 16) & 1) + 0x7FFF
    out = ((u + bias) >> 16).astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float32 holding the same value."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 value (returned as float32)."""
    return bf16_bits_to_f32(f32_to_bf16_bits(x))


def _store(x: np.ndarray, dtype: str) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    return round_to_bf16(x) if dtype == BF16 else x


# ----------------------------------------------------------------------------
# workload descriptions
# ----------------------------------------------------------------------------
@dataclass(frozen=True)
class MatrixSpec:
    rows: int
    cols: int
    name: str = ""


@dataclass(frozen=True)
class ParamSetConfig:
    """A named parameter set: shapes, storage dtypes and value distributions.

    ``variant`` / ``rank`` / ``oversample`` / ``power_iters`` / ``ns_steps``
    name the NormPre settings the workload is measured with; they carry no
    arithmetic here.
    """

    name: str
    matrices: List[MatrixSpec]
    g_dtype: str = BF16
    w_dtype: str = F32
    grad_dist: str = "normal"        # "normal" or "student_t3"
    row_sigma: float = 1.0
    col_sigma: float = 0.0
    prior_momentum: bool = True      # False: M_{t-1} = 0
    w_std: float = 0.02
    variants: tuple = ("G",)
    rank: int = 32
    oversample: int = 8
    power_iters: int = 1
    ns_steps: int = 5
    seed: int = 0
    description: str = ""

    @property
    def n_mats(self) -> int:
        return len(self.matrices)

    @property
    def elements(self) -> int:
        return int(sum(m.rows * m.cols for m in self.matrices))


def _repeat(layers: int, per_layer: List[MatrixSpec]) -> List[MatrixSpec]:
    out = []
    for l in range(layers):
        for s in per_layer:
            out.append(MatrixSpec(s.rows, s.cols, f"l{l}.{s.name}"))
    return out


_GPT2 = _repeat(12, [MatrixSpec(768, 2304, "qkv"), MatrixSpec(768, 768, "attn_proj"),
                     MatrixSpec(768, 3072, "fc"), MatrixSpec(3072, 768, "mlp_proj")])
_LLAMA1B = _repeat(16, [MatrixSpec(2048, 2048, "q"), MatrixSpec(2048, 2048, "k"),
                        MatrixSpec(2048, 2048, "v"), MatrixSpec(2048, 2048, "o"),
                        MatrixSpec(2048, 5504, "gate"), MatrixSpec(2048, 5504, "up"),
                        MatrixSpec(5504, 2048, "down")])
_QWEN3 = _repeat(28, [MatrixSpec(2048, 2048, "q"), MatrixSpec(2048, 1024, "k"),
                      MatrixSpec(2048, 1024, "v"), MatrixSpec(2048, 2048, "o"),
                      MatrixSpec(2048, 6144, "gate"), MatrixSpec(2048, 6144, "up"),
                      MatrixSpec(6144, 2048, "down")])

CONFIGS: Dict[str, ParamSetConfig] = {
    "single_256x1024": ParamSetConfig(
        name="single_256x1024", matrices=[MatrixSpec(256, 1024, "w")],
        g_dtype=F32, w_dtype=F32, grad_dist="normal", row_sigma=1.0, col_sigma=0.0,
        prior_momentum=False, variants=("G", "L"), rank=16, oversample=8, power_iters=1,
        seed=0,
        description="single fp32 256x1024 matrix, N(0,1) x log-normal(1) row scales, "
                    "zero prior momentum"),
    "gpt2_small_G": ParamSetConfig(
        name="gpt2_small_G", matrices=_GPT2, g_dtype=BF16, w_dtype=F32,
        grad_dist="normal", row_sigma=1.0, col_sigma=1.0, variants=("G",),
        description="GPT-2 Small hidden matrices (12 x qkv/attn-proj/fc/mlp-proj), bf16 "
                    "grads N(0,1) x log-normal(1) row and column scales, NormPre-G"),
    "gpt2_small_L": ParamSetConfig(
        name="gpt2_small_L", matrices=_GPT2, g_dtype=BF16, w_dtype=F32,
        grad_dist="normal", row_sigma=1.0, col_sigma=1.0, variants=("L",),
        rank=32, oversample=8, power_iters=1,
        description="GPT-2 Small hidden matrices under NormPre-L (r=32, o=8, p=1)"),
    "llama_1b": ParamSetConfig(
        name="llama_1b", matrices=_LLAMA1B, g_dtype=BF16, w_dtype=F32,
        grad_dist="student_t3", row_sigma=1.0, col_sigma=0.0, variants=("G", "L"),
        description="LLaMA ~1B hidden matrices (16 layers, hidden 2048, SwiGLU 5504), "
                    "bf16 Student-t(3) grads x log-normal(1) row scales"),
    "qwen3_1p7b": ParamSetConfig(
        name="qwen3_1p7b", matrices=_QWEN3, g_dtype=BF16, w_dtype=BF16,
        grad_dist="normal", row_sigma=1.5, col_sigma=1.5, variants=("G", "L"),
        description="Qwen3 ~1.7B hidden matrices (28 layers, GQA k/v 2048x1024, MLP 6144), "
                    "bf16 grads N(0,1) x log-normal(1.5) row and column scales, bf16 weights"),
    # the first two layers of the Qwen3 set: the same shapes, dtypes and value
    # distributions at 1/14 of the size (100M elements, about 1 GB on the
    # device, every per-step buffer still larger than L2), for kernel profiles
    "qwen3_2layers": ParamSetConfig(
        name="qwen3_2layers", matrices=_repeat(2, [MatrixSpec(2048, 2048, "q"), MatrixSpec(2048, 1024, "k"),
                                                  MatrixSpec(2048, 1024, "v"), MatrixSpec(2048, 2048, "o"),
                                                  MatrixSpec(2048, 6144, "gate"), MatrixSpec(2048, 6144, "up"),
                                                  MatrixSpec(6144, 2048, "down")]),
        g_dtype=BF16, w_dtype=BF16, grad_dist="normal", row_sigma=1.5, col_sigma=1.5, variants=("G", "L"),
        description="two Qwen3 ~1.7B layers (the profiling case of the Qwen3 kernels)"),
}


# ----------------------------------------------------------------------------
# drawing
# ----------------------------------------------------------------------------
def _gradient_like(rng: np.random.Generator, cfg: ParamSetConfig, rows: int, cols: int) -> np.ndarray:
    if cfg.grad_dist == "normal":
        z = rng.standard_normal((rows, cols), dtype=np.float32)
    elif cfg.grad_dist == "student_t3":
        # t_3 = xi / sqrt(chi2_3 / 3) with chi2_3 = 2 * Gamma(3/2)
        xi = rng.standard_normal((rows, cols), dtype=np.float32)
        chi2 = 2.0 * rng.standard_gamma(1.5, size=(rows, cols), dtype=np.float32)
        z = xi / np.sqrt(chi2 / np.float32(3.0))
    else:
        raise ValueError(f"unknown gradient distribution {cfg.grad_dist!r}")
    if cfg.row_sigma > 0:
        r = np.exp(np.float32(cfg.row_sigma) * rng.standard_normal(rows, dtype=np.float32))
        z *= r[:, None]
    if cfg.col_sigma > 0:
        c = np.exp(np.float32(cfg.col_sigma) * rng.standard_normal(cols, dtype=np.float32))
        z *= c[None, :]
    return z


def make_matrix(cfg: ParamSetConfig, index: int, seed: Optional[int] = None,
                zero_weight: bool = False) -> Dict[str, np.ndarray]:
    """Draw (G, M_prev, W) for matrix ``index`` of parameter set ``cfg``.

    Returns float32 arrays holding values exactly representable in the storage
    dtype: ``cfg.g_dtype`` for G and for M (a gradient draw, kept in an fp32
    momentum buffer), ``cfg.w_dtype`` for W.
    """
    s = cfg.seed if seed is None else seed
    spec = cfg.matrices[index]
    rows, cols = spec.rows, spec.cols
    g = _store(_gradient_like(np.random.default_rng([s, index, 0]), cfg, rows, cols), cfg.g_dtype)
    if cfg.prior_momentum:
        # momentum after one step from zero = an independent gradient draw
        m = _store(_gradient_like(np.random.default_rng([s, index, 1]), cfg, rows, cols), cfg.g_dtype)
    else:
        m = np.zeros((rows, cols), dtype=np.float32)
    if zero_weight:
        w = np.zeros((rows, cols), dtype=np.float32)
    else:
        w = np.random.default_rng([s, index, 2]).standard_normal((rows, cols), dtype=np.float32)
        w = _store(w * np.float32(cfg.w_std), cfg.w_dtype)
    return {"G": g, "M": m.astype(np.float32), "W": w}


def make_param_set(cfg: ParamSetConfig, seed: Optional[int] = None,
                   indices: Optional[List[int]] = None, workers: int = 0) -> List[Dict[str, np.ndarray]]:
    """Draw every matrix of the set (in parallel threads when workers > 1; each
    matrix has its own random streams, so the values do not depend on it)."""
    idx = list(range(cfg.n_mats) if indices is None else indices)
    if workers and workers > 1 and len(idx) > 1:
        from concurrent.futures import ThreadPoolExecutor
        with ThreadPoolExecutor(max_workers=workers) as ex:
            return list(ex.map(lambda i: make_matrix(cfg, i, seed), idx))
    return [make_matrix(cfg, i, seed) for i in idx]


def custom_config(name: str, shapes, g_dtype: str = F32, w_dtype: str = F32,
                  **kw) -> ParamSetConfig:
    """A parameter set with arbitrary shapes (tests: ragged and odd sizes)."""
    mats = [MatrixSpec(int(r), int(c), f"m{i}") for i, (r, c) in enumerate(shapes)]
    return ParamSetConfig(name=name, matrices=mats, g_dtype=g_dtype, w_dtype=w_dtype, **kw)
