"""Seeded synthetic inputs shared by the tests, the bench and the smoke check.

This package holds no optimizer arithmetic: it only draws gradients, prior
momenta and weights with the shapes and value distributions of the parameter
sets the NormPre step is measured on, and stores them in their storage dtype.
"""
from .inputs import (  # noqa: F401
    CONFIGS,
    MatrixSpec,
    ParamSetConfig,
    bf16_bits_to_f32,
    f32_to_bf16_bits,
    make_matrix,
    make_param_set,
    round_to_bf16,
)
