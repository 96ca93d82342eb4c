"""Seeded synthetic inputs for the MoE expert layer.

This package holds workload shapes and random draws only. It contains none of
the layer's arithmetic, so both the fp64 oracle (``oracle/``) and the CUDA path
(``paper_2506_02965_gb300``) may use it without sharing any of the method.
"""
from .moe_inputs import (  # noqa: F401
    MoEShape,
    SHAPES,
    bf16_round,
    make_inputs,
    make_route_logits,
    party_offsets,
    shape_by_name,
)
