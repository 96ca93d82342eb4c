"""Seed selection for parity runs (test infrastructure; uses only oracle/ and synth/).

Top-k picks are integers decided by floating point. The CUDA path accumulates the
router logits in fp32 on the tensor cores (d/16 accumulation steps of K=16
products, each step adding at most one rounding of the running sum), the oracle in
fp64. ``logit_tol`` bounds their difference per token:

    tau_t = 2 * (d / 16) * 2^-24 * max(1, max_e |z_te|)

(one unit in the last place of the largest partial sum per step, with a factor 2 of
headroom; the tests assert |z_gpu - z_fp64| <= tau_t). A token whose neighbouring
top-(k+1) logits are further apart than 2 tau_t is routed identically by both.
``decided_seed`` returns the first seed, starting from the workload's own, whose every
token is decided that way, so that a full-layer comparison is unique.
"""
from __future__ import annotations

import numpy as np

from oracle import moe_oracle as mo
from synth import moe_inputs as mi


def logit_tol(z, d: int) -> np.ndarray:
    """Per-token bound on |fp32 tensor-core logits - fp64 logits| (shape [T, 1])."""
    z = np.asarray(z, np.float64)
    zmax = np.maximum(1.0, np.abs(z).max(axis=1, keepdims=True))
    return 2.0 * (max(d, 16) / 16.0) * 2.0 ** -24 * zmax


def decided(z, k: int, d: int) -> np.ndarray:
    """Tokens whose top-(k+1) neighbouring logit gaps all exceed twice the bound."""
    return mo.top_margin(z, k) > 2.0 * logit_tol(z, d)[:, 0]


def decided_seed(shape, max_tries: int = 400) -> int:
    for s in range(shape.seed, shape.seed + max_tries):
        inp = mi.make_inputs(shape, seed=s, with_weights=False)
        z = mo.router_logits(inp["x"], inp["w_router"], inp.get("router_bias"), inp["party_offsets"])
        if shape.n_experts == shape.top_k or decided(z, shape.top_k, shape.d_model).all():
            return s
    raise RuntimeError(f"no decided seed for {shape.name} in {max_tries} tries")
