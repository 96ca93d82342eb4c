"""Seed selection for parity runs (test infrastructure; uses only oracle/ and synth/).

Top-k picks are integers decided by floating point. The CUDA path accumulates the
router logits in fp32, the oracle in fp64; the two agree within ``logit_tol(d)``
(a test asserts it). A token whose neighbouring top-(k+1) logits are further apart
than twice that tolerance is routed identically by both. ``decided_seed`` returns
the first seed, starting from the workload's own, whose every token is decided that
way, so that a full-layer comparison is unique.
"""
from __future__ import annotations

import numpy as np

from oracle import moe_oracle as mo
from synth import moe_inputs as mi


def logit_tol(d: int) -> float:
    """Absolute tolerance of fp32-accumulated router logits against fp64 ones.

    Rounding errors of a length-d fp32 dot product of O(1) terms grow like sqrt(d)
    units in the last place of the partial sums; 1e-5 at d = 1024 leaves a wide
    margin over the ~1e-6 such sums show on the layer's input distributions.
    """
    return 1e-5 * (max(d, 1) / 1024.0) ** 0.5


def margins(shape, inp) -> np.ndarray:
    z = mo.router_logits(inp["x"], inp["w_router"], inp.get("router_bias"), inp["party_offsets"])
    return mo.top_margin(z, shape.top_k)


def decided_seed(shape, max_tries: int = 400) -> int:
    tol = logit_tol(shape.d_model)
    for s in range(shape.seed, shape.seed + max_tries):
        inp = mi.make_inputs(shape, seed=s, with_weights=False)
        if shape.n_experts == shape.top_k or margins(shape, inp).min() > 2 * tol:
            return s
    raise RuntimeError(f"no decided seed for {shape.name} in {max_tries} tries")
