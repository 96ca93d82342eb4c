"""Workload shapes and seeded random inputs for the MoE expert layer.

Shapes
------
The five workloads are the layer shapes the throughput and parity runs use:

=====================  =====  =====  ===  =====  ==  ===================================
name                   T      d      E    F      k   notes
=====================  =====  =====  ===  =====  ==  ===================================
tiny_f32               512    256    8    512    2   fp32 everywhere
mid_bf16               4096   1024   16   2816   2   bf16 storage, fp32 accumulation
fine_bf16              8192   2048   64   1408   6   + 2 always-on shared experts (F=1408)
large_zipf_bf16        16384  4096   8    14336  2   router bias gives Zipf(1.2) popularity
party4_bf16            16384  2048   32   5632   2   4 parties x 4096 tokens, one router each
=====================  =====  =====  ===  =====  ==  ===================================

Draw recipe (one ``numpy.random.Generator(PCG64(seed))`` per call, in this order):
x ~ N(0,1) [T,d]; router weights ~ N(0,0.02) [P,E,d]; (Zipf shapes) a random
permutation of expert ranks; W1 ~ N(0,0.02) [E,2F,d] drawn expert by expert;
W2 ~ N(0,0.02) [E,d,F] expert by expert; shared W1s, W2s likewise; upstream
gradient dOut ~ N(0,1) [T,d]. Every draw is float32; for bf16 shapes each value
is then rounded to the nearest bf16 (ties to even), and the rounded values are the
inputs of both the oracle and the GPU path. Default seed = 1000 + workload number.

The Zipf router bias is b_e = -ZIPF_BIAS_SCALE * s * ln(rank_e) with rank_e a
seeded permutation of 1..E, identical for every party. ZIPF_BIAS_SCALE was fitted
once by ``oracle/calibrate_zipf.py`` so that the realised top-2 assignment
fractions of the seeded tokens lie close to rank^-1.2 (normalised).
"""
from __future__ import annotations

from dataclasses import dataclass, replace

import numpy as np

# Fitted by oracle/calibrate_zipf.py (see module docstring); an input constant.
ZIPF_BIAS_SCALE = 1.248


@dataclass(frozen=True)
class MoEShape:
    name: str
    T: int
    d_model: int
    n_experts: int
    d_ff: int
    top_k: int
    dtype: str  # "f32" or "bf16"
    n_parties: int = 1
    n_shared: int = 0
    d_ff_shared: int = 0
    zipf_s: float = 0.0
    normalize_topk: int = 0
    aux_alpha: float = 0.01
    seed: int = 1000

    @property
    def TK(self) -> int:
        return self.T * self.top_k

    @property
    def has_bias(self) -> bool:
        return self.zipf_s > 0.0

    def with_(self, **kw) -> "MoEShape":
        return replace(self, **kw)

    def gemm_flops(self) -> float:
        """Dense-contraction flops of one fwd+bwd of the expert FFNs (18*d*F per row)."""
        f = 18.0 * self.d_model * self.d_ff * self.TK
        f += 18.0 * self.d_model * self.d_ff_shared * self.T * self.n_shared
        return f


SHAPES = {
    1: MoEShape("tiny_f32", 512, 256, 8, 512, 2, "f32", seed=1001),
    2: MoEShape("mid_bf16", 4096, 1024, 16, 2816, 2, "bf16", seed=1002),
    3: MoEShape("fine_bf16", 8192, 2048, 64, 1408, 6, "bf16",
                n_shared=2, d_ff_shared=1408, seed=1003),
    4: MoEShape("large_zipf_bf16", 16384, 4096, 8, 14336, 2, "bf16",
                zipf_s=1.2, seed=1004),
    5: MoEShape("party4_bf16", 16384, 2048, 32, 5632, 2, "bf16",
                n_parties=4, seed=1005),
}


def shape_by_name(name: str) -> MoEShape:
    for s in SHAPES.values():
        if s.name == name:
            return s
    raise KeyError(name)


def bf16_round(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) & np.uint32(0xFFFF0000)
    return r.view(np.float32)


def party_offsets(shape: MoEShape) -> np.ndarray:
    """Token ranges of the parties: party p owns tokens [po[p], po[p+1])."""
    P = shape.n_parties
    if shape.T % P:
        raise ValueError("T must split evenly over the parties")
    return (np.arange(P + 1, dtype=np.int64) * (shape.T // P)).astype(np.int32)


def _normal(rng, shape, scale, dtype):
    a = rng.standard_normal(shape, dtype=np.float32)
    if scale != 1.0:
        a *= np.float32(scale)
    return bf16_round(a) if dtype == "bf16" else a


def make_inputs(shape: MoEShape, seed: int | None = None, with_weights: bool = True) -> dict:
    """Seeded inputs of one layer call (float32 arrays; bf16-representable for bf16 shapes)."""
    seed = shape.seed if seed is None else seed
    rng = np.random.default_rng(seed)
    T, d, E, F, P = shape.T, shape.d_model, shape.n_experts, shape.d_ff, shape.n_parties
    dt = shape.dtype
    out = {"seed": seed}
    out["x"] = _normal(rng, (T, d), 1.0, dt)
    out["w_router"] = _normal(rng, (P, E, d), 0.02, dt)
    if shape.has_bias:
        ranks = rng.permutation(E).astype(np.float64) + 1.0
        b = -ZIPF_BIAS_SCALE * shape.zipf_s * np.log(ranks)
        out["router_bias"] = np.tile(b.astype(np.float32), (P, 1))
        out["zipf_rank"] = ranks.astype(np.int32)
    else:
        out["router_bias"] = None
    out["party_offsets"] = party_offsets(shape)
    if with_weights:
        w1 = np.empty((E, 2 * F, d), np.float32)
        for e in range(E):
            w1[e] = _normal(rng, (2 * F, d), 0.02, dt)
        w2 = np.empty((E, d, F), np.float32)
        for e in range(E):
            w2[e] = _normal(rng, (d, F), 0.02, dt)
        out["w1"], out["w2"] = w1, w2
        S, Fs = shape.n_shared, shape.d_ff_shared
        if S:
            ws1 = np.empty((S, 2 * Fs, d), np.float32)
            for s in range(S):
                ws1[s] = _normal(rng, (2 * Fs, d), 0.02, dt)
            ws2 = np.empty((S, d, Fs), np.float32)
            for s in range(S):
                ws2[s] = _normal(rng, (d, Fs), 0.02, dt)
            out["ws1"], out["ws2"] = ws1, ws2
        else:
            out["ws1"] = out["ws2"] = None
    out["dout"] = _normal(rng, (T, d), 1.0, dt)
    return out


def make_route_logits(T: int, E: int, seed: int, tie_every: int = 7) -> np.ndarray:
    """fp32 router logits with exact ties planted on purpose.

    Rows are N(0,1). Every ``tie_every``-th row copies one logit onto another
    expert (an exact tie at a random rank); every ``3*tie_every``-th row is
    constant (all experts tied); every ``5*tie_every``-th row repeats a value
    across a block of experts around the middle rank.
    """
    rng = np.random.default_rng(seed)
    z = rng.standard_normal((T, E), dtype=np.float32)
    for t in range(0, T, tie_every):
        a, b = rng.choice(E, size=2, replace=False)
        z[t, b] = z[t, a]
    for t in range(1, T, 3 * tie_every):
        z[t, :] = np.float32(0.25)
    for t in range(2, T, 5 * tie_every):
        lo = max(0, E // 2 - 2)
        z[t, lo:lo + min(4, E)] = z[t, lo]
    return z


# ----------------------------------------------------------------------------- training
def party_schedule(n_parties: int, epochs: int, seed: int) -> list:
    """The order in which the parties take their turns: one seeded random permutation
    of 0..n-1 per epoch (the RandomPermutation of Alg. 1), drawn from one generator."""
    rng = np.random.default_rng(seed)
    return [rng.permutation(n_parties).astype(np.int64).tolist() for _ in range(epochs)]


def train_batches(shape: MoEShape, n_parties: int, n_batches: int, seed: int) -> list:
    """Each party's private data D_i: ``n_batches`` batches of shape.T tokens, as
    [(x, y), ...] per party. x ~ N(0,1); the regression target is a fixed random
    linear map of x, y = x R / sqrt(d) with R ~ N(0,1) [d,d] shared by all parties
    (one teacher, so the parties' objectives agree). float32, bf16-rounded for bf16
    shapes. Draw order: R, then party by party, batch by batch, x then nothing else."""
    rng = np.random.default_rng(seed)
    d = shape.d_model
    R = rng.standard_normal((d, d), dtype=np.float32) / np.float32(np.sqrt(d))
    out = []
    for _ in range(n_parties):
        mine = []
        for _ in range(n_batches):
            x = _normal(rng, (shape.T, d), 1.0, shape.dtype)
            y = (x @ R).astype(np.float32)
            mine.append((x, bf16_round(y) if shape.dtype == "bf16" else y))
        out.append(mine)
    return out


def train_init(shape: MoEShape, n_parties: int, seed: int) -> dict:
    """The common initialization of Alg. 1: every party's router W_r[i] and the expert
    pool W1, W2, drawn as in ``make_inputs`` for a shape with n_parties routers."""
    inp = make_inputs(shape.with_(n_parties=n_parties, T=n_parties), seed=seed)
    return {"w_router": inp["w_router"], "w1": inp["w1"], "w2": inp["w2"]}
