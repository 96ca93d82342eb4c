"""The bench's roofline accounting (host only): the algorithmic bytes of the memory-bound
calls and the flops of the expert GEMMs per step, for every workload.

Bytes per token, b bytes per element: gating reads x (d b) and writes probabilities and
picks (4E + 8k); dispatch reads x and writes its k rows (d b + k d b) plus ~12k of
tables; the combine reads k rows and gate weights and writes one row; its backward reads
dOut and the k rows and writes k rows and k gate gradients; the router backward reads
probabilities and their gradients (8E) and x, and writes dx_router; the unpermute-reduce
reads k rows and writes one. The aux loss reads the probabilities (4E). Shared experts
add a row read to the combine and a row read to the unpermute-reduce. The expert GEMMs
are 18 d F flops per routed row (plus 18 d Fs per token and shared expert).
"""
import pytest

import bench
from synth import moe_inputs as mi

# workload: (total algorithmic MB of the memory-bound calls without shared-expert rows,
# expert-GEMM TFLOP per step)
PUBLISHED = {"mid_bf16": (152, 0.425), "fine_bf16": (1290, 3.40), "large_zipf_bf16": (2420, 34.6),
             "party4_bf16": (1220, 6.80)}


@pytest.mark.parametrize("name", sorted(PUBLISHED))
def test_stage_bytes_and_flops(name):
    sh = mi.shape_by_name(name)
    b = 2 if sh.dtype == "bf16" else 4
    T, d, E, k, S = sh.T, sh.d_model, sh.n_experts, sh.top_k, sh.n_shared
    per = bench.stage_bytes(sh)
    assert per["route"] == T * (d * b + 4 * E + 8 * k)
    assert per["aux"] == T * 4 * E
    assert per["dispatch"] == T * (d * b + k * d * b + 12 * k)
    assert per["combine_fwd"] == T * (k * d * b + 4 * k + S * d * b + d * b)
    assert per["combine_bwd"] == T * (d * b + 2 * k * d * b + 4 * k)
    assert per["route_bwd"] == T * (8 * E + 3 * d * b)
    assert per["dispatch_bwd"] == T * (k * d * b + S * d * b + d * b)
    total = bench.mem_bytes_per_step(sh)
    assert total == sum(per.values())
    mb, tflop = PUBLISHED[name]
    shared_rows = 2 * S * d * b * T
    assert abs((total - shared_rows) / 1e6 - mb) <= 0.01 * mb
    assert abs(sh.gemm_flops() / 1e12 - tflop) <= 0.01 * tflop
    assert sh.gemm_flops() == 18.0 * d * (sh.d_ff * T * k + sh.d_ff_shared * T * S)
