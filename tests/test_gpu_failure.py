"""Failure detection on the GPU without faulting it: every mbarrier wait in the
tensor-core kernels is bounded in time. With a 1 ns limit the waits run out, the
kernels record MOE_ERR_TIMEOUT, drain their in-flight copies and MMAs, free TMEM and
return; the same CUDA context then computes correct results again."""
import numpy as np
import pytest
import torch

from oracle import moe_oracle as mo
from synth import moe_inputs as mi
from tests._cmp import TOL, assert_close
from tests.gpu_util import cfg_of, dev, empty, need_gpu, status
from tests.test_gpu_dispatch_combine import picks

pytestmark = pytest.mark.gpu


def _ffn_fwd(L, T=512, d=256, E=4, F=256, k=2):
    idx = picks(T, E, k, "uniform", seed=5)
    counts, off, slot, tok = mo.dispatch_tables(idx, E)
    rng = np.random.default_rng(9)
    x = mi.bf16_round(rng.standard_normal((T, d)).astype(np.float32))
    w1 = mi.bf16_round((rng.standard_normal((E, 2 * F, d)) * 0.05).astype(np.float32))
    w2 = mi.bf16_round((rng.standard_normal((E, d, F)) * 0.05).astype(np.float32))
    sh = mi.MoEShape("f", T, d, E, F, k, "bf16")
    cfg = cfg_of(L, sh)
    TK = T * k
    h, a, y = empty((TK, 2 * F), torch.bfloat16), empty((TK, F), torch.bfloat16), empty((TK, d), torch.bfloat16)
    L.moe_expert_ffn_fwd(cfg, dev(x[tok], torch.bfloat16), dev(off, torch.int32), dev(w1, torch.bfloat16),
                         dev(w2, torch.bfloat16), h, a, y)
    ref = np.zeros((TK, d))
    for e in range(E):
        r = slice(off[e], off[e + 1])
        ref[r] = mo.swiglu_forward(x[tok][r], w1[e], w2[e])[3]
    return y, ref


def test_bounded_wait_timeout_is_reported_and_context_survives():
    L = need_gpu()
    assert status(L) == 0
    L.moe_set_wait_limit_ns(1)
    try:
        # a long contraction (d = 8192, 128 k-blocks per tile): the epilogue's wait for
        # the first accumulator lasts tens of microseconds and runs out
        _ffn_fwd(L, T=256, d=8192, E=2, F=256, k=1)
        code = status(L)
    finally:
        L.moe_set_wait_limit_ns(2_000_000_000)
    assert code == L.MOE_ERR_TIMEOUT
    # the context is intact: the same call now succeeds and matches the oracle
    y, ref = _ffn_fwd(L)
    assert status(L) == 0
    assert_close("y", y, ref, TOL["bf16"])
