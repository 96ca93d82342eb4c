"""moe_dispatch_noalloc: the dispatch entry point for callers that cannot allocate.

Some callers are given only input and output buffers by their host framework (an op
or plugin interface without scratch memory) and cannot call cudaMalloc for the
workspace moe_dispatch needs. moe_dispatch_noalloc keeps that scratch in a fixed
array inside the library. These tests call it through the C ABI and check that its
tables and permuted rows equal those of moe_dispatch on the same inputs, exactly
(integer and copy work), on two calls in a row, and that sizes beyond its fixed
scratch are refused on the host. The tables are also checked directly against the
oracle's dispatch tables (counting, prefix sums and stable slots written out on the CPU).
"""
import numpy as np
import pytest

from oracle import moe_oracle as mo
from synth import moe_inputs as mi
from tests.gpu_util import cfg_of, dev, empty, need_gpu, status

pytestmark = pytest.mark.gpu


def _picks(T, E, k, seed):
    rng = np.random.default_rng(seed)
    return np.stack([rng.permutation(E)[:k] for _ in range(T)]).astype(np.int32)


def _both(L, T, d, E, k, dtype, seed):
    import torch
    sh = mi.MoEShape("na", T, d, E, 128, k, dtype)
    cfg = cfg_of(L, sh)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    picks = _picks(T, E, k, seed)
    xs = np.random.default_rng(seed + 1).standard_normal((T, d)).astype(np.float32)
    idx = dev(picks, torch.int32)
    x = dev(xs, dt)
    ws = L.moe_workspace_size(cfg)
    wsb = torch.empty(ws, dtype=torch.uint8, device="cuda")
    out = []
    for use_ws in (True, False):
        tabs = (empty((E + 1,), torch.int32), empty((T * k,), torch.int32),
                empty((T * k,), torch.int32), empty((T * k, d), dt))
        if use_ws:
            L.moe_dispatch(cfg, idx, x, *tabs, wsb, ws)
        else:
            L.moe_dispatch_noalloc(cfg, idx, x, *tabs)
        out.append(tabs)
    assert status(L) == 0
    return out, picks, x


@pytest.mark.parametrize("T,d,E,k,dtype", [(4096, 1024, 16, 2, "bf16"), (1000, 256, 64, 6, "f32")])
def test_noalloc_dispatch_matches_workspace_dispatch_twice(T, d, E, k, dtype):
    import torch
    L = need_gpu()
    for call, seed in enumerate((11, 12)):  # two calls in a row share the fixed scratch
        (ref, got), picks, x = _both(L, T, d, E, k, dtype, seed)
        for name, a, b in zip(("offsets", "slot_of", "token_of", "x_perm"), ref, got):
            assert torch.equal(a, b), (call, name)
        _, off, slot, tok = mo.dispatch_tables(picks, E)
        assert (got[0].cpu().numpy() == off).all(), call
        assert (got[1].cpu().numpy() == slot.ravel()).all(), call
        assert (got[2].cpu().numpy() == tok).all(), call
        assert torch.equal(got[3], x[torch.as_tensor(tok, device="cuda")]), call


def test_noalloc_dispatch_refuses_sizes_beyond_its_scratch():
    L = need_gpu()
    sh = mi.MoEShape("big", 131072 + 128, 128, 64, 128, 2, "bf16")
    cfg = cfg_of(L, sh)
    with pytest.raises(L.MoEError) as ei:
        L.moe_dispatch_noalloc(cfg, 16, 16, 16, 16, 16, 16)
    assert ei.value.status == L.MOE_ERR_INVALID_ARG
    assert "fixed scratch" in L.moe_last_error()
