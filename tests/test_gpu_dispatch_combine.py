"""GPU dispatch (histogram, offsets, stable slots, gather), combine and their backward
against the oracle, on oracle-made routing tables; planted bad indices must come back
as MOE_ERR_DEVICE_CHECK (the kernels check bounds, nothing faults)."""
import numpy as np
import pytest
import torch

from oracle import moe_oracle as mo
from synth import moe_inputs as mi
from tests._cmp import assert_close, ints
from tests.gpu_util import cfg_of, dev, empty, need_gpu, status

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    return need_gpu()


def picks(T, E, k, pattern, seed=0):
    rng = np.random.default_rng(seed)
    if pattern == "uniform":
        return np.stack([rng.permutation(E)[:k] for _ in range(T)]).astype(np.int32)
    if pattern == "skewed":  # expert 0 (and 1..k-1) in almost every token, last expert unused
        out = []
        for _ in range(T):
            if rng.random() < 0.9:
                out.append(np.arange(k))
            else:
                out.append(rng.permutation(E - 1)[:k])
        return np.asarray(out, np.int32)
    if pattern == "all":  # k == E
        return np.stack([rng.permutation(E) for _ in range(T)]).astype(np.int32)
    if pattern == "edges":  # k == 1: expert sizes at the 16- and 64-row boundaries
        sizes = np.array(EDGE_SIZES[:E])
        assert k == 1 and sizes.sum() == T
        return rng.permutation(np.repeat(np.arange(E), sizes)).astype(np.int32)[:, None]
    raise ValueError(pattern)


# rows per expert around the K=16 MMA step and the 64- and 128-row k-blocks (empty, one
# row, ...)
EDGE_SIZES = [0, 1, 15, 16, 17, 63, 64, 65, 127, 128, 129, 200, 255, 256, 257]


CASES = [(1000, 8, 2, "uniform", "bf16"), (333, 16, 2, "skewed", "bf16"),
         (4096, 64, 6, "uniform", "bf16"), (129, 4, 4, "all", "f32"), (1, 1, 1, "all", "f32"),
         (517, 32, 8, "uniform", "f32")]


@pytest.mark.parametrize("T,E,k,pattern,dtype", CASES)
def test_dispatch_tables_bit_exact(L, T, E, k, pattern, dtype):
    d = 256
    idx = picks(T, E, k, pattern, seed=T + E)
    sh = mi.MoEShape("d", T, d, E, 256, k, dtype)
    cfg = cfg_of(L, sh)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    x = mi.bf16_round(np.random.default_rng(1).standard_normal((T, d)).astype(np.float32))
    ws = L.moe_workspace_size(cfg)
    wsb = torch.empty(ws, dtype=torch.uint8, device="cuda")
    offsets, slot_of, token_of = empty((E + 1,), torch.int32), empty((T * k,), torch.int32), empty((T * k,), torch.int32)
    xp = empty((T * k, d), dt)
    L.moe_dispatch(cfg, dev(idx, torch.int32), dev(x, dt), offsets, slot_of, token_of, xp, wsb, ws)
    assert status(L) == 0
    counts, off, slot, tok = mo.dispatch_tables(idx, E)
    assert (ints(offsets) == off).all()
    assert (ints(slot_of) == slot.ravel()).all()
    assert (ints(token_of) == tok).all()
    assert (xp.float().cpu().numpy() == x[tok]).all()  # a copy: bit-exact


OWNER_CASES = [(1000, 8, 2, 2, "uniform"), (999, 32, 2, 3, "uniform"), (333, 6, 2, 4, "skewed"),
               (4096, 64, 6, 8, "uniform"), (512, 16, 2, 1, "uniform"), (0, 8, 2, 2, "uniform")]


@pytest.mark.parametrize("T,E,k,P,pattern", OWNER_CASES)
def test_owner_dispatch_tables_bit_exact(L, T, E, k, P, pattern):
    """Owner-grouped dispatch: segment order, offsets, slots, token map, the permuted
    copy and the per-(source, owner) send counts against the oracle, bit for bit (P = 1
    gives the expert-major tables; T = 0 still writes the order and zero counts)."""
    d = 256
    idx = picks(T, E, k, pattern, seed=T + E + P) if T else np.zeros((0, k), np.int32)
    sh = mi.MoEShape("o", T, d, E, 256, k, "bf16", n_parties=P)
    cfg = cfg_of(L, sh)
    x = mi.bf16_round(np.random.default_rng(2).standard_normal((max(T, 1), d)).astype(np.float32))[:T]
    po = np.asarray([T * p // P for p in range(P + 1)], np.int32)
    ws = L.moe_workspace_size(cfg)
    wsb = torch.empty(ws, dtype=torch.uint8, device="cuda")
    ge, offsets = empty((E,), torch.int32), empty((E + 1,), torch.int32)
    slot_of, token_of = empty((max(T * k, 1),), torch.int32), empty((max(T * k, 1),), torch.int32)
    xp, send = empty((max(T * k, 1), d), torch.bfloat16), empty((P, P), torch.int32)
    L.moe_dispatch_owner(cfg, dev(idx, torch.int32) if T else None, dev(x, torch.bfloat16) if T else None,
                         dev(po, torch.int32), ge, offsets, slot_of if T else None,
                         token_of if T else None, xp if T else None, send, wsb, ws)
    assert status(L) == 0
    rge, counts, off, slot, tok, rsend = mo.owner_dispatch_tables(idx, E, po)
    assert (ints(ge) == rge).all()
    assert (ints(offsets) == off).all()
    assert (ints(send) == rsend).all()
    if T:
        assert (ints(slot_of) == slot.ravel()).all()
        assert (ints(token_of) == tok).all()
        assert (xp.float().cpu().numpy() == x[tok]).all()


def test_dispatch_detects_bad_index(L):
    T, E, k, d = 300, 8, 2, 128
    idx = picks(T, E, k, "uniform")
    idx[17, 1] = E          # out of range
    idx[40, 1] = idx[40, 0]  # duplicate pick
    sh = mi.MoEShape("d", T, d, E, 128, k, "f32")
    cfg = cfg_of(L, sh)
    ws = L.moe_workspace_size(cfg)
    wsb = torch.empty(ws, dtype=torch.uint8, device="cuda")
    xp = torch.zeros(T * k, d, device="cuda")
    token_of = torch.zeros(T * k, dtype=torch.int32, device="cuda")
    L.moe_dispatch(cfg, dev(idx, torch.int32), torch.zeros(T, d, device="cuda"),
                   empty((E + 1,), torch.int32), empty((T * k,), torch.int32), token_of, xp, wsb, ws)
    assert status(L) == L.MOE_ERR_DEVICE_CHECK
    assert status(L) == 0  # cleared by the read


def _tables(T, E, k, seed):
    idx = picks(T, E, k, "uniform", seed)
    return (idx,) + mo.dispatch_tables(idx, E)


@pytest.mark.parametrize("T,E,k,S,dtype", [(700, 8, 2, 0, "bf16"), (300, 16, 6, 2, "bf16"),
                                           (512, 8, 2, 1, "f32")])
def test_combine_fwd_bwd(L, T, E, k, S, dtype):
    d = 384
    idx, counts, off, slot, tok = _tables(T, E, k, 3)
    rng = np.random.default_rng(4)
    rnd = (lambda *s: mi.bf16_round(rng.standard_normal(s).astype(np.float32))) if dtype == "bf16" \
        else (lambda *s: rng.standard_normal(s).astype(np.float32))
    y, ysh, dout = rnd(T * k, d), rnd(S, T, d), rnd(T, d)
    w = rng.random((T, k)).astype(np.float32)
    sh = mi.MoEShape("c", T, d, E, 256, k, dtype, n_shared=S, d_ff_shared=128 if S else 0)
    cfg = cfg_of(L, sh)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    out = empty((T, d), dt)
    slot_d = dev(slot.ravel(), torch.int32)
    L.moe_combine_fwd(cfg, dev(y, dt), dev(w, torch.float32), slot_d, dev(ysh, dt) if S else None, out)
    dy, dw = empty((T * k, d), dt), empty((T, k), torch.float32)
    L.moe_combine_bwd(cfg, dev(dout, dt), dev(y, dt), dev(w, torch.float32), slot_d, dy, dw)
    assert status(L) == 0
    ref = mo.combine(y.astype(np.float64), w.astype(np.float64), slot) + ysh.astype(np.float64).sum(0)
    tol = 1e-5 if dtype == "f32" else 8e-3  # bf16 output rounding
    assert_close("out", out, ref, tol)
    rdy, rdw = mo.combine_backward(dout, y.astype(np.float64), w.astype(np.float64), slot)
    assert_close("dy", dy, rdy, tol)
    assert_close("dw", dw, rdw, 1e-5)


@pytest.mark.parametrize("T,E,k,P,S,dtype", [(700, 8, 2, 1, 0, "bf16"), (400, 32, 2, 4, 0, "bf16"),
                                             (300, 64, 6, 1, 2, "bf16"), (256, 8, 2, 2, 1, "f32")])
def test_unpermute_reduce_with_router_grad(L, T, E, k, P, S, dtype):
    """dx = the k permuted rows of each token + the router's share + the shared experts'."""
    d = 512
    idx, counts, off, slot, tok = _tables(T, E, k, 5)
    rng = np.random.default_rng(6)
    rnd = (lambda *s: mi.bf16_round(rng.standard_normal(s).astype(np.float32))) if dtype == "bf16" \
        else (lambda *s: rng.standard_normal(s).astype(np.float32))
    dxp, dxsh, dxr = rnd(T * k, d), rnd(S, T, d), rnd(T, d)
    sh = mi.MoEShape("u", T, d, E, 256, k, dtype, n_parties=P, n_shared=S, d_ff_shared=128 if S else 0)
    cfg = cfg_of(L, sh)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    for with_router in (True, False):
        dx = empty((T, d), dt)
        L.moe_dispatch_bwd(cfg, dev(dxp, dt), dev(slot.ravel(), torch.int32),
                           dev(dxr, dt) if with_router else None, dev(dxsh, dt) if S else None, dx)
        assert status(L) == 0
        ref = mo.unpermute_reduce(dxp.astype(np.float64), slot) + dxsh.astype(np.float64).sum(0)
        if with_router:
            ref += dxr.astype(np.float64)
        assert_close("dx", dx, ref, 1e-5 if dtype == "f32" else 8e-3)


def test_combine_detects_bad_slot(L):
    T, E, k, d = 64, 4, 2, 128
    idx, counts, off, slot, tok = _tables(T, E, k, 7)
    slot = slot.copy()
    slot[3, 1] = -5
    slot[9, 0] = T * k
    sh = mi.MoEShape("c", T, d, E, 128, k, "f32")
    cfg = cfg_of(L, sh)
    y = torch.zeros(T * k, d, device="cuda")
    L.moe_combine_fwd(cfg, y, torch.ones(T, k, device="cuda"), dev(slot.ravel(), torch.int32), None,
                      torch.empty(T, d, device="cuda"))
    assert status(L) == L.MOE_ERR_DEVICE_CHECK
