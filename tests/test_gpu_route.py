"""GPU gating (Alg. 7) against the oracle: picks and counts bit-exact on identical fp32
logits (planted ties included), logits within the fp32 accumulation tolerance, and the
per-party aux loss."""
import numpy as np
import pytest
import torch

from oracle import moe_oracle as mo
from oracle import seeds
from synth import moe_inputs as mi
from tests._cmp import assert_close, ints
from tests.gpu_util import cfg_of, dev, empty, need_gpu, status

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    return need_gpu()


def uneven_parties(T, P):
    if P == 1:
        return np.array([0, T], np.int32)
    cuts = sorted(np.random.default_rng(T + P).choice(np.arange(1, T), P - 1, replace=False))
    return np.array([0, *cuts, T], np.int32)


@pytest.mark.parametrize("T,E,k,P,norm", [
    (1000, 8, 2, 1, 0), (777, 16, 2, 1, 1), (513, 64, 6, 1, 0), (300, 4, 4, 1, 0),
    (1024, 32, 2, 4, 0), (5, 3, 1, 1, 0), (129, 64, 8, 3, 1), (1, 2, 2, 1, 0),
    # wide expert pools: lanes hold 4 or 8 experts; P E beyond the shared histogram
    (600, 100, 6, 2, 0), (333, 256, 8, 1, 1), (200, 256, 2, 20, 0)])
def test_route_from_logits_bit_exact(L, T, E, k, P, norm):
    z = mi.make_route_logits(T, E, seed=T * 7 + E, tie_every=3)
    po = uneven_parties(T, P)
    sh = mi.MoEShape("r", T, 128, E, 128, k, "f32", n_parties=P, normalize_topk=norm)
    cfg = cfg_of(L, sh)
    zd = dev(z, torch.float32)
    probs, w = empty((T, E), torch.float32), empty((T, k), torch.float32)
    idx, counts = empty((T, k), torch.int32), empty((P, E), torch.int32)
    pod = dev(po, torch.int32) if P > 1 else None
    L.moe_route_from_logits(cfg, zd, pod, probs, idx, w, counts)
    assert status(L) == 0
    ref_idx = mo.topk_indices(z, k)
    assert (ints(idx) == ref_idx).all()
    assert (ints(counts) == mo.party_counts(ref_idx, E, po)).all()
    p = mo.softmax(z.astype(np.float64))
    assert_close("probs", probs, p, 1e-6)
    assert_close("topk_w", w, mo.gate_weights(p, ref_idx, norm), 1e-6)


@pytest.mark.parametrize("which,T,extra", [
    (1, None, {}), (2, None, {}), (5, 2048, {}), (4, 1024, {}), (3, 1024, {}),
    # 128 tiles, more than one per CTA on some SMs
    (2, 16384, {}),
    # d = 384 (6 k-blocks), three parties of 233 tokens: ragged tiles that end mid-party
    (2, 699, {"d_model": 384, "n_experts": 8, "n_parties": 3}),
    # E = 32 (N = 32), a single partial tile
    (2, 77, {"n_experts": 32}),
    # wide expert pools on the tensor cores (the gating epilogue reads TMEM in chunks):
    # E = 128, E = 130 (scalar stores) with three parties, E = 256
    (2, 700, {"n_experts": 128, "top_k": 6, "d_model": 256}),
    (2, 513, {"n_experts": 130, "top_k": 3, "d_model": 256, "n_parties": 3}),
    (2, 300, {"n_experts": 256, "top_k": 8, "d_model": 128}),
    # fp32 with E > 64: the router products by the CUDA-core GEMM, then the gating
    (1, 300, {"n_experts": 96, "top_k": 4}),
    (1, 257, {"n_experts": 256, "top_k": 8, "n_parties": 1})])
def test_route_matches_oracle(L, which, T, extra):
    """The tensor-core gating (router GEMM with the gating in its epilogue) against the
    fp64 oracle: logits within the accumulation tolerance, picks and counts exact."""
    sh = mi.SHAPES[which]
    if T:
        sh = sh.with_(T=T, **extra)
    sh = sh.with_(seed=seeds.decided_seed(sh))
    inp = mi.make_inputs(sh, with_weights=False)
    dt = torch.bfloat16 if sh.dtype == "bf16" else torch.float32
    Tn, E, k, P = sh.T, sh.n_experts, sh.top_k, sh.n_parties
    cfg = cfg_of(L, sh)
    x, wr = dev(inp["x"], dt), dev(inp["w_router"], dt)
    bias = dev(inp["router_bias"], torch.float32) if inp["router_bias"] is not None else None
    po = dev(inp["party_offsets"], torch.int32) if P > 1 else None
    logits, probs = empty((Tn, E), torch.float32), empty((Tn, E), torch.float32)
    idx, w, counts = empty((Tn, k), torch.int32), empty((Tn, k), torch.float32), empty((P, E), torch.int32)
    L.moe_route(cfg, x, wr, bias, po, logits, probs, idx, w, counts)
    assert status(L) == 0
    ref = mo.route_all(inp, sh)
    err = np.abs(logits.double().cpu().numpy() - ref["logits"])
    assert (err <= seeds.logit_tol(ref["logits"], sh.d_model)).all(), err.max()
    assert (ints(idx) == ref["topk_idx"]).all()
    assert (ints(counts) == ref["party_counts"]).all()
    assert_close("probs", probs, ref["probs"], 1e-4)
    assert_close("topk_w", w, ref["topk_w"], 1e-4)


@pytest.mark.parametrize("P", [1, 4])
def test_aux_loss_matches_oracle(L, P):
    T, E, k = 1024, 16, 2
    rng = np.random.default_rng(P)
    p = mo.softmax(rng.standard_normal((T, E)) * 2)
    idx = mo.topk_indices(np.log(p).astype(np.float32), k)
    po = uneven_parties(T, P)
    cpe = mo.party_counts(idx, E, po)
    loss, coef = mo.aux_loss(p, cpe, po, k, 0.37)
    sh = mi.MoEShape("a", T, 128, E, 128, k, "f32", n_parties=P, aux_alpha=0.37)
    cfg = cfg_of(L, sh)
    gl, gc = empty((P,), torch.float32), empty((P, E), torch.float32)
    L.moe_aux_loss(cfg, dev(p, torch.float32), dev(cpe, torch.int32),
                   dev(po, torch.int32) if P > 1 else None, gl, gc)
    assert status(L) == 0
    assert_close("loss", gl, loss, 1e-5)
    assert_close("coef", gc, coef, 1e-6)
