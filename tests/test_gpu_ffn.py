"""GPU grouped expert GEMMs (ForwardExpert / BackwardExpert of Alg. 6) against the
oracle on oracle-made dispatch tables: ragged expert segments, empty experts, a
skewed split, many tiny experts, F not a multiple of 256, shared experts; bf16 on
the tcgen05 tensor-core kernels, fp32 on the CUDA-core kernels."""
import numpy as np
import pytest
import torch

from oracle import moe_oracle as mo
from synth import moe_inputs as mi
from tests._cmp import TOL, assert_close, assert_close_slices
from tests.gpu_util import cfg_of, dev, empty, need_gpu, status
from tests.test_gpu_dispatch_combine import picks

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    return need_gpu()


CASES = [
    # T, d, E, F, k, pattern, dtype, S, Fs
    (300, 256, 4, 256, 2, "uniform", "bf16", 0, 0),
    (777, 512, 8, 384, 2, "skewed", "bf16", 0, 0),
    (1024, 1024, 16, 2816, 2, "uniform", "bf16", 0, 0),
    (256, 256, 2, 128, 1, "uniform", "bf16", 2, 256),
    (64, 128, 64, 128, 6, "uniform", "bf16", 0, 0),
    (512, 256, 8, 512, 2, "uniform", "f32", 0, 0),
    (100, 64, 3, 96, 2, "skewed", "f32", 1, 40),
]


@pytest.mark.parametrize("case", CASES, ids=[f"{c[6]}-T{c[0]}-d{c[1]}-E{c[2]}-F{c[3]}-k{c[4]}-{c[5]}-S{c[7]}" for c in CASES])
def test_expert_ffn_fwd_bwd(L, case):
    T, d, E, F, k, pattern, dtype, S, Fs = case
    rng = np.random.default_rng(T + d + E)
    rnd = ((lambda s, sc=1.0: mi.bf16_round((rng.standard_normal(s) * sc).astype(np.float32)))
           if dtype == "bf16" else (lambda s, sc=1.0: (rng.standard_normal(s) * sc).astype(np.float32)))
    idx = picks(T, E, k, pattern, seed=T)
    counts, off, slot, tok = mo.dispatch_tables(idx, E)
    x = rnd((T, d))
    w1, w2 = rnd((E, 2 * F, d), 0.05), rnd((E, d, F), 0.05)
    dy = rnd((T * k, d))
    ws1, ws2, dout = (rnd((S, 2 * Fs, d), 0.05), rnd((S, d, Fs), 0.05), rnd((T, d))) if S else (None,) * 3
    xp = x[tok]
    sh = mi.MoEShape("f", T, d, E, F, k, dtype, n_shared=S, d_ff_shared=Fs)
    cfg = cfg_of(L, sh)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    TK = T * k
    g = {n: empty(s, dt) for n, s in dict(h_gu=(TK, 2 * F), act=(TK, F), y=(TK, d), dh=(TK, 2 * F),
                                          dxp=(TK, d), dw1=(E, 2 * F, d), dw2=(E, d, F)).items()}
    if S:
        g.update({n: empty(s, dt) for n, s in dict(h_sh=(S, T, 2 * Fs), a_sh=(S, T, Fs), y_sh=(S, T, d),
                                                     dh_sh=(S, T, 2 * Fs), dx_sh=(S, T, d),
                                                     dws1=(S, 2 * Fs, d), dws2=(S, d, Fs)).items()})
    gs = lambda n: g.get(n)  # noqa: E731
    xd, offd = dev(x, dt), dev(off, torch.int32)
    xpd, w1d, w2d = dev(xp, dt), dev(w1, dt), dev(w2, dt)
    ws1d, ws2d = (dev(ws1, dt), dev(ws2, dt)) if S else (None, None)
    doutd = dev(dout, dt) if S else None
    L.moe_expert_ffn_fwd(cfg, xpd, offd, w1d, w2d, g["h_gu"], g["act"], g["y"], xd if S else None,
                         ws1d, ws2d, gs("h_sh"), gs("a_sh"), gs("y_sh"))
    L.moe_expert_ffn_bwd(cfg, xpd, offd, w1d, w2d, g["h_gu"], g["act"], dev(dy, dt), g["dh"], g["dxp"],
                         g["dw1"], g["dw2"], xd if S else None, doutd, ws1d, ws2d, gs("h_sh"),
                         gs("a_sh"), gs("dh_sh"), gs("dx_sh"), gs("dws1"), gs("dws2"))
    assert status(L) == 0
    tol = TOL[dtype]
    ref = {n: np.zeros(s) for n, s in dict(h_gu=(TK, 2 * F), act=(TK, F), y=(TK, d), dh=(TK, 2 * F),
                                           dxp=(TK, d), dw1=(E, 2 * F, d), dw2=(E, d, F)).items()}
    for e in range(E):
        r = slice(off[e], off[e + 1])
        if off[e + 1] == off[e]:
            continue
        G, U, A, Y = mo.swiglu_forward(xp[r], w1[e], w2[e])
        ref["h_gu"][r] = np.concatenate([G, U], 1)
        ref["act"][r], ref["y"][r] = A, Y
        dH, dX, dW1, dW2 = mo.swiglu_backward(xp[r], w1[e], w2[e], G, U, A, dy[r].astype(np.float64))
        ref["dh"][r], ref["dxp"][r], ref["dw1"][e], ref["dw2"][e] = dH, dX, dW1, dW2
    for n in ref:  # weight gradients expert by expert
        (assert_close_slices if n in ("dw1", "dw2") else assert_close)(n, g[n], ref[n], tol)
    # stage by stage: every contraction and epilogue against fp64 on the GPU's own stored
    # inputs of that stage (bf16 G, U, A, dH), so only its accumulation and output
    # rounding remain: elementwise bound B = 1
    gh = {n: g[n].double().cpu().numpy() for n in ("h_gu", "act", "dh")}
    st = {n: np.zeros_like(ref[n]) for n in ("y", "dh", "dxp", "dw1", "dw2")}
    for e in range(E):
        r = slice(off[e], off[e + 1])
        if off[e + 1] == off[e]:
            continue
        G, U, A, dH = gh["h_gu"][r, :F], gh["h_gu"][r, F:], gh["act"][r], gh["dh"][r]
        st["y"][r] = A @ w2[e].astype(np.float64).T
        dA = dy[r].astype(np.float64) @ w2[e].astype(np.float64)
        sg = mo.sigmoid(G)
        st["dh"][r] = np.concatenate([dA * U * sg * (1.0 + G * (1.0 - sg)), dA * G * sg], 1)
        st["dxp"][r] = dH @ w1[e].astype(np.float64)
        st["dw1"][e] = dH.T @ xp[r].astype(np.float64)
        st["dw2"][e] = dy[r].astype(np.float64).T @ A
    for n in ("y", "dh", "dxp"):
        assert_close(n + " (stage)", g[n], st[n], tol, stage=True)
    for n in ("dw1", "dw2"):
        assert_close_slices(n + " (stage)", g[n], st[n], tol, stage=True)
    for n in ("h_gu", "act"):  # the forward's inputs are exact: the end-to-end reference is the stage's
        assert_close(n + " (stage)", g[n], ref[n], tol, stage=True)
    if pattern == "skewed":  # the last expert got no rows: exact zero weight gradients
        assert off[E] - off[E - 1] == 0
        assert (g["dw1"][E - 1] == 0).all() and (g["dw2"][E - 1] == 0).all()
    for s in range(S):
        G, U, A, Y = mo.swiglu_forward(x, ws1[s], ws2[s])
        dH, dX, dW1, dW2 = mo.swiglu_backward(x, ws1[s], ws2[s], G, U, A, dout.astype(np.float64))
        assert_close("h_sh", g["h_sh"][s], np.concatenate([G, U], 1), tol)
        assert_close("y_sh", g["y_sh"][s], Y, tol)
        assert_close("dh_sh", g["dh_sh"][s], dH, tol)
        assert_close("dx_sh", g["dx_sh"][s], dX, tol)
        assert_close("dws1", g["dws1"][s], dW1, tol)
        assert_close("dws2", g["dws2"][s], dW2, tol)


def test_expert_ffn_is_deterministic(L):
    T, d, E, F, k = 512, 256, 8, 256, 2
    rng = np.random.default_rng(0)
    idx = picks(T, E, k, "uniform")
    counts, off, slot, tok = mo.dispatch_tables(idx, E)
    sh = mi.MoEShape("f", T, d, E, F, k, "bf16")
    cfg = cfg_of(L, sh)
    dt = torch.bfloat16
    xp = dev(rng.standard_normal((T * k, d)), dt)
    w1, w2 = dev(rng.standard_normal((E, 2 * F, d)) * 0.05, dt), dev(rng.standard_normal((E, d, F)) * 0.05, dt)
    dy = dev(rng.standard_normal((T * k, d)), dt)
    offd = dev(off, torch.int32)
    outs = []
    for _ in range(2):
        b = [empty(s, dt) for s in ((T * k, 2 * F), (T * k, F), (T * k, d), (T * k, 2 * F), (T * k, d),
                                     (E, 2 * F, d), (E, d, F))]
        L.moe_expert_ffn_fwd(cfg, xp, offd, w1, w2, b[0], b[1], b[2])
        L.moe_expert_ffn_bwd(cfg, xp, offd, w1, w2, b[0], b[1], dy, b[3], b[4], b[5], b[6])
        outs.append([t.clone() for t in b])
    assert status(L) == 0
    for a, b in zip(*outs):
        assert torch.equal(a, b)


@pytest.mark.parametrize("pairs", [0, 1, 2])
def test_expert_ffn_single_cta_and_pair_tiles(L, pairs):
    """The 256-wide GEMMs in every tile mode: one CTA per 128x256 tile, a CTA pair per
    256x256 tile, or the automatic choice per launch (ragged experts, an empty expert, a
    skewed split, experts ending at every offset of a k-block; d and F of 128 mod 256, so
    that the last pair tile of dA, dW2, GEMM2, dX and dW1 along N holds 128 columns)."""
    L.moe_set_gemm_pairs(pairs)
    try:
        for case in [(777, 512, 8, 512, 2, "skewed", "bf16", 0, 0),
                     (300, 256, 4, 256, 2, "uniform", "bf16", 1, 256),
                     (1024, 1024, 16, 2816, 2, "uniform", "bf16", 0, 0),
                     (777, 384, 8, 384, 2, "skewed", "bf16", 1, 640),
                     (512, 1024, 4, 1408, 2, "skewed", "bf16", 0, 0),
                     # experts of 0, 1, 15, 16, 17, 63, 64, 65, 127, 128, 129, 200, 255, 256,
                     # 257 rows: every way the weight gradients' last k-block (64 rows, 128 for
                     # pair tiles) can end (pairs: zeroed on both CTAs)
                     (1593, 256, 15, 256, 1, "edges", "bf16", 0, 0)]:
            test_expert_ffn_fwd_bwd(L, case)
    finally:
        L.moe_set_gemm_pairs(2)
