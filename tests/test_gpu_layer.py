"""The whole layer, fwd+bwd through the C ABI, against the fp64 oracle.

Full comparisons for the tiny fp32 workload and the mid-size bf16 workload at their
own sizes, and for reduced-T versions of the fine-grained, Zipf and party workloads;
sampled comparisons (per token, per feature column) at the full sizes of those three.
Seeds are chosen by the oracle so that every compared token's routing is decided
beyond the fp32 logit tolerance (oracle.seeds)."""
import numpy as np
import pytest
import torch

from oracle import moe_oracle as mo
from oracle import seeds
from paper_2506_02965_gb300.layer import MoELayer
from synth import moe_inputs as mi
from tests._cmp import TOL, assert_close, assert_close_slices, ints, np64
from tests.gpu_util import need_gpu, status

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    return need_gpu()


def run_layer(sh, inp):
    lay = MoELayer(sh)
    lay.load(inp)
    lay.step()
    torch.cuda.synchronize()
    return lay


def full_compare(lay, inp, sh):
    tol = TOL[sh.dtype]
    fwd = mo.layer_forward(inp, sh)
    bwd = mo.layer_backward(inp, sh, fwd)
    tol_z = seeds.logit_tol(fwd["logits"], sh.d_model)
    assert (np.abs(np64(lay.logits) - fwd["logits"]) <= tol_z).all()
    # integer work: bit-exact
    assert (ints(lay.topk_idx) == fwd["topk_idx"]).all()
    assert (ints(lay.counts) == fwd["party_counts"]).all()
    rows = np.arange(sh.T * sh.top_k)  # GPU permuted row -> oracle (expert-major) row
    if lay.owner_grouped:
        ge, _, off, slot, tok, send = mo.owner_dispatch_tables(fwd["topk_idx"], sh.n_experts,
                                                              inp["party_offsets"])
        assert (ints(lay.group_expert) == ge).all()
        assert (ints(lay.send_counts) == send).all()
        rows = np.empty_like(rows)
        rows[slot.ravel()] = fwd["slot_of"].ravel()
    else:
        off, slot, tok = fwd["offsets"], fwd["slot_of"], fwd["token_of"]
    assert (ints(lay.offsets) == off).all()
    assert (ints(lay.slot_of) == slot.ravel()).all()
    assert (ints(lay.token_of) == tok).all()
    assert (np64(lay.x_perm) == fwd["x_perm"][rows]).all()
    errs = {}
    for name, gpu, ref in [
        ("probs", lay.probs, fwd["probs"]), ("topk_w", lay.topk_w, fwd["topk_w"]),
        ("h_gu", lay.h_gu, fwd["h_gu"][rows]), ("act", lay.act, fwd["act"][rows]),
        ("y_perm", lay.y_perm, fwd["y_perm"][rows]), ("out", lay.out, fwd["out"]),
        ("aux_loss", lay.aux_loss, fwd["aux_loss"]), ("aux_coef", lay.aux_coef, fwd["aux_coef"]),
        ("dy_perm", lay.dy_perm, bwd["dy_perm"][rows]), ("dtopk_w", lay.dtopk_w, bwd["dtopk_w"]),
        ("dh", lay.dh, bwd["dh"][rows]), ("dx_perm", lay.dx_perm, bwd["dx_perm"][rows]),
        ("dw1", lay.dw1, bwd["dw1"]), ("dw2", lay.dw2, bwd["dw2"]),
        ("dlogits", lay.dlogits, bwd["dlogits"]), ("dw_router", lay.dw_router, bwd["dw_router"]),
        ("dbias", lay.dbias, bwd["dbias"]), ("dx_router", lay.dx_router, bwd["dx_router"]),
        ("dx", lay.dx, bwd["dx"]),
    ]:
        per_slice = name in ("dw1", "dw2", "dw_router", "dbias")  # per expert / per party
        errs[name] = (assert_close_slices if per_slice else assert_close)(name, gpu, ref, tol)
    for s in range(sh.n_shared):
        G, U, A, Y = fwd["shared"][s]
        dH, dX, dW1, dW2 = bwd["shared_grads"][s]
        errs[f"y_sh{s}"] = assert_close("y_sh", lay.y_sh[s], Y, tol)
        errs[f"dws1_{s}"] = assert_close("dws1", lay.dws1[s], dW1, tol)
        errs[f"dws2_{s}"] = assert_close("dws2", lay.dws2[s], dW2, tol)
    return errs


def stage_compare(lay, inp, sh):
    """Every stage of the layer against fp64 on the GPU's own stored inputs of that
    stage (bf16 G, U, A, Y, dY, dH, dXp and fp32 gates as the GPU wrote them), so only
    the stage's own accumulation and output rounding remain: elementwise bound B = 1.
    Rows in the GPU's layout (expert-major or owner-grouped)."""
    tol = TOL[sh.dtype]
    bf = sh.dtype == "bf16"
    F, E, k, T = sh.d_ff, sh.n_experts, sh.top_k, sh.T
    g = {n: np64(getattr(lay, n)) for n in ("x_perm", "h_gu", "act", "y_perm", "dy_perm", "dh",
                                            "dx_perm", "topk_w", "dtopk_w", "probs", "dlogits",
                                            "dx_router")}
    off = ints(lay.offsets)
    ge = ints(lay.group_expert) if lay.owner_grouped else np.arange(E)
    slot = ints(lay.slot_of).reshape(T, k)
    w1 = np.asarray(inp["w1"], np.float64)
    w2 = np.asarray(inp["w2"], np.float64)
    dout = np.asarray(inp["dout"], np.float64)
    st = {n: np.zeros_like(g[n]) for n in ("y_perm", "dh", "dx_perm")}
    st["dw1"], st["dw2"] = np.zeros(w1.shape), np.zeros(w2.shape)
    for q in range(E):
        r, e = slice(off[q], off[q + 1]), ge[q]
        if off[q + 1] == off[q]:
            continue
        G, U, A, dY, dH = g["h_gu"][r, :F], g["h_gu"][r, F:], g["act"][r], g["dy_perm"][r], g["dh"][r]
        st["y_perm"][r] = A @ w2[e].T
        dA = dY @ w2[e]
        sg = mo.sigmoid(G)
        st["dh"][r] = np.concatenate([dA * U * sg * (1.0 + G * (1.0 - sg)), dA * G * sg], 1)
        st["dx_perm"][r] = dH @ w1[e]
        st["dw1"][e] = dH.T @ g["x_perm"][r]
        st["dw2"][e] = dY.T @ A
    # combine and its backward on the GPU's expert outputs and gates
    ysh = [np64(lay.y_sh[s2]) for s2 in range(sh.n_shared)]
    st["out"] = mo.combine(g["y_perm"], g["topk_w"], slot) + sum(ysh, np.zeros((T, sh.d_model)))
    st["dy_perm"], st["dtopk_w"] = mo.combine_backward(dout, g["y_perm"], g["topk_w"], slot)
    # gating backward on the GPU's probs and gate gradients; its two products take the
    # bf16 rounding of dlogits as operand on the bf16 path
    rb = mo.router_backward(inp, sh, g["probs"], ints(lay.topk_idx), g["topk_w"], g["dtopk_w"],
                            np64(lay.aux_coef))
    dz = g["dlogits"]
    dz_op = mi.bf16_round(dz.astype(np.float32)).astype(np.float64) if bf else dz
    po = inp["party_offsets"]
    wr = np.asarray(inp["w_router"], np.float64)
    st["dw_router"] = np.stack([dz_op[po[p]:po[p + 1]].T @ np.asarray(inp["x"], np.float64)[po[p]:po[p + 1]]
                                for p in range(sh.n_parties)])
    st["dbias"] = np.stack([dz[po[p]:po[p + 1]].sum(0) for p in range(sh.n_parties)])
    part = mo.party_of_tokens(T, po)
    st["dx_router"] = np.einsum("te,ted->td", dz_op, wr[part])
    dxsh = [np64(lay.dx_sh[s2]) for s2 in range(sh.n_shared)]
    st["dx"] = mo.unpermute_reduce(g["dx_perm"], slot) + g["dx_router"] + sum(dxsh, np.zeros((T, sh.d_model)))
    errs = {}
    for n in ("y_perm", "dh", "dx_perm", "out", "dy_perm", "dtopk_w", "dx_router", "dx"):
        errs[n] = assert_close(n + " (stage)", getattr(lay, n), st[n], tol, stage=True)
    errs["dlogits"] = assert_close("dlogits (stage)", lay.dlogits, rb["dlogits"], tol, stage=True)
    for n in ("dw1", "dw2", "dw_router", "dbias"):
        errs[n] = assert_close_slices(n + " (stage)", getattr(lay, n), st[n], tol, stage=True)
    return errs


SMALL = {
    "tiny_f32": lambda: mi.SHAPES[1],
    "tiny_f32_renorm": lambda: mi.SHAPES[1].with_(normalize_topk=1, aux_alpha=1.0),
    "mid_bf16": lambda: mi.SHAPES[2],
    "mid_bf16_renorm": lambda: mi.SHAPES[2].with_(T=1000, normalize_topk=1),
    "fine_bf16_T512": lambda: mi.SHAPES[3].with_(T=512),
    "large_zipf_bf16_T384": lambda: mi.SHAPES[4].with_(T=384),
    "party4_bf16_T1024": lambda: mi.SHAPES[5].with_(T=1024),
    "all_experts_k_eq_E": lambda: mi.MoEShape("kE", 200, 256, 4, 256, 4, "bf16", seed=77),
    "one_token": lambda: mi.MoEShape("t1", 1, 128, 8, 128, 2, "bf16", seed=78),
    # E % 4 != 0 (CUDA-core router forward), d % 256 != 0 (128-wide tiles; dX and dW1
    # in separate launches), three parties of 233 tokens (router-gradient chunks end
    # inside a 64-token block)
    "odd_E6_d384_parties3": lambda: mi.MoEShape("o6", 699, 384, 6, 256, 2, "bf16", n_parties=3,
                                                seed=79),
    # wide expert pools: E = 128 and 256 (bf16, tensor-core gating with TMEM read in
    # chunks, dz padded to 128 / 256 columns, 128-256 GEMM groups), E = 100 in fp32
    "wide_E128_bf16_parties2": lambda: mi.MoEShape("w128", 640, 256, 128, 128, 4, "bf16",
                                                   n_parties=2, seed=80),
    "wide_E256_bf16": lambda: mi.MoEShape("w256", 512, 128, 256, 128, 8, "bf16", seed=81),
    "wide_E100_f32": lambda: mi.MoEShape("w100", 300, 64, 100, 64, 3, "f32", seed=82),
}


@pytest.mark.parametrize("name", list(SMALL))
def test_layer_full_parity(L, name):
    sh = SMALL[name]()
    sh = sh.with_(seed=seeds.decided_seed(sh))
    inp = mi.make_inputs(sh)
    lay = run_layer(sh, inp)
    assert status(L) == 0
    errs = full_compare(lay, inp, sh)
    print(name, {k: f"{v:.2e}" for k, v in errs.items()})
    serrs = stage_compare(lay, inp, sh)
    print(name, "stage", {k: f"{v:.2e}" for k, v in serrs.items()})


def test_layer_is_deterministic(L):
    sh = mi.SHAPES[2].with_(T=1024)
    inp = mi.make_inputs(sh)
    a = run_layer(sh, inp)
    b = run_layer(sh, inp)
    for n in ("out", "dx", "dw1", "dw2", "dw_router", "dlogits", "dtopk_w", "slot_of"):
        assert torch.equal(getattr(a, n), getattr(b, n)), n


def test_step_from_host_buffers_matches_device_step(L):
    """step_host (x and dOut from pinned host memory, overlapped copies, results back to
    the host) gives the same bits as a step on device-resident inputs, on three steps in
    a row with different inputs each step (so a copy racing a pass would show)."""
    sh = mi.SHAPES[2].with_(T=1024)
    lay = MoELayer(sh)
    lay.load(mi.make_inputs(sh))
    ref = MoELayer(sh)
    ref.load(mi.make_inputs(sh))
    hx = torch.empty(sh.T, sh.d_model, dtype=lay.dt).pin_memory()
    hd, ho, hdx = torch.empty_like(hx).pin_memory(), torch.empty_like(hx).pin_memory(), \
        torch.empty_like(hx).pin_memory()
    hloss = torch.empty(sh.n_parties, dtype=torch.float32).pin_memory()
    for i in range(3):
        inp = mi.make_inputs(sh.with_(seed=sh.seed + 100 + i), with_weights=False)
        hx.copy_(torch.from_numpy(inp["x"]).to(lay.dt))
        hd.copy_(torch.from_numpy(inp["dout"]).to(lay.dt))
        lay.step_host(hx, hd, ho, hdx, hloss)
        torch.cuda.synchronize()
        ref.x.copy_(hx)
        ref.dout.copy_(hd)
        ref.step()
        torch.cuda.synchronize()
        assert torch.equal(ho, ref.out.cpu()), i
        assert torch.equal(hdx, ref.dx.cpu()), i
        assert torch.equal(hloss, ref.aux_loss.cpu()), i
        assert torch.equal(lay.dw1, ref.dw1), i
    assert status(L) == 0


def test_pipelined_host_passes_match_device_steps(L):
    """run_host: five passes with different inputs, uploads and downloads overlapping the
    neighbouring passes' kernels on two copy streams and two device buffer sets; every
    pass's out, dx and aux loss equal a device-resident step on the same inputs, bit for
    bit, and the weight gradients are the last pass's. A copy that raced a pass, or a
    buffer set reused too early, would change some pass's results."""
    sh = mi.SHAPES[2].with_(T=1024)
    lay, ref = MoELayer(sh), MoELayer(sh)
    lay.load(mi.make_inputs(sh))
    ref.load(mi.make_inputs(sh))
    n = 5
    batches = []
    for i in range(n):
        inp = mi.make_inputs(sh.with_(seed=sh.seed + 200 + i), with_weights=False)
        hx = torch.from_numpy(inp["x"]).to(lay.dt).pin_memory()
        hd = torch.from_numpy(inp["dout"]).to(lay.dt).pin_memory()
        batches.append((hx, hd, torch.empty_like(hx).pin_memory(), torch.empty_like(hx).pin_memory(),
                        torch.full((sh.n_parties,), float("nan")).pin_memory()))
    x0 = lay.x
    lay.run_host(batches)
    torch.cuda.synchronize()
    for i, (hx, hd, ho, hdx, hloss) in enumerate(batches):
        ref.x.copy_(hx)
        ref.dout.copy_(hd)
        ref.step()
        torch.cuda.synchronize()
        assert torch.equal(ho, ref.out.cpu()), i
        assert torch.equal(hdx, ref.dx.cpu()), i
        assert torch.equal(hloss, ref.aux_loss.cpu()), i
    assert torch.equal(lay.dw1, ref.dw1) and torch.equal(lay.dw_router, ref.dw_router)
    assert lay.x is x0  # the first buffer set is current again
    assert status(L) == 0


@pytest.mark.parametrize("sh", [mi.SHAPES[5].with_(T=1024), mi.SHAPES[3].with_(T=512, n_parties=2),
                                mi.SHAPES[2].with_(T=1000)], ids=["party4", "fine_P2", "mid_P1"])
def test_owner_grouped_layout_gives_the_same_results(L, sh):
    """The layer with its permuted rows grouped by owner party (moe_dispatch_owner, the
    expert GEMMs told each segment's expert) equals the expert-major layer bit for bit:
    every expert sees the same rows in the same order. The send counts match the picks."""
    inp = mi.make_inputs(sh)
    a, b = MoELayer(sh, owner_grouped=True), MoELayer(sh, owner_grouped=False)
    for lay in (a, b):
        lay.load(inp)
        lay.step()
    torch.cuda.synchronize()
    assert status(L) == 0
    for n in ("out", "dx", "dw1", "dw2", "dw_router", "dbias", "dlogits", "dtopk_w", "aux_loss",
              "topk_idx", "counts"):
        assert torch.equal(getattr(a, n), getattr(b, n)), n
    if sh.n_shared:
        for n in ("dws1", "dws2", "y_sh"):
            assert torch.equal(getattr(a, n), getattr(b, n)), n
    idx = ints(a.topk_idx)
    P = sh.n_parties
    part = mo.party_of_tokens(sh.T, inp["party_offsets"])
    ref = np.zeros((P, P), np.int64)
    np.add.at(ref, (np.repeat(part, sh.top_k), idx.ravel() % P), 1)
    assert (ints(a.send_counts) == ref).all()
    assert (ints(a.group_expert) == sorted(range(sh.n_experts), key=lambda e: (e % P, e))).all()


def test_layer_empty_batch(L):
    sh = mi.MoEShape("empty", 0, 256, 8, 256, 2, "bf16")
    lay = MoELayer(sh)
    inp = mi.make_inputs(sh.with_(T=0))
    lay.load(inp)
    lay.dw1.fill_(1)
    lay.step()
    assert status(L) == 0
    assert (ints(lay.offsets) == 0).all()
    assert (lay.dw1 == 0).all() and (lay.dw2 == 0).all() and (lay.dw_router == 0).all()


@pytest.mark.parametrize("which", [3, 4, 5])
def test_layer_sampled_parity_full_size(L, which):
    """Full-size workloads. Routing of every token; per-party counts, the aux loss and
    its coefficients in full; the gating backward (dlogits, dW_r, db, dx_router) in full
    from the oracle's router backward; sampled tokens' outputs and input gradients, and
    sampled weight-gradient slices, from the oracle one token / one column at a time.

    Reading of "identical inputs" (as for the bit-exact routing test): at these sizes
    some tokens' top-k neighbours lie within the fp32 logit tolerance, so the picks are
    the GPU's (checked equal to the oracle's on every decided token, and a valid top-k
    under the GPU's own logits elsewhere), and the oracle's router backward takes the
    GPU's gate gradients dtopk_w (checked against the oracle on the sampled tokens)."""
    sh = mi.SHAPES[which]
    inp = mi.make_inputs(sh)
    lay = run_layer(sh, inp)
    assert status(L) == 0
    tol = TOL[sh.dtype]
    route = mo.route_all(inp, sh)
    z = route["logits"]
    assert (np.abs(np64(lay.logits) - z) <= seeds.logit_tol(z, sh.d_model)).all()
    decided = seeds.decided(z, sh.top_k, sh.d_model)
    idx = ints(lay.topk_idx)
    assert (idx[decided] == route["topk_idx"][decided]).all()
    # undecided tokens: the GPU picks must still be a valid top-k under its own logits
    gl = np64(lay.logits)
    for t in np.nonzero(~decided)[0]:
        kth = np.sort(gl[t])[::-1][sh.top_k - 1]
        assert (gl[t][idx[t]] >= kth).all()
    flipped = np.nonzero((idx != route["topk_idx"]).any(axis=1))[0]
    touched = set(route["topk_idx"][flipped].ravel().tolist()) | set(idx[flipped].ravel().tolist())
    print(f"{sh.name}: {int((~decided).sum())} undecided tokens, {len(flipped)} routed differently")
    # per-party counts: exact on the picks; the aux loss and its coefficients in full
    po = inp["party_offsets"]
    cnt = mo.party_counts(idx, sh.n_experts, po)
    assert (ints(lay.counts) == cnt).all()
    if not len(flipped):
        assert (ints(lay.counts) == route["party_counts"]).all()
    aux_l, aux_c = mo.aux_loss(route["probs"], cnt, po, sh.top_k, sh.aux_alpha)
    errs = {"aux_loss": assert_close("aux_loss", lay.aux_loss, aux_l, tol),
            "aux_coef": assert_close("aux_coef", lay.aux_coef, aux_c, tol),
            "probs": assert_close("probs", lay.probs, route["probs"], tol)}
    # the gating backward in full
    w_ref = mo.gate_weights(route["probs"], idx, sh.normalize_topk)
    errs["topk_w"] = assert_close("topk_w", lay.topk_w, w_ref, tol)
    rb = mo.router_backward(inp, sh, route["probs"], idx, w_ref, np64(lay.dtopk_w), aux_c)
    errs["dlogits"] = assert_close("dlogits", lay.dlogits, rb["dlogits"], tol)
    errs["dx_router"] = assert_close("dx_router", lay.dx_router, rb["dx_router"], tol)
    for p in range(sh.n_parties):
        errs[f"dw_router{p}"] = assert_close("dw_router", lay.dw_router[p], rb["dw_router"][p], tol)
        errs[f"dbias{p}"] = assert_close("dbias", lay.dbias[p], rb["dbias"][p], tol)
    rng = np.random.default_rng(sh.seed)
    toks = rng.choice(np.nonzero(decided)[0], size=48, replace=False)
    toks = np.concatenate([toks, [0, sh.T - 1]]) if decided[0] and decided[-1] else toks
    rows = mo.sampled_token_rows(inp, sh, route, toks)
    toks_d = torch.as_tensor(toks, device="cuda")
    # per-token rows are compared against the scale of the sampled reference
    errs["out"] = assert_close("out", lay.out[toks_d], rows["out"], tol)
    errs["dx"] = assert_close("dx", lay.dx[toks_d], rows["dx"], tol)
    errs["dtopk_w"] = assert_close("dtopk_w", lay.dtopk_w[toks_d], rows["dtopk_w"], tol)
    errs["dlogits_rows"] = assert_close("dlogits", lay.dlogits[toks_d], rows["dlogits"], tol)
    slot = ints(lay.slot_of).reshape(sh.T, sh.top_k)
    ys = torch.stack([lay.y_perm[torch.as_tensor(slot[t], device="cuda")] for t in toks])
    errs["y"] = assert_close("y", ys, rows["y"], tol)
    dxps = torch.stack([lay.dx_perm[torch.as_tensor(slot[t], device="cuda")] for t in toks])
    errs["dx_perm"] = assert_close("dx_perm", dxps, rows["dx_perm"], tol)
    # weight-gradient slices of experts whose rows no flipped token touched
    F = sh.d_ff
    cols = sorted(rng.choice(F, size=4, replace=False).tolist())
    experts = [e for e in rng.permutation(sh.n_experts)[:6] if e not in touched]
    for e in experts:
        sw = mo.sampled_weight_grads(inp, sh, route, int(e), cols)
        errs[f"dw2_{e}"] = assert_close("dw2 cols", lay.dw2[e][:, cols], sw["dw2_cols"], tol)
        errs[f"dw1g_{e}"] = assert_close("dw1 gate rows", lay.dw1[e][cols], sw["dw1_gate_rows"], tol)
        errs[f"dw1u_{e}"] = assert_close("dw1 up rows", lay.dw1[e][[F + c for c in cols]],
                                         sw["dw1_up_rows"], tol)
    assert (ints(lay.counts).sum() == sh.T * sh.top_k)
    print(sh.name, {k: f"{v:.2e}" for k, v in errs.items()})
