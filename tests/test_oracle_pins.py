"""Pins of the fp64 oracle against facts that do not come from the oracle itself.

Each test checks one part of ``oracle/moe_oracle.py`` against a closed form, an
invariant, brute force on tiny inputs, central finite differences, or an
independently written autograd implementation, chosen so that a dropped term,
wrong sign, wrong index or transposed operand fails at least one of them.
"""
import itertools

import numpy as np
import pytest

from oracle import moe_oracle as mo
from synth import moe_inputs as mi


def tiny_shape(**kw):
    base = dict(name="tiny", T=6, d_model=8, n_experts=4, d_ff=6, top_k=2, dtype="f32",
                n_parties=2, n_shared=1, d_ff_shared=4, aux_alpha=0.7)
    base.update(kw)
    return mi.MoEShape(**base)


def tiny_inputs(shape, seed=3, wscale=0.5, bias=True):
    rng = np.random.default_rng(seed)
    T, d, E, F, P = shape.T, shape.d_model, shape.n_experts, shape.d_ff, shape.n_parties
    inp = dict(
        x=rng.standard_normal((T, d)),
        w_router=wscale * rng.standard_normal((P, E, d)),
        router_bias=(0.3 * rng.standard_normal((P, E)) if bias else None),
        w1=wscale * rng.standard_normal((E, 2 * F, d)),
        w2=wscale * rng.standard_normal((E, d, F)),
        dout=rng.standard_normal((T, d)),
        party_offsets=mi.party_offsets(shape),
    )
    S, Fs = shape.n_shared, shape.d_ff_shared
    inp["ws1"] = wscale * rng.standard_normal((S, 2 * Fs, d)) if S else None
    inp["ws2"] = wscale * rng.standard_normal((S, d, Fs)) if S else None
    return inp


# ------------------------------------------------------------------ softmax / top-k

def test_softmax_sums_to_one_and_two_expert_closed_form():
    rng = np.random.default_rng(0)
    z = rng.standard_normal((50, 7)) * 5
    p = mo.softmax(z)
    assert np.allclose(p.sum(axis=1), 1.0, atol=1e-14)
    assert (p > 0).all()
    z2 = rng.standard_normal((50, 2))
    p2 = mo.softmax(z2)
    sig = 1.0 / (1.0 + np.exp(-(z2[:, 0] - z2[:, 1])))
    assert np.allclose(p2[:, 0], sig, atol=1e-15)


def _brute_topk(zrow, k):
    """Lexicographically best k-permutation under (higher logit, then lower id)."""
    best = None
    for perm in itertools.permutations(range(len(zrow)), k):
        key = tuple(v for e in perm for v in (float(zrow[e]), -e))
        if best is None or key > best[0]:
            best = (key, perm)
    return list(best[1])


@pytest.mark.parametrize("E,k", [(4, 1), (4, 2), (5, 3), (6, 2), (6, 6)])
def test_topk_matches_brute_force_with_planted_ties(E, k):
    z = mi.make_route_logits(40, E, seed=E * 10 + k, tie_every=2)
    idx = mo.topk_indices(z, k)
    for t in range(z.shape[0]):
        assert list(idx[t]) == _brute_topk(z[t], k), t


def test_topk_all_equal_row_picks_lowest_ids():
    z = np.full((3, 8), 0.5, np.float32)
    assert (mo.topk_indices(z, 3) == np.array([0, 1, 2])).all()


def test_gate_weights_paper_vs_renormalised():
    rng = np.random.default_rng(1)
    p = mo.softmax(rng.standard_normal((30, 6)))
    idx = mo.topk_indices(np.log(p).astype(np.float32), 2)
    w = mo.gate_weights(p, idx, 0)
    assert np.allclose(w, np.take_along_axis(p, idx.astype(int), 1))
    assert (w.sum(axis=1) < 1).all()  # paper: not renormalised
    wn = mo.gate_weights(p, idx, 1)
    assert np.allclose(wn.sum(axis=1), 1.0, atol=1e-12)
    assert np.allclose(wn[:, 0] / wn[:, 1], w[:, 0] / w[:, 1])


# ------------------------------------------------------------------ dispatch

@pytest.mark.parametrize("T,E,k", [(1, 1, 1), (9, 4, 2), (64, 8, 3), (200, 16, 2)])
def test_dispatch_tables_brute_force(T, E, k):
    rng = np.random.default_rng(T + E + k)
    idx = np.stack([rng.permutation(E)[:k] for _ in range(T)]).astype(np.int32)
    counts, offsets, slot_of, token_of = mo.dispatch_tables(idx, E)
    assert (counts == np.bincount(idx.ravel(), minlength=E)).all()
    assert counts.sum() == T * k
    assert offsets[0] == 0 and offsets[-1] == T * k
    assert (np.diff(offsets) == counts).all()
    # the permutation equals a stable sort of token-major entries by expert id
    order = np.argsort(idx.ravel(), kind="stable")
    assert (token_of == order // k).all()
    flat = slot_of.ravel()
    assert sorted(flat.tolist()) == list(range(T * k))  # bijection
    assert (flat[order] == np.arange(T * k)).all()
    for e in range(E):  # ascending token id inside each expert segment
        seg = token_of[offsets[e]:offsets[e + 1]]
        assert (np.diff(seg) > 0).all()
    x = rng.standard_normal((T, 5))
    xp = mo.gather_permute(x, token_of)
    # unpermute o permute is the identity, exactly
    for t in range(T):
        for j in range(k):
            assert (xp[slot_of[t, j]] == x[t]).all()


@pytest.mark.parametrize("T,E,k,P", [(1, 1, 1, 1), (12, 4, 2, 2), (99, 8, 3, 3), (200, 32, 2, 4),
                                      (60, 6, 2, 4)])
def test_owner_dispatch_tables(T, E, k, P):
    """Owner-grouped dispatch: segments in (owner = e mod P, expert) order, rows in token
    order; pinned to a library lexsort of the (owner, expert, token) keys, to the plain
    dispatch when P = 1, and to send counts recomputed from the permuted layout."""
    rng = np.random.default_rng(T * 7 + E + k + P)
    idx = np.stack([rng.permutation(E)[:k] for _ in range(T)]).astype(np.int32)
    po = np.linspace(0, T, P + 1).astype(np.int64)
    ge, counts, offsets, slot_of, token_of, send = mo.owner_dispatch_tables(idx, E, po)
    # segment order: owners ascending, experts ascending inside an owner
    assert sorted(ge.tolist(), key=lambda e: (e % P, e)) == ge.tolist()
    assert sorted(ge.tolist()) == list(range(E))
    # the permutation is a stable sort of the (t, j) entries by (owner, expert)
    flat_e = idx.ravel().astype(np.int64)
    flat_t = np.repeat(np.arange(T), k)
    order = np.lexsort((flat_t, flat_e, flat_e % P))
    assert (token_of == flat_t[order]).all()
    assert (slot_of.ravel()[order] == np.arange(T * k)).all()
    for g, e in enumerate(ge):  # segment g holds exactly expert e's rows
        seg = slice(offsets[g], offsets[g + 1])
        assert counts[g] == (flat_e == e).sum()
        assert (idx[token_of[seg]] == e).any(axis=1).all()
    # send counts: totals, per-source totals, and recomputed from the layout
    assert send.sum() == T * k
    assert (send.sum(axis=1) == np.diff(po) * k).all()
    party = np.searchsorted(po, np.arange(T), side="right") - 1
    re = np.zeros((P, P), np.int64)
    for g, e in enumerate(ge):
        for r in range(offsets[g], offsets[g + 1]):
            re[party[token_of[r]], e % P] += 1
    assert (re == send).all()
    if P == 1:
        c1, o1, s1, t1 = mo.dispatch_tables(idx, E)
        assert (counts == c1).all() and (offsets == o1).all()
        assert (slot_of == s1).all() and (token_of == t1).all()


def test_combine_with_identity_experts():
    rng = np.random.default_rng(5)
    T, E, k, d = 40, 6, 3, 7
    x = rng.standard_normal((T, d))
    p = mo.softmax(rng.standard_normal((T, E)))
    idx = mo.topk_indices(np.log(p).astype(np.float32), k)
    _, _, slot_of, token_of = mo.dispatch_tables(idx, E)
    xp = mo.gather_permute(x, token_of)
    wn = mo.gate_weights(p, idx, 1)
    assert np.allclose(mo.combine(xp, wn, slot_of), x, atol=1e-14)
    assert np.allclose(mo.combine(xp, np.ones((T, k)), slot_of), k * x, atol=1e-14)
    assert np.allclose(mo.unpermute_reduce(xp, slot_of), k * x, atol=1e-14)


# ------------------------------------------------------------------ aux loss

def test_aux_loss_closed_forms():
    T, E, k, alpha = 64, 8, 2, 0.37
    probs = np.full((T, E), 1.0 / E)
    counts = np.full((1, E), T * k // E)
    loss, coef = mo.aux_loss(probs, counts, [0, T], k, alpha)
    assert loss[0] == pytest.approx(alpha, rel=1e-14)  # perfectly balanced -> alpha
    assert np.allclose(coef, alpha * E * (1.0 / E) / T)
    probs = np.zeros((T, E)); probs[:, 3] = 1.0
    counts = np.zeros((1, E)); counts[0, 3] = T * k
    loss, _ = mo.aux_loss(probs, counts, [0, T], k, alpha)
    assert loss[0] == pytest.approx(alpha * E, rel=1e-14)  # collapsed -> alpha * E


def test_aux_loss_is_per_party():
    T, E, k = 12, 4, 2
    rng = np.random.default_rng(2)
    probs = mo.softmax(rng.standard_normal((T, E)))
    idx = mo.topk_indices(np.log(probs).astype(np.float32), k)
    po = [0, 4, 12]
    cpe = mo.party_counts(idx, E, po)
    loss, _ = mo.aux_loss(probs, cpe, po, k, 1.0)
    for p in range(2):
        sl = slice(po[p], po[p + 1])
        l1, _ = mo.aux_loss(probs[sl], mo.party_counts(idx[sl], E, [0, po[p + 1] - po[p]]),
                            [0, po[p + 1] - po[p]], k, 1.0)
        assert loss[p] == pytest.approx(l1[0], rel=1e-14)


# ------------------------------------------------------------------ experts

def test_single_expert_top1_is_dense_swiglu_ffn():
    """E = k = 1: the softmax over one expert is 1, so the layer is a dense SwiGLU FFN."""
    torch = pytest.importorskip("torch")
    sh = tiny_shape(n_experts=1, top_k=1, n_parties=1, n_shared=0)
    inp = tiny_inputs(sh, bias=False)
    fwd = mo.layer_forward(inp, sh)
    x = torch.tensor(inp["x"])
    W1 = torch.tensor(inp["w1"][0]); W2 = torch.tensor(inp["w2"][0])
    F = sh.d_ff
    ref = (torch.nn.functional.silu(x @ W1[:F].T) * (x @ W1[F:].T)) @ W2.T
    assert np.allclose(fwd["out"], ref.numpy(), atol=1e-13, rtol=1e-12)
    assert (fwd["topk_w"] == 1.0).all()


def _loss(inp, sh, fwd_ref):
    """Scalar whose gradients the backward returns: <out, dOut> + sum_p L_p, with the
    routing (and the counts f) of the reference point held fixed."""
    fwd = mo.layer_forward(inp, sh)
    assert (fwd["topk_idx"] == fwd_ref["topk_idx"]).all(), "perturbation changed routing"
    return float(np.sum(fwd["out"] * inp["dout"]) + fwd["aux_loss"].sum())


@pytest.mark.parametrize("normalize", [0, 1])
def test_backward_matches_central_finite_differences(normalize):
    sh = tiny_shape(normalize_topk=normalize)
    inp = tiny_inputs(sh, seed=11 + normalize)
    fwd = mo.layer_forward(inp, sh)
    assert mo.top_margin(fwd["logits"], sh.top_k).min() > 1e-3
    bwd = mo.layer_backward(inp, sh, fwd)
    grads = dict(x=bwd["dx"], w_router=bwd["dw_router"], router_bias=bwd["dbias"],
                 w1=bwd["dw1"], w2=bwd["dw2"],
                 ws1=np.stack([g[2] for g in bwd["shared_grads"]]),
                 ws2=np.stack([g[3] for g in bwd["shared_grads"]]))
    h = 1e-6
    rng = np.random.default_rng(99)
    for name, g in grads.items():
        base = inp[name]
        flat_idx = rng.choice(base.size, size=min(base.size, 40), replace=False)
        for fi in flat_idx:
            ii = np.unravel_index(fi, base.shape)
            orig = base[ii]
            base[ii] = orig + h
            lp = _loss(inp, sh, fwd)
            base[ii] = orig - h
            lm = _loss(inp, sh, fwd)
            base[ii] = orig
            num = (lp - lm) / (2 * h)
            assert abs(num - g[ii]) <= 1e-6 * max(1.0, abs(num)), (name, ii, num, g[ii])


def test_gate_and_logit_gradients_finite_differences():
    """dw = d<out,dOut>/dw with the gates as free inputs; dz through the softmax."""
    sh = tiny_shape(n_shared=0)
    inp = tiny_inputs(sh, seed=21)
    fwd = mo.layer_forward(inp, sh)
    bwd = mo.layer_backward(inp, sh, fwd, with_aux=False)
    h = 1e-6
    w = fwd["topk_w"].copy()
    for t in range(sh.T):
        for j in range(sh.top_k):
            wp = w.copy(); wp[t, j] += h
            wm = w.copy(); wm[t, j] -= h
            lp = np.sum(mo.combine(fwd["y_perm"], wp, fwd["slot_of"]) * inp["dout"])
            lm = np.sum(mo.combine(fwd["y_perm"], wm, fwd["slot_of"]) * inp["dout"])
            assert abs((lp - lm) / (2 * h) - bwd["dtopk_w"][t, j]) < 1e-7
    # dlogits: perturb z directly, keeping the picks
    z = fwd["logits"]
    for t in range(sh.T):
        for e in range(sh.n_experts):
            vals = []
            for s in (+h, -h):
                zz = z.copy(); zz[t, e] += s
                ww = mo.gate_weights(mo.softmax(zz), fwd["topk_idx"], sh.normalize_topk)
                vals.append(np.sum(mo.combine(fwd["y_perm"], ww, fwd["slot_of"]) * inp["dout"]))
            assert abs((vals[0] - vals[1]) / (2 * h) - bwd["dlogits"][t, e]) < 1e-7


@pytest.mark.parametrize("normalize", [0, 1])
def test_router_backward_finite_differences(normalize):
    """router_backward (the gating backward for given picks and gate gradients) is the
    gradient of f = sum_tj c_tj w_tj + sum_te a_{p(t),e} p_te with the picks held fixed,
    w and p as Alg. 7 defines them from z = W_r[p] x + b; checked by central differences
    in W_r, b and x, and it agrees with the router part of the full layer backward."""
    sh = tiny_shape(T=8, n_experts=5, top_k=2, normalize_topk=normalize, n_shared=0)
    inp = tiny_inputs(sh, seed=31 + normalize)
    rng = np.random.default_rng(5)
    route = mo.route_all(inp, sh)
    idx = route["topk_idx"]
    c = rng.standard_normal((sh.T, sh.top_k))   # stands in for dL/dw
    a = rng.standard_normal((sh.n_parties, sh.n_experts))  # stands in for dL_aux/dp
    part = mo.party_of_tokens(sh.T, inp["party_offsets"])
    rb = mo.router_backward(inp, sh, route["probs"], idx, route["topk_w"], c, a)

    def f():
        z = mo.router_logits(inp["x"], inp["w_router"], inp["router_bias"], inp["party_offsets"])
        assert (mo.topk_indices(z.astype(np.float32), sh.top_k) == idx).all()
        p = mo.softmax(z)
        w = mo.gate_weights(p, idx, sh.normalize_topk)
        return float(np.sum(c * w) + np.sum(a[part] * p))

    h = 1e-6
    for name, g in (("w_router", rb["dw_router"]), ("router_bias", rb["dbias"]),
                    ("x", rb["dx_router"])):
        base = inp[name]
        for fi in range(base.size):
            ii = np.unravel_index(fi, base.shape)
            orig = base[ii]
            base[ii] = orig + h
            lp = f()
            base[ii] = orig - h
            lm = f()
            base[ii] = orig
            num = (lp - lm) / (2 * h)
            assert abs(num - g[ii]) <= 1e-6 * max(1.0, abs(num)), (name, ii, num, g[ii])
    # the same numbers as the router part of the whole layer's backward
    fwd = mo.layer_forward(inp, sh)
    bwd = mo.layer_backward(inp, sh, fwd)
    rb2 = mo.router_backward(inp, sh, fwd["probs"], fwd["topk_idx"], fwd["topk_w"],
                             bwd["dtopk_w"], fwd["aux_coef"])
    for n in ("dlogits", "dw_router", "dbias", "dx_router"):
        assert np.allclose(rb2[n], bwd[n], atol=1e-13, rtol=1e-12), n


def test_layer_matches_independent_torch_autograd():
    """An independently written torch fp64 layer differentiated by autograd."""
    torch = pytest.importorskip("torch")
    sh = tiny_shape(T=10, n_experts=5, top_k=2)
    inp = tiny_inputs(sh, seed=7)
    fwd = mo.layer_forward(inp, sh)
    bwd = mo.layer_backward(inp, sh, fwd)
    P, F, Fs = sh.n_parties, sh.d_ff, sh.d_ff_shared
    tv = {n: torch.tensor(inp[n], dtype=torch.float64, requires_grad=True)
          for n in ("x", "w_router", "router_bias", "w1", "w2", "ws1", "ws2")}
    po = inp["party_offsets"]

    def ffn(h, W1, W2, Fh):
        return (torch.nn.functional.silu(h @ W1[:Fh].T) * (h @ W1[Fh:].T)) @ W2.T

    outs, aux = [], 0.0
    for p in range(P):
        h = tv["x"][po[p]:po[p + 1]]
        z = h @ tv["w_router"][p].T + tv["router_bias"][p]
        pr = torch.softmax(z, dim=1)
        val, ind = torch.topk(z, sh.top_k, dim=1, sorted=True)
        wsel = torch.gather(pr, 1, ind)
        o = torch.zeros_like(h)
        for r in range(h.shape[0]):
            for j in range(sh.top_k):
                e = int(ind[r, j])
                o[r] = o[r] + wsel[r, j] * ffn(h[r:r + 1], tv["w1"][e], tv["w2"][e], F)[0]
        for s in range(sh.n_shared):
            o = o + ffn(h, tv["ws1"][s], tv["ws2"][s], Fs)
        outs.append(o)
        Tp = h.shape[0]
        cnt = torch.zeros(sh.n_experts, dtype=torch.float64)
        for e in ind.flatten().tolist():
            cnt[e] += 1
        aux = aux + sh.aux_alpha * sh.n_experts * torch.sum(cnt / (Tp * sh.top_k) * pr.mean(0))
        assert (ind.numpy() == fwd["topk_idx"][po[p]:po[p + 1]]).all()
    out = torch.cat(outs)
    assert np.allclose(out.detach().numpy(), fwd["out"], atol=1e-12)
    L = torch.sum(out * torch.tensor(inp["dout"])) + aux
    L.backward()
    for n, g in (("x", bwd["dx"]), ("w_router", bwd["dw_router"]), ("router_bias", bwd["dbias"]),
                 ("w1", bwd["dw1"]), ("w2", bwd["dw2"])):
        assert np.allclose(tv[n].grad.numpy(), g, atol=1e-11, rtol=1e-9), n
    assert np.allclose(tv["ws1"].grad.numpy(), np.stack([g[2] for g in bwd["shared_grads"]]), atol=1e-11)
    assert np.allclose(tv["ws2"].grad.numpy(), np.stack([g[3] for g in bwd["shared_grads"]]), atol=1e-11)


def test_sampled_helpers_agree_with_full_layer():
    """The one-token-at-a-time and one-column-at-a-time evaluations used at large sizes
    reproduce the full-layer tensors."""
    sh = tiny_shape(T=12, n_experts=4, top_k=2, d_ff=8)
    inp = tiny_inputs(sh, seed=4)
    fwd = mo.layer_forward(inp, sh)
    bwd = mo.layer_backward(inp, sh, fwd)
    route = mo.route_all(inp, sh)
    assert (route["topk_idx"] == fwd["topk_idx"]).all()
    toks = [0, 5, 11]
    rows = mo.sampled_token_rows(inp, sh, route, toks)
    assert np.allclose(rows["out"], fwd["out"][toks], atol=1e-12)
    assert np.allclose(rows["dx"], bwd["dx"][toks], atol=1e-12)
    assert np.allclose(rows["dtopk_w"], bwd["dtopk_w"][toks], atol=1e-12)
    assert np.allclose(rows["dlogits"], bwd["dlogits"][toks], atol=1e-12)
    for i, t in enumerate(toks):
        for j in range(sh.top_k):
            r = fwd["slot_of"][t, j]
            assert np.allclose(rows["y"][i, j], fwd["y_perm"][r], atol=1e-12)
            assert np.allclose(rows["dx_perm"][i, j], bwd["dx_perm"][r], atol=1e-12)
    F = sh.d_ff
    for e in range(sh.n_experts):
        cols = [0, 3, F - 1]
        sw = mo.sampled_weight_grads(inp, sh, route, e, cols)
        assert np.allclose(sw["dw2_cols"], bwd["dw2"][e][:, cols], atol=1e-12)
        assert np.allclose(sw["dw1_gate_rows"], bwd["dw1"][e][cols], atol=1e-12)
        assert np.allclose(sw["dw1_up_rows"], bwd["dw1"][e][[F + c for c in cols]], atol=1e-12)


def test_inputs_are_seeded_and_bf16_representable():
    sh = mi.SHAPES[2].with_(T=64, d_model=128, d_ff=128, n_experts=4)
    a = mi.make_inputs(sh)
    b = mi.make_inputs(sh)
    for n in ("x", "w_router", "w1", "w2", "dout"):
        assert (a[n] == b[n]).all()
        assert (mi.bf16_round(a[n]) == a[n]).all()
    c = mi.make_inputs(sh, seed=sh.seed + 1)
    assert not (a["x"] == c["x"]).all()
    # bf16 rounding: ties to even and plain cases
    v = np.array([1.0, 1.00390625, 1.01171875, -2.5, 3.0e-3], np.float32)
    r = mi.bf16_round(v)
    assert r[0] == 1.0 and r[1] == 1.0 and r[2] == 1.015625 and r[3] == -2.5
    assert abs(r[4] - 3.0e-3) / 3.0e-3 < 2 ** -8
