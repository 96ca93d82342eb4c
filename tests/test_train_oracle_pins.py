"""Pins of the training oracle (Alg. 1 on the toy block) against facts that do not come
from the oracle itself: central finite differences, a quadratic whose SGD step has a
closed form, the first-order descent identity of gradient descent (which checks the
whole backward against the forward), brute-force enumeration of Alg. 1's turn order,
and the invariants of "no global broadcast"."""
import itertools

import numpy as np
import pytest

from oracle import train_oracle as to
from synth import moe_inputs as mi


def batch_shape(T=8, **kw):
    base = dict(name="train_tiny", T=T, d_model=8, n_experts=4, d_ff=6, top_k=2, dtype="f32",
                n_parties=1, aux_alpha=0.7)
    base.update(kw)
    return mi.MoEShape(**base)


def rand_params(n, sh, seed=11, wscale=0.5):
    rng = np.random.default_rng(seed)
    E, d, F = sh.n_experts, sh.d_model, sh.d_ff
    return {"w_router": wscale * rng.standard_normal((n, E, d)),
            "w1": wscale * rng.standard_normal((E, 2 * F, d)),
            "w2": wscale * rng.standard_normal((E, d, F))}


def test_mse_zero_at_target_and_finite_differences():
    rng = np.random.default_rng(0)
    out, y = rng.standard_normal((5, 3)), rng.standard_normal((5, 3))
    loss0, g0 = to.mse_loss(y, y)
    assert loss0 == 0.0 and not g0.any()
    loss, g = to.mse_loss(out, y)
    h = 1e-6
    num = np.zeros_like(out)
    for i, j in itertools.product(range(5), range(3)):
        a, b = out.copy(), out.copy()
        a[i, j] += h
        b[i, j] -= h
        num[i, j] = (to.mse_loss(a, y)[0] - to.mse_loss(b, y)[0]) / (2 * h)
    assert np.abs(num - g).max() < 1e-8
    # one token, one feature: (h - y)^2 / 2
    assert to.mse_loss(np.array([[3.0]]), np.array([[1.0]]))[0] == 2.0


def test_sgd_groups_on_a_quadratic_and_the_mask():
    rng = np.random.default_rng(1)
    w, wstar = rng.standard_normal((4, 3, 2)), rng.standard_normal((4, 3, 2))
    grad = w - wstar  # gradient of 0.5 ||w - w*||^2
    counts = np.array([2, 0, 1, 0])
    new = to.sgd_groups(w, grad, 1.0, counts)
    assert np.allclose(new[[0, 2]], wstar[[0, 2]], rtol=0, atol=1e-15)  # lr = 1: the minimum
    assert np.array_equal(new[[1, 3]], w[[1, 3]])       # groups not called: unchanged
    assert np.array_equal(to.sgd_groups(w, grad, 0.0), w)
    half = to.sgd_groups(w, grad, 0.5)
    assert np.allclose(half - wstar, 0.5 * (w - wstar), rtol=0, atol=1e-15)


def _decided_case(n=3, seed=11):
    sh = batch_shape()
    params = rand_params(n, sh, seed)
    (x, y), = mi.train_batches(sh, 1, 1, seed=seed + 1)[0]
    return sh, params, x, y


def test_descent_identity_checks_the_whole_backward():
    """For SGD on exactly the updated parameters, L(theta - lr g) - L(theta) =
    -lr ||g||^2 + O(lr^2); Richardson extrapolation over lr and 2 lr removes the
    second-order term. A wrong sign, a dropped term (aux, router, one of the expert
    weights) or a transposed gradient breaks the identity."""
    sh, params, x, y = _decided_case()
    party = 1
    loss0, _, _, fwd0 = to.batch_loss(params, party, x, y, sh)
    _, rec = to.train_step(params, party, x, y, sh, 0.0)
    called = rec["counts"] > 0
    g2 = (np.sum(rec["dw_router"] ** 2) + np.sum(rec["dw1"][called] ** 2)
          + np.sum(rec["dw2"][called] ** 2))
    assert g2 > 1e-3
    D = []
    for lr in (1e-5, 2e-5):
        new, _ = to.train_step(params, party, x, y, sh, lr)
        loss1, _, _, fwd1 = to.batch_loss(new, party, x, y, sh)
        assert np.array_equal(fwd1["topk_idx"], fwd0["topk_idx"])  # same routing region
        D.append((loss1 - loss0) / lr)
    est = 2 * D[0] - D[1]
    assert abs(est + g2) <= 1e-5 * g2, (est, -g2)


@pytest.mark.parametrize("block", ["w_router", "w1", "w2"])
def test_gradient_of_each_block_against_central_differences(block):
    """Each parameter block's gradient, as train_step applies it, against a central
    difference of the batch objective along a random direction of that block (the
    active party's router only; for the experts, only the called ones move)."""
    sh, params, x, y = _decided_case(n=3, seed=17)
    party = 2
    loss0, _, _, fwd0 = to.batch_loss(params, party, x, y, sh)
    _, rec = to.train_step(params, party, x, y, sh, 0.0)
    rng = np.random.default_rng(99)
    v = np.zeros_like(params[block])
    if block == "w_router":
        v[party] = rng.standard_normal(v[party].shape)
        g = np.zeros_like(v)
        g[party] = rec["dw_router"]
    else:
        called = rec["counts"] > 0
        v[called] = rng.standard_normal(v[called].shape)
        g = rec["d" + block]
    h = 1e-5
    lp = dict(params, **{block: params[block] + h * v})
    lm = dict(params, **{block: params[block] - h * v})
    Lp, _, _, fp = to.batch_loss(lp, party, x, y, sh)
    Lm, _, _, fm = to.batch_loss(lm, party, x, y, sh)
    assert np.array_equal(fp["topk_idx"], fwd0["topk_idx"]) and np.array_equal(fm["topk_idx"], fwd0["topk_idx"])
    num = (Lp - Lm) / (2 * h)
    ana = float(np.sum(g * v))
    assert abs(num - ana) <= 1e-6 * max(1.0, abs(ana)), (block, num, ana)
    assert abs(ana) > 1e-3  # the block matters to the loss


def test_step_changes_only_the_party_router_and_called_experts():
    sh, params, x, y = _decided_case(n=4, seed=23)
    for party in range(4):
        new, rec = to.train_step(params, party, x, y, sh, 0.05)
        for j in range(4):
            same = np.array_equal(new["w_router"][j], params["w_router"][j])
            assert same == (j != party), (party, j)
        for e in range(sh.n_experts):
            for w in ("w1", "w2"):
                same = np.array_equal(new[w][e], params[w][e])
                assert same == (rec["counts"][e] == 0), (party, e, w)
        # parties that update anything: the active one and the hosts of called experts
        brute = {party} | {e % 4 for e in range(sh.n_experts) if rec["counts"][e] > 0}
        assert set(rec["updated_parties"]) == brute


def test_uncalled_expert_keeps_its_bits():
    """A batch whose every token picks experts 0 and 1 (the router strongly prefers
    them) leaves experts 2 and 3 bit for bit as they were."""
    sh, params, x, y = _decided_case(n=2, seed=5)
    params["w_router"][0][:2] = 5.0 * np.sign(x.mean(axis=0))[None, :] + params["w_router"][0][:2]
    x = np.abs(x) * np.sign(x.mean(axis=0))[None, :]
    new, rec = to.train_step(params, 0, x, y, sh, 0.1)
    assert rec["counts"][2] == 0 and rec["counts"][3] == 0
    assert np.array_equal(new["w1"][2:], params["w1"][2:])
    assert np.array_equal(new["w2"][2:], params["w2"][2:])


def test_party_schedule_is_one_permutation_per_epoch():
    sched = mi.party_schedule(5, 7, seed=3)
    assert len(sched) == 7
    for order in sched:
        assert sorted(order) == list(range(5))
    assert sched == mi.party_schedule(5, 7, seed=3)
    assert len({tuple(o) for o in sched}) > 1  # the order changes between epochs


def test_round_robin_order_and_composition():
    """Alg. 1's loop order against brute-force enumeration, and the run equals the
    same train_steps taken one by one."""
    sh = batch_shape(T=6)
    n, B, nb = 3, 2, 3
    params = rand_params(n, sh, seed=31, wscale=0.3)
    batches = mi.train_batches(sh, n, nb, seed=32)
    sched = mi.party_schedule(n, 2, seed=33)
    final, log = to.round_robin_train(params, batches, sched, B, sh, 0.02)
    # enumeration: epoch -> the epoch's permutation -> B consecutive turns of that party,
    # each party's batches read in order and cycled over its nb batches
    seen = {i: 0 for i in range(n)}
    expect = []
    for order in sched:
        for i in order:
            for _ in range(B):
                expect.append((i, seen[i] % nb))
                seen[i] += 1
    assert [(r["party"], r["batch"]) for r in log] == expect
    p = {k: v.copy() for k, v in params.items()}
    for i, b in expect:
        p, _ = to.train_step(p, i, batches[i][b][0], batches[i][b][1], sh, 0.02)
    for k in p:
        assert np.array_equal(p[k], final[k]), k


def test_training_lowers_the_loss():
    """Gradient descent with a small step on a fixed teacher: the mean loss of the last
    epoch is below that of the first."""
    sh = batch_shape(T=16, aux_alpha=0.01)
    n, B = 2, 2
    params = rand_params(n, sh, seed=41, wscale=0.3)
    batches = mi.train_batches(sh, n, 2, seed=42)
    sched = mi.party_schedule(n, 6, seed=43)
    _, log = to.round_robin_train(params, batches, sched, B, sh, 0.1)
    per_epoch = n * B
    first = np.mean([r["loss"] for r in log[:per_epoch]])
    last = np.mean([r["loss"] for r in log[-per_epoch:]])
    assert last < 0.9 * first, (first, last)
