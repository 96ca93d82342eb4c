"""GPU training step of Alg. 1 (toy block) against the training oracle: the SGD update
and the MSE loss kernels, the trainer over several epochs (fp32 and bf16), and the
parameters that must not move (other parties' gating, experts a batch did not call)."""
import numpy as np
import pytest
import torch

from oracle import train_oracle as to
from synth import moe_inputs as mi
from tests._cmp import assert_close
from tests.gpu_util import dev, need_gpu, status

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    return need_gpu()


def ulp(ref, dtype):
    """Spacing of the storage type at |ref| (bf16: 8 significant bits, fp32: 24)."""
    s = np.spacing(np.abs(np.asarray(ref, np.float32)))
    return s * (2.0 ** 16 if dtype == "bf16" else 1.0)


def rounded(a, dtype):
    a = np.asarray(a, np.float32)
    return mi.bf16_round(a) if dtype == "bf16" else a


@pytest.mark.parametrize("dtype,groups,elems,offset", [
    ("bf16", 8, 4096, 0), ("f32", 8, 4096, 0),
    ("bf16", 5, 1001, 0),   # groups not a multiple of the 16-byte vector: element path
    ("f32", 3, 4096, 1),    # misaligned base: element path
    ("bf16", 1, 1 << 20, 0)])
def test_sgd_update_matches_oracle(L, dtype, groups, elems, offset):
    rng = np.random.default_rng(groups * elems + offset)
    w0 = rounded(rng.standard_normal((groups, elems)), dtype)
    g = rounded(rng.standard_normal((groups, elems)), dtype)
    counts = rng.integers(0, 3, groups).astype(np.int32)
    counts[0] = 1
    lr = 0.0371
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    wbuf = dev(np.concatenate([np.zeros(offset, np.float32), w0.ravel()]), tdt)
    gbuf = dev(np.concatenate([np.zeros(offset, np.float32), g.ravel()]), tdt)
    w, gd = wbuf[offset:], gbuf[offset:]
    L.moe_sgd_update(w, gd, groups, elems, dev(counts, torch.int32), lr,
                     L.MOE_BF16 if dtype == "bf16" else L.MOE_F32)
    assert status(L) == 0
    got = w.float().cpu().numpy().reshape(groups, elems)
    ref = to.sgd_groups(w0, g, np.float32(lr), counts)
    for q in range(groups):
        if counts[q] <= 0:
            assert np.array_equal(got[q], w0[q]), q  # not called: not touched
        else:
            assert (np.abs(got[q] - ref[q]) <= ulp(ref[q], dtype)).all(), q
    # without counts every group moves
    w2 = dev(w0, tdt)
    L.moe_sgd_update(w2, dev(g, tdt), groups, elems, None, lr, L.MOE_BF16 if dtype == "bf16" else L.MOE_F32)
    ref2 = to.sgd_groups(w0, g, np.float32(lr))
    assert (np.abs(w2.float().cpu().numpy() - ref2) <= ulp(ref2, dtype)).all()


@pytest.mark.parametrize("elems", [4096, 1001])
def test_sgd_update_with_fp32_master(L, elems):
    """bf16 weights with an fp32 master copy: the master takes the step (within one fp32
    spacing of the oracle), the bf16 weights become the master rounded to bf16 (bit for
    bit), and groups not called keep both copies."""
    groups = 4
    rng = np.random.default_rng(elems)
    m0 = (0.02 * rng.standard_normal((groups, elems))).astype(np.float32)
    g = mi.bf16_round(rng.standard_normal((groups, elems)).astype(np.float32))
    w0 = mi.bf16_round(m0)
    counts = np.array([3, 0, 1, 0], np.int32)
    lr = 1e-4  # steps far below the bf16 spacing of the weights
    m, w = dev(m0, torch.float32), dev(w0, torch.bfloat16)
    L.moe_sgd_update(w, dev(g, torch.bfloat16), groups, elems, dev(counts, torch.int32), lr, L.MOE_BF16,
                     w_master=m)
    assert status(L) == 0
    gm, gw = m.cpu().numpy(), w.float().cpu().numpy()
    ref = to.sgd_groups(m0, g, np.float32(lr), counts)
    for q in range(groups):
        if counts[q] <= 0:
            assert np.array_equal(gm[q], m0[q]) and np.array_equal(gw[q], w0[q]), q
        else:
            assert (np.abs(gm[q] - ref[q]) <= ulp(ref[q], "f32")).all(), q
            assert np.array_equal(gw[q], mi.bf16_round(gm[q])), q
            assert not np.array_equal(gm[q], m0[q])  # the master moved


@pytest.mark.parametrize("dtype,T,d", [("bf16", 1000, 384), ("f32", 77, 36), ("f32", 4096, 1024)])
def test_mse_loss_matches_oracle(L, dtype, T, d):
    rng = np.random.default_rng(T + d)
    out = rounded(rng.standard_normal((T, d)), dtype)
    y = rounded(rng.standard_normal((T, d)), dtype)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    cfg = L.make_config(T, d, 8, 128, 2, dtype=L.MOE_BF16 if dtype == "bf16" else L.MOE_F32)
    ws = torch.empty(L.moe_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    loss = torch.empty(1, device="cuda")
    dout = torch.empty(T, d, dtype=tdt, device="cuda")
    L.moe_mse_loss(cfg, dev(out, tdt), dev(y, tdt), loss, dout, ws, ws.numel())
    assert status(L) == 0
    rl, rg = to.mse_loss(out, y)
    assert abs(loss.item() - rl) <= 1e-5 * rl
    got = dout.float().cpu().numpy()
    bound = ulp(rg, dtype) if dtype == "bf16" else 4 * ulp(rg, dtype)
    assert (np.abs(got - rg) <= bound + 1e-30).all()
    # a second call gives the same bits (fixed-order reduction)
    l2 = torch.empty(1, device="cuda")
    L.moe_mse_loss(cfg, dev(out, tdt), dev(y, tdt), l2, dout, ws, ws.numel())
    assert torch.equal(loss, l2)


def _trainer(sh, n, lr, init, batches):
    from paper_2506_02965_gb300.train import RoundRobinTrainer
    tr = RoundRobinTrainer(sh, n, lr)
    tr.load(init)
    tdt = tr.layer.dt
    dbatches = [[(dev(x, tdt), dev(y, tdt)) for x, y in mine] for mine in batches]
    return tr, dbatches


def _decided_run(sh, n, B, epochs, lr, nb, seed0, margin):
    """Seeds whose every oracle step routes each token with a top-(k+1) logit gap above
    ``margin``, so that the GPU's fp32 logits pick the same experts in the same order
    (the comparison is unique)."""
    for s in range(seed0, seed0 + 100):
        init = mi.train_init(sh, n, seed=s)
        batches = mi.train_batches(sh, n, nb, seed=s + 1)
        sched = mi.party_schedule(n, epochs, seed=s + 2)
        final, log = to.round_robin_train(init, batches, sched, B, sh, lr)
        if min(r["min_margin"] for r in log) > margin:
            return init, batches, sched, final, log
    raise RuntimeError("no decided seed")


def test_trainer_matches_oracle_fp32(L):
    """Alg. 1 with 3 parties, B = 2, two epochs (12 batches) in fp32: turn order, every
    batch's MSE and aux loss, and the final parameters against the oracle."""
    sh = mi.MoEShape("train_f32", 64, 64, 6, 64, 2, "f32", aux_alpha=0.05)
    n, B, epochs, lr = 3, 2, 2, 0.05
    init, batches, sched, final, log = _decided_run(sh, n, B, epochs, lr, nb=3, seed0=500, margin=5e-5)
    tr, dbatches = _trainer(sh, n, lr, init, batches)
    order, losses = tr.run(dbatches, sched, B)
    assert status(L) == 0
    assert order == [(r["party"], r["batch"]) for r in log]
    got = losses.cpu().numpy()
    assert_close("mse", got[:, 0], [r["mse"] for r in log], 1e-4)
    assert_close("aux", got[:, 1], [r["aux"] for r in log], 1e-4)
    assert_close("w_router", tr.w_router, final["w_router"], 1e-4)
    assert_close("w1", tr.w1, final["w1"], 1e-4)
    assert_close("w2", tr.w2, final["w2"], 1e-4)


def test_trainer_bf16_step_by_step(L):
    """bf16 layer with fp32 master weights: two parties, two epochs of one batch each.
    Every step is compared from the same state: the oracle runs the layer on the GPU's
    bf16 weights before the step, and its update is added to the GPU's masters. Each
    master lands within one fp32 spacing of that plus 2% of the largest update of its
    tensor (the bf16 layer's norm-wise tolerance); the bf16 weights are the masters
    rounded, bit for bit; the batch's MSE is within the bf16 tolerance."""
    sh = mi.MoEShape("train_bf16", 256, 128, 8, 128, 2, "bf16", aux_alpha=0.01)
    n, B, epochs, lr = 2, 1, 2, 0.05
    init, batches, sched, _, _ = _decided_run(sh, n, B, epochs, lr, nb=1, seed0=700, margin=2e-4)
    tr, dbatches = _trainer(sh, n, lr, init, batches)
    assert tr.master
    rec = torch.empty(2, device="cuda")
    pairs = (("w_router", "m_router"), ("w1", "m1"), ("w2", "m2"))
    for order in sched:
        for i in order:
            w16 = {k: getattr(tr, k).float().cpu().numpy().astype(np.float64) for k, _ in pairs}
            m32 = {k: getattr(tr, mk).cpu().numpy().astype(np.float64) for k, mk in pairs}
            x, y = batches[i][0]
            ref, r = to.train_step(w16, i, x, y, sh, lr)
            assert r["min_margin"] > 1e-5  # the routing is decided from this state
            tr.step(i, *dbatches[i][0], record=rec)
            assert status(L) == 0
            assert_close("mse", rec[0:1], [r["mse"]], 2e-2)
            for k, mk in pairs:
                delta = ref[k] - w16[k]
                want = m32[k] + delta
                gm = getattr(tr, mk).cpu().numpy()
                bound = ulp(want, "f32") + 2e-2 * np.abs(delta).max() + 1e-12
                assert (np.abs(gm - want) <= bound).all(), (k, i)
                assert np.array_equal(getattr(tr, k).float().cpu().numpy(), mi.bf16_round(gm)), k


def test_uncalled_experts_and_other_parties_do_not_move(L):
    """A batch whose tokens all pick experts 0 and 1: experts 2..5 keep their bits, as
    does the other party's gating; the active party's gating and experts 0, 1 move."""
    sh = mi.MoEShape("train_mask", 32, 64, 6, 64, 2, "f32", aux_alpha=0.01)
    init = mi.train_init(sh, 2, seed=9)
    init["w_router"][1, :2] = 0.5
    (x, y), = mi.train_batches(sh, 1, 1, seed=10)[0]
    x = np.abs(x)
    tr, db = _trainer(sh, 2, 0.1, init, [[(x, y)]])
    xd, yd = db[0][0]
    before = {k: v.clone() for k, v in (("w1", tr.w1), ("w2", tr.w2), ("w_router", tr.w_router))}
    tr.step(1, xd, yd)
    assert status(L) == 0
    counts = tr.layer.counts.cpu().numpy()[0]
    assert counts[0] == sh.T and counts[1] == sh.T and not counts[2:].any()
    for k in ("w1", "w2"):
        now = getattr(tr, k)
        assert torch.equal(now[2:], before[k][2:]), k
        assert not torch.equal(now[:2], before[k][:2]), k
    assert torch.equal(tr.w_router[0], before["w_router"][0])
    assert not torch.equal(tr.w_router[1], before["w_router"][1])
