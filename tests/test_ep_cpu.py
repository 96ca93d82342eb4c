"""Expert parallelism across parties (Sec. 3.2; the "Send" steps of Alg. 3 and Alg. 5)
as world_size 2-4 gloo process groups on this host, one rank per party.

Each rank routes its own tokens with its own gating function, lays its rows out by
host party, and the exchanges of ``paper_2506_02965_gb300.ep`` carry them to the hosts
and back: hidden states forward, expert outputs back, output gradients forward, input
gradients back. The arithmetic on both sides is the fp64 oracle's (the GPU kernels
need a GPU); what is under test is the exchange: split sizes, the order of the rows
on every rank and the permutations between received and expert-major order. Every
rank's results must equal the single-process oracle layer over all parties' tokens:
the same rows reach each expert in the same order, so the results are bit-identical.
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _shape(P, E, k, Tp):
    from synth import moe_inputs as mi
    return mi.MoEShape("ep", P * Tp, 16, E, 8, k, "f32", n_parties=P, aux_alpha=0.3)


def _inputs(sh, seed):
    from synth import moe_inputs as mi
    rng = np.random.default_rng(seed)
    T, d, E, F, P = sh.T, sh.d_model, sh.n_experts, sh.d_ff, sh.n_parties
    return dict(x=rng.standard_normal((T, d)), w_router=0.5 * rng.standard_normal((P, E, d)),
                router_bias=0.3 * rng.standard_normal((P, E)),
                w1=0.5 * rng.standard_normal((E, 2 * F, d)), w2=0.5 * rng.standard_normal((E, d, F)),
                dout=rng.standard_normal((T, d)), party_offsets=mi.party_offsets(sh),
                ws1=None, ws2=None)


def _rank_main(rank, P, E, k, Tp, seed, port, out_dir):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=P)
    from oracle import moe_oracle as mo
    from paper_2506_02965_gb300 import ep

    sh = _shape(P, E, k, Tp)
    inp = _inputs(sh, seed)
    po = inp["party_offsets"]
    rows = slice(po[rank], po[rank + 1])
    Ts = po[rank + 1] - po[rank]
    x = inp["x"][rows]
    one = np.array([0, Ts])
    # --- source side: this party's gating (Alg. 7) on its own tokens
    z = mo.router_logits(x, inp["w_router"][rank:rank + 1], inp["router_bias"][rank:rank + 1], one)
    p = mo.softmax(z)
    idx = mo.topk_indices(z.astype(np.float32), k)
    w = mo.gate_weights(p, idx, sh.normalize_topk)
    cnt = mo.party_counts(idx, E, one)[0]
    tr = ep.DistTransport()  # the GPU party layer's transport, here over gloo
    plan = ep.make_plan(tr.gather_counts(cnt), rank)
    # rows grouped by host party (owner = e mod P): only this party's tokens
    po_local = np.array([0] * (rank + 1) + [Ts] * (P - rank))
    _, _, _, slot, tok, send = mo.owner_dispatch_tables(idx, E, po_local)
    assert list(send[rank]) == plan.send_splits
    x_perm = mo.gather_permute(x, tok)
    # --- hosts: receive hidden states, run the hosted experts (Alg. 6), send outputs back
    xe = ep.exchange(torch.from_numpy(x_perm), plan.send_splits, plan.recv_splits).numpy()[plan.to_expert]
    F = sh.d_ff
    saved = {}
    ye = np.zeros((plan.rows_in, sh.d_model))
    for i, e in enumerate(plan.experts):
        r = slice(plan.offsets[i], plan.offsets[i + 1])
        if r.stop > r.start:
            saved[e] = mo.swiglu_forward(xe[r], inp["w1"][e], inp["w2"][e])
            ye[r] = saved[e][3]
    y_perm = ep.exchange(torch.from_numpy(ye[plan.to_source]), plan.recv_splits,
                         plan.send_splits).numpy()
    out = mo.combine(y_perm, w, slot)
    loss, coef = mo.aux_loss(p, cnt[None], one, k, sh.aux_alpha)
    # --- backward: output gradients to the hosts, input gradients back (Sec. 3.2)
    dy_perm, dw = mo.combine_backward(inp["dout"][rows], y_perm, w, slot)
    dye = tr.exchange(torch.from_numpy(dy_perm), plan.send_splits, plan.recv_splits).numpy()[plan.to_expert]
    dxe = np.zeros((plan.rows_in, sh.d_model))
    dw1, dw2 = {}, {}
    for i, e in enumerate(plan.experts):
        r = slice(plan.offsets[i], plan.offsets[i + 1])
        if r.stop > r.start:
            G, U, A, _ = saved[e]
            _, dX, dW1, dW2 = mo.swiglu_backward(xe[r], inp["w1"][e], inp["w2"][e], G, U, A, dye[r])
            dxe[r], dw1[e], dw2[e] = dX, dW1, dW2
        else:
            dw1[e], dw2[e] = np.zeros((2 * F, sh.d_model)), np.zeros((sh.d_model, F))
    dx_perm = tr.exchange(torch.from_numpy(dxe[plan.to_source]), plan.recv_splits,
                          plan.send_splits).numpy()
    loc = dict(x=x, w_router=inp["w_router"][rank:rank + 1], party_offsets=one)
    rb = mo.router_backward(loc, sh.with_(T=Ts, n_parties=1), p, idx, w, dw, coef)
    dx = mo.unpermute_reduce(dx_perm, slot) + rb["dx_router"]
    dist.barrier()
    dist.destroy_process_group()
    np.savez(os.path.join(out_dir, f"r{rank}.npz"), out=out, dx=dx, loss=loss, dw_router=rb["dw_router"][0],
             dbias=rb["dbias"][0], experts=np.array(plan.experts, np.int64),
             dw1=np.stack([dw1[e] for e in plan.experts]) if plan.experts else np.zeros((0,)),
             dw2=np.stack([dw2[e] for e in plan.experts]) if plan.experts else np.zeros((0,)),
             sent=np.array(plan.send_splits), received=np.array(plan.recv_splits))


@pytest.mark.parametrize("P,E,k,Tp", [(2, 4, 2, 24), (3, 7, 2, 20), (4, 8, 3, 16)])
def test_expert_parallel_exchange_matches_single_process_layer(tmp_path, P, E, k, Tp):
    sys.path.insert(0, ROOT)
    from oracle import moe_oracle as mo
    seed = 100 * P + E
    mp.start_processes(_rank_main, args=(P, E, k, Tp, seed, _free_port(), str(tmp_path)), nprocs=P,
                       join=True, start_method="spawn")
    sh = _shape(P, E, k, Tp)
    inp = _inputs(sh, seed)
    fwd = mo.layer_forward(inp, sh)
    bwd = mo.layer_backward(inp, sh, fwd)
    po = inp["party_offsets"]
    seen = set()
    cross = 0
    for r in range(P):
        got = np.load(tmp_path / f"r{r}.npz")
        rows = slice(po[r], po[r + 1])
        for name, ref in (("out", fwd["out"][rows]), ("dx", bwd["dx"][rows]),
                          ("loss", fwd["aux_loss"][r:r + 1]), ("dw_router", bwd["dw_router"][r]),
                          ("dbias", bwd["dbias"][r])):
            assert np.array_equal(got[name], ref), (r, name)
        for i, e in enumerate(got["experts"]):
            assert e % P == r
            seen.add(int(e))
            assert np.array_equal(got["dw1"][i], bwd["dw1"][e]), (r, e)
            assert np.array_equal(got["dw2"][i], bwd["dw2"][e]), (r, e)
        # what party r sends to each host = the oracle's cross-party send counts
        _, _, _, _, _, send = mo.owner_dispatch_tables(fwd["topk_idx"], E, po)
        assert (got["sent"] == send[r]).all()
        assert (got["received"] == send[:, r]).all()
        cross += int(got["sent"].sum() - got["sent"][r])
    assert seen == set(range(E))
    assert cross > 0  # the exchange really moved rows between parties


def test_plan_permutations_and_splits():
    """Host-side bookkeeping alone: split sums, inverse permutations, expert-major
    offsets, and source blocks in party order inside each expert."""
    sys.path.insert(0, ROOT)
    from paper_2506_02965_gb300 import ep
    rng = np.random.default_rng(0)
    P, E = 3, 8
    C = rng.integers(0, 5, size=(P, E))
    C[1, 4] = 0
    total_recv = 0
    for r in range(P):
        pl = ep.make_plan(C, r)
        assert pl.experts == [e for e in range(E) if e % P == r]
        assert pl.send_splits == [int(C[r, [e for e in range(E) if e % P == o]].sum()) for o in range(P)]
        assert pl.recv_splits == [int(C[s, pl.experts].sum()) for s in range(P)]
        assert (pl.to_source[pl.to_expert] == np.arange(pl.rows_in)).all()
        assert (np.diff(pl.offsets) == C[:, pl.experts].sum(0)).all()
        # label received rows by (source, expert); expert-major order must be sorted by
        # expert position, then source
        lab = []
        for s in range(P):
            for i, e in enumerate(pl.experts):
                lab += [(i, s)] * int(C[s, e])
        lab = [lab[j] for j in pl.to_expert]
        assert lab == sorted(lab)
        total_recv += pl.rows_in
    assert total_recv == C.sum()
    with pytest.raises(ValueError):
        ep.make_plan(C, P)
