"""Expert parallelism on the GPU kernels: every party's share of the layer
(`ep.PartyExpertLayer`: its own gating, dispatch grouped by host party, the exchanges,
the GEMMs of the experts it hosts, the combine, the router backward, the unpermute)
run through the C ABI, against the single-GPU layer on all parties' tokens.

This run has one GPU, so the parties are host threads sharing it, and the exchange
stands in for the network: a barrier (every party has queued its send rows), device
copies of each source's block into each receiver's buffer, a second barrier (every
party has queued its reads before anyone queues more work). All work goes to one
stream in that host order; no kernel waits for another party's kernel. The same rows
reach every expert in the same order as in the single-GPU layer, so outputs, input
gradients and hosted experts' weight gradients are bit-identical; the router weight
gradient is summed over differently chunked tokens (fp32 partials) and is compared
within the stage tolerance.
"""
import threading

import numpy as np
import pytest
import torch

from oracle import seeds
from paper_2506_02965_gb300 import ep
from paper_2506_02965_gb300.layer import MoELayer
from synth import moe_inputs as mi
from tests._cmp import assert_close
from tests.gpu_util import need_gpu, status

pytestmark = pytest.mark.gpu


class LocalExchange:
    """The collectives of P parties that share this process and GPU."""

    def __init__(self, P):
        self.P = P
        self.barrier = threading.Barrier(P, timeout=120)
        self.slots = [None] * P

    def gather_counts(self, rank, counts):
        self.slots[rank] = np.asarray(counts, np.int64)
        self.barrier.wait()
        out = np.stack(self.slots)
        self.barrier.wait()
        return out

    def exchange(self, rank, rows, send_splits, recv_splits):
        self.slots[rank] = (rows, list(send_splits))
        self.barrier.wait()
        parts = []
        for s in range(self.P):
            src, splits = self.slots[s]
            start = int(sum(splits[:rank]))
            parts.append(src[start:start + int(splits[rank])])
        out = torch.cat(parts) if parts else rows[:0]
        assert out.shape[0] == sum(recv_splits)
        self.barrier.wait()
        return out


class PartyTransport:
    def __init__(self, ex, rank):
        self.ex, self.rank = ex, rank

    def gather_counts(self, counts):
        return self.ex.gather_counts(self.rank, counts)

    def exchange(self, rows, send_splits, recv_splits):
        return self.ex.exchange(self.rank, rows, send_splits, recv_splits)


@pytest.mark.parametrize("P,E,k,Tp,d,F,zipf", [(2, 4, 2, 256, 256, 256, 0.0), (3, 8, 2, 200, 128, 256, 0.0),
                                                (4, 8, 3, 384, 256, 512, 1.2), (2, 16, 4, 320, 128, 128, 0.0),
                                                (3, 2, 2, 128, 128, 128, 0.0)])  # party 2 hosts no expert
def test_parties_on_gpu_kernels_match_single_gpu_layer(P, E, k, Tp, d, F, zipf):
    L = need_gpu()
    sh = mi.MoEShape("ep", P * Tp, d, E, F, k, "bf16", n_parties=P, zipf_s=zipf, seed=500 + P)
    sh = sh.with_(seed=seeds.decided_seed(sh))
    inp = mi.make_inputs(sh)
    ref = MoELayer(sh, owner_grouped=True)
    ref.load(inp)
    ref.step()
    torch.cuda.synchronize()
    assert status(L) == 0

    ex = LocalExchange(P)
    po = inp["party_offsets"]
    dt = torch.bfloat16
    parties = []
    for r in range(P):
        rows = slice(po[r], po[r + 1])
        p = ep.PartyExpertLayer(sh, r, P, Tp, PartyTransport(ex, r))
        own = p.experts
        p.load(torch.from_numpy(inp["x"][rows]).to(dt), torch.from_numpy(inp["dout"][rows]).to(dt),
               torch.from_numpy(inp["w_router"][r]).to(dt),
               None if inp["router_bias"] is None else torch.from_numpy(inp["router_bias"][r]),
               torch.from_numpy(inp["w1"][own]).to(dt), torch.from_numpy(inp["w2"][own]).to(dt))
        parties.append(p)
    errors = []

    def run(p):
        try:
            p.step()
        except BaseException as exc:  # reported after the join
            errors.append(exc)
            ex.barrier.abort()

    threads = [threading.Thread(target=run, args=(p,)) for p in parties]
    for t in threads:
        t.start()
    for t in threads:
        t.join(timeout=300)
    assert not errors, errors
    torch.cuda.synchronize()
    assert status(L) == 0

    cross = 0
    for r, p in enumerate(parties):
        assert p.dw1.shape[0] == len(p.experts) and p.dw2.shape[0] == len(p.experts)
        rows = slice(po[r], po[r + 1])
        assert torch.equal(p.topk_idx, ref.topk_idx[rows])
        assert torch.equal(p.counts[0], ref.counts[r])
        assert torch.equal(p.aux_loss[0], ref.aux_loss[r])
        assert torch.equal(p.out, ref.out[rows]), r
        assert torch.equal(p.dtopk_w, ref.dtopk_w[rows]), r
        assert torch.equal(p.dlogits, ref.dlogits[rows]), r
        assert torch.equal(p.dx_router, ref.dx_router[rows]), r
        assert torch.equal(p.dx, ref.dx[rows]), r
        for i, e in enumerate(p.experts):
            assert torch.equal(p.dw1[i], ref.dw1[e]), (r, e)
            assert torch.equal(p.dw2[i], ref.dw2[e]), (r, e)
        assert_close("dw_router", p.dw_router[0], ref.dw_router[r].float().cpu().numpy(), 2e-2, stage=True)
        assert_close("dbias", p.dbias[0], ref.dbias[r].cpu().numpy(), 1e-5, stage=True)
        cross += sum(p.plan.send_splits) - p.plan.send_splits[r]
    assert cross > 0  # rows really went to other parties' experts
