"""Expert parallelism across parties: the "Send" steps of PC-MoE.

In PC-MoE every party hosts a share of the global expert pool (round-robin: expert e
lives on party e mod P, Sec. 3.1) and keeps its gating function local. A party routes
its own tokens and sends each token's hidden state to the host of every expert it
picked (Alg. 3, ProcessExperts). The host runs the expert and returns the output,
which the party sums with its gate weights. In the backward the party sends the
gradient w.r.t. each expert output to the host (Alg. 5, BackwardExperts); the host
back-propagates through the expert, updates it locally and returns one
activation-sized gradient w.r.t. the expert input (Sec. 3.2). There is no all-reduce:
weight gradients never leave their host.

One process per party (rank = party). This module holds the part of that protocol
that is not arithmetic:

  * ``ExchangePlan``: from the per-(source party, expert) row counts, which every
    rank learns with one all-gather of E integers, it derives the split sizes of
    the two all-to-all exchanges and the row permutation between the received
    blocks (source-major) and the expert-major order the grouped expert GEMMs need.
    Inside one expert the rows then follow the sources in party order and, within a
    source, the token order; tokens are party-contiguous, so this is the global
    token order, the same row order as the single-process owner-grouped layout
    (``moe_dispatch_owner``). Weight gradients are then summed over the same rows in
    the same order as on one GPU.
  * ``exchange``: one ``torch.distributed.all_to_all_single`` of row blocks, used
    forward (send rows to their hosts, return expert outputs) and backward (send
    output gradients, return input gradients). NCCL on GPUs, gloo on host tensors.

The source side lays out its rows with ``moe_dispatch_owner`` over its own tokens
(party_offsets with only this party non-empty), which groups them by owner party
and gives send_counts; the host's gathers between received order and expert-major
order use the permutations of the plan. Row gathers are the caller's: the GPU
driver gathers with the library's kernels, the CPU tests with the oracle's.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


def owner_of(e: int, n_parties: int) -> int:
    """The party hosting expert e (round-robin, Sec. 3.1)."""
    return e % n_parties


def owned_experts(rank: int, n_experts: int, n_parties: int) -> list:
    """Experts hosted by `rank`, ascending (the owner-grouped segment order)."""
    return [e for e in range(n_experts) if owner_of(e, n_parties) == rank]


@dataclass
class ExchangePlan:
    """Split sizes and permutations of one rank's exchanges (see the module doc).

    send_splits[o]  rows this rank sends to owner o (its owner-grouped x_perm has them
                    contiguous, owners in order)
    recv_splits[s]  rows this rank receives from source s
    experts         experts this rank hosts (ascending)
    offsets         [len(experts)+1]: expert-major row ranges of the hosted experts
    to_expert       [R]: expert-major row j is received row to_expert[j]
    to_source       [R]: received row i is expert-major row to_source[i] (inverse)
    """
    rank: int
    n_parties: int
    send_splits: list
    recv_splits: list
    experts: list
    offsets: np.ndarray
    to_expert: np.ndarray
    to_source: np.ndarray

    @property
    def rows_in(self) -> int:
        return int(sum(self.recv_splits))

    @property
    def rows_out(self) -> int:
        return int(sum(self.send_splits))


def make_plan(counts, rank: int) -> ExchangePlan:
    """counts[s][e]: rows of source party s picked for expert e (every party's
    per-expert counts, e.g. the all-gathered output of moe_route with P = 1)."""
    C = np.asarray(counts, dtype=np.int64)
    P, E = C.shape
    if not 0 <= rank < P:
        raise ValueError(f"rank {rank} outside [0, {P})")
    if (C < 0).any():
        raise ValueError("negative count")
    by_owner = [owned_experts(o, E, P) for o in range(P)]
    send = [int(C[rank, by_owner[o]].sum()) for o in range(P)]
    mine = by_owner[rank]
    recv = [int(C[s, mine].sum()) for s in range(P)]
    # received layout: source blocks in order; inside a block, experts in `mine` order
    base = np.zeros((P, len(mine)), np.int64)
    pos = 0
    for s in range(P):
        for i, e in enumerate(mine):
            base[s, i] = pos
            pos += C[s, e]
    offsets = np.zeros(len(mine) + 1, np.int64)
    to_expert = np.empty(pos, np.int64)
    j = 0
    for i, e in enumerate(mine):
        for s in range(P):
            n = int(C[s, e])
            to_expert[j:j + n] = base[s, i] + np.arange(n)
            j += n
        offsets[i + 1] = j
    to_source = np.empty_like(to_expert)
    to_source[to_expert] = np.arange(len(to_expert))
    return ExchangePlan(rank, P, send, recv, mine, offsets, to_expert, to_source)


def gather_counts(local_counts, group=None):
    """All-gather every party's per-expert counts [E] -> [P, E] (int64, host)."""
    import torch
    import torch.distributed as dist
    t = torch.as_tensor(np.asarray(local_counts, np.int64))
    world = dist.get_world_size(group)
    dev = "cuda" if dist.get_backend(group) == "nccl" else "cpu"
    t = t.to(dev)
    out = [torch.empty_like(t) for _ in range(world)]
    dist.all_gather(out, t, group=group)
    return torch.stack(out).cpu().numpy()


def exchange(rows, send_splits, recv_splits, group=None):
    """Send row blocks to every rank and receive theirs: block o of `rows` (send_splits[o]
    rows, contiguous, in rank order) goes to rank o; the result holds the blocks
    received from ranks 0..P-1 in order (recv_splits rows each). Backward exchanges
    swap the two split lists."""
    import torch
    import torch.distributed as dist
    if rows.shape[0] != sum(send_splits):
        raise ValueError(f"{rows.shape[0]} rows, splits sum to {sum(send_splits)}")
    out = torch.empty((int(sum(recv_splits)),) + tuple(rows.shape[1:]), dtype=rows.dtype,
                      device=rows.device)
    dist.all_to_all_single(out, rows.contiguous(), output_split_sizes=[int(v) for v in recv_splits],
                           input_split_sizes=[int(v) for v in send_splits], group=group)
    return out


# ----------------------------------------------------------------------------- GPU party
class DistTransport:
    """The exchanges of one rank over torch.distributed (NCCL between GPUs)."""

    def __init__(self, group=None):
        self.group = group

    def gather_counts(self, counts):
        return gather_counts(counts, self.group)

    def exchange(self, rows, send_splits, recv_splits):
        return exchange(rows, send_splits, recv_splits, self.group)


class PartyExpertLayer:
    """One party's share of the MoE layer under expert parallelism, on its own GPU.

    The party holds its tokens x [T_p, d], its gating W_r [E, d] (+ bias), and the
    weights of the experts it hosts (expert e with e mod P == rank, ascending):
    w1 [E_o, 2F, d], w2 [E_o, d, F]. A step runs every kernel of the layer on this GPU
    through the C ABI; `transport` carries the all-gather of the per-expert counts and
    the four row exchanges (hidden states to the hosts, outputs back, output gradients
    to the hosts, input gradients back). Nothing of this party's gating, and no weight
    gradient of a hosted expert, leaves the GPU (Sec. 3.2: no all-reduce).

    Results: out, dx [T_p, d] (this party's tokens); dw_router [E, d], dbias [E];
    dw1, dw2 of the hosted experts; aux_loss [1].
    """

    def __init__(self, shape, rank: int, n_parties: int, tokens: int, transport,
                 device: str = "cuda"):
        import torch
        from . import _lib as L
        self.L, self.torch = L, torch
        self.sh, self.rank, self.P, self.Tp = shape, rank, n_parties, tokens
        self.transport = transport
        self.device = device
        E, d, F, k = shape.n_experts, shape.d_model, shape.d_ff, shape.top_k
        self.dt = torch.bfloat16 if shape.dtype == "bf16" else torch.float32
        self.dtype_code = L.MOE_BF16 if shape.dtype == "bf16" else L.MOE_F32
        self.experts = owned_experts(rank, E, n_parties)
        mk = lambda T, E_, k_, P_=1: L.make_config(T, d, E_, F, k_, P_, 0, 0, shape.normalize_topk,  # noqa: E731
                                                   shape.aux_alpha, self.dtype_code)
        self.cfg = mk(tokens, E, k)                # this party's gating, combine, unpermute
        self.cfg_owner = mk(tokens, E, k, n_parties)  # rows grouped by host party
        z = lambda *s, dtype=None: torch.empty(*s, dtype=dtype or self.dt, device=device)  # noqa: E731
        f32, i32 = torch.float32, torch.int32
        T, TK, Eo = tokens, tokens * k, len(self.experts)
        self.x, self.dout = z(T, d), z(T, d)
        self.w_router, self.router_bias = z(1, E, d), None
        self.w1, self.w2 = z(Eo, 2 * F, d), z(Eo, d, F)  # empty for a party hosting no expert
        self.logits, self.probs = z(T, E, dtype=f32), z(T, E, dtype=f32)
        self.topk_idx, self.topk_w = z(T, k, dtype=i32), z(T, k, dtype=f32)
        self.counts = z(1, E, dtype=i32)
        self.aux_loss, self.aux_coef = z(1, dtype=f32), z(1, E, dtype=f32)
        po = [0] * (rank + 1) + [T] * (n_parties - rank)   # only this party's tokens
        self.party_offsets = torch.tensor(po, dtype=i32, device=device)
        self.group_expert, self.offsets = z(E, dtype=i32), z(E + 1, dtype=i32)
        self.slot_of, self.token_of = z(TK, dtype=i32), z(TK, dtype=i32)
        self.send_counts = z(n_parties, n_parties, dtype=i32)
        self.x_perm, self.y_perm = z(TK, d), z(TK, d)
        self.out = z(T, d)
        self.dy_perm, self.dtopk_w, self.dx_perm = z(TK, d), z(T, k, dtype=f32), z(TK, d)
        self.dlogits, self.dw_router = z(T, E, dtype=f32), z(1, E, d)
        self.dbias, self.dx_router, self.dx = z(1, E, dtype=f32), z(T, d), z(T, d)
        self.dw1, self.dw2 = torch.empty_like(self.w1), torch.empty_like(self.w2)
        self.ws_bytes = max(L.moe_workspace_size(self.cfg), L.moe_workspace_size(self.cfg_owner))
        self.workspace = torch.empty(max(self.ws_bytes, 16), dtype=torch.uint8, device=device)
        self.plan = None

    def load(self, x, dout, w_router, router_bias, w1_owned, w2_owned):
        self.x.copy_(x)
        self.dout.copy_(dout)
        self.w_router.copy_(w_router.reshape(self.w_router.shape))
        if router_bias is not None:
            self.router_bias = router_bias.reshape(1, -1).to(self.device, self.torch.float32).contiguous()
        if self.experts:
            self.w1.copy_(w1_owned)
            self.w2.copy_(w2_owned)

    def _gather(self, src, rows_idx, n_src):
        out = self.torch.empty((len(rows_idx),) + tuple(src.shape[1:]), dtype=src.dtype, device=self.device)
        idx = self.torch.as_tensor(rows_idx, dtype=self.torch.int32, device=self.device)
        self.L.moe_gather_rows(src, idx, len(rows_idx), n_src, src.shape[1], self.dtype_code, out)
        return out

    def _host_cfg(self, rows: int):
        sh = self.sh
        return self.L.make_config(rows, sh.d_model, max(len(self.experts), 1), sh.d_ff, 1, 1, 0, 0,
                                  sh.normalize_topk, sh.aux_alpha, self.dtype_code)

    def forward(self):
        L, torch, pl = self.L, self.torch, None
        L.moe_route(self.cfg, self.x, self.w_router, self.router_bias, None, self.logits, self.probs,
                    self.topk_idx, self.topk_w, self.counts)
        L.moe_aux_loss(self.cfg, self.probs, self.counts, None, self.aux_loss, self.aux_coef)
        self.plan = pl = make_plan(self.transport.gather_counts(self.counts[0].cpu().numpy()), self.rank)
        L.moe_dispatch_owner(self.cfg_owner, self.topk_idx, self.x, self.party_offsets, self.group_expert,
                             self.offsets, self.slot_of, self.token_of, self.x_perm, self.send_counts,
                             self.workspace, self.ws_bytes)
        recv = self.transport.exchange(self.x_perm, pl.send_splits, pl.recv_splits)
        # host: the received rows in expert-major order, the hosted experts' forward
        R = pl.rows_in
        self.xe = self._gather(recv, pl.to_expert, R)
        d, F = self.sh.d_model, self.sh.d_ff
        self.h_gu = torch.empty(R, 2 * F, dtype=self.dt, device=self.device)
        self.act = torch.empty(R, F, dtype=self.dt, device=self.device)
        ye = torch.empty(R, d, dtype=self.dt, device=self.device)
        self.host_offsets = torch.as_tensor(pl.offsets, dtype=torch.int32, device=self.device)
        if R and self.experts:
            L.moe_expert_ffn_fwd(self._host_cfg(R), self.xe, self.host_offsets, self.w1, self.w2, self.h_gu,
                                 self.act, ye)
        back = self._gather(ye, pl.to_source, R)
        self.y_perm = self.transport.exchange(back, pl.recv_splits, pl.send_splits)
        L.moe_combine_fwd(self.cfg, self.y_perm, self.topk_w, self.slot_of, None, self.out)

    def backward(self):
        L, torch, pl = self.L, self.torch, self.plan
        L.moe_combine_bwd(self.cfg, self.dout, self.y_perm, self.topk_w, self.slot_of, self.dy_perm,
                          self.dtopk_w)
        R = pl.rows_in
        dye = self._gather(self.transport.exchange(self.dy_perm, pl.send_splits, pl.recv_splits),
                           pl.to_expert, R)
        d, F = self.sh.d_model, self.sh.d_ff
        dh = torch.empty(R, 2 * F, dtype=self.dt, device=self.device)
        dxe = torch.empty(R, d, dtype=self.dt, device=self.device)
        if self.experts:
            L.moe_expert_ffn_bwd(self._host_cfg(R), self.xe, self.host_offsets, self.w1, self.w2, self.h_gu,
                                 self.act, dye, dh, dxe, self.dw1, self.dw2)
        back = self._gather(dxe, pl.to_source, R)
        self.dx_perm = self.transport.exchange(back, pl.recv_splits, pl.send_splits)
        L.moe_route_bwd(self.cfg, self.x, self.w_router, self.probs, self.topk_idx, self.topk_w, self.dtopk_w,
                        self.aux_coef, None, self.dlogits, self.dw_router, self.dbias, self.dx_router,
                        self.workspace, self.ws_bytes)
        L.moe_dispatch_bwd(self.cfg, self.dx_perm, self.slot_of, self.dx_router, None, self.dx)

    def step(self):
        self.forward()
        self.backward()
