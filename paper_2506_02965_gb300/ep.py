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
