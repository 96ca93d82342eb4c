"""Sequential collaborative training of PC-MoE (Alg. 1) on one GPU, for a toy block whose
only layer is the MoE expert layer.

The n parties share one pool of E experts (expert e is hosted by party e mod n) and each
owns its gating W_r[i] (Alg. 7). In every epoch the parties take turns in a random
order; party i runs B batches of its own tokens. A batch is: the layer's forward with
W_r[i] (LocalForward / ProcessExperts, Alg. 2 and 3), the loss against the batch's
targets (moe_mse_loss: sum ||h - y||^2 / 2T), the layer's backward (Alg. 5 and 6), the
SGD update of W_r[i] (BackwardLocal, Alg. 4) and of every expert the batch called
(BackwardExpert: an expert with no routed token is neither read nor written). Nothing
else changes: there is no global broadcast. Every step runs in the CUDA library on one
stream (no host synchronisation inside a run); the host only picks the turn order and
the batches.

Layouts: W_r [n,E,d]; W1 [E,2F,d]; W2 [E,d,F] (the layer's own buffers); for bf16, fp32
master copies of the three (the SGD updates them and rounds into the bf16 weights, so
that steps below the bf16 spacing are not lost); batches are device tensors x, y [T,d]
of the layer's dtype.
"""
from __future__ import annotations

import numpy as np
import torch

from . import _lib as L
from .layer import MoELayer


class RoundRobinTrainer:
    def __init__(self, shape, n_parties: int, lr: float, device: str = "cuda", master=None):
        """shape: one batch (T tokens of one party: n_parties = 1, no shared experts).
        master: keep fp32 master copies of the parameters that the SGD updates and
        round into the layer's bf16 weights (default: for bf16 shapes)."""
        if shape.n_parties != 1:
            raise ValueError("a batch holds the tokens of one party: shape.n_parties must be 1")
        if shape.n_shared:
            raise ValueError("the toy block has no shared experts")
        if n_parties < 1:
            raise ValueError("n_parties must be >= 1")
        self.shape, self.n, self.lr = shape, int(n_parties), float(lr)
        self.layer = lay = MoELayer(shape, device)
        E, d = shape.n_experts, shape.d_model
        self.w_router = torch.empty(self.n, E, d, dtype=lay.dt, device=device)
        self.mse = torch.empty(1, dtype=torch.float32, device=device)
        self.dtype = L.MOE_BF16 if shape.dtype == "bf16" else L.MOE_F32
        self.master = (shape.dtype == "bf16") if master is None else bool(master)
        if self.master:
            f32 = torch.float32
            self.m_router = torch.empty(self.w_router.shape, dtype=f32, device=device)
            self.m1 = torch.empty(lay.w1.shape, dtype=f32, device=device)
            self.m2 = torch.empty(lay.w2.shape, dtype=f32, device=device)
        else:
            self.m_router = self.m1 = self.m2 = None

    # ------------------------------------------------------------------ parameters
    @property
    def w1(self):
        return self.layer.w1

    @property
    def w2(self):
        return self.layer.w2

    def load(self, init: dict):
        """The common initialization: w_router [n,E,d], w1, w2 as numpy arrays."""
        def put(dst, a):
            dst.copy_(torch.from_numpy(np.ascontiguousarray(a)).to(dst.dtype))

        put(self.w_router, init["w_router"])
        put(self.layer.w1, init["w1"])
        put(self.layer.w2, init["w2"])
        if self.master:
            put(self.m_router, init["w_router"])
            put(self.m1, init["w1"])
            put(self.m2, init["w2"])

    # ------------------------------------------------------------------ one batch
    def step(self, party: int, x, y, stream=None, record=None):
        """One batch of party ``party``: x, y device tensors [T,d] (contiguous, layer
        dtype, 16-byte aligned; used in place, not copied). ``record`` (optional) is a
        device float32 tensor of 2 that receives (MSE, aux loss) of the batch."""
        if not 0 <= party < self.n:
            raise ValueError(f"party {party} outside [0, {self.n})")
        lay, sh = self.layer, self.shape
        main = stream if stream is not None else torch.cuda.current_stream()
        lay.x = x
        lay.w_router = self.w_router[party:party + 1]
        lay.forward(main)
        L.moe_mse_loss(lay.cfg, lay.out, y, self.mse, lay.dout, lay.workspace, lay.ws_bytes,
                       stream=main)
        lay.backward(main)
        E, d, F = sh.n_experts, sh.d_model, sh.d_ff
        # BackwardLocal: the party's gating; BackwardExpert: each called expert
        mr = self.m_router[party] if self.master else None
        L.moe_sgd_update(self.w_router[party], lay.dw_router, 1, E * d, None, self.lr, self.dtype,
                         w_master=mr, stream=main)
        L.moe_sgd_update(lay.w1, lay.dw1, E, 2 * F * d, lay.counts, self.lr, self.dtype,
                         w_master=self.m1, stream=main)
        L.moe_sgd_update(lay.w2, lay.dw2, E, d * F, lay.counts, self.lr, self.dtype,
                         w_master=self.m2, stream=main)
        if record is not None:
            with torch.cuda.stream(main):
                record[0:1].copy_(self.mse)
                record[1:2].copy_(lay.aux_loss)

    # ------------------------------------------------------------------ Alg. 1
    def run(self, batches, schedule, B: int, stream=None):
        """Alg. 1: for each epoch's permutation in ``schedule``, each party in that order
        runs B batches of ``batches[i]`` (its data, read in order and cycled). Returns
        the (party, batch index) of every step and a device tensor [steps, 2] of each
        step's (MSE, aux loss). Queued on the stream; synchronise before reading."""
        if len(batches) != self.n:
            raise ValueError("one list of batches per party")
        steps = sum(len(order) for order in schedule) * B
        log = torch.empty(steps, 2, dtype=torch.float32, device=self.w_router.device)
        used = [0] * self.n
        order_log = []
        for order in schedule:
            if sorted(order) != list(range(self.n)):
                raise ValueError("every epoch's order must be a permutation of the parties")
            for i in order:
                for _ in range(B):
                    b = used[i] % len(batches[i])
                    used[i] += 1
                    x, y = batches[i][b]
                    self.step(i, x, y, stream=stream, record=log[len(order_log)])
                    order_log.append((i, b))
        return order_log, log

    def kernels_per_step(self) -> int:
        """CUDA kernels per batch: the layer's, 2 for the loss, 3 SGD updates."""
        return self.layer.kernels_per_step() + 2 + 3
