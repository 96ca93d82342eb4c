"""One MoE expert layer on the GPU: buffers in HBM and the fwd+bwd call sequence.

torch provides device memory and streams only; every step runs in the CUDA
library through the C ABI (``_lib``). The sequence is the layer's hot path:

  forward : moe_route -> moe_aux_loss -> moe_dispatch -> moe_expert_ffn_fwd -> moe_combine_fwd
  backward: moe_combine_bwd -> moe_expert_ffn_bwd -> moe_route_bwd -> moe_dispatch_bwd

Layouts (row-major): x, out, dout, dx [T,d]; w_router [P,E,d]; w1 [E,2F,d] (gate
rows then up rows); w2 [E,d,F]; x_perm, y_perm, dy_perm, dx_perm [T*k,d];
h_gu, dh [T*k,2F]; act [T*k,F]; shared experts [S,...] likewise.
"""
from __future__ import annotations

import numpy as np
import torch

from . import _lib as L


def overlap_default(shape) -> bool:
    """Whether the aux loss and the router backward run on a second stream beside the
    expert calls. That pays while the expert GEMMs leave SMs idle between and at the end
    of their launches; once every launch fills the GPU for many rounds, the side-stream
    kernels only take SMs from the persistent GEMM grids. Decided by the expert GEMM
    work of one step."""
    return shape.gemm_flops() < OVERLAP_MAX_FLOPS


OVERLAP_MAX_FLOPS = float("inf")


class MoELayer:
    def __init__(self, shape, device: str = "cuda", owner_grouped=None, overlap=None):
        """owner_grouped: lay the permuted rows out by owner party (expert e hosted by
        party e mod P, moe_dispatch_owner) instead of by expert; default: when P > 1.
        overlap: run the aux loss and the router backward on a second stream beside the
        expert calls (True) or in order on the caller's stream (False); default: see
        ``overlap_default``."""
        self.shape = sh = shape
        self.owner_grouped = (sh.n_parties > 1) if owner_grouped is None else bool(owner_grouped)
        self.overlap = overlap_default(sh) if overlap is None else bool(overlap)
        self.device = device
        self.dt = torch.bfloat16 if sh.dtype == "bf16" else torch.float32
        self.cfg = L.make_config(sh.T, sh.d_model, sh.n_experts, sh.d_ff, sh.top_k, sh.n_parties,
                                 sh.n_shared, sh.d_ff_shared, sh.normalize_topk, sh.aux_alpha,
                                 L.MOE_BF16 if sh.dtype == "bf16" else L.MOE_F32)
        T, d, E, F, k, P = sh.T, sh.d_model, sh.n_experts, sh.d_ff, sh.top_k, sh.n_parties
        S, Fs, TK = sh.n_shared, sh.d_ff_shared, sh.T * sh.top_k
        dt, f32, i32 = self.dt, torch.float32, torch.int32

        def z(*s, dtype=dt):
            return torch.empty(*s, dtype=dtype, device=device)

        # parameters and inputs
        self.x, self.dout = z(T, d), z(T, d)
        self.w_router = z(P, E, d)
        self.router_bias = None
        self.party_offsets = z(P + 1, dtype=i32)
        self.w1, self.w2 = z(E, 2 * F, d), z(E, d, F)
        self.ws1 = z(S, 2 * Fs, d) if S else None
        self.ws2 = z(S, d, Fs) if S else None
        # forward
        self.logits, self.probs = z(T, E, dtype=f32), z(T, E, dtype=f32)
        self.topk_idx, self.topk_w = z(T, k, dtype=i32), z(T, k, dtype=f32)
        self.counts = z(P, E, dtype=i32)
        self.aux_loss, self.aux_coef = z(P, dtype=f32), z(P, E, dtype=f32)
        self.offsets = z(E + 1, dtype=i32)
        # owner-grouped layout: the expert of each segment, and the (source party ->
        # owner party) pair counts of the sends
        self.group_expert = z(E, dtype=i32) if self.owner_grouped else None
        self.send_counts = z(P, P, dtype=i32) if self.owner_grouped else None
        self.slot_of, self.token_of = z(TK, dtype=i32), z(TK, dtype=i32)
        self.x_perm = z(TK, d)
        self.h_gu, self.act, self.y_perm = z(TK, 2 * F), z(TK, F), z(TK, d)
        self.h_gu_sh = z(S, T, 2 * Fs) if S else None
        self.act_sh = z(S, T, Fs) if S else None
        self.y_sh = z(S, T, d) if S else None
        self.out = z(T, d)
        # backward
        self.dy_perm, self.dtopk_w = z(TK, d), z(T, k, dtype=f32)
        self.dh, self.dx_perm = z(TK, 2 * F), z(TK, d)
        self.dw1, self.dw2 = z(E, 2 * F, d), z(E, d, F)
        self.dh_sh = z(S, T, 2 * Fs) if S else None
        self.dx_sh = z(S, T, d) if S else None
        self.dws1 = z(S, 2 * Fs, d) if S else None
        self.dws2 = z(S, d, Fs) if S else None
        self.dlogits = z(T, E, dtype=f32)
        self.dw_router = z(P, E, d)
        self.dbias = z(P, E, dtype=f32)
        self.dx_router = z(T, d)
        self.dx = z(T, d)
        # the aux loss and the router backward run beside the expert GEMMs on this stream
        self.side = torch.cuda.Stream(device=device)
        # host<->device copies that overlap the passes (step_host)
        self.copy_stream = torch.cuda.Stream(device=device)
        # device->host copies of pipelined passes (run_host), and their second buffer set
        self.d2h_stream = torch.cuda.Stream(device=device)
        self._io_alt = None
        self.ws_bytes = L.moe_workspace_size(self.cfg)
        self.workspace = torch.empty(max(self.ws_bytes, 16), dtype=torch.uint8, device=device)

    # ------------------------------------------------------------------ inputs
    def load(self, inp: dict):
        """Copy seeded numpy inputs (synth.make_inputs) into the device buffers."""
        def put(dst, a):
            dst.copy_(torch.from_numpy(np.ascontiguousarray(a)).to(dst.dtype))

        put(self.x, inp["x"])
        put(self.dout, inp["dout"])
        put(self.w_router, inp["w_router"])
        put(self.party_offsets, inp["party_offsets"].astype(np.int32))
        if inp.get("router_bias") is not None:
            self.router_bias = torch.empty(self.shape.n_parties, self.shape.n_experts,
                                           dtype=torch.float32, device=self.device)
            put(self.router_bias, inp["router_bias"])
        if "w1" in inp:
            put(self.w1, inp["w1"])
            put(self.w2, inp["w2"])
            if self.shape.n_shared:
                put(self.ws1, inp["ws1"])
                put(self.ws2, inp["ws2"])

    def _po(self):
        return self.party_offsets if self.shape.n_parties > 1 else None

    # ------------------------------------------------------------------ stages
    # One method per C-ABI call of the layer, each on the stream it is given. forward()
    # and backward() chain them with the aux loss and the router backward on the side
    # stream; a caller may also run them one by one on one stream (bench.py times each
    # memory-bound stage that way).
    def route(self, s):
        L.moe_route(self.cfg, self.x, self.w_router, self.router_bias, self._po(), self.logits,
                    self.probs, self.topk_idx, self.topk_w, self.counts, stream=s)

    def aux(self, s):
        L.moe_aux_loss(self.cfg, self.probs, self.counts, self._po(), self.aux_loss,
                       self.aux_coef, stream=s)

    def dispatch(self, s):
        if self.owner_grouped:
            L.moe_dispatch_owner(self.cfg, self.topk_idx, self.x, self.party_offsets,
                                 self.group_expert, self.offsets, self.slot_of, self.token_of,
                                 self.x_perm, self.send_counts, self.workspace, self.ws_bytes,
                                 stream=s)
        else:
            L.moe_dispatch(self.cfg, self.topk_idx, self.x, self.offsets, self.slot_of,
                           self.token_of, self.x_perm, self.workspace, self.ws_bytes, stream=s)

    def ffn_fwd(self, s):
        L.moe_expert_ffn_fwd(self.cfg, self.x_perm, self.offsets, self.w1, self.w2, self.h_gu,
                             self.act, self.y_perm, self.x, self.ws1, self.ws2, self.h_gu_sh,
                             self.act_sh, self.y_sh, group_expert=self.group_expert, stream=s)

    def combine_fwd(self, s):
        L.moe_combine_fwd(self.cfg, self.y_perm, self.topk_w, self.slot_of, self.y_sh, self.out,
                          stream=s)

    def combine_bwd(self, s):
        L.moe_combine_bwd(self.cfg, self.dout, self.y_perm, self.topk_w, self.slot_of,
                          self.dy_perm, self.dtopk_w, stream=s)

    def route_bwd(self, s, with_aux: bool = True):
        L.moe_route_bwd(self.cfg, self.x, self.w_router, self.probs, self.topk_idx, self.topk_w,
                        self.dtopk_w, self.aux_coef if with_aux else None, self._po(),
                        self.dlogits, self.dw_router, self.dbias, self.dx_router, self.workspace,
                        self.ws_bytes, stream=s)

    def ffn_bwd(self, s):
        L.moe_expert_ffn_bwd(self.cfg, self.x_perm, self.offsets, self.w1, self.w2, self.h_gu,
                             self.act, self.dy_perm, self.dh, self.dx_perm, self.dw1, self.dw2,
                             self.x, self.dout, self.ws1, self.ws2, self.h_gu_sh, self.act_sh,
                             self.dh_sh, self.dx_sh, self.dws1, self.dws2,
                             group_expert=self.group_expert, stream=s)

    def dispatch_bwd(self, s):
        L.moe_dispatch_bwd(self.cfg, self.dx_perm, self.slot_of, self.dx_router, self.dx_sh,
                           self.dx, stream=s)

    # the calls of one step in order, with whether each is memory-bound (the expert FFN
    # calls are the tensor-core GEMMs)
    STAGES = (("route", True), ("aux", True), ("dispatch", True), ("ffn_fwd", False),
              ("combine_fwd", True), ("combine_bwd", True), ("route_bwd", True),
              ("ffn_bwd", False), ("dispatch_bwd", True))

    # ------------------------------------------------------------------ passes
    def forward(self, stream=None, mark=None):
        mark = mark or (lambda name: None)
        main = stream if stream is not None else torch.cuda.current_stream()
        self.route(main)
        if self.overlap:
            # the aux loss needs only probs and counts: compute it beside the experts
            fork = torch.cuda.Event()
            fork.record(main)
            self.side.wait_event(fork)
            self.aux(self.side)
            aux_done = torch.cuda.Event()
            aux_done.record(self.side)
        else:
            self.aux(main)
        self.dispatch(main)
        mark("ffn_fwd_begin")
        self.ffn_fwd(main)
        mark("ffn_fwd_end")
        self.combine_fwd(main)
        if self.overlap:
            main.wait_event(aux_done)

    def backward(self, stream=None, with_aux: bool = True, mark=None):
        mark = mark or (lambda name: None)
        main = stream if stream is not None else torch.cuda.current_stream()
        self.combine_bwd(main)
        if self.overlap:
            # the router backward needs only the gate gradients: run it beside the experts
            fork = torch.cuda.Event()
            fork.record(main)
            self.side.wait_event(fork)
            self.route_bwd(self.side, with_aux)
            join = torch.cuda.Event()
            join.record(self.side)
        else:
            self.route_bwd(main, with_aux)
        mark("ffn_bwd_begin")
        self.ffn_bwd(main)
        mark("ffn_bwd_end")
        if self.overlap:
            main.wait_event(join)
        self.dispatch_bwd(main)

    def step(self, stream=None, mark=None):
        """One fwd+bwd pass of the whole layer. ``mark(name)`` (optional) is called at
        the boundaries of the expert-GEMM calls: ffn_fwd_begin/end, ffn_bwd_begin/end."""
        self.forward(stream, mark=mark)
        self.backward(stream, mark=mark)

    def step_host(self, hx, hdout, hout, hdx, hloss, stream=None):
        """One fwd+bwd pass fed from host memory: x and dOut are copied in from the host
        tensors ``hx``, ``hdout`` (pinned for asynchronous copies), out, dx and the aux loss
        are copied back into ``hout``, ``hdx``, ``hloss``. Only x has to arrive before the
        forward and only dx leaves after the backward: dOut's upload runs beside the
        forward and out's download beside the backward, on a copy stream. All copies are
        ordered before the stream's later work, so the next call may reuse every buffer.
        """
        main = stream if stream is not None else torch.cuda.current_stream()
        start = torch.cuda.Event()
        start.record(main)  # the previous pass on this stream is done with dout and out
        with torch.cuda.stream(main):
            self.x.copy_(hx, non_blocking=True)
        self.copy_stream.wait_event(start)
        with torch.cuda.stream(self.copy_stream):
            self.dout.copy_(hdout, non_blocking=True)
        dout_in = torch.cuda.Event()
        dout_in.record(self.copy_stream)
        self.forward(main)
        fwd_done = torch.cuda.Event()
        fwd_done.record(main)
        self.copy_stream.wait_event(fwd_done)
        with torch.cuda.stream(self.copy_stream):
            hout.copy_(self.out, non_blocking=True)
        out_back = torch.cuda.Event()
        out_back.record(self.copy_stream)
        main.wait_event(dout_in)
        self.backward(main)
        with torch.cuda.stream(main):
            hdx.copy_(self.dx, non_blocking=True)
            hloss.copy_(self.aux_loss, non_blocking=True)
        main.wait_event(out_back)

    def run_host(self, batches, stream=None):
        """Several fwd+bwd passes fed from host memory, pipelined: the uploads of pass
        i+1 and the downloads of pass i-1 run on two copy streams beside the kernels of
        pass i. ``batches`` is a sequence of (hx, hdout, hout, hdx, hloss) host tensors as
        in ``step_host`` (pinned); pass i reads hx, hdout of its own tuple and writes its
        hout, hdx, hloss. x, dout, out, dx and the aux loss alternate between two device
        buffer sets; the weight gradients (dw1, dw2, dw_router, dbias) are those of the
        last pass. Returns once every pass is queued; synchronize before reading."""
        main = stream if stream is not None else torch.cuda.current_stream()
        if self._io_alt is None:
            self._io_alt = tuple(torch.empty_like(t) for t in self._io_tensors())
        sets = (self._io_tensors(), self._io_alt)
        h2d, d2h = self.copy_stream, self.d2h_stream
        n = len(batches)
        start = torch.cuda.Event()
        start.record(main)  # earlier work on this stream owns set 0 until here
        h2d.wait_event(start)
        d2h.wait_event(start)
        done = [None] * n      # pass i finished reading its inputs and writing its outputs
        arrived = [None] * n   # pass i's inputs are on the device
        fetched = [None] * n   # pass i's outputs are on the host

        def upload(i):
            hx, hdout = batches[i][0], batches[i][1]
            x, dout = sets[i % 2][0], sets[i % 2][1]
            if i >= 2:
                h2d.wait_event(done[i - 2])
            with torch.cuda.stream(h2d):
                x.copy_(hx, non_blocking=True)
                dout.copy_(hdout, non_blocking=True)
            arrived[i] = torch.cuda.Event()
            arrived[i].record(h2d)

        try:
            if n:
                upload(0)
            for i in range(n):
                if i + 1 < n:
                    upload(i + 1)
                self._set_io(sets[i % 2])
                main.wait_event(arrived[i])
                if i >= 2:
                    main.wait_event(fetched[i - 2])  # set i % 2's outputs are on the host
                self.forward(main)
                self.backward(main)
                done[i] = torch.cuda.Event()
                done[i].record(main)
                d2h.wait_event(done[i])
                hout, hdx, hloss = batches[i][2], batches[i][3], batches[i][4]
                with torch.cuda.stream(d2h):
                    hout.copy_(self.out, non_blocking=True)
                    hdx.copy_(self.dx, non_blocking=True)
                    hloss.copy_(self.aux_loss, non_blocking=True)
                fetched[i] = torch.cuda.Event()
                fetched[i].record(d2h)
        finally:
            self._set_io(sets[0])
        for ev in fetched[-2:]:
            main.wait_event(ev)  # later work on this stream may reuse both sets

    def _io_tensors(self):
        return (self.x, self.dout, self.out, self.dx, self.aux_loss)

    def _set_io(self, t):
        self.x, self.dout, self.out, self.dx, self.aux_loss = t

    def kernels_per_step(self) -> int:
        """CUDA kernels this library launches per step (memsets not counted):
        route 1, aux 1, dispatch 3, expert fwd 2, combine 1, combine bwd 1,
        unpermute-reduce 1; the expert backward as moe_expert_ffn_bwd_kernels reports it
        (its shared experts included); router backward: bf16 5 (dlogits, chunk dbias,
        dW_r partial GEMM, reduce, dx_router GEMM), fp32 4 (dlogits, partials, reduce,
        dx_router GEMM); shared experts add 2 to the forward."""
        bf16 = self.shape.dtype == "bf16"
        return (10 + L.moe_expert_ffn_bwd_kernels(self.cfg) + (5 if bf16 else 4)
                + (2 if self.shape.n_shared else 0))

    def check_status(self, stream=None):
        code = L.moe_device_status(stream)
        if code:
            raise L.MoEError(code, "device", L.moe_status_string(code))

    # ------------------------------------------------------------------ accounting
    def gemm_flops(self) -> float:
        return self.shape.gemm_flops()
