#!/usr/bin/env python
"""Throughput of the MoE expert layer, forward + backward, on GB300.

A step is one pass of the whole layer (gating, aux loss, dispatch, expert FFN
forward, combine, combine backward, expert FFN backward, gating backward,
unpermute-reduce) over one batch of seeded synthetic tokens. The default workload
is large_zipf_bf16, the largest layer that fits one GPU: T=16384 tokens, d=4096,
E=8 SwiGLU experts of F=14336, top-2, router bias giving Zipf(1.2) expert
popularity, bf16 storage with fp32 accumulation (34.6 TFLOP of expert GEMMs per
step).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the fp64 CPU oracle on the host cores

Timing: W untimed warm-up steps, then K steps timed one by one with CUDA events on
the launching stream; L2 is flushed (a 256 MiB write, then a 256 MiB read of another
buffer so that no dirty line is written back inside the step; both outside the events)
before every timed step. Under torchrun each rank runs its own replica (the layer does not
shard; no collective on the data path); the time is the max over ranks and the
value is the tokens of all ranks per second. Prints one JSON line on rank 0.

Rooflines: a second pass runs the layer's calls one after another on one stream,
each bracketed by its own events with L2 flushed before it, and reports every
memory-bound stage's algorithmic bytes / its time against the measured HBM copy
bandwidth, and the expert GEMM calls' algorithmic flops / their time against the
measured bf16 tensor peak.

e2e: the same layer fed from pinned host buffers through MoELayer.run_host, passes
whose host->device uploads (x, dOut) and device->host downloads (out, dx, aux loss)
are all inside one timed region, pipelined with the neighbouring passes' kernels.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from synth import moe_inputs as mi  # noqa: E402

METRIC = "MoE layer fwd+bwd tokens/s on 1 GB300"
FLUSH_BYTES = 256 << 20
# dense bf16 tensor-core rate of one GB300 as NVIDIA states it (without 2:4 sparsity)
NOMINAL_BF16_TFLOPS = 2250.0


def args_():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=60)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="large_zipf_bf16")
    ap.add_argument("--tokens", type=int, default=0,
                    help="override T (a reduced copy of the workload, for ncu captures)")
    ap.add_argument("--experts", type=int, default=0,
                    help="override E (a reduced copy of the workload, for ncu captures)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--train", action="store_true",
                    help="time Alg. 1 training steps (layer + MSE loss + SGD) instead")
    ap.add_argument("--parties", type=int, default=4, help="parties taking turns (--train)")
    ap.add_argument("--lr", type=float, default=0.05, help="SGD step (--train)")
    return ap.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"],
                "bf16_tflops_sustained": p.get("bf16_tflops_sustained"), "source": "measured",
                "sustained_sm_mhz": (p.get("clocks_under_load") or {}).get("sm_mhz_median")}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def reduced_shape(a):
    """The workload's shape, with T and E replaced when --tokens / --experts are given
    (then the name says so and the line is not the workload's)."""
    sh = mi.shape_by_name(a.workload)
    kw = {}
    if a.tokens:
        kw["T"] = a.tokens
    if a.experts:
        kw["n_experts"] = a.experts
    if kw:
        sh = sh.with_(name=sh.name + "_reduced", **kw)
    return sh


def workload_desc(sh):
    s = (f"{sh.name} (T={sh.T}, d={sh.d_model}, E={sh.n_experts}, F={sh.d_ff}, k={sh.top_k}"
         f"{', P=%d' % sh.n_parties if sh.n_parties > 1 else ''}"
         f"{', S=%d shared F=%d' % (sh.n_shared, sh.d_ff_shared) if sh.n_shared else ''})")
    return s


# --------------------------------------------------------------------------- memory bytes
def stage_bytes(sh) -> dict:
    """Algorithmic HBM bytes per step of each memory-bound call: what the layer must
    read and write, per token (b = bytes per activation element), times T:
      route (gating, a1-a3)      read x: d b;              write probs, picks: 4E + 8k
      aux (load-balancing loss)  read probs: 4E
      dispatch (a5-a8)           read x: d b;              write x_perm: k d b; tables: 12k
      combine_fwd (a11)          read y_perm, w: k d b + 4k (+ S d b shared outputs); write out: d b
      combine_bwd (a12)          read dout, y_perm: d b + k d b; write dy_perm, dw: k d b + 4k
      route_bwd (a17)            read probs, dprobs, x, dx-side: 8E + 2 d b; write dx_router: d b
      dispatch_bwd (a18)         read dx_perm: k d b (+ S d b shared dx); write dx: d b
    Re-reads, padding and the weights of the router (P E d b, not per token) do not
    count."""
    b = 2 if sh.dtype == "bf16" else 4
    T, d, E, k, S = sh.T, sh.d_model, sh.n_experts, sh.top_k, sh.n_shared
    per = {
        "route": d * b + 4 * E + 8 * k,
        "aux": 4 * E,
        "dispatch": d * b + k * d * b + 12 * k,
        "combine_fwd": k * d * b + 4 * k + S * d * b + d * b,
        "combine_bwd": d * b + k * d * b + k * d * b + 4 * k,
        "route_bwd": 8 * E + 2 * d * b + d * b,
        "dispatch_bwd": k * d * b + S * d * b + d * b,
    }
    return {n: v * T for n, v in per.items()}


def mem_bytes_per_step(sh) -> float:
    """Algorithmic HBM bytes of all memory-bound calls of one step (stage_bytes summed)."""
    return float(sum(stage_bytes(sh).values()))


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, enabled: bool = True):
        self.proc = None
        self.gpu = gpu_index
        if enabled:
            try:
                self.proc = subprocess.Popen(
                    ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.FIELDS}",
                     "--format=csv,noheader,nounits", "-lms", "50"],
                    stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            except Exception:
                self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = max(mx, float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "samples": len(sm),
                "reasons": sorted(reasons)}


# --------------------------------------------------------------------------- traffic
def gemm_traffic_record(sh):
    """DRAM bytes per grouped-GEMM launch from the committed ncu summary, if it was
    taken on the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", "gemm_traffic.json")
    src = os.path.join(ROOT, "paper_2506_02965_gb300", "csrc", "gemm_tc.cu")
    try:
        rec = json.load(open(path))
        h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        if rec.get("gemm_tc_sha") != h or rec.get("workload") != sh.name:
            return None
        return rec.get("dram_bytes_per_launch")
    except Exception:
        return None


# --------------------------------------------------------------------------- oracle legs
# Both CPU legs (cpu_baseline in our arm's line, and the whole --impl reference arm)
# time the fp64 oracle as it stands on the same sample and with the same policy: the
# first `sample_tokens` tokens of the workload (all experts, fp64 forward + backward),
# the mean over the timed repeats after untimed warm-up repeats. The sample size comes
# from one probe pass so that K + W repeats of it take about REF_BUDGET_S seconds; it
# depends only on the workload and K + W, so both legs of one driver round (the same
# --steps and --warmup) time the same tokens.
REF_BUDGET_S = 150.0
CPU_BASELINE_S = 15.0  # our arm's cpu_baseline: repeats of that sample for about this long


def _oracle_inputs(workload: str):
    import numpy as np
    sh = mi.shape_by_name(workload)
    inp = mi.make_inputs(sh)
    full = {k: (np.asarray(v, np.float64) if isinstance(v, np.ndarray) and v.dtype == np.float32
                else v) for k, v in inp.items()}
    return sh, full


def _oracle_step(sh, full, tokens: int) -> float:
    """One fwd+bwd of the oracle on the first `tokens` tokens; returns seconds."""
    import numpy as np
    from oracle import moe_oracle as mo
    P = sh.n_parties
    tokens = max(P, tokens - tokens % P)
    sub = dict(full)
    sub["x"] = full["x"][:tokens]
    sub["dout"] = full["dout"][:tokens]
    sub["party_offsets"] = (np.arange(P + 1) * (tokens // P)).astype(np.int32)
    s2 = sh.with_(T=tokens)
    t0 = time.perf_counter()
    f = mo.layer_forward(sub, s2)
    mo.layer_backward(sub, s2, f)
    return time.perf_counter() - t0


def oracle_timing(workload: str, steps: int, warmup: int, sample_steps: int,
                  sample_warmup: int, repeats: int | None = None,
                  budget_s: float | None = None) -> dict:
    """Time the oracle: size the sample from (sample_steps + sample_warmup) within
    REF_BUDGET_S, then run `warmup` untimed and `steps` timed repeats of it (or, with
    budget_s, as many timed repeats as fit about budget_s seconds, at least 2)."""
    sh, full = _oracle_inputs(workload)
    P = sh.n_parties
    probe_tok = max(P, 16 - 16 % P)
    _oracle_step(sh, full, probe_tok)             # first touch of the weights
    t_probe = _oracle_step(sh, full, probe_tok)
    t_fixed = _oracle_step(sh, full, P)           # per-step cost that does not scale with T
    per_tok = max(t_probe - t_fixed, 1e-9) / max(probe_tok - P, 1)
    per_step = REF_BUDGET_S / max(1, sample_steps + sample_warmup)
    tokens = int(min(sh.T, max(P, (per_step - t_fixed) / per_tok)))
    tokens = max(P, tokens - tokens % P)
    for _ in range(warmup):
        _oracle_step(sh, full, tokens)
    secs = []
    if budget_s is not None:
        t_end = time.perf_counter() + budget_s
        while len(secs) < 2 or time.perf_counter() < t_end:
            secs.append(_oracle_step(sh, full, tokens))
    else:
        for _ in range(steps):
            secs.append(_oracle_step(sh, full, tokens))
    return {"tokens": tokens, "seconds": secs, "warmup": warmup}


def run_oracle_subprocess(workload: str, steps: int, warmup: int, sample_steps: int,
                          sample_warmup: int, budget_s: float | None = None) -> dict:
    """oracle_timing in a fresh interpreter with every host core for BLAS (the GPU
    process may hold a CUDA context; the oracle needs none)."""
    cores = os.cpu_count() or 1
    env = dict(os.environ, OPENBLAS_NUM_THREADS=str(cores), OMP_NUM_THREADS=str(cores),
               MKL_NUM_THREADS=str(cores), CUDA_VISIBLE_DEVICES="")
    code = (f"import json,sys; sys.path.insert(0,{ROOT!r}); import bench; "
            f"print(json.dumps(bench.oracle_timing({workload!r}, {steps}, {warmup}, "
            f"{sample_steps}, {sample_warmup}, budget_s={budget_s!r})))")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=1800)
    if r.returncode:
        raise RuntimeError(r.stderr[-2000:])
    res = json.loads(r.stdout.strip().splitlines()[-1])
    res["cores"] = cores
    return res


def sample_desc(sh, res) -> str:
    return (f"first {res['tokens']} tokens of {sh.name} (all experts), fp64 fwd+bwd per repeat; "
            f"mean of {len(res['seconds'])} timed repeats after {res['warmup']} untimed; "
            f"sample sized so that --steps + --warmup repeats take ~{REF_BUDGET_S:.0f} s")


def run_reference(a):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    sh = mi.shape_by_name(a.workload)
    res = run_oracle_subprocess(a.workload, a.steps, a.warmup, a.steps, a.warmup)
    ms = 1e3 * statistics.mean(res["seconds"])
    value = res["tokens"] / (ms / 1e3)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": a.gpus, "steps": a.steps, "warmup": a.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded numpy PCG64)",
        "config": {"workload": workload_desc(sh), "sample_tokens": res["tokens"]},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": res["cores"],
                         "kind": "oracle", "sample": sample_desc(sh, res)},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


# --------------------------------------------------------------------------- ranks
def max_over_ranks(vals, world: int, device: str = "cuda"):
    """Element-wise maximum of `vals` over the ranks of the default process group (the
    slowest replica sets the step time). Identity for a single process."""
    if world <= 1:
        return list(vals)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in vals], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


# --------------------------------------------------------------------------- our arm
def train_bench(a):
    """Alg. 1 on one GPU: the parties take turns (a seeded permutation per epoch), one
    batch of the workload's T tokens per turn; a step is the layer's forward and
    backward, the MSE loss and the SGD updates of the active party's gating and of the
    experts its batch called. Inputs resident in HBM; no L2 flush (each step streams
    the expert weights, their gradients and the updated weights, several times L2)."""
    import torch
    from paper_2506_02965_gb300 import _lib as L
    from paper_2506_02965_gb300.train import RoundRobinTrainer

    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    base = mi.shape_by_name(a.workload)
    sh = base.with_(n_parties=1, n_shared=0, d_ff_shared=0)
    n = max(1, a.parties)
    tr = RoundRobinTrainer(sh, n, lr=a.lr)
    tr.load(mi.train_init(sh, n, seed=sh.seed))
    tdt = tr.layer.dt
    batches = [[(torch.from_numpy(x).to("cuda", tdt), torch.from_numpy(y).to("cuda", tdt))
                for x, y in mine] for mine in mi.train_batches(sh, n, 1, seed=sh.seed + 1)]
    w_epochs = max(1, -(-max(3, a.warmup) // n))
    t_epochs = max(1, -(-a.steps // n))
    sched = mi.party_schedule(n, w_epochs + t_epochs, seed=sh.seed + 2)
    tr.run(batches, sched[:w_epochs], 1)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    _, log = tr.run(batches, sched[w_epochs:], 1)
    e1.record()
    torch.cuda.synchronize()
    tr.layer.check_status()
    steps = t_epochs * n
    ms = e0.elapsed_time(e1) / steps
    # the SGD updates alone (counts of the last batch), for their HBM fraction
    lay, E, d, F = tr.layer, sh.n_experts, sh.d_model, sh.d_ff
    called = int((lay.counts > 0).sum().item())
    nb = 2 if sh.dtype == "bf16" else 4
    # per element: read w (or the fp32 master) and dw, write w (and the master)
    per_elem = (4 + nb + 4 + nb) if tr.master else 3 * nb
    sgd_bytes = per_elem * (called * 3 * F * d + E * d)
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 20
    g0.record()
    for _ in range(reps):  # lr = 0: the same traffic, parameters unchanged
        L.moe_sgd_update(tr.w_router[0], lay.dw_router, 1, E * d, None, 0.0, tr.dtype,
                         w_master=tr.m_router[0] if tr.master else None)
        L.moe_sgd_update(lay.w1, lay.dw1, E, 2 * F * d, lay.counts, 0.0, tr.dtype, w_master=tr.m1)
        L.moe_sgd_update(lay.w2, lay.dw2, E, d * F, lay.counts, 0.0, tr.dtype, w_master=tr.m2)
    g1.record()
    torch.cuda.synchronize()
    sgd_ms = g0.elapsed_time(g1) / reps
    pk = peaks()
    losses = log.cpu().numpy()
    line = {"metric": "Alg. 1 training step (MoE layer fwd+bwd + MSE + SGD) tokens/s on 1 GB300",
            "value": sh.T / (ms / 1e3), "unit": "tokens/s", "n_gpus": 1, "steps": steps,
            "warmup": w_epochs * n, "ms_per_step": ms, "higher_is_better": True,
            "dtype": sh.dtype, "data": "synthetic (seeded numpy PCG64, regression on a fixed random teacher)",
            "config": {"workload": f"{workload_desc(sh)}, {n} parties taking turns, B=1, SGD lr={a.lr}"
                                    + (", fp32 master weights" if tr.master else ""),
                       "l2": "not flushed: every step streams the weights and their gradients (> L2)"},
            "sgd": {"ms_per_step": sgd_ms, "bytes": sgd_bytes, "achieved_gbs": sgd_bytes / sgd_ms / 1e6,
                    "peak_gbs": pk["hbm_gbs"], "frac": sgd_bytes / sgd_ms / 1e6 / pk["hbm_gbs"]},
            "loss_first_last": [float(losses[0].sum()), float(losses[-1].sum())],
            "gpu_launches": steps * tr.kernels_per_step()}
    print(json.dumps(line), flush=True)


def main():
    a = args_()
    if a.impl == "reference":
        run_reference(a)
        return
    if a.train:
        train_bench(a)
        return
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if world > 1:
            dist.barrier()

    from paper_2506_02965_gb300.layer import MoELayer
    sh = reduced_shape(a)
    inp = mi.make_inputs(sh)
    lay = MoELayer(sh)
    lay.load(inp)
    for name in ("w1", "w2", "ws1", "ws2"):  # on the device now; x and dOut stay for e2e
        inp.pop(name, None)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    # after the flush write, a read of another buffer larger than L2 leaves it holding
    # clean lines: the timed call then starts cold without paying for the write-back of
    # the flush's dirty lines
    clean = torch.ones(FLUSH_BYTES // 4, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()

    for i in range(max(3, a.warmup)):
        flush.fill_(i & 0xFF)
        clean.sum()
        lay.step()
    torch.cuda.synchronize()
    lay.check_status()

    K = a.steps
    # headline: K steps exactly as a user runs them, each bracketed by two events
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    clocks = ClockSampler(local, enabled=not a.no_clocks)
    time.sleep(0.3 if clocks.proc else 0)
    barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    for i in range(K):
        flush.fill_(i & 0xFF)
        clean.sum()
        ev[i][0].record(stream)
        lay.step()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    barrier()
    wall = time.perf_counter() - t_wall
    clk = clocks.stop()
    lay.check_status()
    ms = statistics.mean([e0.elapsed_time(e1) for e0, e1 in ev])

    # rooflines: the layer's calls one after another on one stream, each bracketed by
    # its own events with L2 flushed before it (not the headline: the step overlaps the
    # aux loss and the router backward with the expert calls on a side stream)
    Ks = max(3, min(K, 20))
    names = [n for n, _ in lay.STAGES]
    evs = [{n: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for n in names} for _ in range(Ks)]
    barrier()
    torch.cuda.synchronize()
    for i in range(Ks):
        for j, n in enumerate(names):
            flush.fill_((i + j) & 0xFF)
            clean.sum()
            evs[i][n][0].record(stream)
            getattr(lay, n)(stream)
            evs[i][n][1].record(stream)
    torch.cuda.synchronize()
    lay.check_status()
    stage_ms = {n: statistics.mean([e[n][0].elapsed_time(e[n][1]) for e in evs]) for n in names}
    red = max_over_ranks([ms] + [stage_ms[n] for n in names], world)
    ms, stage_ms = red[0], dict(zip(names, red[1:]))
    gms = stage_ms["ffn_fwd"] + stage_ms["ffn_bwd"]
    value = world * sh.T / (ms / 1e3)

    # e2e: host buffers in, host results out, through the same public calls. The passes
    # are pipelined (MoELayer.run_host): pass i+1's uploads and pass i-1's downloads run
    # on copy streams beside pass i's kernels; every pass's copies are in the timed
    # region. No L2 flush between these passes: each one streams the expert weights and
    # writes their gradients (several times L2) through the cache.
    e2e = None
    if not a.no_e2e:
        hx = torch.from_numpy(inp["x"]).to(lay.dt).pin_memory()
        hd = torch.from_numpy(inp["dout"]).to(lay.dt).pin_memory()
        outs = [(torch.empty_like(hx).pin_memory(), torch.empty_like(hx).pin_memory(),
                 torch.empty(sh.n_parties, dtype=torch.float32).pin_memory()) for _ in range(2)]
        Ke = max(3, min(K, 40))
        batches = [(hx, hd) + outs[i % 2] for i in range(Ke)]
        lay.run_host(batches[:max(3, a.warmup)], stream=stream)  # warm-up of the pipelined path
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier()
        torch.cuda.synchronize()
        e0.record(stream)
        lay.run_host(batches, stream=stream)
        e1.record(stream)
        torch.cuda.synchronize()
        ems = e0.elapsed_time(e1) / Ke
        ems = max_over_ranks([ems], world)[0]
        nb = 2 if sh.dtype == "bf16" else 4
        e2e = {"value": world * sh.T / (ems / 1e3), "unit": "tokens/s",
               "h2d_bytes_per_step": 2 * sh.T * sh.d_model * nb,
               "d2h_bytes_per_step": 2 * sh.T * sh.d_model * nb + 4 * sh.n_parties,
               "ms_per_step": ems, "passes": "pipelined: copies on two streams beside the kernels",
               "l2": "not flushed: every pass streams the expert weights and writes their gradients (> L2)"}
        lay.check_status()

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    pk = peaks()
    gemm_flops = sh.gemm_flops()
    achieved = gemm_flops / (gms / 1e3) / 1e12
    # expert-GEMM launches: GEMM1, GEMM2 (+2 for shared experts), then the backward's as
    # the library reports them (dA with dW2 in one launch, dX as CTA pairs beside dW1 on
    # the tensor cores by default; four on the CUDA cores; shared experts' four)
    from paper_2506_02965_gb300 import _lib as L
    n_gemm = 2 + L.moe_expert_ffn_bwd_kernels(lay.cfg) + (2 if sh.n_shared else 0)
    traffic = gemm_traffic_record(sh)
    fwd_flops, bwd_flops = gemm_flops / 3.0, 2.0 * gemm_flops / 3.0
    roofline = {"bound": "tensor", "kernel": "grouped_gemm_kernel (tcgen05, all expert GEMM launches)",
                "achieved": achieved, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                "frac": achieved / pk["bf16_tflops"], "traffic": traffic,
                "peak_source": f"{pk['source']} bf16 burst (torch.matmul 8192^3, best of 10)",
                "peak_sustained": pk["bf16_tflops_sustained"],
                "peak_sustained_sm_mhz": pk.get("sustained_sm_mhz"),
                "frac_sustained": (achieved / pk["bf16_tflops_sustained"]
                                   if pk["bf16_tflops_sustained"] else None),
                "peak_nominal": NOMINAL_BF16_TFLOPS,
                "frac_nominal": achieved / NOMINAL_BF16_TFLOPS,
                "flops_per_step": gemm_flops, "ms_per_step": gms,
                "launches_per_step": n_gemm,
                "calls": {"ffn_fwd": {"ms": stage_ms["ffn_fwd"],
                                      "tflops": fwd_flops / stage_ms["ffn_fwd"] / 1e9},
                          "ffn_bwd": {"ms": stage_ms["ffn_bwd"],
                                      "tflops": bwd_flops / stage_ms["ffn_bwd"] / 1e9}},
                "timing": "CUDA events around moe_expert_ffn_fwd and moe_expert_ffn_bwd, "
                          f"mean of {Ks} serial passes"}
    sb = stage_bytes(sh)
    mem_stages = {n: {"bytes": sb[n], "ms": stage_ms[n],
                      "gbs": sb[n] / (stage_ms[n] / 1e3) / 1e9,
                      "frac": sb[n] / (stage_ms[n] / 1e3) / 1e9 / pk["hbm_gbs"]} for n in sb}
    mem_bytes = sum(sb.values())
    mem_ms = sum(stage_ms[n] for n in sb)
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": a.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": sh.dtype,
        "data": "synthetic (seeded numpy PCG64, workload shapes, random-init weights)",
        "config": {"workload": workload_desc(sh), "global_batch": world * sh.T,
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                   "l2": "flushed before every timed step (256 MiB write, then a 256 MiB read so "
                         "that no dirty line is left)"},
        "roofline": roofline,
        "roofline_mem": {"bound": "hbm", "achieved": mem_bytes / (mem_ms / 1e3) / 1e9,
                         "peak": pk["hbm_gbs"], "unit": "GB/s",
                         "frac": mem_bytes / (mem_ms / 1e3) / 1e9 / pk["hbm_gbs"],
                         "peak_source": f"{pk['source']} HBM copy bandwidth",
                         "bytes_per_step": mem_bytes, "ms_per_step": mem_ms,
                         "stages": mem_stages,
                         "timing": "CUDA events around each memory-bound call, L2 flushed "
                                   "(256 MiB write, then a 256 MiB read so that no dirty line "
                                   f"is left) before each, mean of {Ks} serial passes"},
        "serial_ms_per_step": sum(stage_ms.values()),
        "gpu_launches": K * lay.kernels_per_step(),
        "wall_s_timed": wall,
    }
    if e2e:
        line["e2e"] = e2e
    if clk:
        line["clocks"] = clk
    if world == 1 and not a.no_cpu_baseline:
        try:
            cb = run_oracle_subprocess(a.workload, 0, 1, a.steps, a.warmup, budget_s=CPU_BASELINE_S)
            v = cb["tokens"] / statistics.mean(cb["seconds"])
            line["cpu_baseline"] = {"value": v, "unit": "tokens/s", "cores": cb["cores"],
                                    "kind": "oracle", "sample": sample_desc(sh, cb)}
        except Exception as ex:  # reported, not fatal
            line["cpu_baseline"] = {"error": str(ex)[-300:]}
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
