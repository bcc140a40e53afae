#!/usr/bin/env python
"""Benchmark of the Stream-Factorized Attention hot path on GB300.

One step = one pass of the hot path over one synthetic batch of the
Qwen3-8B-class layer (B=1, L=4096 tokens, n=4 -> 16384 positions, Hq=32, Hkv=8,
Dh=128, bf16, intra-stream / WITHIN mask):
  expansion gather (4 tables of 151936 x 4096)  -> sfa_fwd -> sfa_bwd_row_terms
  -> sfa_bwd_main -> sfa_bwd_finalize, with sfa_bwd_clear on a side stream beside
  the forward.
Metric: attention FLOPs over visible pairs only (forward 4*Dh, backward 10*Dh per
pair and query head) per second of the whole step, in TFLOP/s.

The same JSON line also carries: the dominant kernel's roofline, the end-to-end
number through the C ABI with host buffers, the CPU oracle baseline, and under
"extras" the CROSS (full cross-stream) layer of the same shape, the expansion-factor
sweep, the LOCAL (sliding-window) layer at windows of 1024 and 4096 positions, the
HBM bandwidth of the expansion backward and the final-stream selection and of the
decoding step over the expanded KV cache, the final-stream-only layer (the L
final-stream queries against all nL keys), and the large-MoE-class stack (L=8192,
n=4, Hq=64: 7 WITHIN + 1 CROSS layers, forward + backward).

--impl reference times the fp64 CPU oracle on a bounded sample of the same
workload (the paper publishes no implementation to run).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2607_08186_gb300.inputs import AttnShape, CROSS, LOCAL, SHAPES, WITHIN, WITHIN_NAIVE, attn_inputs  # noqa: E402

METRIC = "SFA fwd+bwd TFLOP/s (visible pairs) at n=4, % of bf16 peak; scaling vs n"
WORKLOAD = "qwen3_8b_n4"
GATHER_V, GATHER_D = 151936, 4096
FWD_FLOP, BWD_FLOP = 4, 10  # per visible pair, per query head, times Dh
MODE_NAME = {WITHIN: "WITHIN", CROSS: "CROSS", LOCAL: "LOCAL", WITHIN_NAIVE: "WITHIN_naive"}


# ---------------------------------------------------------------- FLOP model
def visible_pairs(s: AttnShape, mode: int, window: int = 0) -> int:
    """Visible (query, key) pairs per (batch, head): WITHIN n*L(L+1)/2 (Eq. 4),
    CROSS nL(nL+1)/2 (Fig. 2a), LOCAL sum_p min(p+1, w) (Fig. 2b).  The naive WITHIN
    schedule computes the WITHIN result: its pairs are WITHIN's."""
    if mode in (WITHIN, WITHIN_NAIVE):
        return s.n * s.L * (s.L + 1) // 2
    if mode == CROSS:
        return s.nL * (s.nL + 1) // 2
    w = min(window, s.nL)
    return w * (w + 1) // 2 + (s.nL - w) * w


def attn_flops(s: AttnShape, mode: int, per_pair: int, window: int = 0) -> float:
    return float(per_pair) * s.Dh * visible_pairs(s, mode, window) * s.Hq * s.B


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"bf16": p["bf16_tflops"], "bf16_sustained": p["bf16_tflops_sustained"],
                "hbm": p["hbm_gbs"], "src": "measured"}
    except Exception:
        return {"bf16": 1900.0, "bf16_sustained": 1700.0, "hbm": 6800.0, "src": "fallback"}


# ---------------------------------------------------------------- distributed
def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return ws, rank, local


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def reduce_max(x: float, ws: int) -> float:
    """Max of a per-rank number over all ranks (the job's time is its slowest rank)."""
    if ws <= 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, seconds_per_rank: float, ws: int) -> tuple[float, float]:
    """Weak scaling: every rank processes its own batch; value = all ranks' units / slowest time."""
    t = reduce_max(seconds_per_rank, ws)
    return units_per_rank * ws / t, t


# ---------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clock / throttle samples while the timed region runs."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None
        self.path = os.path.join("/tmp", f"hdsfa_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for ln in f:
                parts = [p.strip() for p in ln.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for nm, val in zip(names, parts[5:9]):
                    if val.lower() == "active":
                        reasons.add(nm)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ---------------------------------------------------------------- the step
class HotPath:
    """Device buffers and the five launches of one step."""

    def __init__(self, s: AttnShape, mode: int, dev, with_gather: bool = True, seed: int = 1, window: int = 0):
        from paper_2607_08186_gb300 import binding
        self.b = binding
        self.s, self.mode, self.dev, self.window = s, mode, dev, window
        q, k, v, do = attn_inputs(s, seed=seed)
        self.host_in = [t.pin_memory() for t in (q, k, v, do)]
        self.q, self.k, self.v, self.do = (t.to(dev, non_blocking=False) for t in self.host_in)
        self.o = torch.empty_like(self.q)
        self.lse = torch.empty(s.B, s.Hq, s.nL, dtype=torch.float32, device=dev)
        self.dq, self.dk, self.dv = torch.empty_like(self.q), torch.empty_like(self.k), torch.empty_like(self.v)
        self.ws = torch.empty(binding.sfa_bwd_workspace_bytes(s.B, s.L, s.n, s.Hq, s.Hkv, s.Dh, mode),
                              dtype=torch.uint8, device=dev)
        self.with_gather = with_gather
        if with_gather:
            g = torch.Generator(device=dev)
            g.manual_seed(seed + 100)
            # n embedding tables ~ N(0, 0.02), Qwen3-8B-sized (V x D = 0.62B per table)
            self.tables = (torch.randn(s.n, GATHER_V, GATHER_D, generator=g, device=dev,
                                       dtype=torch.float32) * 0.02).to(torch.bfloat16)
            gi = torch.Generator().manual_seed(seed + 200)
            self.host_ids = torch.randint(0, GATHER_V, (s.B, s.L), generator=gi,
                                          dtype=torch.int64).to(torch.int32).pin_memory()
            self.ids = self.host_ids.to(dev)
            self.x = torch.empty(s.B, s.nL, GATHER_D, dtype=torch.bfloat16, device=dev)
        self.host_out = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
                         for t in (self.o, self.lse, self.dq, self.dk, self.dv)]
        # the dQ accumulator is cleared on a side stream beside the forward (it needs
        # nothing from it), after the previous step's finalize has read it
        self.side = torch.cuda.Stream(device=dev)
        self.ev_start, self.ev_clear, self.ev_fin = torch.cuda.Event(), torch.cuda.Event(), torch.cuda.Event()
        self.launches_per_step = 5 + (1 if with_gather else 0)

    def _bufs(self):
        return {"q": self.q, "k": self.k, "v": self.v, "do": self.do, "ids": getattr(self, "ids", None),
                "o": self.o, "lse": self.lse, "dq": self.dq, "dk": self.dk, "dv": self.dv}

    def step(self, ev=None, bufs=None, stream=None):
        b, s = self.b, self.s
        t = bufs or self._bufs()
        main = stream if stream is not None else torch.cuda.current_stream()
        # the side stream's clear starts only once this step has started on the main
        # stream (so it is inside a timed step) and the previous step's dQ is out
        self.ev_start.record(main)
        self.side.wait_event(self.ev_start)
        self.side.wait_event(self.ev_fin)
        b.sfa_bwd_clear(s.B, s.L, s.n, s.Hq, s.Hkv, s.Dh, self.mode, self.ws, stream=self.side)
        self.ev_clear.record(self.side)
        if self.with_gather:
            b.hd_expand_embed(self.tables, t["ids"], self.x, stream=stream)
        if ev is not None:
            ev[0].record()
        b.sfa_fwd(t["q"], t["k"], t["v"], t["o"], t["lse"], s.n, self.mode, window=self.window, stream=stream)
        if ev is not None:
            ev[1].record()
        b.sfa_bwd_row_terms(t["o"], t["do"], t["lse"], s.n, self.mode, self.ws, s.Hkv, stream=stream)
        main.wait_event(self.ev_clear)
        if ev is not None:
            ev[2].record()
        b.sfa_bwd_main(t["q"], t["k"], t["v"], t["do"], t["dk"], t["dv"], s.n, self.mode, self.ws,
                       window=self.window, stream=stream)
        if ev is not None:
            ev[3].record()
        b.sfa_bwd_finalize(t["dq"], s.n, self.mode, self.ws, s.Hkv, stream=stream)
        self.ev_fin.record(main)

    def e2e(self, steps: int, warmup: int, ws: int) -> float:
        """Seconds per step end to end with host buffers: every step copies its inputs
        host -> device (pinned), runs the five launches and copies its results device ->
        host.  Three streams overlap step k+1's upload and step k-1's download with step
        k's compute; two device buffer sets, ordered by events, keep them apart."""
        sets = [self._bufs()]
        sets.append({name: (None if t is None else torch.empty_like(t)) for name, t in sets[0].items()})
        s_in, s_cmp, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
        n = warmup + steps
        ev = {key: [torch.cuda.Event() for _ in range(n)] for key in ("in", "cmp", "out")}
        ins = ("q", "k", "v", "do") + (("ids",) if self.with_gather else ())
        host_in = list(self.host_in) + ([self.host_ids] if self.with_gather else [])
        outs = ("o", "lse", "dq", "dk", "dv")
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        barrier(ws)
        torch.cuda.synchronize()
        for i in range(n):
            if i == warmup:
                s_in.wait_event(ev["out"][i - 1]) if i > 0 else None
                t0.record(s_in)
            d = sets[i & 1]
            with torch.cuda.stream(s_in):
                if i >= 2:
                    s_in.wait_event(ev["cmp"][i - 2])  # step i-2 has read this set's inputs
                for name, src in zip(ins, host_in):
                    d[name].copy_(src, non_blocking=True)
                ev["in"][i].record(s_in)
            s_cmp.wait_event(ev["in"][i])
            if i >= 2:
                s_cmp.wait_event(ev["out"][i - 2])  # this set's previous results are out
            self.step(bufs=d, stream=s_cmp)
            ev["cmp"][i].record(s_cmp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev["cmp"][i])
                for dst, name in zip(self.host_out, outs):
                    dst.copy_(d[name], non_blocking=True)
                ev["out"][i].record(s_out)
        t1.record(s_out)
        torch.cuda.synchronize()
        barrier(ws)
        return t0.elapsed_time(t1) / 1e3 / steps

    def io_bytes(self):
        h2d = sum(t.numel() * t.element_size() for t in self.host_in)
        if self.with_gather:
            h2d += self.host_ids.numel() * 4
        d2h = sum(t.numel() * t.element_size() for t in self.host_out)
        return h2d, d2h


class L2Flush:
    """Writes a buffer of twice the L2 size, so the next timed region starts with none of
    its inputs in L2."""

    def __init__(self, dev):
        self.nbytes = 2 * torch.cuda.get_device_properties(dev).L2_cache_size
        self.buf = torch.empty(self.nbytes, dtype=torch.uint8, device=dev)

    def __call__(self):
        self.buf.zero_()


def timed_steps(step, iters: int, warmup: int, flush: L2Flush, ws: int = 1, nev: int = 4):
    """Median device time (s) of `iters` calls of step(ev): each call bracketed by its own
    CUDA events on the launching stream, the L2 flushed between calls outside the events,
    `warmup` untimed calls first; ev holds `nev` events the step may record inside.
    Returns (median step s, the per-step inner events)."""
    for _ in range(warmup):
        step(None)
        flush()
    torch.cuda.synchronize()
    barrier(ws)
    torch.cuda.synchronize()
    se = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(iters)]
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(nev)] for _ in range(iters)]
    for i in range(iters):
        flush()
        se[i][0].record()
        step(evs[i])
        se[i][1].record()
    torch.cuda.synchronize()
    barrier(ws)
    return statistics.median(a.elapsed_time(b) for a, b in se) / 1e3, evs


def measure_layer(s: AttnShape, mode: int, dev, iters=10, warmup=3, window: int = 0, flush=None):
    """fwd, bwd-main and fwd+bwd times of one layer (no gather), seconds: medians over
    `iters` steps with the L2 flushed between them."""
    hp = HotPath(s, mode, dev, with_gather=False, seed=7, window=window)
    flush = flush or L2Flush(dev)
    total, evs = timed_steps(lambda ev: hp.step(ev), iters, warmup, flush)
    fwd = statistics.median(e[0].elapsed_time(e[1]) for e in evs) / 1e3
    bwd = statistics.median(e[2].elapsed_time(e[3]) for e in evs) / 1e3
    del hp
    torch.cuda.empty_cache()
    return {"fwd_s": fwd, "bwd_main_s": bwd, "step_s": total}


# ---------------------------------------------------------------- bandwidth ops
def time_op(fn, sets: int, iters=21, warmup=3):
    """Device time (s) per call of fn(k), k = call index: `iters` calls back to back
    between two events, the call k using buffer set k % sets (sets chosen so that
    consecutive calls touch more than the 129 MB L2 and read from HBM)."""
    for k in range(warmup):
        fn(k % sets)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for k in range(iters):
        fn(k % sets)
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / 1e3 / iters


def time_graph(fn, sets: int, reps: int = 7, warmup: int = 3):
    """Device time (s) per call of fn(k) when `reps` rounds over the `sets` buffer sets
    are captured once as a CUDA graph and replayed: what a serving loop that replays
    its step graph pays, without the host's launch cost per call."""
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        for k in range(warmup):
            fn(k % sets)
    torch.cuda.current_stream().wait_stream(stream)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for k in range(reps * sets):
            fn(k % sets)
    graph.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    graph.replay()
    b.record()
    torch.cuda.synchronize()
    del graph
    return a.elapsed_time(b) / 1e3 / (reps * sets)


def measure_expansion_backward(dev, hbm_peak: float, V: int = GATHER_V):
    """Expansion backward (adjoint of Eq. 1) and final-stream selection (Eq. 2) with
    its adjoint at the step's shapes: L=4096 tokens, n=4, D=4096, V=151936.
    Algorithmic bytes: expansion backward reads dX (n*L*D bf16) and the ids and
    reads + writes the fp32 rows of the distinct ids (U*n*D*8); its apply part (the
    row sums after the id-only plan) the same without the ids; selection reads and
    writes L*D bf16; its adjoint reads L*D and writes n*L*D bf16.  Three buffer sets
    rotate so that no call finds its inputs in L2."""
    from paper_2607_08186_gb300 import binding, inputs
    B, L, n, D = 1, 4096, 4, GATHER_D
    S = 3
    g = torch.Generator(device=dev)
    g.manual_seed(31)
    dX = [torch.randn(B, n * L, D, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
          for _ in range(S)]
    dE = torch.zeros(n, V, D, dtype=torch.float32, device=dev)
    ws = torch.empty(binding.hd_expand_embed_bwd_workspace_bytes(B, L), dtype=torch.uint8, device=dev)
    out = {}
    for name, zipf in (("uniform_ids", 0.0), ("zipf1_ids", 1.0)):
        ids = inputs.token_ids(B, L, V, seed=31, zipf=zipf).to(dev)
        U = int(torch.unique(ids).numel())
        t = time_op(lambda k: binding.hd_expand_embed_bwd(dX[k], ids, dE, ws), S)
        nbytes = B * n * L * D * 2 + B * L * 4 + U * n * D * 8
        binding.hd_expand_embed_bwd_plan(ids, V, ws)
        t_apply = time_op(lambda k: binding.hd_expand_embed_bwd_apply(dX[k], dE, ws, L), S)
        t_plan = time_op(lambda k: binding.hd_expand_embed_bwd_plan(ids, V, ws), S)
        ab = nbytes - B * L * 4
        out[f"expand_bwd_{name}"] = {"ms": t * 1e3, "distinct_ids": U, "bytes": nbytes,
                                     "gbs": nbytes / t / 1e9, "frac_hbm": nbytes / t / 1e9 / hbm_peak,
                                     "plan_ms": t_plan * 1e3, "apply_ms": t_apply * 1e3,
                                     "apply_gbs": ab / t_apply / 1e9,
                                     "apply_frac_hbm": ab / t_apply / 1e9 / hbm_peak}
    del dE
    y = [torch.empty(B, L, D, dtype=torch.bfloat16, device=dev) for _ in range(S)]
    t = time_op(lambda k: binding.hd_select_final_stream(dX[k], y[k], n), S)
    nbytes = 2 * B * L * D * 2
    out["select_final"] = {"ms": t * 1e3, "bytes": nbytes, "gbs": nbytes / t / 1e9,
                           "frac_hbm": nbytes / t / 1e9 / hbm_peak}
    t = time_op(lambda k: binding.hd_select_final_stream_bwd(y[k], dX[k], n), S)
    nbytes = B * L * D * 2 + B * n * L * D * 2
    out["select_final_bwd"] = {"ms": t * 1e3, "bytes": nbytes, "gbs": nbytes / t / 1e9,
                               "frac_hbm": nbytes / t / 1e9 / hbm_peak}
    out["workload"] = (f"B={B} L={L} n={n} V={V} D={D}; 21 calls back to back over {S} rotating "
                       "buffer sets (no call finds its inputs in L2)")
    del dX, y, ws
    torch.cuda.empty_cache()
    return out


def measure_moe_stack(dev, pk, steps: int = 3, warmup: int = 1):
    """Large-MoE-class attention stack: B=1, L=8192 tokens, n=4 (32768 positions), Hq=64,
    Hkv=8, Dh=128; 7 WITHIN layers then 1 CROSS layer, forward + backward of every layer
    with its own Q, K, V, dO (device-generated N(0,1)).  TMFLOP/s over visible pairs of the
    whole stack, per step; each layer's inputs and outputs are > 0.5 GB (beyond L2)."""
    from paper_2607_08186_gb300 import binding
    s = AttnShape(1, 8192, 4, 64, 8, 128)
    modes = [WITHIN] * 7 + [CROSS]
    g = torch.Generator(device=dev)
    g.manual_seed(61)

    def rnd(*shape):
        return torch.randn(*shape, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)

    layers = []
    for mode in modes:
        q, k, v, do = rnd(s.B, s.nL, s.Hq, s.Dh), rnd(s.B, s.nL, s.Hkv, s.Dh), rnd(s.B, s.nL, s.Hkv, s.Dh), \
            rnd(s.B, s.nL, s.Hq, s.Dh)
        t = {"mode": mode, "q": q, "k": k, "v": v, "do": do, "o": torch.empty_like(q),
             "lse": torch.empty(s.B, s.Hq, s.nL, dtype=torch.float32, device=dev),
             "dq": torch.empty_like(q), "dk": torch.empty_like(k), "dv": torch.empty_like(v),
             "ws": torch.empty(binding.sfa_bwd_workspace_bytes(s.B, s.L, s.n, s.Hq, s.Hkv, s.Dh, mode),
                               dtype=torch.uint8, device=dev)}
        layers.append(t)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(len(modes) + 1)] for _ in range(steps)]

    def run(ev=None):
        for i, t in enumerate(layers):
            if ev is not None:
                ev[i].record()
            binding.sfa_fwd(t["q"], t["k"], t["v"], t["o"], t["lse"], s.n, t["mode"])
            binding.sfa_bwd(t["q"], t["k"], t["v"], t["o"], t["lse"], t["do"], t["dq"], t["dk"], t["dv"], s.n,
                            t["mode"], t["ws"])
        if ev is not None:
            ev[-1].record()

    for _ in range(warmup):
        run()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for i in range(steps):
        run(evs[i])
    t1.record()
    torch.cuda.synchronize()
    sec = t0.elapsed_time(t1) / 1e3 / steps
    flops = sum(attn_flops(s, m, FWD_FLOP + BWD_FLOP) for m in modes)
    within_ms = statistics.mean(e[i].elapsed_time(e[i + 1]) for e in evs for i in range(7))
    cross_ms = statistics.mean(e[7].elapsed_time(e[8]) for e in evs)
    del layers
    torch.cuda.empty_cache()
    return {"workload": "moe_large_n4 stack: B=1 L=8192 n=4 (32768 positions) Hq=64 Hkv=8 Dh=128, "
                        "7 WITHIN + 1 CROSS layers, fwd+bwd (prep, main, finalize) per layer",
            "ms_per_stack": sec * 1e3, "flops_per_stack": flops, "tflops": flops / sec / 1e12,
            "frac": flops / sec / 1e12 / pk["bf16"], "frac_of_sustained": flops / sec / 1e12 / pk["bf16_sustained"],
            "within_layer_ms": within_ms, "within_layer_tflops": attn_flops(s, WITHIN, 14) / within_ms / 1e9,
            "cross_layer_ms": cross_ms, "cross_layer_tflops": attn_flops(s, CROSS, 14) / cross_ms / 1e9}


def final_pairs(L: int, n: int, mode: int, window: int = 0) -> int:
    """Visible pairs per (batch, head) of the final-stream problem: query t at position
    t*n + n-1 sees (t+1)*n keys (CROSS), t+1 (WITHIN: stream n-1 only), or
    min((t+1)*n, w) (LOCAL)."""
    if mode == WITHIN:
        return L * (L + 1) // 2
    if mode == CROSS:
        return n * L * (L + 1) // 2
    return sum(min((t + 1) * n, window) for t in range(L))


def measure_final_layer(dev, bf16_peak: float, iters: int = 10, flush=None):
    """Final-stream-only layer (Sec. 3.1 KV-mirror layers: the L final-stream queries against
    all nL keys), L=4096, n=4, with Qwen3-8B-class heads (Hq=32, Hkv=8, Dh=128) and the 80B
    configuration's heads (Hq=24, Hkv=2, Dh=256, Table 6): fwd and bwd TFLOP/s over
    visible pairs; medians over `iters` calls with the L2 flushed between them."""
    from paper_2607_08186_gb300 import binding
    B, L, n = 1, 4096, 4
    flush = flush or L2Flush(dev)
    g = torch.Generator(device=dev)
    g.manual_seed(51)

    def rnd(*shape):
        return torch.randn(*shape, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)

    out = {"workload": f"final-stream layer B={B} L={L} n={n} ({n * L} key positions)"}
    for name, Hq, Hkv, Dh in (("qwen3_8b", 32, 8, 128), ("80b", 24, 2, 256)):
        q, do = rnd(B, L, Hq, Dh), rnd(B, L, Hq, Dh)
        k, v = rnd(B, n * L, Hkv, Dh), rnd(B, n * L, Hkv, Dh)
        o, lse = torch.empty_like(q), torch.empty(B, Hq, L, dtype=torch.float32, device=dev)
        dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
        res = {"heads": f"Hq={Hq} Hkv={Hkv} Dh={Dh}"}
        for mode in (WITHIN, CROSS):
            ws = torch.empty(binding.sfa_bwd_final_workspace_bytes(B, L, n, Hq, Hkv, Dh, mode), dtype=torch.uint8,
                             device=dev)
            tf, _ = timed_steps(lambda ev: binding.sfa_fwd_final(q, k, v, o, lse, mode), iters, 3, flush)
            tb, _ = timed_steps(lambda ev: binding.sfa_bwd_final(q, k, v, o, lse, do, dq, dk, dv, mode, ws),
                                iters, 3, flush)
            pairs = final_pairs(L, n, mode) * Hq * B
            res[MODE_NAME[mode]] = {"fwd_ms": tf * 1e3, "bwd_ms": tb * 1e3,
                                    "fwd_tflops": FWD_FLOP * Dh * pairs / tf / 1e12,
                                    "bwd_tflops": BWD_FLOP * Dh * pairs / tb / 1e12,
                                    "fwd_frac": FWD_FLOP * Dh * pairs / tf / 1e12 / bf16_peak,
                                    "bwd_frac": BWD_FLOP * Dh * pairs / tb / 1e12 / bf16_peak}
        out[name] = res
        del q, do, k, v, o, lse, dq, dk, dv, ws
        torch.cuda.empty_cache()
    return out


def measure_decode(dev, hbm_peak: float, quick: bool = False):
    """Decoding step (Sec. 3.2), n=4: the new token's 4 positions against a context of T
    tokens (4T cached positions) for batch B, WITHIN and CROSS layers, with Qwen3-8B-class
    heads (Hq=32, Hkv=8, Dh=128) and, unless quick, the 80B configuration's heads (Hq=24,
    Hkv=2, Dh=256) and the 617B configuration's (Hq=96, Hkv=8, Dh=128) of Table 6.
    Algorithmic bytes: the visible cached K and V rows (B*T*n*Hkv*Dh*2 bytes each) plus
    q and o; rotating cache sets keep every call out of L2.  `us` is the device time per
    step of the calls replayed from a CUDA graph (how a serving loop runs the step);
    `us_eager` the same calls launched one by one from Python, where at batch 1 the
    host's launch cost per call is about the kernels' time."""
    from paper_2607_08186_gb300 import binding
    n = 4
    heads = {"qwen3_8b": (32, 8, 128, [(1, 8192), (4, 8192), (16, 8192), (1, 32768), (16, 32768)]),
             "80b": (24, 2, 256, [(1, 8192), (16, 8192), (1, 32768), (16, 32768)]),
             "617b": (96, 8, 128, [(1, 8192), (16, 8192)])}
    if quick:
        heads = {"qwen3_8b": (32, 8, 128, [(1, 8192), (16, 8192)])}
    res = {}
    g = torch.Generator(device=dev)
    g.manual_seed(41)
    for name, (Hq, Hkv, Dh, grid) in heads.items():
        out = []
        for B, T in grid:
            cache_bytes = 2 * B * T * n * Hkv * Dh * 2
            S = max(1, min(3, -(-400_000_000 // cache_bytes)))
            sets = []
            for _ in range(S):
                kc = torch.randn(B, T * n, Hkv, Dh, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
                vc = torch.randn(B, T * n, Hkv, Dh, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
                q = torch.randn(B, n, Hq, Dh, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)
                sets.append((q, kc, vc))
            lens = torch.full((B,), T, dtype=torch.int32, device=dev)
            o = torch.empty(B, n, Hq, Dh, dtype=torch.bfloat16, device=dev)
            lse = torch.empty(B, Hq, n, dtype=torch.float32, device=dev)
            row = {"B": B, "context_tokens": T, "cached_positions": T * n}
            for mode in (WITHIN, CROSS):
                ws = torch.empty(binding.sfa_decode_workspace_bytes(B, T, n, Hq, Hkv, Dh, mode), dtype=torch.uint8,
                                 device=dev)
                call = (lambda k: binding.sfa_decode(sets[k][0], sets[k][1], sets[k][2], lens, o, n, mode, ws,
                                                     max_tokens=T, lse=lse))
                t = time_graph(call, S)
                te = time_op(call, S)
                nbytes = cache_bytes + 2 * B * n * Hq * Dh * 2
                row[MODE_NAME[mode]] = {"us": t * 1e6, "gbs": nbytes / t / 1e9,
                                        "frac_hbm": nbytes / t / 1e9 / hbm_peak, "us_eager": te * 1e6}
            out.append(row)
            del sets, o, lse
            torch.cuda.empty_cache()
        res[name] = {"heads": f"Hq={Hq} Hkv={Hkv} Dh={Dh}", "rows": out}
    return {"workload": "decode step, n=4, all sequences at the context length; "
                        "bytes = cached K+V rows read + q + o", **res}


# ---------------------------------------------------------------- ncu traffic record
# ABI phase -> (kernel symbol, source file) of the implementation the library runs.
KERNEL_OF = {
    "sfa_fwd": ("hdsfa::tcfwd::fwd_kernel<128, false>", "sfa_fwd_tc.cu"),
    "sfa_bwd_main": ("hdsfa::tcbwd::bwd_kernel<128, false>", "sfa_bwd_tc.cu"),
}


def source_hash(fname: str) -> str:
    """sha256 prefix of a kernel's source file plus the device headers it includes."""
    h = hashlib.sha256()
    for part in (fname, "tc_common.cuh", "common.cuh"):
        with open(os.path.join(ROOT, "paper_2607_08186_gb300", "csrc", part), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def traffic_record(phase: str):
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) of the
    kernel behind `phase`, from the ncu record profiles/traffic.json, if it was
    captured on the current source of that kernel's file (else None)."""
    sym, fname = KERNEL_OF[phase]
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rows = json.load(f).get("rows", [])
    for r in rows:
        if r.get("kernel") == sym and r.get("source") == fname:
            return float(r["dram_bytes_per_launch"]) if r.get("sha16") == source_hash(fname) else None
    return None


# ---------------------------------------------------------------- CPU oracle baseline
def oracle_prefix_sample(L_prefix: int, mode: int):
    """fp64 oracle fwd + bwd of the benchmark layer restricted to its first
    L_prefix tokens (all heads).  Returns (seconds, visible-pair FLOPs)."""
    import oracle
    full = SHAPES[WORKLOAD]
    sp = AttnShape(full.B, L_prefix, full.n, full.Hq, full.Hkv, full.Dh)
    q, k, v, do = attn_inputs(sp, seed=1)
    t = time.perf_counter()
    oracle.sfa_fwd(q, k, v, sp.n, mode)
    oracle.sfa_bwd(q, k, v, do, sp.n, mode)
    dt = time.perf_counter() - t
    return dt, attn_flops(sp, mode, FWD_FLOP + BWD_FLOP), sp


def cpu_baseline(target_s: float = 12.0, mode: int = WITHIN):
    import oracle
    oracle.build()
    L0 = 64
    t0, _, _ = oracle_prefix_sample(L0, mode)
    Lp = int(L0 * math.sqrt(max(target_s, 0.5) / max(t0, 1e-3)))
    Lp = max(L0, min(SHAPES[WORKLOAD].L, (Lp // 16) * 16))
    dt, fl, sp = oracle_prefix_sample(Lp, mode)
    return {"value": fl / dt / 1e12, "unit": "TFLOP/s", "cores": oracle.num_threads(), "kind": "oracle",
            "sample": (f"fp64 oracle fwd+bwd of the {MODE_NAME[mode]} layer on its first {Lp} tokens "
                       f"({sp.nL} positions, Hq={sp.Hq}, Hkv={sp.Hkv}, Dh={sp.Dh}); "
                       f"{dt:.1f} s for {fl:.3e} visible-pair FLOPs")}


def run_reference(args, ws, rank):
    if rank != 0:
        return
    import oracle
    oracle.build()
    budget = 150.0 / max(1, args.steps + args.warmup)
    L0 = 64
    t0, _, _ = oracle_prefix_sample(L0, WITHIN)
    Lp = int(L0 * math.sqrt(max(budget, 0.3) / max(t0, 1e-3)))
    Lp = max(16, min(SHAPES[WORKLOAD].L, (Lp // 16) * 16))
    for _ in range(args.warmup):
        oracle_prefix_sample(Lp, WITHIN)
    times, fl, sp = [], 0.0, None
    for _ in range(args.steps):
        dt, fl, sp = oracle_prefix_sample(Lp, WITHIN)
        times.append(dt)
    mean = sum(times) / len(times)
    val = fl / mean / 1e12
    s = SHAPES[WORKLOAD]
    sample = (f"each step: fp64 oracle fwd+bwd of the WITHIN layer on its first {Lp} tokens "
              f"({sp.nL} positions, Hq={sp.Hq}, Hkv={sp.Hkv}, Dh={sp.Dh})")
    print(json.dumps({
        "metric": METRIC, "value": val, "unit": "TFLOP/s", "impl": "reference", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": mean * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{WORKLOAD}_within: B={s.B} L={s.L} n={s.n} ({s.nL} positions) "
                               f"Hq={s.Hq} Hkv={s.Hkv} Dh={s.Dh}, WITHIN mask", "sample": sample},
        "cpu_baseline": {"value": val, "unit": "TFLOP/s", "cores": oracle.num_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# ---------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-extras", action="store_true", help="skip the extras (CROSS / LOCAL layers, n sweep, expansion backward) and the CPU baseline")
    ap.add_argument("--expand-bwd-only", action="store_true",
                    help="time only the expansion backward and final-stream selection (JSON line)")
    ap.add_argument("--moe-only", action="store_true",
                    help="time only the large-MoE-class 8-layer stack (JSON line)")
    ap.add_argument("--final-only", action="store_true",
                    help="time only the final-stream-only layer (JSON line)")
    ap.add_argument("--decode-only", action="store_true",
                    help="time only the decoding step over the serving grid (JSON line)")
    ap.add_argument("--vocab", type=int, default=GATHER_V,
                    help="table rows V for --expand-bwd-only (smaller V for traffic captures)")
    ap.add_argument("--layer-only", choices=["within", "cross", "local"], default=None,
                    help="time only one attention layer (fwd + bwd, no gather / e2e / extras); "
                         "the small case used for kernel profiles")
    ap.add_argument("--head-dim", type=int, choices=[128, 256], default=128,
                    help="with --layer-only: 128 = the Qwen3-8B-class layer, 256 = the 80B-class "
                         "layer (B=1, L=4096, n=4, Hq=24, Hkv=2)")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    ws, rank, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, ws, rank)
        return
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_08186_gb300 import build
    if rank == 0 or ws == 1:
        build.build()
    barrier(ws)
    s = SHAPES[WORKLOAD]
    pk = peaks()
    if args.moe_only:
        r = measure_moe_stack(dev, pk, steps=args.steps if args.steps < 20 else 3)
        if rank == 0:
            print(json.dumps(r), flush=True)
        return
    if args.final_only:
        r = measure_final_layer(dev, pk["bf16"], iters=max(10, args.steps))
        if rank == 0:
            print(json.dumps(r), flush=True)
        return
    if args.decode_only:
        r = measure_decode(dev, pk["hbm"])
        if rank == 0:
            print(json.dumps(r), flush=True)
        return
    if args.expand_bwd_only:
        r = measure_expansion_backward(dev, pk["hbm"], V=args.vocab)
        if rank == 0:
            print(json.dumps(r), flush=True)
        return
    if args.layer_only:
        mode = {"within": WITHIN, "cross": CROSS, "local": LOCAL}[args.layer_only]
        w = 4096 if mode == LOCAL else 0
        ls, name = (s, WORKLOAD) if args.head_dim == 128 else (AttnShape(1, 4096, 4, 24, 2, 256), "80b_dh256_n4")
        r = measure_layer(ls, mode, dev, iters=args.steps, warmup=args.warmup, window=w)
        fl = attn_flops(ls, mode, FWD_FLOP + BWD_FLOP, w)
        if rank == 0:
            print(json.dumps({"layer": f"{name}_{args.layer_only}", "ms": r["step_s"] * 1e3,
                              "tflops": fl / r["step_s"] / 1e12, "fwd_ms": r["fwd_s"] * 1e3,
                              "fwd_tflops": attn_flops(ls, mode, FWD_FLOP, w) / r["fwd_s"] / 1e12,
                              "bwd_main_ms": r["bwd_main_s"] * 1e3}), flush=True)
        return
    hp = HotPath(s, WITHIN, dev, with_gather=True, seed=1)
    flops_step = attn_flops(s, WITHIN, FWD_FLOP + BWD_FLOP)

    # device-resident timed region: K steps, each bracketed by CUDA events on the
    # launching stream, the L2 flushed (2 x L2 written) between steps outside the events;
    # the step time is the median over the K steps
    flush = L2Flush(dev)
    clocks = ClockSampler(local)
    for _ in range(args.warmup):
        hp.step()
        flush()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    sec, evs = timed_steps(lambda ev: hp.step(ev), args.steps, 0, flush, ws)
    clk = clocks.stop()
    value, sec_max = job_throughput(flops_step, sec, ws)
    fwd_s = statistics.median(e[0].elapsed_time(e[1]) for e in evs) / 1e3
    bwd_s = statistics.median(e[2].elapsed_time(e[3]) for e in evs) / 1e3
    bwd_flops = attn_flops(s, WITHIN, BWD_FLOP)
    fwd_flops = attn_flops(s, WITHIN, FWD_FLOP)
    dom = "sfa_bwd_main" if bwd_s >= fwd_s else "sfa_fwd"
    dom_flops, dom_s = (bwd_flops, bwd_s) if dom == "sfa_bwd_main" else (fwd_flops, fwd_s)
    achieved = dom_flops / dom_s / 1e12
    tr = traffic_record(dom)

    # end to end through the C ABI with host buffers
    e2e_s = hp.e2e(max(5, args.steps // 2), 3, ws)
    e2e_val, _ = job_throughput(flops_step, e2e_s, ws)
    h2d, d2h = hp.io_bytes()
    launches = hp.launches_per_step * args.steps
    del hp
    torch.cuda.empty_cache()

    out = {
        "metric": METRIC, "value": value / 1e12, "unit": "TFLOP/s", "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": sec_max * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": (f"{WORKLOAD}_within: B={s.B} L={s.L} n={s.n} ({s.nL} positions) "
                                f"Hq={s.Hq} Hkv={s.Hkv} Dh={s.Dh}, WITHIN mask, fwd+bwd, plus the "
                                f"expansion gather of {s.n} tables {GATHER_V}x{GATHER_D}"),
                   "flops_per_step": flops_step, "flop_model": "fwd 4*Dh + bwd 10*Dh per visible pair per head",
                   "l2": (f"inputs larger than L2 (Q 134 MB, dO 134 MB, K+V 67 MB, gather tables 5 GB), and "
                          f"the L2 flushed between steps ({flush.nbytes / 1e6:.0f} MB written, outside the "
                          "steps' events)"),
                   "timing": (f"median of {args.steps} steps, each bracketed by CUDA events on the launching "
                              f"stream after {args.warmup} warm-up steps; max over ranks"),
                   "parallelism": f"replicas x{ws}"},
        "pct_of_peak": 100.0 * value / 1e12 / pk["bf16"],
        # the same step counted without the backward's QK^T recompute (bwd 8*Dh per pair)
        "strict_flop_model": {"per_pair": "fwd 4*Dh + bwd 8*Dh", "value": value / 1e12 * 12 / 14,
                              "unit": "TFLOP/s"},
        "roofline": {"kernel": f"{dom} ({KERNEL_OF[dom][0]})", "bound": "tensor", "achieved": achieved, "peak": pk["bf16"],
                     "unit": "TFLOP/s", "frac": achieved / pk["bf16"],
                     "frac_of_sustained": achieved / pk["bf16_sustained"],
                     "peak_source": f"{pk['src']} bf16 dense burst", "traffic": tr,
                     "algorithmic_flops_per_launch": dom_flops, "avg_launch_ms": dom_s * 1e3},
        "kernels_ms": {"sfa_fwd": fwd_s * 1e3, "sfa_bwd_main": bwd_s * 1e3},
        "e2e": {"value": e2e_val / 1e12, "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e_s * 1e3},
        "gpu_launches": launches,
        "clocks": clk,
    }
    if not args.no_extras and rank == 0 and ws == 1:
        extras = {}
        r = measure_layer(s, CROSS, dev, flush=flush)
        fl = attn_flops(s, CROSS, FWD_FLOP + BWD_FLOP)
        extras["cross_layer"] = {"workload": f"{WORKLOAD}_cross", "tflops": fl / r["step_s"] / 1e12,
                                 "fwd_tflops": attn_flops(s, CROSS, FWD_FLOP) / r["fwd_s"] / 1e12,
                                 "bwd_main_tflops": attn_flops(s, CROSS, BWD_FLOP) / r["bwd_main_s"] / 1e12,
                                 "ms": r["step_s"] * 1e3}
        sweep = []
        for n in (1, 2, 4, 8):
            sn = AttnShape(1, 4096, n, 32, 8, 128)
            row = {"n": n}
            # WITHIN_naive: WITHIN's mask per pair over the full causal tile schedule (no
            # stream-tile skipping), FLOPs counted over WITHIN's visible pairs
            for mode in (WITHIN, CROSS, WITHIN_NAIVE):
                r = measure_layer(sn, mode, dev, flush=flush)
                fl = attn_flops(sn, mode, FWD_FLOP + BWD_FLOP)
                row[MODE_NAME[mode]] = {"ms": r["step_s"] * 1e3, "tflops": fl / r["step_s"] / 1e12}
            row["skipping_speedup"] = row["WITHIN_naive"]["ms"] / row["WITHIN"]["ms"]
            sweep.append(row)
        base = sweep[0]["WITHIN"]["ms"]
        for row in sweep:
            row["WITHIN_cost_vs_n1"] = row["WITHIN"]["ms"] / base
        extras["n_sweep"] = sweep
        loc = []
        for w in (1024, 4096):
            r = measure_layer(s, LOCAL, dev, window=w, flush=flush)
            fl = attn_flops(s, LOCAL, FWD_FLOP + BWD_FLOP, w)
            loc.append({"window_positions": w, "ms": r["step_s"] * 1e3, "tflops": fl / r["step_s"] / 1e12,
                        "fwd_tflops": attn_flops(s, LOCAL, FWD_FLOP, w) / r["fwd_s"] / 1e12,
                        "bwd_main_tflops": attn_flops(s, LOCAL, BWD_FLOP, w) / r["bwd_main_s"] / 1e12})
        extras["local_layer"] = {"workload": f"{WORKLOAD}_local", "windows": loc}
        # head dim 256 (80B-class heads: 24 query over 2 K/V heads): the head-dim-256
        # tcgen05 forward and backward kernels
        s80 = AttnShape(1, 4096, 4, 24, 2, 256)
        r = measure_layer(s80, WITHIN, dev, flush=flush)
        fl = attn_flops(s80, WITHIN, FWD_FLOP + BWD_FLOP)
        extras["head_dim_256_layer"] = {
            "workload": "B=1 L=4096 n=4 Hq=24 Hkv=2 Dh=256, WITHIN, fwd+bwd (head-dim-256 tcgen05 kernels)",
            "ms": r["step_s"] * 1e3, "tflops": fl / r["step_s"] / 1e12,
            "fwd_tflops": attn_flops(s80, WITHIN, FWD_FLOP) / r["fwd_s"] / 1e12,
            "bwd_main_tflops": attn_flops(s80, WITHIN, BWD_FLOP) / r["bwd_main_s"] / 1e12}
        extras["expansion_backward"] = measure_expansion_backward(dev, pk["hbm"])
        extras["decode"] = measure_decode(dev, pk["hbm"], quick=True)
        extras["final_stream_layer"] = measure_final_layer(dev, pk["bf16"], flush=flush)
        extras["moe_stack"] = measure_moe_stack(dev, pk)
        out["extras"] = extras
        out["cpu_baseline"] = cpu_baseline()
    if rank == 0:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
