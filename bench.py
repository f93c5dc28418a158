#!/usr/bin/env python3
"""Benchmark of the DART hot path on GB300.

One step = one pass of the whole prefill hot path of a DART block over one
batch of seeded synthetic input: dart_chunk_scan (chunked SSD scan with chunk
state memories) followed by dart_sma_forward (state-memory attention and the
gated merge), on the long-context workload B1 H32 L16384 P64 N128 S256
(64 chunk memories per head). The JSON line also carries the decode step
(B64 H32, 64 cached memories = 2 GiB) measured against HBM bandwidth.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl dart|reference]

Under torchrun (N > 1) every rank runs its own replica of the workload
(the path shards over independent (batch, head) units and has no exchange
step), so scaling is weak and value = all ranks' tokens / max rank time.
``--impl reference`` times the CPU oracle (fp64, OpenMP) on a bounded sample
of the same workload; it is the only other place this file runs the oracle.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import re
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "DART layer prefill tokens/s at L=16K and % bf16 TC peak; decode % HBM BW"
PREFILL = "prefill_l16k"
DECODE = "decode_b64"
L2_FLUSH_BYTES = 256 << 20  # > 129 MB L2
NOMINAL_HBM_GBS = 7900.0


def _peaks() -> dict:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=float(p["hbm_gbs"]), bf16=float(p["bf16_tflops"]),
                    bf16_sus=float(p["bf16_tflops_sustained"]), source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


def sma_pairs(w) -> int:
    """(token, memory) pairs summed over batch and heads: token t sees t // S memories."""
    S, M = w.chunk, w.nchunks
    return w.batch * w.heads * S * (M * (M - 1) // 2)


def sma_flops(w) -> float:
    """Algorithmic SMA flops: per pair the key read (N x P) and value read (N x P)."""
    return sma_pairs(w) * 4.0 * w.dstate * w.headdim


def scan_flops(w) -> float:
    """Algorithmic scan flops per (b, chunk, h): chunk state 2 S N P, inter-chunk
    output 2 S N P, causal-half intra-chunk scores S(S+1)/2 x 2N (shared by the
    heads of a group) and their application S(S+1)/2 x 2P."""
    S, N, P = w.chunk, w.dstate, w.headdim
    per_ch = 4.0 * S * N * P + S * (S + 1) * P
    per_grp = S * (S + 1) * N
    return w.batch * w.nchunks * (w.heads * per_ch + w.groups * per_grp)


def scan_bytes(w) -> float:
    """Algorithmic HBM bytes of the forward scan with bf16 token inputs and fp32
    outputs: X, B, C (bf16) and dt read once; Y_ssd, the chunk memories and their
    inverse RMS (fp32) written once."""
    T = w.batch * w.seqlen
    reads = T * (w.heads * w.headdim * 2 + 2 * w.groups * w.dstate * 2 + w.heads * 4)
    writes = T * w.heads * w.headdim * 4 + w.batch * w.nchunks * w.heads * w.dstate * (w.headdim + 1) * 4
    return float(reads + writes)


def decode_bytes(w, m_cap) -> int:
    """HBM bytes one decode step must move: the whole cache of completed memories,
    the running state (read + write), the partial memory (write; read unless the
    token starts a chunk) and the per-token vectors."""
    B, H, N, P = w.batch, w.heads, w.dstate, w.headdim
    es = 2 if w.dtype == "bf16" else 4
    nh = min(w.pos // w.chunk, m_cap)
    cache = B * nh * H * N * P * es
    state = 2 * B * H * N * P * 4
    part = (1 if w.pos % w.chunk == 0 else 2) * B * H * N * P * 4
    app = B * H * N * P * es if (w.pos + 1) % w.chunk == 0 else 0
    tok = B * H * (P * es + P * 4 + 3 * 4) + B * w.groups * (3 * w.dstate + P) * es
    return cache + state + part + app + tok


class Clocks:
    """nvidia-smi sampler for the timed region (start before, stop after)."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (FileNotFoundError, OSError):
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self) -> dict:
        rows = []
        if self.path and os.path.exists(self.path):
            for ln in open(self.path):
                parts = [p.strip() for p in ln.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "samples": len(rows), "reasons": reasons}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(value: float, world: int, device) -> float:
    """Largest value over all ranks (the slowest rank sets whole-job time)."""
    if world == 1:
        return value
    import torch
    import torch.distributed as dist

    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


# ----------------------------------------------------------------- oracle legs

def oracle_sample(w, inp: dict, heads: int):
    """Run the oracle's whole prefill path on the first ``heads`` heads of the
    workload (every token); returns (seconds, threads)."""
    import oracle

    sl = {k: inp[k][:, :, :heads] for k in ("X", "dt", "z")}
    A = inp["A"][:heads]
    t0 = time.perf_counter()
    Yssd, _ = oracle.ssd_recurrence(sl["X"], sl["dt"], A, inp["Bm"], inp["Cm"])
    dH = oracle.chunk_memories(sl["X"], sl["dt"], A, inp["Bm"], w.chunk)
    R, lse = oracle.sma(dH, inp["Q"], inp["Cm"], inp["E"], w.chunk, w.eps)
    oracle.merge(Yssd, sl["z"], R)
    return time.perf_counter() - t0, oracle.num_threads()


def run_reference(args) -> None:
    world, rank, _ = _dist()
    if rank != 0:
        return
    import oracle
    from paper_2608_02032_gb300.workloads import WORKLOADS, prefill_inputs

    w = WORKLOADS[PREFILL]
    inp = prefill_inputs(w)
    # one head per oracle thread: its recurrence and memories run over independent
    # (batch, head) units, so fewer heads than threads would leave cores idle
    heads = args.ref_heads or max(1, min(w.heads, oracle.num_threads()))
    for _ in range(args.warmup):
        oracle_sample(w, inp, heads)
    times = []
    threads = 1
    for _ in range(args.steps):
        t, threads = oracle_sample(w, inp, heads)
        times.append(t)
    per_step = sum(times) / len(times)
    # tokens/s of the full workload: the sample covers heads / H of its (token, head) work
    value = w.tokens / (per_step * w.heads / heads)
    sample = (f"{heads} of {w.heads} heads, all {w.seqlen} tokens, full prefill path "
              f"(recurrence, memories, SMA, merge) per step")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": per_step * 1e3, "higher_is_better": True,
        "ms_per_full_workload_extrapolated": per_step * w.heads / heads * 1e3,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": _config(w),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def _config(w) -> dict:
    return {"workload": f"{w.name}: {w.notes}", "batch": w.batch, "seqlen": w.seqlen,
            "heads": w.heads, "groups": w.groups, "headdim": w.headdim, "dstate": w.dstate,
            "chunk": w.chunk, "memories": w.nchunks, "inputs": "bf16", "accumulate": "f32",
            "memories_and_outputs": "f32",
            "l2": "flushed (256 MiB write) between timed steps", "parallelism": "replicas",
            "clocks": "sampled every 200 ms over ~1 s of untimed steps and the timed steps after them"}


# ------------------------------------------------------------------- GPU leg

def run_dart(args) -> None:
    import torch

    from paper_2608_02032_gb300 import binding as Bd
    from paper_2608_02032_gb300.workloads import (WORKLOADS, decode_cache_slab, decode_state_slab,
                                                  decode_token_inputs, prefill_inputs)

    world, rank, local = _dist()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (the DART library has no CPU path)")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=dev)
    Bd.lib()
    peaks = _peaks()
    w = WORKLOADS[args.workload]
    inp = prefill_inputs(w)
    tdt = torch.bfloat16
    Bsz, L, H, G, P, N, S = w.batch, w.seqlen, w.heads, w.groups, w.headdim, w.dstate, w.chunk
    M = w.nchunks
    names_in = ("X", "Bm", "Cm", "Q", "E", "z")
    d_in = {k: inp[k].to(dev, tdt).contiguous() for k in names_in}
    d_in["dt"] = inp["dt"].to(dev).contiguous()
    d_in["A"] = inp["A"].to(dev).contiguous()
    dims = Bd.make_dims(Bsz, L, H, G, P, N, S, Bd.DART_BF16, eps=w.eps)
    # bf16 token inputs; memories and outputs fp32 (fp32 accumulation throughout)
    Yssd = torch.empty(Bsz, L, H, P, dtype=torch.float32, device=dev)
    Mem = torch.empty(Bsz, M, H, N, P, dtype=torch.float32, device=dev)
    rM = torch.empty(Bsz, M, H, N, dtype=torch.float32, device=dev)
    Y = torch.empty_like(Yssd)
    lse = torch.empty(Bsz, L, H, dtype=torch.float32, device=dev)
    ws = torch.empty(Bd.dart_workspace_size(dims, Bd.DART_OP_CHUNK_SCAN), dtype=torch.uint8, device=dev)
    ws_sma = torch.empty(max(Bd.dart_workspace_size(dims, Bd.DART_OP_SMA_FORWARD), 256),
                         dtype=torch.uint8, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    # the scan writes the SMA's operand tiles (dart_chunk_scan_with_tiles) where both
    # calls run on the tensor cores; the SMA call is then the SMA kernel alone
    n_tiles = Bd.dart_sma_tiles_size(dims)
    tiles = torch.empty(max(n_tiles, 256), dtype=torch.uint8, device=dev)

    # the SMA kernel may start under the scan's last kernel (programmatic dependent
    # launch); the split timing puts a one-element kernel of torch's between the two
    # calls, which that kernel cannot overlap, so each call is timed on its own
    sep = torch.zeros(1, dtype=torch.float32, device=dev)

    def step(split=False):
        if n_tiles > 0:
            Bd.dart_chunk_scan_with_tiles(dims, d_in["X"], d_in["dt"], d_in["A"], d_in["Bm"], d_in["Cm"], Yssd,
                                          Mem, rM, None, tiles, ws, stream)
        else:
            Bd.dart_chunk_scan(dims, d_in["X"], d_in["dt"], d_in["A"], d_in["Bm"], d_in["Cm"], Yssd, Mem,
                               rM, None, ws, stream)
        evs = None
        if split:
            evs = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            evs[0].record(stream)
            sep.add_(1.0)
            evs[1].record(stream)
        if n_tiles > 0:
            Bd.dart_sma_forward_with_tiles(dims, tiles, d_in["Q"], d_in["Cm"], d_in["E"], d_in["z"], Yssd, Y,
                                           None, lse, stream)
        else:
            Bd.dart_sma_forward(dims, Mem, rM, d_in["Q"], d_in["Cm"], d_in["E"], d_in["z"], Yssd, Y, None,
                                lse, ws_sma, stream)
        return evs

    for _ in range(args.warmup):
        step()
        step(split=True)
    torch.cuda.synchronize()

    # ---- kernel-level timing, inputs resident in HBM
    evs = []
    with Clocks(local) as clk:
        # the timed steps take milliseconds and nvidia-smi samples every 200 ms: keep
        # the GPU on this workload for ~1 s of untimed steps first, so that most
        # samples see it under load, then time the K steps right after
        t_load = time.perf_counter()
        while time.perf_counter() - t_load < 1.0:
            flush.random_(0, 255)
            step()
            torch.cuda.synchronize()
        barrier(world)
        torch.cuda.synchronize()
        launches0 = Bd.dart_launch_count()  # the timed steps' launches only
        t_wall = time.perf_counter()
        for _ in range(args.steps):
            flush.random_(0, 255)  # untimed: evict L2 between steps
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            step()
            e1.record(stream)
            evs.append((e0, e1))
        torch.cuda.synchronize()
        barrier(world)
        t_wall = time.perf_counter() - t_wall
        launches = Bd.dart_launch_count() - launches0
        # the same steps again with the calls apart: the scan's and the SMA's own times
        split = []
        for _ in range(args.steps):
            flush.random_(0, 255)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            mid = step(split=True)
            e1.record(stream)
            split.append((e0, mid[0], mid[1], e1))
        torch.cuda.synchronize()
    step_ms = [a.elapsed_time(b) for a, b in evs]
    scan_ms = [a.elapsed_time(b) for a, b, _, _ in split]
    sma_ms = [c.elapsed_time(d) for _, _, c, d in split]
    ms = sum(step_ms) / len(step_ms)
    ms_max = max_over_ranks(ms, world, dev)
    value = world * w.tokens / (ms_max / 1e3)
    sma_avg = sum(sma_ms) / len(sma_ms)
    scan_avg = sum(scan_ms) / len(scan_ms)
    achieved = sma_flops(w) / (sma_avg / 1e3) / 1e12
    clocks = clk.summary()

    # ---- end to end through the C ABI: pinned host inputs in, Y back out
    # (dart_prefill_host: the copies overlap the kernels head group by head group)
    h_in = {k: inp[k].to(tdt).pin_memory() for k in names_in}
    h_in["dt"] = inp["dt"].pin_memory()
    h_in["A"] = inp["A"].pin_memory()
    h_out = torch.empty(Y.shape, dtype=Y.dtype).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in h_in.values())
    d2h = h_out.numel() * h_out.element_size()
    ws_host = torch.empty(Bd.dart_workspace_size(dims, Bd.DART_OP_PREFILL_HOST), dtype=torch.uint8, device=dev)
    e2e_ms = []
    for it in range(args.warmup + args.steps):
        flush.random_(0, 255)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        Bd.dart_prefill_host(dims, h_in["X"], h_in["dt"], h_in["A"], h_in["Bm"], h_in["Cm"], h_in["Q"],
                             h_in["E"], h_in["z"], h_out, ws_host, stream)
        e1.record(stream)
        e1.synchronize()
        if it >= args.warmup:
            e2e_ms.append(e0.elapsed_time(e1))
    e2e_avg = max_over_ranks(sum(e2e_ms) / len(e2e_ms), world, dev)
    e2e_value = world * w.tokens / (e2e_avg / 1e3)

    # ---- decode step (HBM bound)
    dec = None
    if not args.no_decode:
        dec = bench_decode(args, dev, world, peaks, Bd, WORKLOADS[args.decode_workload], decode_cache_slab,
                           decode_state_slab, decode_token_inputs)
    del flush
    # ---- training step (forward + backward)
    train = None
    if not args.no_train:
        # the training workload is a sweep over the chunk size: one leg per S
        train = [bench_train(args, dev, world, peaks, Bd, WORKLOADS[name], prefill_inputs)
                 for name in args.train_workload.split(",")]

    # ---- the whole block (projections, convolution, hot path, norm) at the L = 16K shape
    block = None
    if not args.no_block:
        block = bench_block(args, dev, world, peaks, Bd)

    # ---- CPU oracle on a bounded sample (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle

        ch = args.cpu_heads or max(1, min(w.heads, oracle.num_threads()))
        secs, threads = oracle_sample(w, inp, ch)
        cpu = {"value": w.tokens / (secs * w.heads / ch), "unit": "tokens/s",
               "cores": threads, "kind": "oracle",
               "sample": f"{ch} of {w.heads} heads, all {w.seqlen} tokens, full "
                         f"prefill path (recurrence, memories, SMA, merge), {secs:.1f} s"}

    if rank == 0:
        traffic = _traffic_from_profiles() if n_tiles > 0 else None
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic", "config": _config(w),
            "roofline": {"kernel": "sma_tc_kernel (dart_sma_forward_with_tiles; its operand tiles come from "
                                   "the scan's chunk-state kernel)" if n_tiles > 0 else "sma_forward",
                         "bound": "tensor", "achieved": achieved,
                         "peak": peaks["bf16"], "unit": "TFLOP/s",
                         "frac": achieved / peaks["bf16"],
                         "frac_of_sustained": achieved / peaks["bf16_sus"],
                         "peak_source": f"{peaks['source']} bf16 dense (burst)",
                         "algorithmic_flops_per_launch": sma_flops(w),
                         "ms_per_launch": sma_avg, "traffic": traffic},
            "layer": {"scan_ms": scan_avg, "sma_ms": sma_avg,
                      "timing": "scan_ms and sma_ms from the same steps with the two calls kept apart "
                                "(an event and a one-element kernel between them); ms_per_step from "
                                "steps where the SMA kernel may start under the scan's last wave",
                      "scan_roofline": {"bound": "hbm", "algorithmic_bytes": scan_bytes(w),
                                        "achieved": scan_bytes(w) / (scan_avg / 1e3) / 1e9,
                                        "peak": peaks["hbm"], "unit": "GB/s",
                                        "frac": scan_bytes(w) / (scan_avg / 1e3) / 1e9 / peaks["hbm"]},
                      "layer_tflops": (sma_flops(w) + scan_flops(w)) / (ms / 1e3) / 1e12,
                      "layer_frac": (sma_flops(w) + scan_flops(w)) / (ms / 1e3) / 1e12 / peaks["bf16"]},
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "ms_per_step": e2e_avg},
            "gpu_launches": launches, "clocks": clocks, "wall_s_timed": t_wall,
            "decode": dec,
            "train": train,
            "block": block,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


def bench_decode(args, dev, world, peaks, Bd, w, cache_slab, state_slab, token_inputs):
    import torch

    tdt = torch.bfloat16
    m_cap = w.mem + 1
    cache = torch.empty(w.batch, m_cap, w.heads, w.dstate, w.headdim, dtype=tdt, device=dev)
    state = torch.empty(w.batch, w.heads, w.dstate, w.headdim, dtype=torch.float32, device=dev)
    for b in range(w.batch):
        cache[b] = cache_slab(w, b, m_cap).to(dev, tdt)
        state[b] = state_slab(w, b).to(dev)
    partial = torch.zeros_like(state)
    tok = token_inputs(w)
    t = {k: tok[k].to(dev, tdt) for k in ("x", "b", "c", "q", "e", "z")}
    t["dt"], t["A"] = tok["dt"].to(dev), tok["A"].to(dev)
    y = torch.empty(t["x"].shape, dtype=torch.float32, device=dev)
    lse = torch.empty(w.batch, w.heads, dtype=torch.float32, device=dev)
    dims = Bd.make_dims(w.batch, 1, w.heads, w.groups, w.headdim, w.dstate, w.chunk, Bd.DART_BF16,
                        mem_dtype=Bd.DART_BF16, out_dtype=Bd.DART_F32, eps=w.eps)
    stream = torch.cuda.current_stream(dev)

    def step():
        Bd.dart_decode_step(dims, w.pos, m_cap, cache, state, partial, t["x"], t["dt"], t["A"], t["b"],
                            t["c"], t["q"], t["e"], t["z"], y, lse, None, stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    barrier(world)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):  # the 2 GiB cache is far larger than L2
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, world, dev)
    nbytes = decode_bytes(w, m_cap)
    gbs = nbytes / (ms / 1e3) / 1e9
    del cache, state, partial
    torch.cuda.empty_cache()
    return {"workload": f"{w.name}: {w.notes}", "tokens_per_s": world * w.batch / (ms / 1e3),
            "ms_per_step": ms, "bytes_per_step": nbytes,
            "roofline": {"kernel": "decode_step", "bound": "hbm", "achieved": gbs,
                         "peak": peaks["hbm"], "unit": "GB/s", "frac": gbs / peaks["hbm"],
                         "frac_of_nominal": gbs / NOMINAL_HBM_GBS,
                         "peak_source": f"{peaks['source']} copy bandwidth",
                         "traffic": _traffic_from_profiles("decode_step_decode_b64.md", "decode.cu")
                         if w.name == DECODE else None}}


def bench_block(args, dev, world, peaks, Bd):
    """One whole DART block forward (dart_block_forward) on the DART 380M block
    shape at L = 16K: in-projection, convolution, scan, SMA + merge, D skip, gated
    RMSNorm, out-projection; inputs and weights resident in HBM."""
    import torch

    from paper_2608_02032_gb300.workloads import BLOCK_WORKLOADS, block_inputs

    w = BLOCK_WORKLOADS["block_l16k"]
    inp = block_inputs(w)
    d = {k: v.to(dev) for k, v in inp.items()}
    for k in ("U", "W_in", "W_out"):
        d[k] = d[k].to(torch.bfloat16)
    dims = Bd.make_block_dims(w.batch, w.seqlen, w.d_model, w.heads, w.groups, w.headdim, w.dstate, w.chunk,
                              w.conv, Bd.DART_BF16, w.eps, w.norm_eps)
    out = torch.empty(w.batch, w.seqlen, w.d_model, dtype=torch.bfloat16, device=dev)
    ws = torch.empty(Bd.dart_block_workspace_size(dims), dtype=torch.uint8, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        Bd.dart_block_forward(dims, d["U"], d["W_in"], d["conv_w"], d["conv_b"], d["dt_bias"], d["A_log"],
                              d["D"], d["norm_w"], d["W_out"], out, ws, stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    barrier(world)
    times = []
    for _ in range(args.steps):
        flush.random_(0, 255)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        times.append((e0, e1))
    torch.cuda.synchronize()
    ms = max_over_ranks(sum(a.elapsed_time(b) for a, b in times) / len(times), world, dev)
    T = w.tokens
    proj = 2.0 * T * w.d_model * (w.d_in_proj + w.d_inner)
    pw = block_path_workload(w)
    flops = proj + sma_flops(pw) + scan_flops(pw)
    del ws, flush
    torch.cuda.empty_cache()
    return {"workload": f"{w.name}: {w.notes}", "tokens_per_s": world * T / (ms / 1e3), "ms_per_step": ms,
            "flops_per_step": flops, "tflops": flops / (ms / 1e3) / 1e12,
            "frac_of_peak": flops / (ms / 1e3) / 1e12 / peaks["bf16"],
            "peak_source": f"{peaks['source']} bf16 dense (burst)",
            "flops_model": "projections 2 T d_model (D_in + d_inner) + SMA + scan algorithmic flops"}


def block_path_workload(bw):
    """The hot-path workload inside a block workload (for the flop counts)."""
    from paper_2608_02032_gb300.workloads import Workload

    return Workload(bw.name, bw.batch, bw.heads, bw.seqlen, bw.headdim, bw.dstate, bw.chunk, groups=bw.groups)


def bench_train(args, dev, world, peaks, Bd, w, prefill_inputs):
    """One training step of the layer: forward (scan, SMA + merge, keeping the SMA
    logits) and backward (SMA from those logits, scan) on the training workload,
    inputs resident in HBM."""
    import torch

    inp = prefill_inputs(w, with_grad=True)
    tdt = torch.bfloat16
    Bsz, L, H, G, P, N, S = w.batch, w.seqlen, w.heads, w.groups, w.headdim, w.dstate, w.chunk
    M = w.nchunks
    d = {k: inp[k].to(dev, tdt).contiguous() for k in ("X", "Bm", "Cm", "Q", "E", "z", "dY")}
    d["dt"], d["A"] = inp["dt"].to(dev).contiguous(), inp["A"].to(dev).contiguous()
    dims = Bd.make_dims(Bsz, L, H, G, P, N, S, Bd.DART_BF16, eps=w.eps)
    f32 = dict(dtype=torch.float32, device=dev)
    Yssd, Y = torch.empty(Bsz, L, H, P, **f32), torch.empty(Bsz, L, H, P, **f32)
    Mem, rM = torch.empty(Bsz, M, H, N, P, **f32), torch.empty(Bsz, M, H, N, **f32)
    lse = torch.empty(Bsz, L, H, **f32)
    dM = torch.empty(Bsz, M, H, N, P, **f32)
    dQ, dC = torch.empty(Bsz, L, G, N, **f32), torch.empty(Bsz, L, G, N, **f32)
    dE, dz = torch.empty(Bsz, L, G, P, **f32), torch.empty(Bsz, L, H, **f32)
    dX, ddt = torch.empty(Bsz, L, H, P, **f32), torch.empty(Bsz, L, H, **f32)
    dA, dB = torch.empty(H, **f32), torch.empty(Bsz, L, G, N, **f32)
    logits = torch.empty(Bsz, H, M, L, **f32)  # the SMA logits, kept by the forward for the backward
    wsz = lambda op: torch.empty(max(Bd.dart_workspace_size(dims, op), 256), dtype=torch.uint8, device=dev)
    ws_scan, ws_sma = wsz(Bd.DART_OP_CHUNK_SCAN), wsz(Bd.DART_OP_SMA_FORWARD)
    ws_sbwd, ws_cbwd = wsz(Bd.DART_OP_SMA_BACKWARD), wsz(Bd.DART_OP_SCAN_BACKWARD)
    stream = torch.cuda.current_stream(dev)

    def step(evs=None):
        def mark():
            if evs is not None:
                evs.append(torch.cuda.Event(enable_timing=True))
                evs[-1].record(stream)

        mark()
        Bd.dart_chunk_scan(dims, d["X"], d["dt"], d["A"], d["Bm"], d["Cm"], Yssd, Mem, rM, None, ws_scan,
                           stream)
        mark()
        Bd.dart_sma_forward_with_logits(dims, Mem, rM, d["Q"], d["Cm"], d["E"], d["z"], Yssd, Y, None, lse,
                                        logits, ws_sma, stream)
        mark()
        Bd.dart_sma_backward_with_logits(dims, Mem, rM, d["Q"], d["Cm"], d["E"], d["z"], lse, logits, d["dY"],
                                         dM, dQ, dC, dE, dz, ws_sbwd, stream)
        mark()
        Bd.dart_chunk_scan_backward(dims, d["X"], d["dt"], d["A"], d["Bm"], d["Cm"], d["dY"], dM, dX,
                                    ddt, dA, dB, dC, ws_cbwd, stream)
        mark()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    barrier(world)
    runs = []
    for _ in range(args.steps):  # every step reads and writes far more than L2
        evs = []
        step(evs)
        runs.append(evs)
    torch.cuda.synchronize()
    phase = [sum(r[i].elapsed_time(r[i + 1]) for r in runs) / len(runs) for i in range(4)]
    ms = max_over_ranks(sum(phase), world, dev)
    flops = 4 * sma_flops(w) + 3 * scan_flops(w)
    tf = flops / (ms / 1e3) / 1e12
    return {"workload": f"{w.name}: {w.notes}", "tokens_per_s": world * w.tokens / (ms / 1e3),
            "ms_per_step": ms,
            "phase_ms": {"scan_fwd": phase[0], "sma_fwd": phase[1], "sma_bwd": phase[2],
                         "scan_bwd": phase[3]},
            "roofline": {"kernel": "layer fwd+bwd", "bound": "tensor", "achieved": tf,
                         "peak": peaks["bf16_sus"], "unit": "TFLOP/s", "frac": tf / peaks["bf16_sus"],
                         "peak_source": f"{peaks['source']} bf16 dense (sustained)",
                         "algorithmic_flops_per_step": flops,
                         "flops_model": "4 x SMA forward + 3 x scan forward (backward ~3x / 2x)",
                         "traffic": None}}


def _traffic_from_profiles(profile: str = "sma_forward_prefill_l16k.md", source: str = "sma_tc.cu"):
    """DRAM bytes per launch of a kernel from its committed ncu summary, while the
    source hash recorded there matches the current kernel source (else null)."""
    path = os.path.join(ROOT, "profiles", profile)
    src = os.path.join(ROOT, "paper_2608_02032_gb300", "csrc", source)
    try:
        with open(path) as f:
            text = f.read()
        with open(src, "rb") as f:
            digest = hashlib.sha256(f.read()).hexdigest()
    except OSError:
        return None
    mb = re.search(r"^dram_bytes_per_launch: (\d+)$", text, re.M)
    mh = re.search(r"^source_sha256: ([0-9a-f]{64})$", text, re.M)
    if mb is None or mh is None or mh.group(1) != digest:
        return None
    return int(mb.group(1))


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("dart", "reference"), default="dart")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-train", action="store_true")
    ap.add_argument("--no-block", action="store_true")
    ap.add_argument("--decode-workload", default=DECODE, help="decode workload (a smaller one for profiling)")
    ap.add_argument("--train-workload", default="train_b8_l4k_s256,train_b8_l4k_s128",
                    help="comma-separated training workloads (one leg each)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-heads", type=int, default=0,
                    help="heads in the oracle CPU sample (default: one per oracle thread)")
    ap.add_argument("--ref-heads", type=int, default=0,
                    help="heads per reference-arm step (default: one per oracle thread)")
    ap.add_argument("--workload", default=PREFILL, help="prefill workload (smaller ones for profiling)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "dart":
        print("note: at least 3 warm-up steps are required; using 3", file=sys.stderr)
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_dart(args)


if __name__ == "__main__":
    main()
