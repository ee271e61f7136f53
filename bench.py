"""Benchmark of the MiKV decode hot path on GB300.

A step = one decode token through every layer of the workload: per layer, insert the new KV pair,
attend over the mixed-precision cache (bf16 important set + low-bit retained set), update the
accumulated-attention scores, pick the least important slot and quantize/pack it into the retained set.
The metric is the compressed-KV bytes the attention reads per step divided by the step time (GB/s),
with ms per step alongside. Inputs are seeded synthetic tensors resident in HBM before timing; the cache
(tens of GB) is far larger than L2, so no flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload mistral-7b|llama2-7b|llama2-13b|tiny]
  python bench.py --impl reference ...   # the CPU oracle on a bounded sample of the same workload

Multi-GPU (torchrun, one process per GPU): the (batch, head) units are independent, so every rank runs
its own batch of the workload with no data-path collective (weak scaling); ranks only meet at the
timing barrier and a max-reduce of the elapsed time.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

import mikv_inputs as mi  # noqa: E402

METRIC = "decode-attn compressed-KV GB/s and % of GB300 HBM peak; us per decode step"
UNIT = "GB/s"
DEFAULT_WORKLOAD = "mistral-7b"
L2_BYTES = 129 * 10 ** 6          # GB300 L2
L2_FLUSH_BYTES = 1024 << 20       # flush buffer: a 512 MiB write, then a 512 MiB read (each far larger than L2)


ATTN_SOURCES = ["mikv_attention.cuh", "mikv_attention.cu", "mikv_attn_h16.cu", "mikv_device.cuh", "mikv_internal.h",
                "mikv_rows.cuh"]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "attention_traffic.json")


def _code_only(text: str) -> str:
    """C++ source without its comments and with whitespace collapsed: what the compiler sees of it (a change
    of a comment alone leaves the kernel, and so its profile, as it was)."""
    import re
    out, i, n = [], 0, len(text)
    while i < n:
        if text.startswith("//", i):
            j = text.find("\n", i)
            i = n if j < 0 else j
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            i = n if j < 0 else j + 2
        elif text[i] in "\"'":  # string and character literals are kept whole
            q, j = text[i], i + 1
            while j < n and text[j] != q:
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        else:
            out.append(text[i])
            i += 1
    return re.sub(r"\s+", " ", "".join(out)).strip()


def attention_source_sha256() -> str:
    """Hash of the attention kernel's sources, comments left out."""
    import hashlib
    h = hashlib.sha256()
    for f in ATTN_SOURCES:
        with open(os.path.join(ROOT, "paper_2402_18096_gb300", "csrc", f), encoding="utf-8") as fh:
            h.update(_code_only(fh.read()).encode())
    return h.hexdigest()


def profiled_traffic_ratio(workload: str):
    """DRAM bytes (read + write) per algorithmic byte of the attention kernel on `workload`, from the
    committed ncu figures (profiles/attention_traffic.json), if they were taken on this workload and on the
    current kernel sources; else None (counters of another kernel or shape do not apply)."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    try:
        with open(TRAFFIC_FILE) as f:
            d = json.load(f)
        if d.get("kernel_source_sha256") != attention_source_sha256() or workload not in d.get("workloads", []):
            return None
        return float(d["dram_bytes_per_algorithmic_byte"])
    except (OSError, KeyError, ValueError, TypeError):
        return None


def flush_l2(scrub: torch.Tensor):
    """Evict L2: write the first half of `scrub` (larger than L2), then read its second half, so that the dirty
    lines of the write are written back before whatever follows (only clean lines of `scrub` remain)."""
    half = scrub.numel() // 2
    scrub[:half].add_(1)
    scrub[half:].max()


def timed_with_flush(fn, n: int, scrub: torch.Tensor, stream) -> float:
    """Milliseconds of n calls fn(i), each timed alone with CUDA events on `stream` after an L2 flush
    (flush_l2) has evicted whatever the previous call left in L2."""
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    for i in range(n):
        flush_l2(scrub)
        evs[i][0].record(stream)
        fn(i)
        evs[i][1].record(stream)
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in evs)


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = os.path.join("/tmp", f"mikv_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx = max(mx, float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        return dist, rank, world, local
    return None, 0, 1, local


def max_over_ranks(dist, x: float, device="cuda") -> float:
    """The slowest rank's time: every rank contributes x, all receive the maximum."""
    if dist is None:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def rank_workload(w, rank: int):
    """Weak scaling: every rank runs the same shape on its own batch (its own seeds)."""
    return mi.scaled(w, seed=w.seed + 7919 * rank)


def build_model(w, steps_cap: int, dev, rank: int):
    """All layers' caches, built from seeded prefill tensors with the library's own kernels."""
    import paper_2402_18096_gb300 as pkg
    from paper_2402_18096_gb300.layer import MixedPrecisionLayer
    shape = pkg.shape_for_context(w.batch, w.heads_q, w.heads_kv, w.bits, w.group, w.context, w.ratio, steps_cap,
                                  hi_bits=w.hi_bits, k_channel_group=64 if w.k_channel else 0)
    wr = rank_workload(w, rank)  # each rank owns a different batch
    layers, ms, in_bytes = [], [], 0
    for li in range(w.layers):
        k, v = mi.prefill_kv(wr, li, dev)
        scores = mi.initial_scores(wr, li, dev)
        q_pre = mi.prefill_queries(wr, li, dev)
        in_bytes = sum(x.numel() * x.element_size() for x in (k, v, scores, q_pre))
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        ev[0].record()
        layers.append(MixedPrecisionLayer.from_prefill(shape, k, v, scores, q_pre, device=dev))
        ev[1].record()
        ev[1].synchronize()
        ms.append(ev[0].elapsed_time(ev[1]))
        del k, v, scores, q_pre
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    # cache build (balancer, selection, gather of the important rows, quantize/pack of the rest) per layer;
    # the first layer also pays one-time costs and is left out when there are others
    t = statistics.median(ms[1:] if len(ms) > 1 else ms)
    build = {"ms_per_layer": round(t, 3), "input_bytes_per_layer": in_bytes,
             "input_gbs": round(in_bytes / (t * 1e-3) / 1e9, 1),
             "inputs": "prefill q, k, v (bf16) and importance scores (fp32), each read once"}
    return shape, layers, build


def run_mikv(args):
    import paper_2402_18096_gb300 as pkg
    dist, rank, world, local = _dist()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    pkg.load()
    w = mi.WORKLOADS[args.workload]
    if args.batch:
        w = mi.scaled(w, batch=args.batch)
    if args.layers:
        w = mi.scaled(w, layers=args.layers)
    K, W = args.steps, args.warmup
    e2e_steps = max(2, K // 2)
    steps_cap = W + K + W + e2e_steps + 4
    shape, layers, build = build_model(w, steps_cap, dev, rank)
    L = len(layers)
    # per-step decode inputs, resident on the device
    n_in = W + K
    inputs = [[mi.decode_inputs(rank_workload(w, rank), li, s, dev) for li in range(L)]
              for s in range(n_in)]
    out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream()

    def step(s):
        for li, layer in enumerate(layers):
            q, kn, vn = inputs[s][li]
            layer.step(q, kn, vn, out)

    for s in range(W):
        step(s)
    torch.cuda.synchronize()
    for layer in layers:
        pkg.mikv_workspace_check(layer.ws)

    n_lo_before = [layer.n_lo for layer in layers]
    # a cache that L2 would hold between steps is timed step by step after an L2 flush
    cache_total = sum(layer.cache.nbytes_attended(layer.n_lo) for layer in layers)
    scrub = torch.zeros(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev) if cache_total < 2 * L2_BYTES else None
    clocks = ClockSampler(torch.cuda.current_device()) if rank == 0 else None
    if clocks:
        clocks.start()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    if scrub is None:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for s in range(K):
            step(W + s)
        e1.record(stream)
        torch.cuda.synchronize()
        step_ms = e0.elapsed_time(e1)
    else:  # a cache that fits in L2: every timed step starts from a flushed L2 (the flush is not timed)
        step_ms = timed_with_flush(lambda s: step(W + s), K, scrub, stream)
    if dist:
        dist.barrier()
    clk = clocks.stop() if clocks else None
    # bytes attended over the K steps (the attention of step s reads n_lo + s retained rows per layer)
    grow = 1 if w.bits else 0
    bytes_per_step = sum(layer.cache.nbytes_attended(n0 + grow * s) for layer, n0 in zip(layers, n_lo_before)
                         for s in range(K)) / K
    # per-channel keys: a step whose demotion completes a group of 64 adds one quantization launch per layer
    kch_launches = sum(1 for n0 in n_lo_before for s in range(K) if w.k_channel and (n0 + s) % 64 == 63)
    ms = step_ms / K
    ms = max_over_ranks(dist, ms)
    for layer in layers:
        pkg.mikv_workspace_check(layer.ws)

    # ---- dominant kernel alone: decode attention (split-K kernel + merge), same caches, events on stream
    ws_attn = [torch.zeros(pkg.mikv_workspace_bytes(shape, pkg.WS_ATTENTION, layer.n_lo) + 256, dtype=torch.uint8,
                           device=dev) for layer in layers[:1]]
    q0 = inputs[0][0][0]
    def attend_all(_=None):
        for layer in layers:
            pkg.mikv_decode_attention(layer.cache, layer.n_lo, q0, layer.sm_scale, out, ws_attn[0])

    attn_reps = max(2, -(-16 // L))  # at least 16 launches
    attend_all()  # untimed: the first launches of this entry point's kernels (module loading, attributes)
    torch.cuda.synchronize()
    if scrub is None:
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for _ in range(attn_reps):
            attend_all()
        a1.record(stream)
        torch.cuda.synchronize()
        attn_ms = a0.elapsed_time(a1) / (attn_reps * L)
    else:
        attn_ms = timed_with_flush(attend_all, max(attn_reps, K), scrub, stream) / (max(attn_reps, K) * L)
    attn_bytes = sum(layer.cache.nbytes_attended(layer.n_lo) for layer in layers) / L

    # ---- end to end through the C ABI with host buffers: H2D inputs, D2H outputs, every step
    # every layer's (q, k_new, v_new) of a step sit in one pinned host buffer and arrive in one copy
    per_in = [inputs[0][li] for li in range(L)]
    sizes = [t.numel() for trip in per_in for t in trip]
    host_flat = torch.cat([t.reshape(-1).cpu() for trip in per_in for t in trip]).pin_memory()
    dev_flat = torch.empty_like(host_flat, device=dev)
    views = list(torch.split(dev_flat, sizes))
    dev_in = [[views[3 * li + j].view(per_in[li][j].shape) for j in range(3)] for li in range(L)]
    host_out = torch.empty(L, w.batch, w.heads_q, w.head_dim, dtype=torch.bfloat16).pin_memory()
    dev_out = torch.empty(L, w.batch, w.heads_q, w.head_dim, dtype=torch.bfloat16, device=dev)
    h2d = host_flat.numel() * host_flat.element_size()
    d2h = host_out.numel() * host_out.element_size()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    e2e_s = 0.0
    for s in range(e2e_steps):
        if scrub is not None:  # flushed L2 before every step, outside the timed span
            flush_l2(scrub)
            torch.cuda.current_stream().synchronize()
        t0 = time.perf_counter()
        dev_flat.copy_(host_flat, non_blocking=True)
        for li, layer in enumerate(layers):
            layer.step(dev_in[li][0], dev_in[li][1], dev_in[li][2], dev_out[li])
        host_out.copy_(dev_out, non_blocking=True)
        torch.cuda.current_stream().synchronize()
        e2e_s += time.perf_counter() - t0
    e2e_ms = e2e_s * 1e3 / e2e_steps
    e2e_ms = max_over_ranks(dist, e2e_ms)
    for layer in layers:
        pkg.mikv_workspace_check(layer.ws)

    peak, peak_kind = _peaks()
    ratio = profiled_traffic_ratio(w.name)
    traffic = None if ratio is None else int(ratio * attn_bytes)
    value = world * bytes_per_step / (ms * 1e-3) / 1e9
    achieved = attn_bytes / (attn_ms * 1e-3) / 1e9
    line = {
        "metric": METRIC,
        "value": round(value, 1),
        "unit": UNIT,
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": round(ms, 4),
        "us_per_step": round(ms * 1e3, 1),
        "pct_of_hbm_peak": round(100 * value / world / peak, 1),
        "hbm_peak_gbs": peak,
        "hbm_peak_kind": peak_kind,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16+int%d" % w.bits,
        "data": "synthetic",
        "config": {"workload": w.name, "batch": w.batch, "layers": L, "heads_q": w.heads_q, "heads_kv": w.heads_kv,
                   "context": w.context, "bits": w.bits, "group": w.group, "importance_ratio": w.ratio,
                   "compressed_bytes_per_step": int(bytes_per_step), "l2": ("cache larger than L2, no flush" if scrub is None else
                         f"cache smaller than L2: L2 flushed before every timed step and launch (not timed) by a "
                         f"{L2_FLUSH_BYTES >> 21} MiB write and a {L2_FLUSH_BYTES >> 21} MiB read; per-step CUDA "
                         "events summed"),
                   "parallelism": f"replicas{world}"},
        "roofline": {"kernel": "decode attention (split-K + merge)", "bound": "hbm", "achieved": round(achieved, 1),
                     "peak": peak, "unit": "GB/s", "frac": round(achieved / peak, 3),
                     "traffic": traffic, "bytes_per_launch": int(attn_bytes), "avg_launch_us": round(attn_ms * 1e3, 2)},
        "e2e": {"value": round(world * bytes_per_step / (e2e_ms * 1e-3) / 1e9, 1), "unit": UNIT,
                "ms_per_step": round(e2e_ms, 4), "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        # per layer step: attention (with the new token's insertion) and the fused tail; a coded important set
        # quantizes the new token in a kernel of its own
        "gpu_launches": K * L * (2 if w.hi_bits >= 16 else 3) + kch_launches,
        "cache_build": build,
    }
    if clk:
        line["clocks"] = clk
    if rank == 0 and world == 1 and not args.no_cpu_baseline:  # the host baseline is an N = 1 figure
        line["cpu_baseline"] = cpu_baseline(w, seconds=args.cpu_seconds)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


# ------------------------------------------------------------------ CPU oracle (reference arm)

def _oracle_head(w, b, h, steps_cap):
    """Oracle cache of one (batch row, KV head) built from seeded prefill tensors of that head (drawn on
    the GPU when there is one, only to save time, then copied to the host)."""
    import numpy as np
    import oracle
    gen_dev = "cuda" if torch.cuda.is_available() else "cpu"
    G = w.heads_q // w.heads_kv
    k, v = mi.prefill_kv(w, 0, gen_dev, heads=[h])
    scores = mi.initial_scores(w, 0, gen_dev, rows=[b], heads=[h]).cpu()
    q_pre = mi.prefill_queries(w, 0, gen_dev, heads=list(range(h * G, (h + 1) * G)))
    bal = None if w.k_channel else oracle.balancer(mi.bf16_bits(q_pre), mi.bf16_bits(k))
    ks, vs = mi.bf16_bits(k[b:b + 1]), mi.bf16_bits(v[b:b + 1])
    sc = scores.numpy()
    del k, v, q_pre
    k_b = oracle.budget(w.context, w.ratio)  # the oracle's own importance-ratio rule
    lo_cap = _lo_cap(w.context - k_b + steps_cap, w.k_channel)
    dem, kept = oracle.select_demote(sc, w.context - k_b)
    if w.k_channel:  # per-channel retained keys: no balancer, the last incomplete group staged in bf16
        c = oracle.empty_cache(1, 1, w.head_dim, w.bits, w.group, k_b + 1, lo_cap, k_channel=True)
        oracle.gather_hi(c, ks, vs, kept, src_scores=sc)
        oracle.append_retained(c, ks, vs, dem, 0)
    else:
        c = oracle.empty_cache(1, 1, w.head_dim, w.bits, w.group, k_b + 1, lo_cap, hi_bits=w.hi_bits)
        oracle.gather_hi(c, ks, vs, kept, src_scores=sc, balancer_=bal)
        oracle.quantize_pack(c, ks, vs, dem, 0, balancer_=bal)
    return c, bal, np.array([[k_b]], np.int32)


def _lo_cap(rows: int, k_channel: bool) -> int:
    q = 64 if k_channel else 16
    return max(q, (rows + q - 1) // q * q)


def _oracle_step(w, c, bal, slots, n_lo, pos, q, kn, vn):
    """One decode step of one KV head on the oracle, in the library's order."""
    import numpy as np
    import oracle
    G = w.heads_q // w.heads_kv
    oracle.insert_token(c, kn, vn, pos, slots, balancer_=bal)
    _, hl, ml = oracle.decode_attention(c, q, n_lo, 1 / math.sqrt(w.head_dim), balancer_=bal)
    hc = oracle.budget(w.context, w.ratio) + 1
    acc = oracle.update_importance(c["acc"][:, :, :hc], hl[:, :, :hc].astype(np.float32), ml.astype(np.float32), G)
    c["acc"][:, :, :hc] = acc
    dem, _ = oracle.select_demote(acc, 1, c["hi_tok"][:, :, :hc], want_kept=False)
    if w.k_channel:
        oracle.append_retained(c, c["k_hi"], c["v_hi"], dem, n_lo, src_tok=c["hi_tok"])
    else:
        oracle.demote_hi(c, dem[:, :, 0], n_lo, balancer_=bal)
    return dem[0]


def _head_bytes(w, n_lo):
    import oracle
    hi_cap = oracle.budget(w.context, w.ratio) + 1
    lo = 2 * (w.head_dim * w.bits // 8 + 4 * (w.head_dim // w.group))
    if w.k_channel:  # keys: codes per token, (alpha, beta) per channel and 64 tokens; staged rows in bf16
        lo = 2 * w.head_dim * w.bits // 8 + 4 * (w.head_dim // w.group) + 4 * w.head_dim // 64
        return hi_cap * 4 * w.head_dim + (n_lo // 64 * 64) * lo + (n_lo % 64) * 4 * w.head_dim
    hi = 4 * w.head_dim if w.hi_bits >= 16 else 2 * (w.head_dim * w.hi_bits // 8 + 4 * (w.head_dim // 64))
    return hi_cap * hi + n_lo * lo


def _oracle_steps(w, c, bal, slots, seconds: float, steps=None):
    """Whole decode steps of one KV head on the oracle until `seconds` of oracle time (or `steps` steps)
    have passed; returns (compressed bytes attended, oracle seconds, steps). Input generation is untimed."""
    G = w.heads_q // w.heads_kv
    import oracle
    n_lo = w.context - oracle.budget(w.context, w.ratio)
    done_bytes, elapsed, n = 0, 0.0, 0
    while (steps is None and elapsed < seconds) or (steps is not None and n < steps):
        q, kn, vn = mi.decode_inputs(w, 0, n, "cpu", rows=[0], kv_heads=[0])
        qb = mi.bf16_bits(q[:, :G])
        kb, vb = mi.bf16_bits(kn[:, :1]), mi.bf16_bits(vn[:, :1])
        t0 = time.perf_counter()
        slots = _oracle_step(w, c, bal, slots, n_lo, w.context + n, qb, kb, vb)
        elapsed += time.perf_counter() - t0
        done_bytes += _head_bytes(w, n_lo)
        n_lo += 1
        n += 1
        if n_lo >= c["k_codes"].shape[2]:
            break
    return done_bytes, elapsed, n


def _oracle_core(w, c, bal, slots, seconds, ready, start, out):
    """One host core of the all-cores sample: the single-core sample's steps on its own copy of the head."""
    torch.set_num_threads(1)
    try:
        import oracle  # noqa: F401  (built by the parent)
        ready.put(os.getpid())
        if not start.wait(timeout=600):
            out.put(None)
            return
        out.put(_oracle_steps(w, c, bal, slots, seconds))
    except Exception as e:  # reported to the parent, which then leaves the all-cores figure out
        out.put(repr(e))


def _all_cores(w, c, bal, slots, seconds: float):
    """The same single-head decode steps on every host core at once (one spawned process per core, each on
    its own copy of the head's cache, started together): the sum of the per-core rates, or None with the
    reason if the processes cannot be run."""
    import multiprocessing as mp
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    if cores < 2:
        return None, "one host core"
    ctx = mp.get_context("spawn")  # a fresh interpreter per core: nothing inherited from the CUDA parent
    ready, out, start = ctx.Queue(), ctx.Queue(), ctx.Event()
    procs = [ctx.Process(target=_oracle_core, args=(w, c, bal, slots, seconds, ready, start, out), daemon=True)
             for _ in range(cores)]
    def collect(q, n, deadline):  # n items from q, giving up at the deadline or when a process died
        got = []
        while len(got) < n:
            if time.time() > deadline:
                raise TimeoutError("host-core processes did not answer in time")
            try:
                got.append(q.get(timeout=1.0))
            except Exception:
                if any(p.exitcode not in (None, 0) for p in procs):
                    raise RuntimeError("a host-core process exited early")
        return got

    try:
        for p in procs:
            p.start()
        collect(ready, len(procs), time.time() + 180)
        start.set()
        res = collect(out, len(procs), time.time() + seconds + 120)
    except Exception as e:
        return None, repr(e)
    finally:
        for p in procs:
            p.join(timeout=30)
            if p.is_alive():
                p.kill()
    bad = [r for r in res if not isinstance(r, tuple)]
    if bad:
        return None, str(bad[0])
    rate = sum(b / t for b, t, _ in res if t > 0)
    return {"value": round(rate / 1e9, 4), "cores": cores, "steps": sum(n for _, _, n in res)}, None


def cpu_baseline(w, seconds: float = 15.0, steps=None, all_cores: bool = True):
    """The oracle, as it stands, on a bounded sample: whole decode steps of single KV heads, first on one
    core, then on every host core at once (one process per core). `value` is the all-cores rate when it
    could be measured, else the single-core rate."""
    import oracle
    oracle.build()
    c, bal, slots = _oracle_head(w, 0, 0, 64)
    c0 = {k: a.copy() for k, a in c.items()}  # the single-core run advances its copy of the cache
    s0 = slots.copy()
    done_bytes, elapsed, n = _oracle_steps(w, c, bal, slots, seconds, steps)
    single = done_bytes / elapsed / 1e9
    line = {"value": round(single, 4), "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{n} whole decode steps of one KV head (batch row 0, head 0, layer 0) of {w.name}; "
                      f"single-threaded C, fp64 attention; bytes = that head's compressed KV",
            "ms_per_head_step": round(1e3 * elapsed / n, 3), "single_core_value": round(single, 4)}
    if all_cores:
        par, why = _all_cores(w, c0, bal, s0, seconds / 2)
        if par:
            line.update(value=par["value"], cores=par["cores"])
            line["sample"] = (f"the same single-head decode steps on {par['cores']} host cores at once (one "
                              f"process per core, {par['steps']} steps in all, about {seconds / 2:.0f} s of oracle "
                              f"time each; sum of the per-core rates), after {n} steps on one core")
        else:
            line["all_cores_unavailable"] = why
    return line


def run_sweep(args):
    """Every point of the batch-64 sweep (bits x importance ratio x group): whole decode steps on one
    layer (insert, attention, importance update, one demotion per head), plus attention alone."""
    import paper_2402_18096_gb300 as pkg
    from paper_2402_18096_gb300.layer import MixedPrecisionLayer
    dev = torch.device("cuda")
    pkg.load()
    peak, peak_kind = _peaks()
    points = []
    for w in mi.sweep_workloads():
        K, W = args.steps, args.warmup
        shape = pkg.shape_for_context(w.batch, w.heads_q, w.heads_kv, w.bits, w.group, w.context, w.ratio, K + W + 4,
                                      hi_bits=w.hi_bits)
        k, v = mi.prefill_kv(w, 0, dev)
        sc = mi.initial_scores(w, 0, dev)
        qp = mi.prefill_queries(w, 0, dev)
        layer = MixedPrecisionLayer.from_prefill(shape, k, v, sc, qp, device=dev)
        del k, v, qp
        ins = [mi.decode_inputs(w, 0, s, dev) for s in range(K + W)]
        out = torch.empty(w.batch, w.heads_q, w.head_dim, dtype=torch.bfloat16, device=dev)
        for s in range(W):
            layer.step(*ins[s], out)
        torch.cuda.synchronize()
        b0 = layer.cache.nbytes_attended(layer.n_lo)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for s in range(K):
            layer.step(*ins[W + s], out)
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / K
        nbytes = (b0 + layer.cache.nbytes_attended(layer.n_lo)) / 2 - (layer.cache.nbytes_attended(1)
                                                                     - layer.cache.nbytes_attended(0)) / 2
        ws = torch.zeros(pkg.mikv_workspace_bytes(shape, pkg.WS_ATTENTION, layer.n_lo) + 256, dtype=torch.uint8,
                         device=dev)
        pkg.mikv_decode_attention(layer.cache, layer.n_lo, ins[0][0], layer.sm_scale, out, ws)  # untimed first call
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record()
        for _ in range(K):
            pkg.mikv_decode_attention(layer.cache, layer.n_lo, ins[0][0], layer.sm_scale, out, ws)
        a1.record()
        torch.cuda.synchronize()
        attn_ms = a0.elapsed_time(a1) / K
        ab = layer.cache.nbytes_attended(layer.n_lo)
        pkg.mikv_workspace_check(layer.ws)
        pkg.mikv_workspace_check(ws)
        points.append({"bits": w.bits, "group": w.group, "ratio": w.ratio, "compressed_bytes": int(nbytes),
                       "us_per_step": round(ms * 1e3, 1), "step_gbs": round(nbytes / ms / 1e6, 1),
                       "attn_us": round(attn_ms * 1e3, 1), "attn_gbs": round(ab / attn_ms / 1e6, 1),
                       "attn_frac": round(ab / attn_ms / 1e6 / peak, 3)})
        del layer, ins
        torch.cuda.empty_cache()
    print(json.dumps({"sweep": "batch 64, 32 heads, T 4096, one layer; bits x ratio x group",
                      "metric": METRIC, "unit": UNIT, "peak": peak, "peak_kind": peak_kind, "steps": args.steps,
                      "warmup": args.warmup, "points": points}), flush=True)


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = mi.WORKLOADS[args.workload]
    K, W = args.steps, args.warmup
    import oracle
    oracle.build()
    G = w.heads_q // w.heads_kv
    c, bal, slots = _oracle_head(w, 0, 0, W + K + 4)
    n_lo = w.context - oracle.budget(w.context, w.ratio)
    times, nbytes = [], []
    for s in range(W + K):
        q, kn, vn = mi.decode_inputs(w, 0, s, "cpu", rows=[0], kv_heads=[0])
        qb, kb, vb = mi.bf16_bits(q[:, :G]), mi.bf16_bits(kn[:, :1]), mi.bf16_bits(vn[:, :1])
        t0 = time.perf_counter()
        slots = _oracle_step(w, c, bal, slots, n_lo, w.context + s, qb, kb, vb)
        dt = time.perf_counter() - t0
        if s >= W:
            times.append(dt)
            nbytes.append(_head_bytes(w, n_lo))
        n_lo += 1
    value = sum(nbytes) / sum(times) / 1e9
    ms = 1e3 * sum(times) / K
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT, "n_gpus": args.gpus,
        "steps": K, "warmup": W, "ms_per_step": round(ms, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64 attention, f32 quantizer", "data": "synthetic",
        "config": {"workload": w.name, "sample": "one KV head (batch row 0, head 0) of layer 0 per step"},
        "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"{K} whole decode steps of one KV head of {w.name}, single-threaded C"},
        "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_prefill(args):
    """Prefill importance (mikv_prefill_scores) for one layer of the workload: the accumulated causal
    attention of every prefill token; tensor-core roofline against the measured bf16 peak."""
    import paper_2402_18096_gb300 as pkg
    from paper_2402_18096_gb300.layer import workspace
    w = mi.WORKLOADS[args.workload]
    if args.batch:
        w = mi.scaled(w, batch=args.batch)
    dev = torch.device("cuda")
    pkg.load()
    k, _ = mi.prefill_kv(w, 0, dev)
    q = mi.prefill_queries(w, 0, dev)
    shape = pkg.Shape(w.batch, w.heads_q, w.heads_kv, 2, 32, 1, 16)
    out = torch.empty(w.batch, w.heads_kv, w.context, device=dev)
    ws = workspace(pkg.mikv_workspace_bytes(shape, pkg.WS_PREFILL, w.context), dev)
    for _ in range(args.warmup):
        pkg.mikv_prefill_scores(shape, q, k, out, ws)
    torch.cuda.synchronize()
    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        pkg.mikv_prefill_scores(shape, q, k, out, ws)
    e1.record()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    pkg.mikv_workspace_check(ws)
    ms = e0.elapsed_time(e1) / args.steps
    T = w.context
    # algorithmic work: two passes (row statistics, column sums) over the causal triangle of Q K^T
    flops = 2.0 * w.batch * w.heads_q * (T * (T + 1) / 2) * 2 * w.head_dim
    tflops = flops / ms / 1e9
    # a timed loop of a second or more runs under the power cap: it is compared with the sustained bf16 peak,
    # shorter ones against the burst peak
    sustained = ms * args.steps >= 1000.0
    peak, kind = None, "fallback"
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            mp = json.load(f)
        if sustained and "bf16_tflops_sustained" in mp:
            peak, kind = float(mp["bf16_tflops_sustained"]), "measured"
        else:
            peak, kind, sustained = float(mp["bf16_tflops"]), "measured", False
    if peak is None:
        peak = 1700.0 if sustained else 1900.0
    print(json.dumps({
        "metric": "prefill importance (accumulated causal attention) TFLOP/s", "value": round(tflops, 1),
        "unit": "TFLOP/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_layer": round(ms, 3),
        "higher_is_better": True, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "batch": w.batch, "heads_q": w.heads_q, "heads_kv": w.heads_kv, "context": T},
        "roofline": {"kernel": "prefill_rows_kernel + prefill_cols_kernel", "bound": "tensor", "achieved": round(tflops, 1),
                     "peak": peak, "peak_kind": kind + (" bf16 sustained" if sustained else " bf16 burst"), "unit": "TFLOP/s",
                     "frac": round(tflops / peak, 3)},
        "clocks": clocks}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mikv", choices=["mikv", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(mi.WORKLOADS))
    ap.add_argument("--batch", type=int, default=0, help="smaller batch (profiling cases only)")
    ap.add_argument("--layers", type=int, default=0, help="fewer layers (profiling cases only)")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true", help="the batch-64 bits x ratio x group sweep (one layer)")
    ap.add_argument("--prefill", action="store_true", help="prefill importance scores of one layer")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "mikv" and not (args.batch or args.layers):
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    elif args.sweep:
        run_sweep(args)
    elif args.prefill:
        run_prefill(args)
    else:
        run_mikv(args)


if __name__ == "__main__":
    main()
