#!/usr/bin/env python
"""Benchmark: incremental-prefill attention at 120K cached tokens, one layer.

Workload (the 120K-context step): 64 query heads, 4 KV heads, head_dim 128,
bf16, RoPE base 1e6, page size 64.  The cache holds a 4,096-token static
prefix plus 256-token chunks; the first timed step starts at 122,880 cached
tokens.  A step appends a 256-token state chunk, attends a 512-token task
suffix over the whole cache and truncates the suffix (section III-D), through
the C-ABI library: by default in one pass (csr_append_chunk_attend_suffix, then
csr_truncate_suffix; --step separate issues csr_append_chunk and
csr_attend_suffix instead); the chunk is then invalidated again (csr_rewind, host-only)
so that every step sees exactly 122,880 cached tokens.  Inputs are seeded synthetic N(0,1) bf16 tensors already
resident in HBM; the KV cache (about 252 MB) is larger than the 129 MB L2, so
no flush is needed between steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  `value` is the device-timed microseconds per
layer-step (lower is better), `e2e` the same through the public API with the
step's inputs copied from pinned host memory and its outputs copied back
inside the timed region.  `roofline` is the attention kernel's achieved
TFLOP/s (algorithmic FLOPs / its CUDA-event time) against the measured bf16
peak; `cpu_baseline` times the fp64 CPU oracle on a bounded sample of the
same step.  With N > 1 (torchrun) every rank runs an independent replica
(the path does not shard: one layer's cache lives on one GPU); `value` is the
whole job's time per layer-step, the slowest replica's step time divided by N
(N layer-steps per step time), and config.replica_us_per_step the step time
itself.  `--impl reference` times the fp64 oracle alone.
"""
from __future__ import annotations

import argparse
import hashlib
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

METRIC = "µs/layer and % roofline, incremental-prefill attention at 120K cached tokens"
UNIT = "us/layer"
HQ, HKV, D, P, BASE = 64, 4, 128, 64, 1e6
PREFIX, CHUNK, SUFFIX, L0 = 4096, 256, 512, 122880
LAYERS_PROXY = 94
WORKLOAD_NAME = ("120K-context step: append 256-token chunk + attend 512-token suffix + truncate, "
                 "122,880 cached tokens, 64 q / 4 kv heads, head_dim 128, page 64, bf16, 1 layer")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "attention_120k_traffic.txt")
ATTN_SRC = os.path.join(ROOT, "paper_2605_07325_gb300", "csrc", "kernels_attn.cu")


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            m = json.load(f)
        return float(m["hbm_gbs"]), float(m["bf16_tflops"]), float(m["bf16_tflops_sustained"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, 1900.0, 1700.0, "fallback"


def _attention_source_hash() -> str:
    with open(ATTN_SRC, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def _traffic_per_launch(fused: bool):
    """DRAM bytes per attention launch of the step from the committed ncu
    summary (the fused step's single launch, or the mean of the separate
    step's two), if it was taken on the current kernel source; else None."""
    try:
        with open(TRAFFIC_FILE) as f:
            kv = dict(line.strip().split("=", 1) for line in f
                      if "=" in line and not line.startswith("#"))
        if kv.get("kernel_source_sha256_16") != _attention_source_hash():
            return None
        if fused:
            return float(kv["dram_bytes_per_launch_fused"])
        return float(kv["dram_bytes_per_step"]) / 2
    except (OSError, KeyError, ValueError):
        return None


# ------------------------------------------------------------------ replicas
def reduce_max_over_ranks(values, device=None):
    """Max over ranks of each value (the slowest replica defines the time);
    identity when torch.distributed is not initialised or has one rank."""
    import torch
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t.cpu()]


# --------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.proc = None
        self.first = ""
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={gpu_id}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            # wait for the first sample: nvidia-smi's start-up (driver queries)
            # must not fall inside the timed region
            self.first = self.proc.stdout.readline()
            time.sleep(0.3)
        except OSError:
            self.proc = None

    def stop(self, t0: float, t1: float):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=10)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in (self.first + out).splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                rows.append((ts, float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return None
        inside = [r for r in rows if t0 - 1 <= r[0] <= t1 + 1] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i, v in enumerate(r[3]) if v == "Active"})
        return {"sm_mhz": statistics.median(r[1] for r in inside),
                "sm_max_mhz": max(r[2] for r in inside), "reasons": reasons,
                "samples": len(inside)}


# ------------------------------------------------------------------ oracle leg
def _oracle_cache(seed: int = 7):
    """Rotated keys and values of a 122,880-token cache for the oracle."""
    import numpy as np
    from oracle import oracle as orc
    from paper_2605_07325_gb300 import synth
    rng = np.random.default_rng(seed)
    k = synth.bf16_to_f64(synth.bf16_bits(rng.standard_normal((L0, HKV, D), dtype=np.float32)))
    v = synth.bf16_to_f64(synth.bf16_bits(rng.standard_normal((L0, HKV, D), dtype=np.float32)))
    k = orc.rope(k, np.arange(L0), BASE)
    return k, v


def _oracle_step_sample(k_cache, v_cache, n_chunk: int, n_suffix: int, seed: int):
    """Time the oracle on n_chunk tokens of the chunk and n_suffix tokens of
    the suffix (all 64 query heads), and return (seconds, sampled pairs,
    full-step pairs) so the time can be scaled to the whole step."""
    import numpy as np
    from oracle import oracle as orc
    from paper_2605_07325_gb300 import costmodel, synth
    rng = np.random.default_rng(seed)
    new = CHUNK + SUFFIX
    q = synth.bf16_to_f64(synth.bf16_bits(rng.standard_normal((new, HQ, D), dtype=np.float32)))
    kn = synth.bf16_to_f64(synth.bf16_bits(rng.standard_normal((new, HKV, D), dtype=np.float32)))
    vn = synth.bf16_to_f64(synth.bf16_bits(rng.standard_normal((new, HKV, D), dtype=np.float32)))
    pos_new = np.arange(L0, L0 + new)
    sel = np.concatenate([np.arange(n_chunk), CHUNK + np.arange(n_suffix)])
    t0 = time.perf_counter()
    kn_rot = orc.rope(kn, pos_new, BASE)                         # all new keys
    q_rot = orc.rope(q[sel], pos_new[sel], BASE)                 # sampled queries
    k_all = np.concatenate([k_cache, kn_rot])
    v_all = np.concatenate([v_cache, vn])
    kpos = np.arange(L0 + new)
    orc.attention(q_rot, pos_new[sel], k_all, v_all, kpos, 1.0 / math.sqrt(D))
    secs = time.perf_counter() - t0
    sampled = int(sum(L0 + int(s) + 1 for s in sel))
    full = costmodel.query_key_pairs(L0, new)
    return secs, sampled, full


def _oracle_config_tiny() -> float:
    """The tiny correctness case in full through the oracle (8 q / 2 kv heads,
    d 64, page 16, base 1e4): a 256-token prefix, three 256-token chunks, a
    32-token suffix, truncate, one more chunk, the suffix again; every output
    computed.  Returns seconds."""
    from oracle import oracle as orc
    from paper_2605_07325_gb300 import synth
    t0 = time.perf_counter()
    o = orc.OracleCSR(8, 2, 64, 16, 1e4, pool_pages=256)
    blk = lambda seed, n: synth.block(seed, n, 8, 2, 64).f64()
    o.init_static(*blk(0, 256))
    for i in range(3):
        o.append_chunk(*blk(1 + i, 256))
    o.attend_suffix(*blk(100, 32))
    o.truncate_suffix()
    o.append_chunk(*blk(4, 256))
    o.attend_suffix(*blk(101, 32))
    o.truncate_suffix()
    return time.perf_counter() - t0


def _oracle_config_8k() -> float:
    """One step of the 8K-context case in full through the oracle (64 q / 4 kv
    heads, d 128, page 64, base 1e6): over a 2,048-token prefix + 48 chunks
    of 128 (cache bookkeeping only while filling), append a 128-token chunk,
    attend a 64-token suffix, truncate.  Returns the step's seconds."""
    from oracle import oracle as orc
    from paper_2605_07325_gb300 import synth
    o = orc.OracleCSR(HQ, HKV, D, P, BASE, pool_pages=(8192 + 256) // P + 8)
    blk = lambda seed, n: synth.block(seed, n, HQ, HKV, D).f64()
    o.attend = False
    o.init_static(*blk(200, 2048))
    for i in range(48):
        o.append_chunk(*blk(201 + i, 128))
    o.attend = True
    chunk, suffix = blk(300, 128), blk(301, 64)
    t0 = time.perf_counter()
    o.append_chunk(*chunk)
    o.attend_suffix(*suffix)
    o.truncate_suffix()
    return time.perf_counter() - t0


def cpu_baseline(target_s: float = 15.0):
    """The oracle as it stands, on this host's cores: the 120K step on a
    bounded sample scaled by query-key pairs to microseconds per layer-step
    (extrapolated), and the tiny and 8K cases in full."""
    from oracle import oracle as orc
    k, v = _oracle_cache()
    s1, p1, full = _oracle_step_sample(k, v, 1, 1, seed=11)       # calibration
    per_pair = s1 / p1
    tokens = max(2, min(CHUNK + SUFFIX, int(target_s / (per_pair * (L0 + 300)))))
    n_c = min(CHUNK, tokens // 2)
    n_s = min(SUFFIX, tokens - n_c)
    secs, pairs, full = _oracle_step_sample(k, v, n_c, n_s, seed=12)
    us = secs * full / pairs * 1e6
    cores = orc.default_threads()
    tiny_s = _oracle_config_tiny()
    step8k_s = _oracle_config_8k()
    return {"value": us, "unit": UNIT, "cores": cores, "kind": "oracle",
            "extrapolated": True, "sampled_fraction": pairs / full, "sample_seconds": secs,
            "sample": (f"fp64 C oracle: RoPE of the step's 768 new keys + attention of {n_c} chunk "
                       f"and {n_s} suffix query tokens (all 64 heads) over 122,880+ keys, "
                       f"{secs:.1f} s, scaled by query-key pairs to the full step"),
            "configs": [
                {"config": "tiny correctness case: full session (prefix 256, 3 chunks of 256, "
                           "suffix 32, truncate, chunk, suffix), 8 q / 2 kv heads, d 64",
                 "seconds": tiny_s, "cores": cores, "extrapolated": False},
                {"config": "8K-context step: append 128 + attend 64 + truncate over 8,192 cached, "
                           "64 q / 4 kv heads, d 128", "us_per_step": step8k_s * 1e6,
                 "cores": cores, "extrapolated": False},
                {"config": WORKLOAD_NAME, "us_per_step": us, "cores": cores, "extrapolated": True,
                 "sampled_fraction": pairs / full}]}


def run_reference(args):
    """--impl reference: the fp64 oracle timed alone on the host cores.  Each
    step runs a bounded sample of the 120K step; `value` scales it by
    query-key pairs to the whole step (extrapolated: true), `ms_per_step` is
    the time a step actually took."""
    from oracle import oracle as orc
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    k, v = _oracle_cache()
    s1, p1, _ = _oracle_step_sample(k, v, 1, 1, seed=11)
    budget = 150.0 / max(1, args.steps + args.warmup)              # seconds per step
    tokens = max(2, int(budget / (s1 / p1 * (L0 + 300))))
    n_c, n_s = tokens // 2, tokens - tokens // 2
    vals, spent, fracs = [], [], []
    for i in range(args.warmup + args.steps):
        secs, pairs, full = _oracle_step_sample(k, v, n_c, n_s, seed=100 + i)
        if i >= args.warmup:
            vals.append(secs * full / pairs * 1e6)
            spent.append(secs)
            fracs.append(pairs / full)
    value = statistics.mean(vals)
    cores = orc.default_threads()
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": statistics.mean(spent) * 1e3, "higher_is_better": False, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "extrapolated": True, "sampled_fraction": statistics.mean(fracs),
            "config": {"workload": WORKLOAD_NAME},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "extrapolated": True, "sampled_fraction": statistics.mean(fracs),
                             "sample": f"per step: {n_c} chunk + {n_s} suffix query tokens "
                                       f"({statistics.mean(spent):.2f} s actually spent per step, "
                                       "ms_per_step), scaled by query-key pairs to the whole step "
                                       "(value)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# -------------------------------------------------------------------- GPU leg
def run_ours(args):
    import torch
    import torch.distributed as dist
    from paper_2605_07325_gb300 import costmodel, csr

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    K, W = args.steps, args.warmup
    fill = args.fill_chunk
    fill_chunks = (L0 - PREFIX) // fill
    max_tokens = L0 + CHUNK + SUFFIX
    pool_pages = math.ceil(max_tokens / P) + 16
    cfg = csr.make_config(HQ, HKV, D, P, BASE, max_new_tokens=PREFIX, pool_pages=pool_pages,
                          max_seq_tokens=max_tokens + P,
                          fg_chunk_tiles=args.fg_chunk_tiles,
                          flags=csr.FLAG_SCHEDULE_LOCAL if args.schedule == "local" else 0)
    stream = torch.cuda.Stream(device=dev, priority=-1)
    gen = torch.Generator(device=dev).manual_seed(1234 + rank)

    def rnd(n, h):
        return torch.randn((n, h, D), generator=gen, device=dev, dtype=torch.float32).to(torch.bfloat16)

    with torch.cuda.stream(stream):
        ctx = csr.Context(cfg, device=str(dev), stream=stream)
        pq, pk, pv = rnd(PREFIX, HQ), rnd(PREFIX, HKV), rnd(PREFIX, HKV)
        ctx.init_static(pq, pk, pv, stream=stream)
        fq = rnd(fill, HQ)
        fout = torch.empty((fill, HQ, D), dtype=torch.bfloat16, device=dev)
        for _ in range(fill_chunks):
            ctx.append_chunk(fq, rnd(fill, HKV), rnd(fill, HKV), out=fout, stream=stream)
        sets = []
        for _ in range(4):   # the step's tokens: the chunk (first 256), then the suffix
            sets.append(dict(q=rnd(CHUNK + SUFFIX, HQ), k=rnd(CHUNK + SUFFIX, HKV),
                             v=rnd(CHUNK + SUFFIX, HKV),
                             o=torch.empty((CHUNK + SUFFIX, HQ, D), dtype=torch.bfloat16, device=dev)))
    stream.synchronize()
    assert ctx.layout()[1] == L0, ctx.layout()[1]
    fused = args.step == "fused"

    def run_step(s):
        # one step of the robot loop: state chunk, task suffix, drop the suffix;
        # then invalidate the cache after L0 (host-only) so every step sees 122,880
        # cached tokens
        if fused:
            ctx.append_chunk_attend_suffix(s["q"], s["k"], s["v"], CHUNK, out=s["o"], stream=stream)
        else:
            c, x = slice(0, CHUNK), slice(CHUNK, CHUNK + SUFFIX)
            ctx.append_chunk(s["q"][c], s["k"][c], s["v"][c], out=s["o"][c], stream=stream)
            ctx.attend_suffix(s["q"][x], s["k"][x], s["v"][x], out=s["o"][x], stream=stream)
        ctx.truncate_suffix()
        ctx.rewind(L0)

    def step(i):
        run_step(sets[i % len(sets)])

    for i in range(W):
        step(i)
    stream.synchronize()
    assert ctx.layout()[1] == L0

    # ------------------------------------------------ device-timed region
    props = torch.cuda.get_device_properties(dev)
    uuid = getattr(props, "uuid", None)
    gpu_id = f"GPU-{uuid}" if uuid is not None else os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[local]
    sampler = ClockSampler(gpu_id)
    launches0 = ctx.kernel_launches()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t_wall0 = time.time()
    e0.record(stream)
    for i in range(K):
        step(i)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    t_wall1 = time.time()
    if world > 1:
        dist.barrier()
    ms_total = e0.elapsed_time(e1)
    launches = ctx.kernel_launches() - launches0
    clocks = sampler.stop(t_wall0, t_wall1)
    # the same K steps again with an event pair around every kernel launch
    # (the library's timing): the per-kernel device times of the roofline.
    # They are a second timed region because the events sit between launches
    # the library otherwise chains with programmatic dependent launch (a
    # launch's first CTAs start on the SMs the previous one's last CTAs free)
    ctx.set_timing(True)
    torch.cuda.synchronize(dev)
    e4, e5 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e4.record(stream)
    for i in range(K):
        step(i)
    e5.record(stream)
    torch.cuda.synchronize(dev)
    ms_instrumented = e4.elapsed_time(e5)
    ktimes = ctx.get_timing()
    ctx.set_timing(False)

    # ------------------------------------------------ end to end, host buffers
    host = []
    for s in sets:
        host.append({k: s[k].cpu().pin_memory() for k in ("q", "k", "v")})
        host[-1]["o"] = torch.empty((CHUNK + SUFFIX, HQ, D), dtype=torch.bfloat16).pin_memory()
    # two staging sets: step i's inputs go up and step i-1's output comes down on a
    # copy stream while the compute stream runs the step before; the stream order
    # on the copy stream (upload i+1 after download i-1) keeps a staging set from
    # being overwritten while a step still reads it
    stage = [{k: torch.empty_like(v) for k, v in sets[0].items()} for _ in range(2)]
    copy_stream = torch.cuda.Stream(device=dev)
    h2d = sum(sets[0][k].numel() * 2 for k in ("q", "k", "v"))
    d2h = (CHUNK + SUFFIX) * HQ * D * 2
    up_done = [torch.cuda.Event() for _ in range(2)]
    step_done = [torch.cuda.Event() for _ in range(2)]

    def upload(i):
        h, b = host[i % len(host)], i % 2
        with torch.cuda.stream(copy_stream):
            for k in ("q", "k", "v"):
                stage[b][k].copy_(h[k], non_blocking=True)
        up_done[b].record(copy_stream)

    def download(i):
        h, b = host[i % len(host)], i % 2
        copy_stream.wait_event(step_done[b])
        with torch.cuda.stream(copy_stream):
            h["o"].copy_(stage[b]["o"], non_blocking=True)

    def run_e2e(n, start=None, end=None):
        if start is not None:
            start.record(stream)
        if n == 0:
            if end is not None:
                end.record(stream)
            return
        copy_stream.wait_stream(stream)
        upload(0)
        for i in range(n):
            b = i % 2
            stream.wait_event(up_done[b])
            with torch.cuda.stream(stream):
                run_step(stage[b])
            step_done[b].record(stream)
            if i > 0:
                download(i - 1)
            if i + 1 < n:
                upload(i + 1)
        download(n - 1)
        stream.wait_stream(copy_stream)
        if end is not None:
            end.record(stream)

    run_e2e(W)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    run_e2e(K, e2, e3)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    ms_e2e = e2.elapsed_time(e3)
    flags = ctx.device_status()

    ms_total, ms_e2e = reduce_max_over_ranks([ms_total, ms_e2e], device=dev)

    # ------------------------------------------------ roofline of the attention kernel
    hbm, peak_burst, peak_sust, peak_kind = _peaks()
    # the timed steps covered L = L0 + 256 i for the chunk and + 256 for the suffix
    step_flops = (costmodel.attention_flops(HQ, D, L0, CHUNK) +
                  costmodel.attention_flops(HQ, D, L0 + CHUNK, SUFFIX))
    flops = step_flops * K
    att_ms, att_n = ktimes["attention"]
    achieved = flops / (att_ms * 1e-3) / 1e12 if att_ms > 0 else None
    traffic = _traffic_per_launch(fused)
    step_floor = (costmodel.floor_seconds(costmodel.attention_flops(HQ, D, L0, CHUNK),
                                          costmodel.call_bytes(HQ, HKV, D, L0, CHUNK), peak_burst, hbm) +
                  costmodel.floor_seconds(costmodel.attention_flops(HQ, D, L0 + CHUNK, SUFFIX),
                                          costmodel.call_bytes(HQ, HKV, D, L0 + CHUNK, SUFFIX),
                                          peak_burst, hbm)) * 1e6
    us_step = ms_total / K * 1e3
    # the whole job: `world` replicas each process one layer-step per step time
    us_job = us_step / world
    line = {
        "metric": METRIC, "value": us_job, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": W, "ms_per_step": ms_total / K, "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: seeded N(0,1) bf16 Q/K/V (torch CUDA generator), resident in HBM",
        "config": {"workload": WORKLOAD_NAME, "cached_tokens": L0,
                   "step_calls": ("csr_append_chunk_attend_suffix + csr_truncate_suffix" if fused else
                                  "csr_append_chunk + csr_attend_suffix + csr_truncate_suffix"),
                   "step_flops": step_flops,
                   "l2": "inputs larger than L2: the 252 MB KV cache is streamed every step",
                   "replicas": world, "replica_us_per_step": us_step,
                   "foreground_ctas": ctx.cfg.num_ctas or props.multi_processor_count,
                   "kernel_events": "value: K steps timed whole, no per-kernel events; roofline."
                                    "achieved: the same K steps again with a CUDA event pair around "
                                    "every kernel launch (the events sit between launches the "
                                    "library otherwise chains with programmatic dependent launch)",
                   "instrumented_us_per_step": ms_instrumented / K * 1e3},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak_burst, "unit": "TFLOP/s",
                     "frac": (achieved / peak_burst) if achieved else None,
                     "traffic": traffic,
                     "kernel": "attn_pair_kernel<128, true>: the whole call in one cooperative "
                               "launch (RoPE + paged append, tcgen05 QK^T and PV over TMA-staged "
                               "paged K/V, cut units merged by their last pieces)",
                     "launches": att_n, "avg_launch_us": att_ms / max(1, att_n) * 1e3,
                     "peak_source": f"bf16_tflops ({peak_kind}, burst)",
                     "frac_of_sustained": (achieved / peak_sust) if achieved else None},
        "step_roofline": {"floor_us": step_floor, "frac": step_floor / us_step,
                          "note": "max(FLOPs / bf16 peak, bytes / HBM peak) per call, summed over the step"},
        "ttft_proxy_94_layers_ms": us_step * LAYERS_PROXY / 1e3,
        "kernels": {k: {"ms_total": v[0], "launches": v[1]} for k, v in ktimes.items() if v[1]},
        "e2e": {"value": ms_e2e / K * 1e3 / world, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "copies": "pinned host -> device inputs and device -> host output of every step, "
                          "on a copy stream overlapping the neighbouring steps' compute"},
        "gpu_launches": launches,
        "clocks": clocks,
        "device_error_flags": flags,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline()
    if rank == 0:
        print(json.dumps(line), flush=True)
    ctx.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


# ------------------------------------------------------------------ ASR leg
ASR_CAP, ASR_EVICT = 131072, 32768


def run_asr(args):
    """The ASR cycle run: cache capped at 131,072 tokens (4,096-token prefix),
    foreground steps (256-token chunk + 512-token suffix + truncate; one fused
    call, or two with --step separate) at a fixed cadence; reaching the cap
    evicts the oldest 32,768 tokens of chunks and
    rebuilds the retained ~98K tokens on a low-priority stream (Algorithm 1),
    then swaps.  --asr-cap / --asr-evict / --asr-chunk change the setting (the
    paper's robot run: 100-token chunks, tau_mem = 110K, the oldest half of the
    chunks evicted: --asr-chunk 100 --asr-cap 110000 --asr-evict 52952).  Reports foreground step latency during and outside rebuilds
    and checks that every post-swap layout is consistent (distinct page ids,
    disjoint from the free list, pool fully accounted for); the layouts are
    compared with the oracle's allocator in the GPU tests."""
    import numpy as np
    import torch
    from paper_2605_07325_gb300 import csr

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    # N_max of App. D: the active version may grow past tau_mem while the rebuild and its
    # catch-up run (Eq. oom_time); one eviction's worth of headroom covers back-to-back steps
    cap, evict, chunk = args.asr_cap, args.asr_evict, args.asr_chunk
    n_max = cap + evict
    pool_pages = (2 * n_max) // P + 64
    cfg = csr.make_config(HQ, HKV, D, P, BASE, max_new_tokens=PREFIX, pool_pages=pool_pages,
                          max_seq_tokens=n_max, cap_tokens=cap,
                          evict_tokens=evict, n_catchup=0,
                          rebuild_tiles_per_cta=args.asr_rebuild_tiles,
                          flags=csr.FLAG_UNPACED_REBUILD if args.asr_unpaced else 0,
                          rebuild_duty=args.asr_duty)
    fg = torch.cuda.Stream(device=dev, priority=-1)     # high priority
    lo = torch.cuda.Stream(device=dev, priority=0)      # low priority (rebuild, R_2)
    gen = torch.Generator(device=dev).manual_seed(4321)

    def rnd(n, h):
        return torch.randn((n, h, D), generator=gen, device=dev, dtype=torch.float32).to(torch.bfloat16)

    chunks = {}

    def provider(cid, n):
        q, k, v = chunks[cid]
        return q, k, v, None

    def reconciling():
        try:
            ctx.layout(csr.VERSION_PENDING)
            return True
        except csr.CsrError:
            return False

    def layout_consistent():
        pt, length = ctx.layout()
        free = ctx.free_pages()
        return (len(set(pt)) == len(pt) and not set(pt) & set(free)
                and len(pt) + len(free) == pool_pages and len(pt) == -(-length // P))

    with torch.cuda.stream(fg):
        ctx = csr.Context(cfg, device=str(dev), stream=fg)
        ctx.set_reconciler(provider, lo)
        ctx.init_static(rnd(PREFIX, HQ), rnd(PREFIX, HKV), rnd(PREFIX, HKV), stream=fg)
        fout = torch.empty((chunk, HQ, D), dtype=torch.bfloat16, device=dev)
        while ctx.layout()[1] + chunk < cap:
            q, k, v = rnd(chunk, HQ), rnd(chunk, HKV), rnd(chunk, HKV)
            chunks[len(chunks)] = (q, k, v)      # ids are 0, 1, 2, ... in append order
            ctx.append_chunk(q, k, v, out=fout, stream=fg)
        sq, sk, sv = rnd(SUFFIX, HQ), rnd(SUFFIX, HKV), rnd(SUFFIX, HKV)
        so = torch.empty((SUFFIX, HQ, D), dtype=torch.bfloat16, device=dev)
        step_out = torch.empty((chunk + SUFFIX, HQ, D), dtype=torch.bfloat16, device=dev)
    fg.synchronize()
    fused = args.step == "fused"

    period = 1.0 / args.asr_cadence_hz if args.asr_cadence_hz > 0 else 0.0
    records, rebuilds, layout_ok = [], [], True
    cycles, step = 0, 0
    rb_start = None
    peak_len = 0
    next_t = time.perf_counter()
    while cycles < args.asr_cycles:
        with torch.cuda.stream(fg):
            q, k, v = rnd(chunk, HQ), rnd(chunk, HKV), rnd(chunk, HKV)
            if fused:   # the task's tokens as one block: the chunk, then the suffix
                qs, ks, vs = torch.cat([q, sq]), torch.cat([k, sk]), torch.cat([v, sv])
        fg.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0 = time.perf_counter()
        # the task starts by polling the reconciliation (the swap happens between tasks)
        st = ctx.poll_swap(fg)
        was = st == csr.RECON_RUNNING            # (the poll's answer: no host work in the timed region)
        if st == csr.RECON_SWAPPED:
            t_sw = time.perf_counter()
            layout_ok = layout_ok and layout_consistent()
            rebuilds.append(t_sw - rb_start)
            cycles += 1
            t0 += time.perf_counter() - t_sw     # the layout check is the bench's, not the step's
        e0.record(fg)
        chunks[len(chunks)] = (q, k, v)          # before the call: it may start a rebuild
        if fused:
            _, _, cid = ctx.append_chunk_attend_suffix(qs, ks, vs, chunk, out=step_out, stream=fg)
        else:
            _, _, cid = ctx.append_chunk(q, k, v, out=fout, stream=fg)
            ctx.attend_suffix(sq, sk, sv, out=so, stream=fg)
        assert cid == len(chunks) - 1
        ctx.truncate_suffix()   # with the fused call, an eviction due starts here
        e1.record(fg)
        e1.synchronize()
        t1 = time.perf_counter()
        now = reconciling()
        if now and not was:
            rb_start = time.perf_counter()   # the library started it inside append_chunk
        length = ctx.layout()[1]
        peak_len = max(peak_len, length)
        during = was or now
        records.append((t1 - t0, e0.elapsed_time(e1) / 1e3, during, length))
        step += 1
        if period:
            next_t += period
            time.sleep(max(0.0, next_t - time.perf_counter()))
    flags = ctx.device_status()

    def pct(xs, q):
        return float(np.percentile(np.array(xs) * 1e3, q)) if xs else None

    dur = [r[0] for r in records if r[2]]
    out = [r[0] for r in records if not r[2]]
    dev_dur = [r[1] for r in records if r[2]]
    dev_out = [r[1] for r in records if not r[2]]
    # A rebuild runs while the cache is at its largest (from tau_mem until the
    # swap), the steps outside it over every length down to the post-eviction
    # one: the like-for-like baseline is the outside steps over caches at
    # least as long as the shortest one a rebuild ran beside (less 2,048).
    band = min((r[3] for r in records if r[2]), default=0) - 2048
    out_m = [r[0] for r in records if not r[2] and r[3] >= band]
    dev_out_m = [r[1] for r in records if not r[2] and r[3] >= band]
    line = {
        "workload": (f"ASR cycle run: cap {cap:,} tokens, 4,096-token prefix, {chunk}-token chunks + "
                     f"512-token suffix per step, evict oldest {evict:,} tokens, rebuild on a "
                     "low-priority stream, 64 q / 4 kv heads, d 128, page 64, 1 layer"),
        "step_calls": ("csr_append_chunk_attend_suffix + csr_truncate_suffix" if fused else
                       "csr_append_chunk + csr_attend_suffix + csr_truncate_suffix"),
        "cadence_hz": args.asr_cadence_hz, "rebuild_tiles_per_cta": args.asr_rebuild_tiles or 16,
        "rebuild_pacing": "all tasks at once" if args.asr_unpaced else
                          "one task in flight, started after the foreground work",
        "rebuild_duty": args.asr_duty,
        "cycles": cycles, "steps": step,
        "steps_during_rebuild": len(dur),
        "fg_ms_host": {"p50_outside": pct(out, 50), "p99_outside": pct(out, 99),
                       "p50_during": pct(dur, 50), "p99_during": pct(dur, 99)},
        "fg_ms_device": {"p50_outside": pct(dev_out, 50), "p99_outside": pct(dev_out, 99),
                         "p50_during": pct(dev_dur, 50), "p99_during": pct(dev_dur, 99)},
        "matched_outside": {"min_cached_tokens": band, "steps": len(out_m),
                            "host_p50": pct(out_m, 50), "host_p99": pct(out_m, 99),
                            "device_p50": pct(dev_out_m, 50), "device_p99": pct(dev_out_m, 99)},
        "rebuild_to_swap_s": {"mean": statistics.mean(rebuilds) if rebuilds else None,
                              "max": max(rebuilds) if rebuilds else None,
                              "note": "eviction to the poll (start of a step) that swapped"},
        "peak_cached_tokens": peak_len, "n_max_tokens": n_max,
        "layout_consistent": layout_ok,
        "device_error_flags": flags,
    }
    if out and dur:
        line["p99_increase_during_rebuild_all_lengths"] = pct(dur, 99) / pct(out, 99) - 1.0
    if out_m and dur:
        line["p99_increase_during_rebuild"] = pct(dur, 99) / pct(out_m, 99) - 1.0
        line["p99_increase_during_rebuild_device"] = pct(dev_dur, 99) / pct(dev_out_m, 99) - 1.0
    # App. D viability: the rebuild (warm-up + catch-up, here eviction -> swap)
    # must end before the cache, growing at X_dot tokens/s from tau_mem, reaches N_max
    if rebuilds and period:
        x_dot = chunk / period
        dt_mem = (n_max - cap) / x_dot
        line["viability"] = {"x_dot_tokens_per_s": x_dot, "dt_mem_s": dt_mem,
                             "dt_rebuild_max_s": max(rebuilds),
                             "holds": max(rebuilds) <= dt_mem and peak_len <= n_max}
        # the library's own check (csr_check_viability) for an eviction started
        # now, from the rebuild pace it observed on the last reconciliation
        try:
            line["viability_library"] = ctx.check_viability(evict, x_dot)
        except csr.CsrError as e:
            line["viability_library"] = {"error": str(e)}
    print(json.dumps(line), flush=True)
    ctx.close()
    return 0 if layout_ok and flags == 0 else 1


# ------------------------------------------------------------- unordered leg
def run_unordered(args):
    """Per-layer analogue of the paper's unordered baseline (Table II,
    'Unord.'): the whole prompt is dynamic, so every step recomputes the
    cache from scratch -- a causal prefill of the 4,096-token prefix, the
    chunks and the 512-token suffix (123,648 tokens, in 4,096-token blocks) --
    against the CSR step (append 256 + attend 512 + truncate over 122,880
    cached tokens) measured in the same run."""
    import torch
    from paper_2605_07325_gb300 import costmodel, csr

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    total = L0 + CHUNK + SUFFIX
    cfg = csr.make_config(HQ, HKV, D, P, BASE, max_new_tokens=4096,
                          pool_pages=total // P + 16, max_seq_tokens=total + P)
    stream = torch.cuda.Stream(device=dev, priority=-1)
    gen = torch.Generator(device=dev).manual_seed(777)

    def rnd(n, h):
        return torch.randn((n, h, D), generator=gen, device=dev, dtype=torch.float32).to(torch.bfloat16)

    blocks = []
    left = total
    while left > 0:
        n = min(4096, left)
        blocks.append((rnd(n, HQ), rnd(n, HKV), rnd(n, HKV),
                       torch.empty((n, HQ, D), dtype=torch.bfloat16, device=dev)))
        left -= n
    times = []
    with torch.cuda.stream(stream):
        for step in range(args.warmup + max(5, args.steps // 100)):
            ctx = csr.Context(cfg, device=str(dev), stream=stream)
            stream.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            q, k, v, o = blocks[0]
            ctx.init_static(q, k, v, out=o, stream=stream)
            for q, k, v, o in blocks[1:]:
                ctx.append_chunk(q, k, v, out=o, stream=stream)
            e1.record(stream)
            stream.synchronize()
            if step >= args.warmup:
                times.append(e0.elapsed_time(e1))
            assert ctx.device_status() == 0
            ctx.close()
    unordered_ms = statistics.mean(times)
    flops = costmodel.attention_flops(HQ, D, 0, total)
    line = {"workload": "unordered baseline: full causal prefill of 123,648 tokens per step, "
                        "64 q / 4 kv heads, d 128, page 64, bf16, 1 layer",
            "unordered_ms_per_layer": unordered_ms, "steps": len(times),
            "unordered_ms_min": min(times), "unordered_ms_max": max(times),
            "unordered_ms_stdev": statistics.stdev(times) if len(times) > 1 else 0.0,
            "tflops": flops / (unordered_ms * 1e-3) / 1e12,
            "note": "compare with the CSR step (value of the default bench line) measured "
                    "in the same process below"}
    csr_args = argparse.Namespace(**vars(args))
    csr_args.no_cpu_baseline = True
    csr_args.steps = min(args.steps, 100)
    import io
    import contextlib
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        run_ours(csr_args)
    csr_line = json.loads(buf.getvalue().strip().splitlines()[-1])
    line["csr_us_per_layer"] = csr_line["value"]
    line["speedup_csr_over_unordered"] = unordered_ms * 1e3 / csr_line["value"]
    line["paper_context"] = ("paper Table II, 120K tokens: unordered 14.67 s vs CSR M=1024 0.56 s "
                             "(26x), end-to-end TTFT of a 235B model on 4xH100")
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- sweep leg
SWEEP_L = (16384, 32768, 65536, 98304, 131072)
SWEEP_N = (16, 64, 256, 1024, 4096)


def run_sweep(args):
    """One attend call of n new tokens over L cached tokens for every sweep
    point: device time per call (mean over K >= 20 back-to-back calls, and
    the median and p99 of K single calls), the attention kernel's time,
    achieved TFLOP/s and GB/s, and the fraction of the roofline floor
    max(FLOPs / bf16 peak, bytes / HBM peak)."""
    import torch
    from paper_2605_07325_gb300 import costmodel, csr

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    hbm, peak, _, kind = _peaks()
    max_L = max(args.sweep_l or SWEEP_L)
    path_flags = {"auto": 0, "fused": csr.FLAG_FUSED_ALWAYS, "three": csr.FLAG_FUSED_NEVER}[args.sweep_path]
    cfg = csr.make_config(HQ, HKV, D, P, BASE, max_new_tokens=4096,
                          pool_pages=(max_L + 4096) // P + 16, max_seq_tokens=max_L + 4096 + P,
                          flags=path_flags)
    stream = torch.cuda.Stream(device=dev, priority=-1)
    gen = torch.Generator(device=dev).manual_seed(99)

    def rnd(n, h):
        return torch.randn((n, h, D), generator=gen, device=dev, dtype=torch.float32).to(torch.bfloat16)

    K, W = max(20, args.steps // 10), args.warmup
    sweep_n = args.sweep_n or SWEEP_N
    points = []
    with torch.cuda.stream(stream):
        ctx = csr.Context(cfg, device=str(dev), stream=stream)
        ctx.init_static(rnd(PREFIX, HQ), rnd(PREFIX, HKV), rnd(PREFIX, HKV), stream=stream)
        fill_q = rnd(4096, HQ)
        fill_o = torch.empty((4096, HQ, D), dtype=torch.bfloat16, device=dev)
        blocks = {n: (rnd(n, HQ), rnd(n, HKV), rnd(n, HKV),
                      torch.empty((n, HQ, D), dtype=torch.bfloat16, device=dev)) for n in sweep_n}
        for L in (args.sweep_l or SWEEP_L):
            while ctx.layout()[1] < L:
                ctx.append_chunk(fill_q, rnd(4096, HKV), rnd(4096, HKV), out=fill_o, stream=stream)
            assert ctx.layout()[1] == L
            for n in sweep_n:
                q, k, v, o = blocks[n]
                for _ in range(W):
                    ctx.attend_suffix(q, k, v, out=o, stream=stream)
                    ctx.truncate_suffix()
                # one call inside an NVTX range "probe": what an ncu capture of a
                # sweep point selects (--nvtx --nvtx-include probe/)
                stream.synchronize()
                torch.cuda.nvtx.range_push("probe")
                ctx.attend_suffix(q, k, v, out=o, stream=stream)
                ctx.truncate_suffix()
                stream.synchronize()
                torch.cuda.nvtx.range_pop()
                # whole calls, untimed inside (the library's per-kernel events
                # would add their own cost to short calls) ...
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                for _ in range(K):
                    ctx.attend_suffix(q, k, v, out=o, stream=stream)
                    ctx.truncate_suffix()
                e1.record(stream)
                stream.synchronize()
                us = e0.elapsed_time(e1) / K * 1e3
                # ... the latency of single calls (an event pair around each:
                # consecutive calls no longer overlap) ...
                ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                      for _ in range(K)]
                for a, b_ in ev:
                    a.record(stream)
                    ctx.attend_suffix(q, k, v, out=o, stream=stream)
                    ctx.truncate_suffix()
                    b_.record(stream)
                stream.synchronize()
                lat = sorted(a.elapsed_time(b_) * 1e3 for a, b_ in ev)
                # ... then the per-kernel split from a third, event-timed pass
                ctx.set_timing(True)
                for _ in range(K):
                    ctx.attend_suffix(q, k, v, out=o, stream=stream)
                    ctx.truncate_suffix()
                stream.synchronize()
                t = ctx.get_timing()
                ctx.set_timing(False)
                f = costmodel.attention_flops(HQ, D, L, n)
                b = costmodel.call_bytes(HQ, HKV, D, L, n)
                floor = costmodel.floor_seconds(f, b, peak, hbm) * 1e6
                att_us = t["attention"][0] / max(1, t["attention"][1]) * 1e3
                pt = {"L": L, "n": n, "us_per_call": us, "calls": K,
                      "us_median": lat[len(lat) // 2], "us_p99": lat[min(len(lat) - 1, int(0.99 * len(lat)))],
                      "attention_us": att_us,
                      "rope_append_us": t["rope_append"][0] / K * 1e3, "merge_us": t["merge"][0] / K * 1e3,
                      "tflops": f / (us * 1e-6) / 1e12, "gbs": b / (us * 1e-6) / 1e9,
                      "floor_us": floor, "bound": "tensor" if f / (peak * 1e12) > b / (hbm * 1e9) else "hbm",
                      "roofline_frac": floor / us}
                points.append(pt)
                print(json.dumps(pt), flush=True)
    status = ctx.device_status()
    ctx.close()
    oracle_points = _sweep_oracle(args, points) if args.sweep_oracle else []
    print(json.dumps({"sweep": "L x n, one attend call each", "path": args.sweep_path,
                      "peaks": {"bf16_tflops": peak, "hbm_gbs": hbm,
                      "source": kind}, "points": len(points),
                      "min_frac": min(p["roofline_frac"] for p in points),
                      "oracle_points": len(oracle_points),
                      "device_error_flags": status}), flush=True)
    return 0


def _sweep_oracle(args, points):
    """The oracle column of the sweep: the fp64 C oracle on the same call (RoPE
    of the n new queries and keys, attention of all 64 heads over L + n keys)
    in full, on the host cores, for n in {16, 256} at every L."""
    import numpy as np
    from oracle import oracle as orc
    from paper_2605_07325_gb300 import synth
    ls = sorted(args.sweep_l or SWEEP_L)
    ns = [n for n in (16, 256) if n in (args.sweep_n or SWEEP_N)]
    if not ns:
        return []
    rng = np.random.default_rng(5)
    cap = max(ls) + max(ns)
    bf = lambda shape: synth.bf16_to_f64(synth.bf16_bits(rng.standard_normal(shape, dtype=np.float32)))
    k_all = np.empty((cap, HKV, D))
    v_all = np.empty((cap, HKV, D))
    for i in range(0, cap, 4096):                 # the cache: rotated keys, values (not timed)
        m = min(4096, cap - i)
        k_all[i:i + m] = orc.rope(bf((m, HKV, D)), np.arange(i, i + m), BASE)
        v_all[i:i + m] = bf((m, HKV, D))
    kpos = np.arange(cap)
    gpu = {(p["L"], p["n"]): p["us_per_call"] for p in points}
    out = []
    for L in ls:
        for n in ns:
            q, kn, vn = bf((n, HQ, D)), bf((n, HKV, D)), bf((n, HKV, D))
            pos = np.arange(L, L + n)
            t0 = time.perf_counter()
            q_rot = orc.rope(q, pos, BASE)
            k_all[L:L + n] = orc.rope(kn, pos, BASE)
            v_all[L:L + n] = vn
            orc.attention(q_rot, pos, k_all[:L + n], v_all[:L + n], kpos[:L + n], 1.0 / math.sqrt(D))
            secs = time.perf_counter() - t0
            pt = {"L": L, "n": n, "oracle_us": secs * 1e6, "cores": orc.default_threads(),
                  "extrapolated": False, "kind": "oracle (fp64 C, all 64 heads, in full)"}
            if (L, n) in gpu:
                pt["gpu_us"] = gpu[(L, n)]
                pt["oracle_over_gpu"] = secs * 1e6 / gpu[(L, n)]
            out.append(pt)
            print(json.dumps(pt), flush=True)
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--step", choices=["fused", "separate"], default="fused",
                    help="how a step calls the library: separate (csr_append_chunk then "
                         "csr_attend_suffix) or fused (csr_append_chunk_attend_suffix, one pass)")
    ap.add_argument("--schedule", choices=["default", "local"], default="default",
                    help="fused launch's piece schedule: the idle-interval construction, or "
                         "least-advanced-first steps where they balance (CSR_FLAG_SCHEDULE_LOCAL)")
    ap.add_argument("--fg-chunk-tiles", type=int, default=0,
                    help="key tiles per attention work item (0: the library's cost model)")
    ap.add_argument("--fill-chunk", type=int, default=CHUNK, choices=[256, 512, 1024, 2048, 4096],
                    help="chunk size used to fill the cache before timing (fewer launches "
                         "for profiler captures); the timed steps are unchanged")
    ap.add_argument("--asr", action="store_true",
                    help="run the ASR cycle workload instead of the 120K step line")
    ap.add_argument("--asr-cycles", type=int, default=10)
    ap.add_argument("--asr-cap", type=int, default=ASR_CAP, help="tau_mem in tokens")
    ap.add_argument("--asr-evict", type=int, default=ASR_EVICT, help="tokens evicted per cycle")
    ap.add_argument("--asr-chunk", type=int, default=CHUNK, help="tokens per state chunk")
    ap.add_argument("--asr-rebuild-tiles", type=int, default=0,
                    help="key tiles per rebuild CTA (0: the library default, 16)")
    ap.add_argument("--asr-duty", type=float, default=0.0,
                    help="share of wall time the rebuild may occupy the GPU (0 = no limit)")
    ap.add_argument("--asr-unpaced", action="store_true",
                    help="enqueue every rebuild task at once (default: one in flight, started "
                         "after the foreground work)")
    ap.add_argument("--asr-cadence-hz", type=float, default=2.0,
                    help="foreground step rate; 0 runs steps back to back")
    ap.add_argument("--sweep", action="store_true",
                    help="run the L x n sweep instead of the 120K step line")
    ap.add_argument("--sweep-l", type=int, nargs="*", default=None,
                    help="cached lengths of the sweep (default: 16K 32K 64K 96K 128K)")
    ap.add_argument("--sweep-n", type=int, nargs="*", default=None,
                    help="new-token counts of the sweep (default: 16 64 256 1024 4096)")
    ap.add_argument("--sweep-path", choices=["auto", "fused", "three"], default="auto",
                    help="with --sweep: the library's choice of foreground path, or one forced")
    ap.add_argument("--sweep-oracle", action="store_true",
                    help="with --sweep: also time the fp64 oracle in full on every L at n = 16 and 256")
    ap.add_argument("--unordered", action="store_true",
                    help="time the unordered baseline (full recompute per step) beside CSR")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.sweep:
        return run_sweep(args)
    if args.unordered:
        return run_unordered(args)
    if args.asr:
        return run_asr(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
