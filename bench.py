"""Benchmark of the SemKV packed mixed-precision KV cache on GB300.

Workload (default, --config b16x64k): one layer of the Llama-3.1-8B KV shape (8 KV
heads, 32 query heads, head_dim 128), batch 16 x 65536-token context, affine 6/5
levels with the top 26% of tokens (Zipf(1.1) scores) at 6 levels, block B = 128.
Inputs are seeded synthetic tensors (fp16 N(0,1) K/V with 4 outlier channels x8 per
head), standing in for LongBench prompts run through the model.  Other --config
values measure the other workloads (tiny, b1x32k, l32x128k, blk4k, tq32k).

One step = one pass of the generation-time hot path over the batch:
  A6  block-exact deferred quantization of a block of 128 staged tokens
      (semkv_append_block: top-r rank in the block, quantize, pack, append), and
  A7  decode attention for all query heads over the whole cache (the prompt + the
      appended block), for every layer of the config, split-K + combine.
The appended slots are reused every step (counts rewound), so the work per step is
constant.  In the block-wise config (blk4k) a step stages ONE generated token, runs
the block append when the stage is full, and decodes over the pools plus the fp16
stage.  The prompt's own rank + quantize (A1-A5 at full size) is timed apart and
reported as quantize_gbs.

value = algorithmic bytes of the step (records and staged fp16 rows read by decode
attention, q and out, plus the appended block's fp16 K/V read and records written) /
step time, in GB/s.  The default workload moves 722 MB of records per step, more
than the 129 MB L2; workloads smaller than twice the L2 are timed step by step with
an L2 flush (a 512 MB write) between steps, outside the timed events.  roofline:
decode attention's bytes per step / its mean time (CUDA events on the launching
stream) against the measured HBM copy peak.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time

for _v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")   # the CPU oracle baseline runs on one core

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_28911_gb300 import synthetic  # noqa: E402

METRIC = ("packed-KV decode attention µs/step and HBM GB/s (% of peak); quantize GB/s")

_LLAMA = "8 KV heads, 32 q heads, d=128"
CONFIGS = {
    # base 0 = affine, 1 = TQ-MSE; mode "block": stage + append a 128-token block per
    # step; "token": stage one token per step, append when the stage is full
    "b16x64k": dict(base=0, B=16, T=65536, NL=1, H=8, Hq=32, L_hi=6, L_lo=5, r=(26, 100),
                    block=128, seed=3, mode="block",
                    desc=f"batch 16 x 64K context, 1 layer of the Llama-3.1-8B KV shape "
                         f"({_LLAMA}), affine 6/5 levels at r=26%"),
    "b4x64k": dict(base=0, B=4, T=65536, NL=1, H=8, Hq=32, L_hi=6, L_lo=5, r=(26, 100),
                   block=128, seed=3, mode="block",
                   desc=f"batch 4 x 64K context, 1 layer of the Llama-3.1-8B KV shape "
                        f"({_LLAMA}), affine 6/5 levels at r=26% (profiling size: 180 MB "
                        f"of records, above L2)"),
    "b1x32k": dict(base=0, B=1, T=32768, NL=1, H=8, Hq=32, L_hi=6, L_lo=5, r=(26, 100),
                   block=128, seed=2, mode="block",
                   desc=f"batch 1 x 32K context, 1 layer of the Llama-3.1-8B KV shape "
                        f"({_LLAMA}), affine 6/5 levels at r=26%"),
    "tiny": dict(base=0, B=1, T=1024, NL=1, H=1, Hq=4, L_hi=5, L_lo=5, r=(0, 100), block=128,
                 seed=0, mode="block",
                 desc="1 layer, 1 KV head, 4 q heads, 1024 tokens, uniform 5-level affine"),
    "l32x128k": dict(base=0, B=1, T=131072, NL=32, H=8, Hq=32, L_hi=6, L_lo=5, r=(26, 100),
                     block=128, seed=3, mode="block",
                     desc=f"batch 1 x 128K context, all 32 layers of the Llama-3.1-8B KV shape "
                          f"({_LLAMA}), affine 6/5 levels at r=26%, every layer decoded"),
    "blk4k": dict(base=0, B=1, T=4096, NL=1, H=8, Hq=32, L_hi=6, L_lo=5, r=(26, 100),
                  block=128, seed=4, mode="token",
                  desc=f"4K-token prompt + generated tokens one per step, block-wise "
                       f"deferred quantization every 128 tokens, 1 layer ({_LLAMA}), affine 6/5"),
    "had32k": dict(base=2, B=1, T=32768, NL=1, H=8, Hq=32, L_hi=6, L_lo=5, r=(26, 100),
                   block=128, seed=6, mode="block",
                   desc=f"batch 1 x 32K context, 1 layer of the Llama-3.1-8B KV shape "
                        f"({_LLAMA}), Hadamard-rotated affine 6/5 levels at r=26%"),
    "hb16x64k": dict(base=2, B=16, T=65536, NL=1, H=8, Hq=32, L_hi=6, L_lo=5, r=(26, 100),
                     block=128, seed=3, mode="block",
                     desc=f"batch 16 x 64K context, 1 layer of the Llama-3.1-8B KV shape "
                          f"({_LLAMA}), Hadamard-rotated affine 6/5 levels at r=26%"),
    "tqd32k": dict(base=3, B=1, T=32768, NL=1, H=8, Hq=32, L_hi=4, L_lo=3, r=(3, 4), block=128,
                   seed=5, mode="block",
                   desc=f"batch 1 x 32K context, 1 layer of the Mistral-7B KV shape ({_LLAMA}), "
                        f"TurboQuant-MSE-style base with a dense random rotation at 4/3 levels, "
                        f"r=75%"),
    "tq32k": dict(base=1, B=1, T=32768, NL=1, H=8, Hq=32, L_hi=4, L_lo=3, r=(3, 4), block=128,
                  seed=5, mode="block",
                  desc=f"batch 1 x 32K context, 1 layer of the Mistral-7B KV shape ({_LLAMA}), "
                       f"rotated TurboQuant-MSE-style base at 4/3 levels, r=75%"),
}
L2_BYTES = 129 * 2**20


def profiled_traffic(config_name: str):
    """DRAM bytes per decode launch from the committed ncu summary, or None when the
    summary does not cover this workload or the decode kernel source has changed since
    the counters were taken (its sha256 prefix is recorded beside the figure)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "decode_kernel_b4x64k.md")
    src = os.path.join(ROOT, "paper_2608_28911_gb300", "csrc", "decode.cu")
    try:
        text = open(path).read()
        digest = hashlib.sha256(open(src, "rb").read()).hexdigest()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch_%s: (\d+)" % re.escape(config_name), text)
    h = re.search(r"source_sha256_prefix: ([0-9a-f]+)", text)
    if not m or not h or not digest.startswith(h.group(1)):
        return None
    return int(m.group(1))


def max_over_ranks(values, device=None):
    """Each value's maximum over the ranks of the default process group (the values
    themselves in a single process): the job is as slow as its slowest replica."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t.cpu()]


def job_gbs(bytes_per_rank: float, world: int, seconds: float) -> float:
    """Whole-job throughput: every replica moves bytes_per_rank in `seconds`."""
    return bytes_per_rank * world / seconds / 1e9


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples taken while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.25)
        return self

    def __exit__(self, *exc):
        time.sleep(0.15)
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in self.lines:
            parts = [p.strip() for p in l.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------ GPU arm ---------

def build_workload(cfg, dev):
    import torch
    from paper_2608_28911_gb300 import semkv
    B, T, NL, H, Hq = cfg["B"], cfg["T"], cfg["NL"], cfg["H"], cfg["Hq"]
    r_num, r_den = cfg["r"]
    blk = cfg["block"]
    n_high = semkv.semkv_high_count_floor(T, r_num, r_den)
    n_high_blk = semkv.semkv_block_high_count(blk, r_num, r_den)
    signs = (synthetic.signs(cfg["seed"], NL, H)
             if cfg["base"] in (semkv.BASE_TQ, semkv.BASE_AFFINE_HAD) else None)
    rot = synthetic.rotations(cfg["seed"], NL, H) if cfg["base"] == semkv.BASE_TQ_DENSE else None
    desc = semkv.QuantDesc(cfg["base"], cfg["L_hi"], cfg["L_lo"], signs=signs, device=dev,
                           rotation=rot)
    cache = semkv.KVCache(desc, B, NL, H, Hq, hi_cap=n_high + n_high_blk,
                          lo_cap=T - n_high + blk - n_high_blk, block=blk, device=dev)
    k = torch.empty((B, NL, H, T, 128), dtype=torch.float16, device=dev)
    v = torch.empty_like(k)
    scores = torch.empty((B, T), dtype=torch.float32, device=dev)
    big = NL * H * T > 2**24   # draw large caches on the device, layer by layer
    for b in range(B):   # one seeded stream per sequence keeps host memory small
        sd = cfg["seed"] * 100 + b
        if big:
            for l in range(NL):
                kl, vl = synthetic.kv_layer_device(sd, l, 1, H, T, dev)
                k[b, l].copy_(kl[0])
                v[b, l].copy_(vl[0])
        else:
            kb, vb = synthetic.kv(sd, 1, NL, H, T)
            k[b].copy_(torch.from_numpy(kb[0]))
            v[b].copy_(torch.from_numpy(vb[0]))
        scores[b].copy_(torch.from_numpy(synthetic.scores_zipf(sd, 1, T)[0]))
    return dict(desc=desc, cache=cache, k=k, v=v, scores=scores, n_high=n_high,
                n_high_blk=n_high_blk)


def decode_bytes(cfg, desc, hi, lo, stage_n):
    """Algorithmic bytes of one decode attention call (one layer): the records of both
    pools, the staged fp16 rows, q and out."""
    from paper_2608_28911_gb300 import semkv
    B, H, Hq = cfg["B"], cfg["H"], cfg["Hq"]
    rh = semkv.semkv_record_bytes(desc.base, desc.levels_hi)
    rl = semkv.semkv_record_bytes(desc.base, desc.levels_lo)
    return B * H * (hi * rh + lo * rl + stage_n * 2 * 128 * 2) + B * Hq * 128 * (2 + 4)


def append_bytes(cfg, desc):
    """Algorithmic bytes of one block append: the block's fp16 K/V read, its scores,
    and its records written."""
    from paper_2608_28911_gb300 import semkv
    B, NL, H, blk = cfg["B"], cfg["NL"], cfg["H"], cfg["block"]
    rh = semkv.semkv_record_bytes(desc.base, desc.levels_hi)
    rl = semkv.semkv_record_bytes(desc.base, desc.levels_lo)
    nh_b = semkv.semkv_block_high_count(blk, *cfg["r"])
    return B * NL * H * (blk * 2 * 128 * 2 + nh_b * rh + (blk - nh_b) * rl) + B * blk * 4


def pre_decode_work(k, cache, blk, token_mode, base_counts, r_num, r_den, desc,
                    blocks_k, blocks_v, blocks_s, nblocks, semkv):
    """The host and device work of step k that precedes its decode calls: staging and,
    when due, the block append (with the appended slots rewound first)."""
    if not token_mode:
        # the block's K/V and scores already sit in device buffers laid out as the
        # stage (the caller's): point the cache's stage at them
        j = k % nblocks
        cache.s.hi_count, cache.s.lo_count, cache.s.n_tokens = base_counts
        cache.s.stage_k = blocks_k[j].data_ptr()
        cache.s.stage_v = blocks_v[j].data_ptr()
        cache.s.stage_score = blocks_s[j].data_ptr()
        cache.s.stage_n = blk
        semkv.semkv_append_block(desc, cache, r_num, r_den)
    else:
        n = cache.s.stage_n
        if n == 0:
            cache.s.hi_count, cache.s.lo_count, cache.s.n_tokens = base_counts
        j = k % (nblocks * blk)
        cache.stage_k[:, :, :, n].copy_(blocks_k[:, :, :, j])
        cache.stage_v[:, :, :, n].copy_(blocks_v[:, :, :, j])
        cache.stage_score[:, n].copy_(blocks_s[:, j])
        cache.s.stage_n = n + 1
        if cache.s.stage_n == blk:
            semkv.semkv_append_block(desc, cache, r_num, r_den)


def gpu_arm(args, cfg, rank, world):
    import torch
    from paper_2608_28911_gb300 import semkv
    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    w = build_workload(cfg, dev)
    desc, cache = w["desc"], w["cache"]
    B, T, NL, H, Hq, blk = cfg["B"], cfg["T"], cfg["NL"], cfg["H"], cfg["Hq"], cfg["block"]
    r_num, r_den = cfg["r"]
    token_mode = cfg["mode"] == "token"

    # ---- prompt: rank + quantize + pack (A1-A5), timed for quantize GB/s
    is_high = torch.empty((B, T), dtype=torch.uint8, device=dev)
    slot = torch.empty((B, T), dtype=torch.int32, device=dev)
    qt = []
    for it in range(4):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        semkv.semkv_rank_assign(w["scores"], w["n_high"], is_high, slot)
        semkv.semkv_quantize_pack(desc, w["k"], w["v"], is_high, slot, w["n_high"], cache)
        e1.record(stream)
        torch.cuda.synchronize()
        if it > 0:
            qt.append(e0.elapsed_time(e1) * 1e-3)
    rh = semkv.semkv_record_bytes(desc.base, desc.levels_hi)
    rl = semkv.semkv_record_bytes(desc.base, desc.levels_lo)
    q_bytes = B * NL * H * (T * 2 * 128 * 2 + w["n_high"] * rh + (T - w["n_high"]) * rl) + B * T * 4
    quantize_gbs = q_bytes / statistics.median(qt) / 1e9
    # the value-norm indicator over the prompt's V cache (Sec. 3.3), the cheapest scorer
    vn = torch.empty((B, T), dtype=torch.float32, device=dev)
    st_ = []
    for it in range(4):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        semkv.semkv_score_kv_norm(w["v"], vn)
        e1.record(stream)
        torch.cuda.synchronize()
        if it > 0:
            st_.append(e0.elapsed_time(e1) * 1e-3)
    score_gbs = (B * NL * H * T * 128 * 2 + B * T * 4) / statistics.median(st_) / 1e9
    # fake quantization of the prompt's K and V at the selected precisions (Sec. 4.1;
    # not provided for the dense-rotation base)
    fake_gbs = None
    if cfg["base"] != semkv.BASE_TQ_DENSE:
        ko, vo = torch.empty_like(w["k"]), torch.empty_like(w["v"])
        ft = []
        for it in range(4):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            e0.record(stream)
            semkv.semkv_fake_quant(desc, w["k"], w["v"], ko, vo, is_high=is_high)
            e1.record(stream)
            torch.cuda.synchronize()
            if it > 0:
                ft.append(e0.elapsed_time(e1) * 1e-3)
        fake_gbs = (B * NL * H * T * 128 * 2 * 4 + B * T) / statistics.median(ft) / 1e9
        del ko, vo
    del w["k"], w["v"]
    torch.cuda.empty_cache()

    # ---- generation-time step
    nblocks = 4
    gk, gv = synthetic.kv(cfg["seed"] * 100 + 99, B, NL, H, blk * nblocks)
    gs = synthetic.scores_zipf(cfg["seed"] * 100 + 99, B, blk * nblocks)
    if token_mode:
        blocks_k = torch.from_numpy(gk).to(dev)
        blocks_v = torch.from_numpy(gv).to(dev)
        blocks_s = torch.from_numpy(gs).to(dev)
    else:  # per block, contiguous in the stage layout [B][NL][H][blk][128]
        blocks_k = [torch.from_numpy(np.ascontiguousarray(gk[:, :, :, j * blk:(j + 1) * blk])).to(dev)
                    for j in range(nblocks)]
        blocks_v = [torch.from_numpy(np.ascontiguousarray(gv[:, :, :, j * blk:(j + 1) * blk])).to(dev)
                    for j in range(nblocks)]
        blocks_s = [torch.from_numpy(np.ascontiguousarray(gs[:, j * blk:(j + 1) * blk])).to(dev)
                    for j in range(nblocks)]
    q_all = torch.from_numpy(np.stack([synthetic.queries(cfg["seed"], B, Hq, step=i)
                                       for i in range(nblocks)])).to(dev)
    out = torch.empty((B, Hq, 128), dtype=torch.float32, device=dev)
    ws = cache.workspace()
    scale = 1.0 / math.sqrt(128)
    base_counts = (cache.s.hi_count, cache.s.lo_count, cache.s.n_tokens)
    nh_b = semkv.semkv_block_high_count(blk, r_num, r_den)
    # launches per decode call: (query rotation,) pools, combine (plus the stage kernel
    # while tokens are staged)
    plain = cfg["base"] == semkv.BASE_AFFINE
    dec_launch = (0 if plain else 1) + 1 + 1
    # a block append: the block rank (which also writes the slot -> token maps), quantize
    app_launch = 2

    def decode_all(qv, ev=None):
        if ev is not None:
            ev[0].record(stream)
        for layer in range(NL):
            semkv.semkv_decode_attention(desc, cache, layer, qv, out, scale, ws)
        if ev is not None:
            ev[1].record(stream)

    def q_for(i):
        return q_all[(i // blk) % nblocks] if token_mode else q_all[i % nblocks]

    def step(i, ev=None):
        pre_decode(i)
        decode_all(q_for(i), ev)

    def pre_decode(i):
        pre_decode_work(i, cache, blk, token_mode, base_counts, r_num, r_den, desc,
                        blocks_k, blocks_v, blocks_s, nblocks, semkv)

    if not token_mode:
        dec_bytes = NL * decode_bytes(cfg, desc, base_counts[0] + nh_b,
                                      base_counts[1] + blk - nh_b, 0)
        app_bytes = append_bytes(cfg, desc)
        launches_per_step = app_launch + NL * dec_launch
    else:
        # over a cycle of blk steps: stages 1..blk-1 hold that many fp16 rows, the
        # last step decodes the appended block from the pools
        cyc = sum(decode_bytes(cfg, desc, base_counts[0], base_counts[1], n) for n in range(1, blk))
        cyc += decode_bytes(cfg, desc, base_counts[0] + nh_b, base_counts[1] + blk - nh_b, 0)
        dec_bytes = NL * cyc / blk
        app_bytes = append_bytes(cfg, desc) / blk
        launches_per_step = (app_launch + NL * (dec_launch + 1) * (blk - 1) + NL * dec_launch) / blk

    flush = NL * dec_bytes < 2 * L2_BYTES
    scrub = torch.empty(512 * 2**20, dtype=torch.uint8, device=dev) if flush else None

    for i in range(args.warmup):
        step(i)
    if token_mode:   # start the timed steps at a block boundary
        while cache.s.stage_n != 0:
            step(0)
    torch.cuda.synchronize()

    if args.graph:
        # replay each distinct step from CUDA graphs, as a serving loop would: the same
        # kernels on the same data without the per-call host work.  Captured in step
        # order, so the host-side counts evolve exactly as in the direct calls; the
        # pre-decode part and the decode part are separate graphs so events can time
        # the decode between them.
        n_distinct = blk if token_mode else nblocks
        parts = []
        for k in range(n_distinct):
            ga, gd = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
            with torch.cuda.graph(ga):
                pre_decode(k)
            with torch.cuda.graph(gd):
                decode_all(q_for(k))
            parts.append((ga, gd))
        # block mode: each step also as ONE graph (the append and the decode together, so
        # the programmatic dependent launches overlap their boundary too), which times
        # the step; the pairs above time the decode alone.  (Every block-mode step rewinds
        # the counts first, so capturing the steps again finds the same host state.)
        whole = []
        if not token_mode:
            for k in range(n_distinct):
                gw = torch.cuda.CUDAGraph()
                with torch.cuda.graph(gw):
                    pre_decode(k)
                    decode_all(q_for(k))
                whole.append(gw)
        torch.cuda.synchronize()

        def step(i, ev=None, _parts=parts):   # noqa: F811 (the graph replay of the step)
            ga, gd = _parts[i % len(_parts)]
            ga.replay()
            if ev is not None:
                ev[0].record(stream)
            gd.replay()
            if ev is not None:
                ev[1].record(stream)
        for i in range(args.warmup):
            step(i)
        torch.cuda.synchronize()
        if whole:
            def step_whole(i, _whole=whole):
                _whole[i % len(_whole)].replay()
            for i in range(args.warmup):
                step_whole(i)
            torch.cuda.synchronize()

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize()

    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    # the step as a whole (one graph per step where there is one), and the decode alone
    # (its calls bracketed by events); the same steps, timed twice
    step_timed = step_whole if (args.graph and not token_mode) else step
    dec_loop = args.graph and not token_mode
    with ClockSampler(dev.index) as clk:
        if not flush:
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            barrier()
            t0.record(stream)
            for i in range(args.steps):
                if dec_loop:
                    step_timed(i)
                else:
                    step(i, evs[i])
            t1.record(stream)
            barrier()
            elapsed = t0.elapsed_time(t1) * 1e-3
        else:
            # small workloads: time each step alone, the L2 flushed in between
            sev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(args.steps)]
            barrier()
            for i in range(args.steps):
                scrub.fill_(i & 0xFF)
                sev[i][0].record(stream)
                if dec_loop:
                    step_timed(i)
                else:
                    step(i, evs[i])
                sev[i][1].record(stream)
            barrier()
            elapsed = sum(a.elapsed_time(b) for a, b in sev) * 1e-3
        if dec_loop:
            # the decode alone: the same steps replayed as (append, decode) graph pairs
            barrier()
            for i in range(args.steps):
                if flush:
                    scrub.fill_(i & 0xFF)
                step(i, evs[i])
            barrier()
    dec_times = [a.elapsed_time(b) * 1e-3 for a, b in evs]
    err = int(cache.dev_error.item())
    # the cache's own stage buffers again (the steps above pointed it at the blocks)
    cache.s.stage_k, cache.s.stage_v = cache.stage_k.data_ptr(), cache.stage_v.data_ptr()
    cache.s.stage_score = cache.stage_score.data_ptr()

    # ---- end to end through the public API with host buffers
    # contiguous pinned host buffers per block (per token in the block-wise workload),
    # as a serving loop would hand them over
    if not token_mode:
        pin_k = [torch.from_numpy(np.ascontiguousarray(gk[:, :, :, j * blk:(j + 1) * blk])).pin_memory()
                 for j in range(nblocks)]
        pin_v = [torch.from_numpy(np.ascontiguousarray(gv[:, :, :, j * blk:(j + 1) * blk])).pin_memory()
                 for j in range(nblocks)]
        pin_s = [torch.from_numpy(np.ascontiguousarray(gs[:, j * blk:(j + 1) * blk])).pin_memory()
                 for j in range(nblocks)]
        h2d = (blk * B * NL * H * 128 * 2 * 2) + blk * B * 4 + B * Hq * 128 * 2
    else:
        ntok = nblocks * blk
        pin_k = torch.from_numpy(np.ascontiguousarray(np.moveaxis(gk, 3, 0))).pin_memory()
        pin_v = torch.from_numpy(np.ascontiguousarray(np.moveaxis(gv, 3, 0))).pin_memory()
        pin_s = torch.from_numpy(np.ascontiguousarray(gs.T)).pin_memory()
        h2d = B * NL * H * 128 * 2 * 2 + B * 4 + B * Hq * 128 * 2
    pin_q = q_all.cpu().pin_memory()
    pin_out = torch.empty((B, Hq, 128), dtype=torch.float32).pin_memory()
    d2h = B * Hq * 128 * 4
    qdev = torch.empty((B, Hq, 128), dtype=torch.float16, device=dev)
    tok_k = torch.empty((B, NL, H, 128), dtype=torch.float16, device=dev)
    tok_v = torch.empty_like(tok_k)
    tok_s = torch.empty((B,), dtype=torch.float32, device=dev)

    def step_e2e(i):
        if not token_mode:
            j = i % nblocks
            cache.s.hi_count, cache.s.lo_count, cache.s.n_tokens = base_counts
            cache.stage_k.copy_(pin_k[j], non_blocking=True)
            cache.stage_v.copy_(pin_v[j], non_blocking=True)
            cache.stage_score.copy_(pin_s[j], non_blocking=True)
            qdev.copy_(pin_q[j], non_blocking=True)
            cache.s.stage_n = blk
            semkv.semkv_append_block(desc, cache, r_num, r_den)
        else:
            n = cache.s.stage_n
            if n == 0:
                cache.s.hi_count, cache.s.lo_count, cache.s.n_tokens = base_counts
            j = i % ntok
            tok_k.copy_(pin_k[j], non_blocking=True)
            tok_v.copy_(pin_v[j], non_blocking=True)
            tok_s.copy_(pin_s[j], non_blocking=True)
            qdev.copy_(pin_q[(i // blk) % nblocks], non_blocking=True)
            cache.stage_token(tok_k, tok_v, tok_s)
            if cache.s.stage_n == blk:
                semkv.semkv_append_block(desc, cache, r_num, r_den)
        for layer in range(NL):
            semkv.semkv_decode_attention(desc, cache, layer, qdev, out, scale, ws)
        pin_out.copy_(out, non_blocking=True)

    # Block mode overlaps the copies with the compute, as a serving loop would: a copy
    # stream uploads step i+1's block and queries into the other of two staging
    # buffers (the cache's stage pointers are the caller's) while step i runs, and
    # reads step i's output back after it; every copy stays inside the timed region.
    copy_s = torch.cuda.Stream()
    nbuf = 2
    bufs = [dict(k=torch.empty_like(cache.stage_k), v=torch.empty_like(cache.stage_v),
                 s=torch.empty_like(cache.stage_score), q=torch.empty_like(qdev),
                 o=torch.empty_like(out)) for _ in range(nbuf)]
    pin_outs = [torch.empty_like(pin_out).pin_memory() for _ in range(nbuf)]
    up_ev = [torch.cuda.Event() for _ in range(nbuf)]
    done_ev = [torch.cuda.Event() for _ in range(nbuf)]

    def upload(i):
        j, bb = i % nblocks, bufs[i % nbuf]
        with torch.cuda.stream(copy_s):
            if i >= nbuf:
                copy_s.wait_event(done_ev[i % nbuf])  # step i - 2 is done with this buffer
            bb["k"].copy_(pin_k[j], non_blocking=True)
            bb["v"].copy_(pin_v[j], non_blocking=True)
            bb["s"].copy_(pin_s[j], non_blocking=True)
            bb["q"].copy_(pin_q[j], non_blocking=True)
            up_ev[i % nbuf].record(copy_s)

    def compute(i):
        bb = bufs[i % nbuf]
        stream.wait_event(up_ev[i % nbuf])
        cache.s.hi_count, cache.s.lo_count, cache.s.n_tokens = base_counts
        cache.s.stage_k, cache.s.stage_v = bb["k"].data_ptr(), bb["v"].data_ptr()
        cache.s.stage_score = bb["s"].data_ptr()
        cache.s.stage_n = blk
        semkv.semkv_append_block(desc, cache, r_num, r_den)
        for layer in range(NL):
            semkv.semkv_decode_attention(desc, cache, layer, bb["q"], bb["o"], scale, ws)
        done_ev[i % nbuf].record(stream)
        with torch.cuda.stream(copy_s):
            copy_s.wait_event(done_ev[i % nbuf])
            pin_outs[i % nbuf].copy_(bb["o"], non_blocking=True)

    def run_pipelined(n):
        upload(0)
        for i in range(n):
            if i + 1 < n:
                upload(i + 1)
            compute(i)

    e2e_steps = max(3, min(args.steps, 200))
    if token_mode:
        e2e_steps = max(blk, (e2e_steps // blk) * blk)
        cache.s.stage_n = 0
        for i in range(blk):
            step_e2e(i)
    else:
        run_pipelined(3)
        torch.cuda.synchronize()
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    if token_mode:
        for i in range(e2e_steps):
            step_e2e(i)
    else:
        run_pipelined(e2e_steps)
        stream.wait_stream(copy_s)  # the last read-back is inside the timed region
    e1.record(stream)
    barrier()
    e2e_time = e0.elapsed_time(e1) * 1e-3 / e2e_steps
    if not token_mode:
        # the pipelined loop computes what the serial one does: recheck its last step
        torch.cuda.synchronize()
        cache.s.stage_k, cache.s.stage_v = cache.stage_k.data_ptr(), cache.stage_v.data_ptr()
        cache.s.stage_score = cache.stage_score.data_ptr()
        got = pin_outs[(e2e_steps - 1) % nbuf].clone()
        step_e2e(e2e_steps - 1)
        torch.cuda.synchronize()
        if not torch.equal(got, pin_out):
            raise RuntimeError("pipelined end-to-end step differs from the serial step")

    elapsed, e2e_time = max_over_ranks([elapsed, e2e_time], device=dev)
    return dict(elapsed=elapsed, dec_times=dec_times, dec_bytes=dec_bytes, app_bytes=app_bytes,
                quantize_gbs=quantize_gbs, score_gbs=score_gbs, fake_gbs=fake_gbs,
                clocks=clk.summary(), err=err,
                e2e_time=e2e_time,
                h2d=h2d, d2h=d2h, flush=flush, launches=launches_per_step * args.steps)


# ------------------------------------------------------------ CPU oracle ------

def oracle_sample(cfg, budget_s: float, max_steps: int | None = None, pair: int = 0):
    """The CPU oracle as it stands on a bounded sample of the same workload: one
    (sequence, KV head) of the batch (`pair`) and one layer, at full context -- append
    one block and run fp64 decode attention for that head's query heads -- repeated
    until the time budget (or max_steps) is spent.  Returns (GB/s of algorithmic bytes,
    sample description, steps, seconds)."""
    import oracle
    T, Hq, H, blk = cfg["T"], cfg["Hq"], cfg["H"], cfg["block"]
    base = cfg["base"]
    r_num, r_den = cfg["r"]
    G = Hq // H
    b, h = divmod(pair % (cfg["B"] * H), H)
    n_high = oracle.high_count_floor(T, r_num, r_den)
    nh_b = oracle.block_high_count(blk, r_num, r_den)
    oc = oracle.Cache(base=base, L_hi=cfg["L_hi"], L_lo=cfg["L_lo"], batch=1, layers=1, kv_heads=1,
                      q_heads=G, block=blk, hi_cap=((n_high + nh_b + 15) // 16) * 16,
                      lo_cap=((T - n_high + blk + 15) // 16) * 16)
    if base in (oracle.BASE_TQ, oracle.BASE_AFFINE_HAD):
        oc.signs = np.ascontiguousarray(synthetic.signs(cfg["seed"], 1, H)[:, h:h + 1])
    if base == oracle.BASE_TQ_DENSE:
        oc.rotation = np.ascontiguousarray(synthetic.rotations(cfg["seed"], 1, H)[:, h:h + 1])
    if base in (oracle.BASE_TQ, oracle.BASE_TQ_DENSE):
        _, c32, t32, _ = oracle.lloyd_max_gaussian(cfg["L_hi"])
        oc.cb_hi = (c32, t32)
        _, c32, t32, _ = oracle.lloyd_max_gaussian(cfg["L_lo"])
        oc.cb_lo = (c32, t32)
    kb, vb = synthetic.kv_layer(cfg["seed"] * 100 + b, 0, 1, H, T)
    s = synthetic.scores_zipf(cfg["seed"] * 100 + b, 1, T)
    oracle.quantize_prompt(oc, synthetic.f16_bits(kb[:, None, h:h + 1]),
                           synthetic.f16_bits(vb[:, None, h:h + 1]), s, r_num, r_den)
    gk, gv = synthetic.kv(cfg["seed"] * 100 + 99, 1, 1, H, blk)
    gs = synthetic.scores_zipf(cfg["seed"] * 100 + 99, 1, blk)
    q = synthetic.f16_bits(synthetic.queries(cfg["seed"], 1, Hq)[:, h * G:(h + 1) * G])
    counts = (oc.hi_count, oc.lo_count, oc.n_tokens)
    rh, rl = oracle.record_bytes(base, cfg["L_hi"]), oracle.record_bytes(base, cfg["L_lo"])
    per_step = ((n_high + nh_b) * rh + (T - n_high + blk - nh_b) * rl + G * 128 * 6
                + blk * 2 * 128 * 2 + nh_b * rh + (blk - nh_b) * rl + blk * 4)
    steps, t_start = 0, time.perf_counter()
    while True:
        oc.hi_count, oc.lo_count, oc.n_tokens = counts
        oc.stage_k[0, 0, 0, :blk] = synthetic.f16_bits(gk[0, 0, h])
        oc.stage_v[0, 0, 0, :blk] = synthetic.f16_bits(gv[0, 0, h])
        oc.stage_score[0, :blk] = gs[0]
        oc.stage_n = blk
        oracle.append_block(oc, r_num, r_den)
        oracle.decode_attention(oc, 0, q, 1 / math.sqrt(128))
        steps += 1
        el = time.perf_counter() - t_start
        if (max_steps is not None and steps >= max_steps) or (max_steps is None and el >= budget_s):
            break
    sample = (f"1 of {cfg['B'] * H} (sequence, KV head) pairs, 1 of {cfg['NL']} layers, at "
              f"full {T}-token context: append one {blk}-token block + fp64 decode attention "
              f"for its {G} query heads, x{steps} repetitions")
    return per_step * steps / el / 1e9, sample, steps, el


def _oracle_worker(args):
    """One process of the multi-core baseline (module level, so a spawned process can
    import it): the oracle on its own (sequence, KV head) pair."""
    cfg_name, budget_s, max_steps, pair = args
    gbs, _, steps, el = oracle_sample(CONFIGS[cfg_name], budget_s, max_steps, pair)
    return gbs * el * 1e9, steps, el


def host_cpus():
    """(usable cores, CPU model) of this host."""
    n = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    model = ""
    try:
        r = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10)
        m = re.search(r"Model name:\s*(.+)", r.stdout)
        model = m.group(1).strip() if m else ""
    except (OSError, subprocess.SubprocessError):
        pass
    if not model:
        try:
            for line in open("/proc/cpuinfo"):
                if line.lower().startswith(("model name", "cpu part")):
                    model = line.split(":", 1)[1].strip()
                    break
        except OSError:
            pass
    return n, model


def oracle_sample_cores(cfg_name, budget_s: float, max_steps: int | None = None, cores=None):
    """The oracle as it stands on every host core at once: one spawned process per core,
    each on its own (sequence, KV head) pair of the workload (the pairs are independent,
    as on the GPU).  Returns (GB/s of all processes' bytes over the wall time, sample,
    cores, CPU model, wall seconds)."""
    import multiprocessing as mp
    n, model = host_cpus()
    n = cores or n
    cfg = CONFIGS[cfg_name]
    pairs = cfg["B"] * cfg["H"]
    ctx = mp.get_context("spawn")    # a fresh interpreter per process: no CUDA state inherited
    t0 = time.perf_counter()
    with ctx.Pool(n) as pool:
        res = pool.map(_oracle_worker, [(cfg_name, budget_s, max_steps, i % pairs) for i in range(n)])
    wall = time.perf_counter() - t0
    total_bytes = sum(r[0] for r in res)
    busy = max(r[2] for r in res)
    sample = (f"{n} processes, one per core, each on its own (sequence, KV head) pair of "
              f"{pairs}, 1 of {cfg['NL']} layers, at full {cfg['T']}-token context: append one "
              f"{cfg['block']}-token block + fp64 decode attention, "
              f"x{min(r[1] for r in res)}-{max(r[1] for r in res)} repetitions each")
    return total_bytes / busy / 1e9, sample, n, model, wall


# ------------------------------------------------------------------ main ------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="b16x64k", choices=sorted(CONFIGS))
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--graph", action=argparse.BooleanOptionalAction, default=True,
                    help="replay the device-resident steps from CUDA graphs (the e2e steps "
                         "always call the API directly)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    cfg = CONFIGS[args.config]
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    peaks, peak_kind = load_peaks()
    config = {"workload": cfg["desc"], "batch": cfg["B"], "context": cfg["T"],
              "layers": cfg["NL"], "kv_heads": cfg["H"], "q_heads": cfg["Hq"],
              "levels": [cfg["L_hi"], cfg["L_lo"]], "r": f"{cfg['r'][0]}/{cfg['r'][1]}",
              "block": cfg["block"],
              "base": {0: "affine", 1: "TQ-MSE", 2: "Hadamard-rotated affine",
                       3: "TQ-MSE, dense rotation"}[cfg["base"]],
              "step": "one generated token staged per step, block append every 128 steps"
              if cfg["mode"] == "token" else "append one 128-token block + decode every layer"}

    if args.impl == "reference":
        if rank != 0:
            return
        # every host core runs the oracle on its own pair; a step = one block append +
        # decode on each of them
        steps = args.warmup + args.steps
        gbs, sample, cores, model, wall = oracle_sample_cores(args.config, 0, max_steps=steps)
        line = {"impl": "reference", "metric": METRIC, "value": gbs, "unit": "GB/s",
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": wall / steps * 1e3, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config,
                "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": cores, "kind": "oracle",
                                 "cpu": model, "sample": sample},
                "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
        dist.init_process_group("nccl")
    r = gpu_arm(args, cfg, rank, world)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    if rank != 0:
        return
    config["l2"] = ("flushed between timed steps (512 MB write, outside the events)" if r["flush"]
                    else "inputs larger than L2 (records read per step > 2 x 129 MB)")
    step_s = r["elapsed"] / args.steps
    step_bytes = r["dec_bytes"] + r["app_bytes"]
    dec_mean = sum(r["dec_times"]) / len(r["dec_times"])
    achieved = r["dec_bytes"] / dec_mean / 1e9
    peak = peaks["hbm_gbs"]
    line = {
        "metric": METRIC, "value": job_gbs(step_bytes, world, step_s), "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f16 codes x f16 -> f32 (mma), f32 softmax",
        "data": "synthetic", "config": config,
        "decode_us_per_step": dec_mean * 1e6,
        "decode_gbs": achieved,
        "decode_frac_of_peak": achieved / peak,
        "decode_frac_of_nominal_8tbs": achieved / 8000.0,
        "quantize_gbs": r["quantize_gbs"],
        "value_norm_score_gbs": r["score_gbs"],
        "fake_quant_gbs": r["fake_gbs"],
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": profiled_traffic(args.config),
                     "kernel": {0: "decode_affine_fast_kernel + combine_wide_kernel",
                                2: "qrot_kernel + decode_affine_fast_kernel + combine_wide_kernel",
                                1: "qrot_kernel + decode_kernel<1> + combine_wide_kernel",
                                3: "qrot_dense_kernel + decode_kernel<1> + combine_kernel<dense>"}[cfg["base"]]
                               + " (semkv_decode_attention)",
                     "peak_kind": f"{peak_kind} hbm_gbs"},
        "e2e": {"value": job_gbs(step_bytes, world, r["e2e_time"]), "unit": "GB/s",
                "h2d_bytes_per_step": r["h2d"], "d2h_bytes_per_step": r["d2h"]},
        "gpu_launches": int(round(r["launches"])),
        "clocks": r["clocks"],
        "device_error": r["err"],
    }
    if world == 1 and args.cpu_seconds > 0:
        # the oracle on every host core (the baseline), and on one core alongside
        gbs, sample, cores, model, _ = oracle_sample_cores(args.config, args.cpu_seconds / 2)
        gbs1, sample1, _, _ = oracle_sample(cfg, args.cpu_seconds / 2)
        line["cpu_baseline"] = {"value": gbs, "unit": "GB/s", "cores": cores, "kind": "oracle",
                                "cpu": model, "sample": sample,
                                "single_core": {"value": gbs1, "unit": "GB/s", "sample": sample1}}
    print(json.dumps(line))


if __name__ == "__main__":
    main()
