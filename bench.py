#!/usr/bin/env python
"""Benchmark of the GPU-resident LLM prefix (blocks [0, k) of a 7B-class backbone).

One step = one frame through the prefix: a 2304-token prefill of blocks [0, 16) (all
projections, attention and KV writes on the tensor-core path) and the boundary hand-off of
h^(16) [2304, 4096] bf16 to pinned host memory on a side stream, overlapped with the next
frame's prefill (the GPU side of the cross-frame pipeline, Sec. IV-C). A decode phase then
times 64 single-token steps of the same 16 blocks against a 2304-position context.

Inputs are seeded synthetic tensors of the workload's shapes (the paper's Bench2Drive frames
and Orion weights are not available): weights ~ N(0, 0.02), hidden states ~ N(0, 1).

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Under torchrun each rank runs an independent replica (the prefix has no exchange step on one
GPU); the slowest rank's time is reported and ``value`` counts all ranks' tokens.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "prefix prefill tokens/s & % bf16 TC peak; decode µs/step & HBM GB/s (1 GB300)"
WORKLOAD = "7b_prefix16_2304tok"
DECODE_WORKLOAD = "7b_decode16_ctx2304"
PIPELINE_WORKLOAD = "7b_pipeline32_3072tok"
BLOCK_WORKLOAD = "7b_block_1024tok"
PIPELINE_SPLITS = (8, 16, 24)
HYBRID_SPLIT = 31  # GPU blocks [0, 31), the last block on the host cores
HYBRID_ZONE_MIN = 28  # dynamic zone [28, 32] of the scheduled run


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return d["hbm_gbs"], d["bf16_tflops"], d["bf16_tflops_sustained"], "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# ------------------------------------------------------------------------------------------
# distributed plumbing (replicas; only the barrier and the max-reduce of the time cross ranks)
# ------------------------------------------------------------------------------------------
class Dist:
    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None

    def init(self, backend: str):
        if self.world > 1:
            import torch.distributed as dist
            dist.init_process_group(backend=backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, x: float, device=None) -> float:
        if not self.pg:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64, device=device)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


# ------------------------------------------------------------------------------------------
# clocks sampled during the timed region
# ------------------------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        # raw samples go to $VLA_ARTIFACT_DIR (default: artifacts/ at the repository root)
        out = os.environ.get("VLA_ARTIFACT_DIR", os.path.join(ROOT, "artifacts"))
        self.path = os.path.join(out, f"clocks_{os.getpid()}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict | None:
        if not self.proc:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, smax, reasons = [], 0.0, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax = max(smax, float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------------------
# CPU oracle timing (baseline and reference arm): only here and in the tests is oracle/ run
# ------------------------------------------------------------------------------------------
_ORACLE_W = {}


def oracle_prefill_time(n_tokens: int, seed: int = 0) -> tuple[float, int]:
    """Seconds for the float64 oracle to run one 7B-class block over the first ``n_tokens``
    tokens of the workload's frame (weights converted outside the timed region)."""
    import oracle
    wl = synth.WORKLOADS[WORKLOAD]
    s = wl.shape
    if seed not in _ORACLE_W:
        _ORACLE_W[seed] = oracle.LayerWeights.from_bf16(synth.layer_weights(s, seed, 0))
    w = _ORACLE_W[seed]
    x = oracle.bf16_to_f64(synth.hidden_states(n_tokens, s.hidden, seed, min(n_tokens, wl.visual_tokens),
                                               wl.visual_scale))
    cache = oracle.KVCache([0], s.n_kv_heads, s.head_dim, n_tokens)
    t0 = time.perf_counter()
    oracle.block_forward(x, w, cache, 0, s)
    return time.perf_counter() - t0, os.cpu_count() or 1


def oracle_decode_time(dwl) -> float:
    """Seconds for the float64 oracle to run one decode step of one 7B-class block against the
    decode workload's random context (weights and context converted outside the timed region)."""
    import oracle
    s = dwl.shape
    if dwl.seed not in _ORACLE_W:
        _ORACLE_W[dwl.seed] = oracle.LayerWeights.from_bf16(synth.layer_weights(s, dwl.seed, 0))
    w = _ORACLE_W[dwl.seed]
    kb, vb = synth.random_kv(dwl.prefill_ctx, s, dwl.seed, 0)
    cache = oracle.KVCache([0], s.n_kv_heads, s.head_dim, dwl.prefill_ctx + 1)
    cache.fill(0, oracle.bf16_to_f64(kb), oracle.bf16_to_f64(vb))
    x = oracle.bf16_to_f64(synth.decode_hidden(0, s.hidden, dwl.seed))
    t0 = time.perf_counter()
    oracle.decode_step(x, {0: w}, 0, 1, cache, s)
    return time.perf_counter() - t0


def cpu_threads() -> int:
    for v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(v, "").isdigit():
            return int(os.environ[v])
    if hasattr(os, "sched_getaffinity"):
        return len(os.sched_getaffinity(0))
    return os.cpu_count() or 1


def run_reference(args, dist: Dist):
    """The oracle as it stands, timed on the host cores (rank 0 only). One step is a bounded
    sample of the workload: one of its blocks over the whole frame (every token, so the
    quadratic attention term is the workload's); the workload's step is that block time times
    its block count."""
    if dist.rank != 0:
        return
    wl = synth.WORKLOADS[WORKLOAD]
    M, L = wl.n_tokens, wl.prefix_layers
    for _ in range(args.warmup):
        oracle_prefill_time(M)
    t = 0.0
    for _ in range(args.steps):
        dt, _ = oracle_prefill_time(M)
        t += dt
    per_step = t / args.steps
    tok_s = M / (per_step * L)
    sample = (f"1 of {L} blocks over the full {M}-token frame per step ({per_step:.2f} s), the workload's "
              f"step taken as {L}x that (float64 numpy oracle)")
    line = {"impl": "reference", "metric": METRIC, "value": tok_s, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_step * 1e3,
            "ms_per_workload_step": per_step * L * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "blocks": L, "tokens": M, "hidden": 4096},
            "cpu_baseline": {"value": tok_s, "unit": "tokens/s", "cores": cpu_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": tok_s, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------------
# GPU arm
# ------------------------------------------------------------------------------------------
def to_dev(bits, torch):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def _traffic(kernel_key: str):
    """DRAM bytes per launch of a kernel from the committed ncu summary, if it was taken on
    the current source of that kernel (else None)."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            d = json.load(f)[kernel_key]
        src = open(os.path.join(ROOT, d["source"]), "rb").read()
        if hashlib.sha256(src).hexdigest()[:16] != d["source_sha256_16"]:
            return None
        return d["dram_bytes_per_launch"]
    except Exception:
        return None


def _dec_gateup(dstages: dict, s, D: int) -> dict | None:
    """Decode's largest kernel (gate/up GEMV + SwiGLU): weight bytes per launch over its
    average launch time in the stage-timed pass (plain launches, no graph overlap)."""
    ms, n = dstages.get("dec_gateup", (0.0, 0))
    if not n:
        return None
    f_pad = (s.ffn + 255) // 256 * 256
    nbytes = 2 * f_pad * D * 2
    us = ms / n * 1e3
    return {"kernel": "gemv_kernel<kGemvSwiGLU> (gate/up + SwiGLU)", "bytes_per_launch": nbytes,
            "avg_launch_us": us, "achieved_gbs": nbytes / (us * 1e-6) / 1e9, "traffic": _traffic("dec_gateup"),
            "timing": "stage-timed pass: plain launches, without the graph's programmatic overlap"}


def _pipeline_frames(vla, pl, xs, Mp, D, stream, choose_split, on_done=None) -> list:
    """Submits every frame as soon as a ring slot is free (split from choose_split(backlog)),
    collects them in order; returns each frame's stage times."""
    res, f = [], 0
    while len(res) < len(xs):
        while f < len(xs):
            try:
                vla.vla_pipeline_submit(pl, f, xs[f], Mp, choose_split(f - len(res)), stream)
            except vla.VlaError as e:
                if e.name != "VLA_ERR_BUSY":
                    raise
                break
            f += 1
        out = np.empty((Mp, D), dtype=np.uint16)
        fid, t = vla.vla_pipeline_collect(pl, out, 600000)
        assert fid == len(res)
        if on_done:
            on_done(t)
        res.append(t.as_dict())
    return res


def hybrid_pipeline(vla, p, s, pwl, xs, stream, seed: int, k: int, zone_min: int, torch) -> dict:
    """Frames of the pipeline workload through vla_pipeline (GPU blocks [0, k), CPU blocks
    [k, N)); per-frame T_G, T_X, T_C (Eq. 8-10) and the steady interval between frames (Eq. 13).
    Then the same frames with the split chosen per frame by the scheduler (Sec. IV-D) over the
    dynamic zone [zone_min, N], starting from zone_min + 2."""
    D, N, Mp = s.hidden, pwl.n_layers, pwl.n_tokens
    threads = cpu_threads()
    t0 = time.perf_counter()
    cfg = vla.VlaConfig(hidden=D, n_heads=s.n_heads, n_kv_heads=s.n_kv_heads, head_dim=s.head_dim, ffn=s.ffn,
                        rms_eps=s.rms_eps, rope_base=s.rope_base, max_ctx=Mp)
    cpu = vla.vla_cpu_model_create(cfg, [synth.layer_weights(s, seed, l) for l in range(zone_min, N)], zone_min,
                                   threads)
    t_create = time.perf_counter() - t0
    pl = vla.vla_pipeline_create(p, cpu, Mp, 2)
    sched = vla.vla_scheduler_create(N, zone_min, N, zone_min + 2, max_step=1, alpha=0.5)
    try:
        res = _pipeline_frames(vla, pl, xs, Mp, D, stream, lambda backlog: k)
        def choose(backlog):
            return vla.vla_scheduler_next(sched, backlog=backlog)

        sres = _pipeline_frames(vla, pl, xs + xs, Mp, D, stream, choose,
                                on_done=lambda t: vla.vla_scheduler_observe(sched, t))
        est = vla.vla_scheduler_estimates(sched)
    finally:
        vla.vla_scheduler_destroy(sched)
        vla.vla_pipeline_destroy(pl)
        vla.vla_cpu_model_destroy(cpu)
    tg = statistics.median(r["t_gpu_ms"] for r in res)
    tx = statistics.median(r["t_xfer_ms"] for r in res)
    tc = statistics.median(r["t_cpu_ms"] for r in res)
    done = [r["t_done_s"] for r in res]
    interval = statistics.median(b - a for a, b in zip(done[1:-1], done[2:])) * 1e3 if len(done) > 2 else None
    waits = [(r["t_ready_s"] - r["t_start_s"]) * 1e3 for r in res[1:]]
    block_flops = 2.0 * Mp * (s.n_heads * s.head_dim * D + 2 * s.n_kv_heads * s.head_dim * D +
                              D * s.n_heads * s.head_dim + 3 * s.ffn * D) + 2.0 * Mp * Mp * s.head_dim * s.n_heads
    sdone = [r["t_done_s"] for r in sres]
    return {"split": k, "gpu_blocks": k, "cpu_blocks": N - k, "frames": len(res), "tokens": Mp,
            "t_gpu_ms": tg, "t_xfer_ms": tx, "t_cpu_ms": tc,
            "steady_interval_ms": interval, "eq13_max_ms": max(tg, tx + tc), "eq12_serial_ms": tg + tx + tc,
            "cpu_wait_for_gpu_ms": waits,
            "cpu_suffix_gflops": block_flops * (N - k) / (tc * 1e-3) / 1e9, "cpu_threads": threads,
            "cpu_model_create_s": t_create,
            "note": "depth-2 ring; interval = median gap between consecutive frame completions after the "
                    "first two; the CPU suffix is the library's C++ block on the host cores",
            "scheduled": {"zone": [zone_min, N], "splits": [r["split"] for r in sres],
                          "interval_ms": [round((b - a) * 1e3, 3) for a, b in zip(sdone, sdone[1:])],
                          "est_ms_per_block": {"gpu": est[0], "cpu": est[1], "xfer_ms": est[2]},
                          "note": "split chosen per frame by the scheduler from observed stage times "
                                  "(at most one block per frame), no co-tenant load"}}


def run_ours(args, dist: Dist):
    import torch

    import paper_2608_14586_gb300 as vla
    torch.cuda.set_device(dist.local)
    dist.init("nccl")
    vla.build()
    vla.load()
    hbm_peak, bf16_burst, bf16_sust, peak_src = _peaks()
    wl = synth.WORKLOADS[WORKLOAD]
    dwl = synth.WORKLOADS[DECODE_WORKLOAD]
    s = wl.shape
    L = args.blocks or wl.prefix_layers
    M = wl.n_tokens
    D = s.hidden
    pwl = synth.WORKLOADS[PIPELINE_WORKLOAD]
    dec_steps = dwl.decode_steps
    pipeline_on = not args.no_pipeline and dist.world == 1
    max_ctx = max(M, dwl.prefill_ctx + dec_steps + 8, pwl.n_tokens if pipeline_on else 0)
    seed = wl.seed
    # the model holds every block of the 32-block stack when the pipeline phase runs (its
    # splits go past block 16); the prefill and decode phases use blocks [0, L)
    n_model = max(L, pwl.n_layers) if pipeline_on else L

    # ---- model: the prefix blocks (seeded synthetic weights), library-owned copies
    layers = []
    for l in range(n_model):
        layers.append({k: to_dev(v, torch) for k, v in synth.layer_weights(s, seed, l).items()})
    cfg = vla.VlaConfig(hidden=D, n_heads=s.n_heads, n_kv_heads=s.n_kv_heads, head_dim=s.head_dim, ffn=s.ffn,
                        rms_eps=s.rms_eps, rope_base=s.rope_base, max_ctx=max_ctx)
    p = vla.vla_prefix_create(cfg, layers)
    del layers
    torch.cuda.empty_cache()
    kv = vla.vla_kv_create(p, 0, L, max_ctx)

    xb = synth.hidden_states(M, D, seed, wl.visual_tokens, wl.visual_scale)
    x = to_dev(xb, torch)
    outs = [torch.empty((M, D), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    pinned = [torch.empty((M, D), dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    main = torch.cuda.current_stream()
    side = torch.cuda.Stream()
    ready = [torch.cuda.Event() for _ in range(2)]
    done = [torch.cuda.Event() for _ in range(2)]
    for e in done:
        e.record(side)
    launches = [0]

    def step(i: int, x_in):
        b = i & 1
        main.wait_event(done[b])                   # frame i-2's copy of this buffer has landed
        vla.vla_kv_reset(kv, main)                  # a new frame starts at position 0
        vla.vla_prefix_prefill(p, x_in, M, 0, L, kv, outs[b], main)
        launches[0] += vla.vla_last_launch_count(p) + 1
        ready[b].record(main)
        vla.vla_boundary_to_host(outs[b], M, D, pinned[b], side, ready[b], done[b])

    for i in range(args.warmup):
        step(i, x)
    torch.cuda.synchronize()

    gpu_id = os.environ.get("CUDA_VISIBLE_DEVICES", str(dist.local)).split(",")[0] \
        if dist.world == 1 else str(dist.local)
    clocks = ClockSampler(gpu_id)
    clocks.start()
    # ---- timed region: events bracket only the dominant kernel (gate/up GEMM)
    dist.barrier()
    torch.cuda.synchronize()
    launches[0] = 0
    vla.vla_prefix_stage_times(p)
    vla.vla_prefix_set_timing(p, ["gemm_gateup"])
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_start.record(main)
    for i in range(args.steps):
        step(i, x)
    main.wait_event(done[(args.steps - 1) & 1])
    t_end.record(main)
    torch.cuda.synchronize()
    vla.vla_prefix_set_timing(p, ())
    dist.barrier()
    ms = t_start.elapsed_time(t_end) / args.steps
    ms = dist.max(ms, "cuda")
    gu_ms, gu_n = vla.vla_prefix_stage_times(p)["gemm_gateup"]
    prefill_launches = launches[0]
    assert vla.vla_last_async_error(p) == 0

    # ---- diagnostic pass (not the timed region): every stage's average launch time
    vla.vla_prefix_set_timing(p, "all")
    for i in range(max(3, args.steps // 4)):
        step(i, x)
    torch.cuda.synchronize()
    vla.vla_prefix_set_timing(p, ())
    stages = vla.vla_prefix_stage_times(p)

    # roofline of the dominant kernel: gate/up projection + SwiGLU (51% of the GEMM flops)
    gu_flops = 2.0 * M * (2 * s.ffn) * D
    gu_tflops = gu_flops / (gu_ms / gu_n * 1e-3) / 1e12 if gu_n else 0.0
    block_flops = 2.0 * M * (s.n_heads * s.head_dim * D + 2 * s.n_kv_heads * s.head_dim * D +
                             D * s.n_heads * s.head_dim + 3 * s.ffn * D) + 2.0 * M * M * s.head_dim * s.n_heads
    step_tflops = block_flops * L / (ms * 1e-3) / 1e12

    # ---- end to end through the C ABI with host buffers (H2D of the frame, D2H of h^(k)), as a
    # streaming loop runs it: each step's frame goes up on its own stream while the previous
    # step computes (two device input buffers), and each result comes back on a side stream
    e2e = None
    if not args.no_e2e:
        host_in = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).pin_memory()
        x_devs = [torch.empty_like(x) for _ in range(2)]
        up = torch.cuda.Stream()
        in_ready = [torch.cuda.Event() for _ in range(2)]
        in_free = [torch.cuda.Event() for _ in range(2)]

        def upload(i):  # frame of step i into x_devs[i & 1], once the prefill that read it is done
            b = i & 1
            if i >= 2:
                up.wait_event(in_free[b])
            vla.vla_frame_to_device(host_in, M, D, x_devs[b], up)
            in_ready[b].record(up)

        def e2e_step(i):
            b = i & 1
            upload(i + 1)  # the next step's frame overlaps this step's compute
            main.wait_event(in_ready[b])
            main.wait_event(done[b])
            vla.vla_kv_reset(kv, main)
            vla.vla_prefix_prefill(p, x_devs[b], M, 0, L, kv, outs[b], main)
            in_free[b].record(main)
            ready[b].record(main)
            vla.vla_boundary_to_host(outs[b], M, D, pinned[b], side, ready[b], done[b])

        upload(0)
        for i in range(args.warmup):
            e2e_step(i)
        torch.cuda.synchronize()
        dist.barrier()
        t0 = time.perf_counter()
        for i in range(args.warmup, args.warmup + args.steps):  # one upload and one download per step
            e2e_step(i)
        done[(args.warmup + args.steps - 1) & 1].synchronize()
        torch.cuda.synchronize()
        e2e_ms = (time.perf_counter() - t0) * 1e3 / args.steps
        e2e_ms = dist.max(e2e_ms, "cuda")
        # the boundary that reached the host equals the device result
        last = (args.warmup + args.steps - 1) & 1
        assert torch.equal(pinned[last].view(torch.int16).cpu(), outs[last].view(torch.int16).cpu())
        e2e = {"value": M * dist.world / (e2e_ms * 1e-3), "unit": "tokens/s", "ms_per_step": e2e_ms,
               "h2d_bytes_per_step": M * D * 2, "d2h_bytes_per_step": M * D * 2}

    # ---- latency until one frame's boundary h^(16) is in host memory: the prefix followed by
    # a device-to-host copy, vs the prefix whose last epilogue stores it to the host itself
    boundary = None
    if not args.no_e2e:
        hb = torch.empty((M, D), dtype=torch.bfloat16).pin_memory()

        def frame_to_host(fused: bool) -> float:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(main)
            vla.vla_kv_reset(kv, main)
            if fused:
                vla.vla_prefix_prefill_to_host(p, x, M, 0, L, kv, outs[0], hb, main)
            else:
                vla.vla_prefix_prefill(p, x, M, 0, L, kv, outs[0], main)
                vla.vla_boundary_to_host(outs[0], M, D, hb, main)
            e1.record(main)
            torch.cuda.synchronize()
            return e0.elapsed_time(e1)

        lat = {}
        for fused in (False, True):
            for _ in range(2):
                frame_to_host(fused)
            lat[fused] = statistics.median(frame_to_host(fused) for _ in range(max(5, args.steps // 3)))
            assert torch.equal(hb.view(torch.int16), outs[0].view(torch.int16).cpu())
        boundary = {"bytes": M * D * 2, "prefix_then_copy_ms": lat[False], "fused_store_ms": lat[True],
                    "note": "one frame, from launch until h^(16) is in page-locked host memory (median)"}

    # ---- decode: 64 single-token steps against a 2304-position random context, in a cache
    # sized for the workload (2304 + 64 steps)
    decode = None
    if not args.no_decode:
        ctx0 = dwl.prefill_ctx
        vla.vla_kv_destroy(kv)
        max_ctx = ctx0 + dec_steps + 8
        kv = vla.vla_kv_create(p, 0, L, max_ctx)
        for l in range(L):
            kb, vb = synth.random_kv(ctx0, s, dwl.seed, l)
            kp, vp = vla.vla_kv_data(kv, l)
            for ptr, bits in ((kp, kb), (vp, vb)):
                src = to_dev(bits, torch)  # [Hkv, ctx0, dh] -> rows of the [Hkv, max_ctx, dh] plane
                for g in range(s.n_kv_heads):
                    dst = _dev_view(ptr + g * max_ctx * s.head_dim * 2, ctx0 * s.head_dim, torch)
                    dst.copy_(src[g].reshape(-1))
        torch.cuda.synchronize()
        xd = to_dev(np.stack([synth.decode_hidden(t, D, dwl.seed)[0] for t in range(dec_steps)]), torch)
        yd = torch.empty((1, D), dtype=torch.bfloat16, device="cuda")

        def decode_run():
            vla.vla_kv_set_length(kv, ctx0, main)
            n = 1
            for t in range(dec_steps):
                vla.vla_prefix_decode(p, xd[t:t + 1], 0, L, kv, yd, main)
                n += vla.vla_last_launch_count(p)
            return n

        for _ in range(max(1, args.warmup // 2)):
            decode_run()
        torch.cuda.synchronize()
        dist.barrier()
        d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        d0.record(main)
        reps = max(1, args.steps // 8)
        dec_launches = 0
        for _ in range(reps):
            dec_launches += decode_run()
        d1.record(main)
        torch.cuda.synchronize()
        dist.barrier()
        dec_us = d0.elapsed_time(d1) * 1e3 / (reps * dec_steps)
        dec_us = dist.max(dec_us, "cuda")
        assert vla.vla_last_async_error(p) == 0
        vla.vla_prefix_set_timing(p, "all")
        decode_run()
        torch.cuda.synchronize()
        vla.vla_prefix_set_timing(p, ())
        dstages = vla.vla_prefix_stage_times(p)
        # batched decode: B sequences with the same 2304-position context, one step each per
        # launch of the whole range (the weights streamed once for the batch)
        batched = []
        extra = [vla.vla_kv_create(p, 0, L, max_ctx) for _ in range(3)]
        for kvb in extra:
            for l in range(L):
                src_k, src_v = vla.vla_kv_data(kv, l)
                dst_k, dst_v = vla.vla_kv_data(kvb, l)
                n = s.n_kv_heads * max_ctx * s.head_dim
                _dev_view(dst_k, n, torch).copy_(_dev_view(src_k, n, torch))
                _dev_view(dst_v, n, torch).copy_(_dev_view(src_v, n, torch))
        torch.cuda.synchronize()
        for B in (2, 4):
            kvs = [kv] + extra[:B - 1]
            xb_dev = to_dev(np.concatenate([synth.decode_hidden(t, D, dwl.seed + b) for b in range(B)
                                            for t in range(1)], axis=0), torch)
            yb_dev = torch.empty_like(xb_dev)

            def batch_run():
                for k in kvs:
                    vla.vla_kv_set_length(k, ctx0, main)
                for t in range(dec_steps):
                    vla.vla_prefix_decode_batch(p, xb_dev, 0, L, kvs, yb_dev, main)

            batch_run()
            torch.cuda.synchronize()
            b0, b1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            b0.record(main)
            for _ in range(reps):
                batch_run()
            b1.record(main)
            torch.cuda.synchronize()
            us = b0.elapsed_time(b1) * 1e3 / (reps * dec_steps)
            batched.append({"batch": B, "us_per_step": us, "tokens_per_s": B / (us * 1e-6),
                            "speedup_vs_batch1": B * dec_us / us})
        assert vla.vla_last_async_error(p) == 0
        for kvb in extra:
            vla.vla_kv_destroy(kvb)
        weight_bytes = L * 2 * (s.n_heads * s.head_dim * D + 2 * s.n_kv_heads * s.head_dim * D +
                                D * s.n_heads * s.head_dim + 3 * s.ffn * D)
        avg_ctx = ctx0 + (dec_steps + 1) / 2
        kv_bytes = L * 2 * s.n_kv_heads * s.head_dim * 2 * avg_ctx
        dec_bytes = weight_bytes + kv_bytes
        dec_gbs = dec_bytes / (dec_us * 1e-6) / 1e9
        decode = {"workload": DECODE_WORKLOAD, "blocks": L, "us_per_step": dec_us, "bytes_per_step": dec_bytes,
                  "attention_plan": vla.vla_kv_decode_plan(kv),
                  "hbm_gbs": dec_gbs,
                  "roofline": {"bound": "hbm", "achieved": dec_gbs, "peak": hbm_peak, "unit": "GB/s",
                               "frac": dec_gbs / hbm_peak, "peak_source": f"{peak_src} copy bandwidth",
                               "traffic": None},
                  "dominant_kernel": _dec_gateup(dstages, s, D),
                  "batched": batched,
                  "gpu_launches_per_step": dec_launches / (reps * dec_steps),
                  "stages_us_per_launch": {k: round(v[0] / v[1] * 1e3, 2) for k, v in dstages.items() if v[1]}}
    # ---- one 7B block over a 1024-token frame (768 visual rows at 2x scale + 256 text rows)
    block1k = None
    if not args.no_block1k:
        bwl = synth.WORKLOADS[BLOCK_WORKLOAD]
        Mb = bwl.n_tokens
        xb1 = to_dev(synth.hidden_states(Mb, D, bwl.seed, bwl.visual_tokens, bwl.visual_scale), torch)
        yb1 = torch.empty_like(xb1)
        kv1 = vla.vla_kv_create(p, 0, 1, Mb)

        def one_block():
            vla.vla_kv_reset(kv1, main)
            vla.vla_prefix_prefill(p, xb1, Mb, 0, 1, kv1, yb1, main)

        for _ in range(args.warmup):
            one_block()
        torch.cuda.synchronize()
        # back-to-back frames: the block's 354 MB of weights exceed L2, so each frame streams
        # them from HBM again (no flush needed)
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(max(10, args.steps) + 1)]
        evs[0].record(main)
        for i in range(1, len(evs)):
            one_block()
            evs[i].record(main)
        torch.cuda.synchronize()
        times = [evs[i - 1].elapsed_time(evs[i]) for i in range(1, len(evs))]
        assert vla.vla_last_async_error(p) == 0
        vla.vla_kv_destroy(kv1)
        b_ms = statistics.median(times)
        b_flops = 2.0 * Mb * (s.n_heads * s.head_dim * D + 2 * s.n_kv_heads * s.head_dim * D +
                              D * s.n_heads * s.head_dim + 3 * s.ffn * D) + 2.0 * Mb * Mb * s.head_dim * s.n_heads
        block1k = {"workload": BLOCK_WORKLOAD, "tokens": Mb, "us_per_frame": b_ms * 1e3, "tokens_per_s": Mb / (b_ms * 1e-3),
                   "tflops": b_flops / (b_ms * 1e-3) / 1e12, "frac_of_peak": b_flops / (b_ms * 1e-3) / 1e12 / bf16_burst,
                   "peak": bf16_burst, "peak_source": f"{peak_src} bf16 burst (a single block timed alone)",
                   "timing": "median of per-frame CUDA events over back-to-back frames; weights 354 MB > L2"}

    # ---- pipeline (4 frames x 3072 tokens; prefix [0, k) of a 32-block stack for k = 8/16/24):
    # frame t's boundary copy runs on the side stream under frame t+1's prefix
    pipeline = None
    if pipeline_on:
        Mp = pwl.n_tokens
        kvp = vla.vla_kv_create(p, 0, pwl.n_layers, Mp)
        xs = [to_dev(synth.hidden_states(Mp, D, f, pwl.visual_tokens, pwl.visual_scale), torch)
              for f in range(pwl.frames)]
        hp = [torch.empty((Mp, D), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
        pp = [torch.empty((Mp, D), dtype=torch.bfloat16).pin_memory() for _ in range(2)]
        frame_flops = 2.0 * Mp * (s.n_heads * s.head_dim * D + 2 * s.n_kv_heads * s.head_dim * D +
                                  D * s.n_heads * s.head_dim + 3 * s.ffn * D) + 2.0 * Mp * Mp * s.head_dim * s.n_heads
        splits = []
        for k in PIPELINE_SPLITS:
            def frames(copy: bool):
                for f in range(pwl.frames):
                    b = f & 1
                    main.wait_event(done[b])
                    vla.vla_kv_reset(kvp, main)
                    vla.vla_prefix_prefill(p, xs[f], Mp, 0, k, kvp, hp[b], main)
                    if copy:
                        ready[b].record(main)
                        vla.vla_boundary_to_host(hp[b], Mp, D, pp[b], side, ready[b], done[b])

            frames(True)
            torch.cuda.synchronize()
            res = {}
            for copy in (False, True):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(main)
                frames(copy)
                if copy:
                    main.wait_event(done[(pwl.frames - 1) & 1])
                e1.record(main)
                torch.cuda.synchronize()
                res[copy] = e0.elapsed_time(e1) / pwl.frames
            assert torch.equal(pp[(pwl.frames - 1) & 1].view(torch.int16).cpu(),
                               hp[(pwl.frames - 1) & 1].view(torch.int16).cpu())
            tf = frame_flops * k / (res[False] * 1e-3) / 1e12
            splits.append({"k": k, "ms_per_frame": res[True], "prefix_only_ms_per_frame": res[False],
                           "copy_exposed_ms_per_frame": res[True] - res[False], "tflops": tf,
                           "frac_of_peak": tf / bf16_burst, "frac_of_sustained": tf / bf16_sust,
                           "boundary_bytes": Mp * D * 2})
        assert vla.vla_last_async_error(p) == 0
        vla.vla_kv_destroy(kvp)
        pipeline = {"workload": PIPELINE_WORKLOAD, "frames": pwl.frames, "tokens": Mp, "blocks_total": pwl.n_layers,
                    "note": "wall time per frame of the GPU prefix with the boundary copy to pinned host memory "
                            "overlapped on a side stream, vs the prefix alone",
                    "splits": splits}

        # ---- hybrid pipeline (Sec. IV-C, Eq. 12-14): GPU prefix [0, k) of frame t+1 while the
        # host cores run the suffix [k, 32) of frame t, frames handed over in order
        if not args.no_hybrid:
            try:
                pipeline["hybrid"] = hybrid_pipeline(vla, p, s, pwl, xs, main, seed, HYBRID_SPLIT, HYBRID_ZONE_MIN,
                                                     torch)
            except Exception as e:  # the GPU-only figures above stand; the line says what failed
                pipeline["hybrid"] = {"error": f"{type(e).__name__}: {e}"}
    clock_info = clocks.stop()

    # ---- CPU oracle baseline (rank 0, N = 1 only): 1 block over the whole 2304-token frame
    cpu = None
    if dist.rank == 0 and dist.world == 1 and not args.no_cpu_baseline and decode is not None:
        t_dec = oracle_decode_time(dwl)
        decode["cpu_baseline"] = {"value": t_dec * L * 1e6, "unit": "us/step", "cores": cpu_threads(),
                                  "kind": "oracle",
                                  "sample": f"one decode step of 1 of {L} blocks at context {dwl.prefill_ctx} "
                                            f"({t_dec:.2f} s), extrapolated x{L}; float64 numpy oracle"}
    if dist.rank == 0 and dist.world == 1 and not args.no_cpu_baseline:
        t_cpu, _ = oracle_prefill_time(M)
        cpu = {"value": M / (t_cpu * L), "unit": "tokens/s", "cores": cpu_threads(), "kind": "oracle",
               "sample": f"1 of {L} blocks over the full {M}-token frame ({t_cpu:.1f} s), extrapolated x{L} "
                         f"blocks; float64 numpy oracle"}

    if dist.rank == 0:
        tok_s = M * dist.world / (ms * 1e-3)
        line = {
            "metric": METRIC, "value": tok_s, "unit": "tokens/s", "n_gpus": dist.world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": WORKLOAD if L == wl.prefix_layers else f"{WORKLOAD} ({L} blocks)",
                       "blocks": L, "tokens": M, "hidden": D,
                       "heads": f"{s.n_heads}q/{s.n_kv_heads}kv x {s.head_dim}", "ffn": s.ffn,
                       "boundary_bytes": M * D * 2, "l2": "weights 5.67 GB streamed per step > 129 MB L2",
                       "parallelism": f"replicas x{dist.world}"},
            "roofline": {"kernel": "gemm_gateup (tcgen05, SwiGLU epilogue)", "bound": "tensor",
                         "achieved": gu_tflops, "peak": bf16_burst, "unit": "TFLOP/s", "frac": gu_tflops / bf16_burst,
                         "peak_source": f"{peak_src} bf16 burst (the timed region is well under a second)",
                         "peak_sustained": bf16_sust, "frac_of_sustained": gu_tflops / bf16_sust,
                         "traffic": _traffic("gemm_gateup"),
                         "flops_per_launch": gu_flops, "avg_launch_ms": gu_ms / max(gu_n, 1)},
            "step_tflops": step_tflops, "step_frac_of_peak": step_tflops / bf16_burst,
            "step_frac_of_sustained": step_tflops / bf16_sust,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": prefill_launches,
            "clocks": clock_info,
            "stages_ms_per_launch": {k: round(v[0] / v[1], 4) for k, v in stages.items() if v[1]},
            "decode": decode,
            "pipeline": pipeline,
            "block_1024": block1k,
            "boundary": boundary,
        }
        line["summary"] = _summary(line, stages, s, M, D, bf16_burst, hbm_peak)
        print(json.dumps(line), flush=True)
    vla.vla_kv_destroy(kv)
    vla.vla_prefix_destroy(p)
    dist.close()


def _summary(line: dict, stages: dict, s, M: int, D: int, bf16_burst: float, hbm_peak: float) -> dict:
    """The headline figures again, short, as the JSON line's last key (a log that keeps only
    the end of the line still shows them)."""
    r = line["roofline"]
    out = {"prefill": {"tokens_s": round(line["value"]), "ms_step": round(line["ms_per_step"], 3),
                       "gateup_frac_burst": round(r["frac"], 3), "step_frac_burst": round(line["step_frac_of_peak"], 3)}}
    attn = stages.get("attn_prefill")
    if attn and attn[1]:
        ms = attn[0] / attn[1]
        fl = 2.0 * M * M * s.head_dim * s.n_heads
        out["prefill"]["attn_us"] = round(ms * 1e3, 1)
        out["prefill"]["attn_frac_burst"] = round(fl / (ms * 1e-3) / 1e12 / bf16_burst, 3)
    for name in ("gemm_qkv", "gemm_o", "gemm_down"):
        st = stages.get(name)
        if st and st[1]:
            out["prefill"][name + "_us"] = round(st[0] / st[1] * 1e3, 1)
    d = line.get("decode")
    if d:
        out["decode"] = {"us_step": round(d["us_per_step"], 1), "hbm_gbs": round(d["hbm_gbs"]),
                         "frac_hbm": round(d["hbm_gbs"] / hbm_peak, 3),
                         "attn_us": d["stages_us_per_launch"].get("dec_attn")}
    b = line.get("block_1024")
    if b:
        out["block_1024"] = {"us": round(b["us_per_frame"], 1), "frac_burst": round(b["frac_of_peak"], 3)}
    pl = line.get("pipeline")
    if pl:
        out["pipeline_ms_per_frame"] = {str(x["k"]): round(x["ms_per_frame"], 2) for x in pl["splits"]}
    if line.get("e2e"):
        out["e2e_tokens_s"] = round(line["e2e"]["value"])
    c = line.get("clocks")
    if c:
        out["clocks"] = {"sm_mhz": c["sm_mhz"], "reasons": c["reasons"]}
    return out


class _CudaArray:
    def __init__(self, ptr: int, numel: int):
        self.__cuda_array_interface__ = {"data": (int(ptr), False), "shape": (int(numel),), "typestr": "<i2",
                                         "strides": None, "version": 3}


def _dev_view(ptr, numel, torch):
    return torch.as_tensor(_CudaArray(ptr, numel), device="cuda").view(torch.bfloat16)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--blocks", type=int, default=0, help="prefix depth (default: the workload's 16)")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-pipeline", action="store_true")
    ap.add_argument("--no-block1k", action="store_true")
    ap.add_argument("--no-hybrid", action="store_true", help="skip the GPU prefix + CPU suffix pipeline")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    dist = Dist()
    if args.impl == "reference":
        run_reference(args, dist)
    else:
        run_ours(args, dist)


if __name__ == "__main__":
    main()
