"""Per-stage timing of the prefix library on seeded synthetic 7B-class blocks.

    python -m paper_2608_14586_gb300.profile prefill --blocks 1 --tokens 2304 --steps 3
    python -m paper_2608_14586_gb300.profile decode --blocks 2 --ctx 2304 --steps 4

Stage timing (vla_prefix_set_timing) launches every kernel directly on the stream with an
event pair around it (decode then runs without its captured graph and without programmatic
dependent launch), so each launch is a separate, individually profiled kernel; the printed
numbers are per-launch averages of the timed stages.
"""
from __future__ import annotations

import argparse
import json

import numpy as np

import synth

from . import (VlaConfig, build, load, vla_kv_create, vla_kv_data, vla_kv_decode_plan, vla_kv_destroy,
               vla_kv_set_length,
               vla_last_async_error, vla_prefix_create, vla_prefix_decode, vla_prefix_destroy, vla_prefix_prefill,
               vla_prefix_set_timing, vla_prefix_stage_times)


def _dev(bits, torch):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("mode", choices=("prefill", "decode"))
    ap.add_argument("--blocks", type=int, default=1)
    ap.add_argument("--tokens", type=int, default=2304, help="prefill tokens per call")
    ap.add_argument("--ctx", type=int, default=2304, help="decode: pre-filled context positions")
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--seed", type=int, default=0)
    a = ap.parse_args(argv)
    import torch
    build()
    load()
    s = synth.B7
    max_ctx = a.tokens if a.mode == "prefill" else a.ctx + a.steps + 8
    layers = [{k: _dev(v, torch) for k, v in synth.layer_weights(s, a.seed, l).items()} for l in range(a.blocks)]
    cfg = VlaConfig(hidden=s.hidden, n_heads=s.n_heads, n_kv_heads=s.n_kv_heads, head_dim=s.head_dim, ffn=s.ffn,
                    rms_eps=s.rms_eps, rope_base=s.rope_base, max_ctx=max_ctx)
    p = vla_prefix_create(cfg, layers)
    del layers
    kv = vla_kv_create(p, 0, a.blocks, max_ctx)
    try:
        vla_prefix_set_timing(p, "all")
        if a.mode == "prefill":
            x = _dev(synth.hidden_states(a.tokens, s.hidden, a.seed), torch)
            y = torch.empty_like(x)
            for _ in range(a.steps):
                vla_kv_set_length(kv, 0)
                vla_prefix_prefill(p, x, a.tokens, 0, a.blocks, kv, y)
        else:
            for l in range(a.blocks):
                kb, vb = synth.random_kv(a.ctx, s, a.seed, l)
                kp, vp = vla_kv_data(kv, l)
                for ptr, bits in ((kp, kb), (vp, vb)):
                    src = _dev(bits, torch)
                    for g in range(s.n_kv_heads):
                        n = a.ctx * s.head_dim
                        dst = torch.as_tensor(_Raw(ptr + g * max_ctx * s.head_dim * 2, n), device="cuda")
                        dst.copy_(src[g].reshape(-1).view(torch.int16))
            torch.cuda.synchronize()
            vla_kv_set_length(kv, a.ctx)
            y = torch.empty((1, s.hidden), dtype=torch.bfloat16, device="cuda")
            for t in range(a.steps):
                vla_prefix_decode(p, _dev(synth.decode_hidden(t, s.hidden, a.seed), torch), 0, a.blocks, kv, y)
        torch.cuda.synchronize()
        vla_prefix_set_timing(p, ())
        if vla_last_async_error(p) != 0:
            raise RuntimeError("device-side timeout reported")
        times = vla_prefix_stage_times(p)
        print(json.dumps({"mode": a.mode, "blocks": a.blocks, "steps": a.steps, "attention_plan": vla_kv_decode_plan(kv),
                          "us_per_launch": {k: round(v[0] / v[1] * 1e3, 2) for k, v in times.items() if v[1]},
                          "launches": {k: v[1] for k, v in times.items() if v[1]}}))
    finally:
        vla_kv_destroy(kv)
        vla_prefix_destroy(p)


class _Raw:
    def __init__(self, ptr: int, numel: int):
        self.__cuda_array_interface__ = {"data": (int(ptr), False), "shape": (int(numel),), "typestr": "<i2",
                                         "strides": None, "version": 3}


if __name__ == "__main__":
    main()
