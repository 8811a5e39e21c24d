"""The cross-frame asynchronous pipeline of Sec. IV-C (include/vla_cpu.h): the GPU prefix
[0, p) of frame t+1 overlaps the CPU suffix [p, N) of frame t; frames come out in order with
their ids; each frame may use its own split point. Outputs equal the hand-composed path
(GPU prefill, boundary copy, CPU prefill) bit for bit and the float64 oracle within the
block tolerance."""
import numpy as np
import pytest

import oracle
import synth
from helpers import COS_FINAL, REL_L2_BLOCK, Model, cos_sim, rel_l2, sync, to_dev, vla_cfg

pytestmark = pytest.mark.gpu


def _bits(t):
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _composed(vla, m, cpu, x, M, split, L, max_ctx):
    """GPU [0, split) -> host bits -> CPU [split, L), with fresh caches."""
    import torch
    kv = vla.vla_kv_create(m.handle, 0, L, max_ctx)
    h = torch.empty_like(x)
    vla.vla_prefix_prefill(m.handle, x, M, 0, split, kv if split else None, h)
    sync()
    hb = _bits(h)
    vla.vla_kv_destroy(kv)
    _, c0, _ = vla.vla_cpu_model_info(cpu)
    ckv = vla.vla_cpu_kv_create(cpu, c0, L, max_ctx)
    y = np.empty_like(hb)
    vla.vla_cpu_prefill(cpu, hb, M, split, L, ckv, y)
    vla.vla_cpu_kv_destroy(ckv)
    return y


def _run_frames(vla, pl, xs, M, splits, stream):
    """Submits every frame as soon as a slot is free; returns [(frame_id, y, times)]."""
    out, f = [], 0
    while len(out) < len(xs):
        while f < len(xs):
            try:
                vla.vla_pipeline_submit(pl, 100 + f, xs[f], M, splits[f], stream)
            except vla.VlaError as e:
                assert e.name == "VLA_ERR_BUSY"
                break
            f += 1
        y = np.empty((M, xs[0].shape[1]), dtype=np.uint16)
        fid, t = vla.vla_pipeline_collect(pl, y, 120000)
        out.append((fid, y, t.as_dict()))
    return out


def test_tiny_pipeline_per_frame_split_matches_oracle(vla_lib):
    vla = vla_lib
    import torch
    s, L, M, max_ctx = synth.TINY, 3, 64, 64
    splits = [1, 2, 3, 1, 2]
    m = Model(s, L, 4, max_ctx, gain="random")
    cpu = vla.vla_cpu_model_create(vla_cfg(s, max_ctx), m.bits[1:], 1, 4)
    try:
        xb = [synth.hidden_states(M, s.hidden, 40 + f) for f in range(len(splits))]
        xs = [to_dev(b) for b in xb]
        stream = torch.cuda.current_stream()
        pl = vla.vla_pipeline_create(m.handle, cpu, M, 2)
        try:
            res = _run_frames(vla, pl, xs, M, splits, stream)
            assert vla.vla_pipeline_in_flight(pl) == 0
        finally:
            vla.vla_pipeline_destroy(pl)
        assert [r[0] for r in res] == [100 + f for f in range(len(splits))]
        for f, (fid, y, t) in enumerate(res):
            assert t["split"] == splits[f] and t["n_tokens"] == M
            assert t["t_submit_s"] <= t["t_ready_s"] <= t["t_done_s"] and t["t_start_s"] <= t["t_ready_s"]
            np.testing.assert_array_equal(y, _composed(vla, m, cpu, xs[f], M, splits[f], L, max_ctx))
            cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)
            ref = oracle.prefix_forward(oracle.bf16_to_f64(xb[f]), m.weights64(), 0, L, cache, s)
            got = oracle.bf16_to_f64(y)
            assert rel_l2(got, ref) < REL_L2_BLOCK
            assert cos_sim(got, ref) > COS_FINAL
        # a pipeline destroyed with frames in flight finishes them first and frees everything
        pl = vla.vla_pipeline_create(m.handle, cpu, M, 3)
        for f in range(3):
            vla.vla_pipeline_submit(pl, f, xs[f], M, splits[f], stream)
        assert vla.vla_pipeline_in_flight(pl) == 3
        vla.vla_pipeline_destroy(pl)
        sync()
        assert vla.vla_last_async_error(m.handle) == 0
    finally:
        vla.vla_cpu_model_destroy(cpu)
        m.close()


def test_7b_pipeline_overlaps_gpu_prefix_with_cpu_suffix(vla_lib):
    """Four 512-token frames through a 4-block 7B-class stack, CPU holding blocks [2, 4):
    splits 3, 2, 4, 3. The GPU prefix and boundary copy of frame t+1 run while the CPU still
    runs frame t's suffix; a full ring refuses a submit with BUSY."""
    vla = vla_lib
    import torch
    s, L, M = synth.B7, 4, 512
    splits = [3, 2, 4, 3]
    m = Model(s, L, 6, M)
    cpu = vla.vla_cpu_model_create(vla_cfg(s, M), m.bits[2:], 2, 0)
    try:
        xs = [to_dev(synth.hidden_states(M, s.hidden, 60 + f, 448, 1.0)) for f in range(len(splits))]
        stream = torch.cuda.current_stream()
        pl = vla.vla_pipeline_create(m.handle, cpu, M, 2)
        try:
            vla.vla_pipeline_submit(pl, 7, xs[0], M, splits[0], stream)
            vla.vla_pipeline_submit(pl, 8, xs[1], M, splits[1], stream)
            with pytest.raises(vla.VlaError) as ei:
                vla.vla_pipeline_submit(pl, 9, xs[2], M, splits[2], stream)
            assert ei.value.name == "VLA_ERR_BUSY"
            with pytest.raises(vla.VlaError) as ei:
                vla.vla_pipeline_submit(pl, 9, xs[2], M, 1, stream)  # below the CPU model's first block
            assert ei.value.name == "VLA_ERR_RANGE"
            # frame 7's suffix (one CPU block over 512 tokens) is far from done right after submit
            with pytest.raises(vla.VlaError) as ei:
                vla.vla_pipeline_collect(pl, None, 0)
            assert ei.value.name == "VLA_ERR_TIMEOUT"
            assert vla.vla_pipeline_in_flight(pl) == 2  # a timed-out collect leaves the frame queued
            res = []
            for _ in range(2):
                y = np.empty((M, s.hidden), dtype=np.uint16)
                fid, t = vla.vla_pipeline_collect(pl, y, 120000)
                res.append((fid, y, t.as_dict()))
            rest = _run_frames(vla, pl, xs[2:], M, splits[2:], stream)
        finally:
            vla.vla_pipeline_destroy(pl)
        assert [r[0] for r in res] == [7, 8] and [r[0] for r in rest] == [100, 101]
        ys = [r[1] for r in res] + [r[1] for r in rest]
        times = [r[2] for r in res] + [r[2] for r in rest]
        # frame 1 was enqueued before frame 0's suffix finished, and its prefix and boundary
        # copy ran under that suffix: the CPU stage took frame 1 up without waiting for the GPU
        assert times[1]["t_submit_s"] < times[0]["t_done_s"]
        assert times[1]["t_ready_s"] - times[1]["t_start_s"] < 0.05
        assert times[0]["t_cpu_ms"] > 20 * times[1]["t_gpu_ms"]
        for t in times:
            assert t["t_gpu_ms"] > 0 and t["t_cpu_ms"] >= 0 and t["t_xfer_ms"] >= 0
        for f in range(len(splits)):
            np.testing.assert_array_equal(ys[f], _composed(vla, m, cpu, xs[f], M, splits[f], L, M))
        # CPU and GPU arithmetic agree to rounding: the all-GPU frame against a 2-block CPU suffix
        kv = vla.vla_kv_create(m.handle, 0, L, M)
        yg = torch.empty_like(xs[1])
        vla.vla_prefix_prefill(m.handle, xs[1], M, 0, L, kv, yg)
        sync()
        vla.vla_kv_destroy(kv)
        g = oracle.bf16_to_f64(_bits(yg))
        assert rel_l2(oracle.bf16_to_f64(ys[1]), g) < REL_L2_BLOCK
        assert vla.vla_last_async_error(m.handle) == 0
    finally:
        vla.vla_cpu_model_destroy(cpu)
        m.close()


def test_scheduler_drives_the_split_of_the_pipeline(vla_lib):
    """Phi (Sec. IV-D) on the live pipeline: from observed stage times it moves the boundary
    one block per frame toward the cheaper side, here the GPU (a tiny block costs the host
    cores far more than the GPU), and stops at the zone's end; every frame stays correct."""
    vla = vla_lib
    import torch
    s, L, M, max_ctx = synth.TINY, 3, 64, 64
    m = Model(s, L, 8, max_ctx)
    cpu = vla.vla_cpu_model_create(vla_cfg(s, max_ctx), m.bits[1:], 1, 2)
    sched = vla.vla_scheduler_create(L, 1, L, 1, max_step=1, alpha=1.0)
    try:
        xs = [to_dev(synth.hidden_states(M, s.hidden, 80 + f)) for f in range(5)]
        stream = torch.cuda.current_stream()
        pl = vla.vla_pipeline_create(m.handle, cpu, M, 1)  # depth 1: each split sees the last frame
        splits = []
        try:
            for f in range(5):
                k = vla.vla_scheduler_next(sched)
                splits.append(k)
                vla.vla_pipeline_submit(pl, f, xs[f], M, k, stream)
                y = np.empty((M, s.hidden), dtype=np.uint16)
                fid, t = vla.vla_pipeline_collect(pl, y, 120000)
                assert fid == f
                vla.vla_scheduler_observe(sched, t)
                np.testing.assert_array_equal(y, _composed(vla, m, cpu, xs[f], M, k, L, max_ctx))
        finally:
            vla.vla_pipeline_destroy(pl)
        assert splits == [1, 2, 3, 3, 3], splits  # no move before the first observation
        g_ms, c_ms, _ = vla.vla_scheduler_estimates(sched)
        assert 0 < g_ms < c_ms
    finally:
        vla.vla_scheduler_destroy(sched)
        vla.vla_cpu_model_destroy(cpu)
        m.close()
