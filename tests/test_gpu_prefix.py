"""Block-range parity of vla_prefix_prefill / vla_prefix_decode against the float64 oracle,
and the partition identity of Eq. 6 on the GPU."""
import numpy as np
import pytest

import oracle
import synth
from helpers import sync, COS_FINAL, REL_L2_BLOCK, Model, cos_sim, from_dev, kv_planes, rel_l2, to_dev

pytestmark = pytest.mark.gpu


def _kv_planes(vla, kv, layer, shape, max_ctx, n):
    """(K, V) float64 [Hkv, n, dh] read from the library's cache."""
    k, v = kv_planes(vla, kv, layer, shape, max_ctx)
    return from_dev(k[:, :n]), from_dev(v[:, :n])


def test_tiny_two_blocks_chained_and_partition_identity(vla_lib):
    import torch
    vla = vla_lib
    wl = synth.WORKLOADS["tiny_2blk_64tok"]
    s = wl.shape
    M, L, k = wl.n_tokens, wl.n_layers, wl.prefix_layers
    max_ctx = 128
    m = Model(s, L, wl.seed, max_ctx)
    try:
        xb = synth.hidden_states(M, s.hidden, wl.seed)
        x = to_dev(xb)
        # oracle: [0, L) with per-block outputs and the cache
        cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)
        per_block = []
        ref = oracle.prefix_forward(oracle.bf16_to_f64(xb), m.weights64(), 0, L, cache, s, per_block=per_block)
        # GPU: [0, k) then [k, L) with the boundary in between (Eq. 6)
        kv = vla.vla_kv_create(m.handle, 0, L, max_ctx)
        h = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, x, M, 0, k, kv, h)
        y = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, h, M, k, L, kv, y)
        sync()
        assert vla.vla_last_async_error(m.handle) == 0
        assert rel_l2(from_dev(h), per_block[k - 1]) < REL_L2_BLOCK
        assert rel_l2(from_dev(y), ref) < REL_L2_BLOCK
        assert cos_sim(from_dev(y), ref) > COS_FINAL
        for l in range(L):
            K, V = _kv_planes(vla, kv, l, s, max_ctx, M)
            assert rel_l2(K, cache.k[l][:, :M]) < REL_L2_BLOCK
            assert rel_l2(V, cache.v[l][:, :M]) < REL_L2_BLOCK
        assert vla.vla_kv_length(kv) == M
        # GPU partition identity: [0, L) in one call equals the split run, bit for bit
        kv2 = vla.vla_kv_create(m.handle, 0, L, max_ctx)
        y2 = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, x, M, 0, L, kv2, y2)
        sync()
        assert torch.equal(y.view(torch.int16), y2.view(torch.int16))
        vla.vla_kv_destroy(kv)
        vla.vla_kv_destroy(kv2)
    finally:
        m.close()


def test_7b_block_1024_tokens(vla_lib):
    import torch
    vla = vla_lib
    wl = synth.WORKLOADS["7b_block_1024tok"]
    s = wl.shape
    M = wl.n_tokens
    m = Model(s, 1, wl.seed, 2048)
    try:
        xb = synth.hidden_states(M, s.hidden, wl.seed, wl.visual_tokens, wl.visual_scale)
        x = to_dev(xb)
        cache = oracle.KVCache([0], s.n_kv_heads, s.head_dim, M)
        ref = oracle.prefix_forward(oracle.bf16_to_f64(xb), m.weights64(), 0, 1, cache, s)
        kv = vla.vla_kv_create(m.handle, 0, 1, M)
        y = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, x, M, 0, 1, kv, y)
        sync()
        assert vla.vla_last_async_error(m.handle) == 0
        got = from_dev(y)
        assert rel_l2(got, ref) < REL_L2_BLOCK
        assert cos_sim(got, ref) > COS_FINAL
        K, V = _kv_planes(vla, kv, 0, s, M, M)
        assert rel_l2(K, cache.k[0][:, :M]) < REL_L2_BLOCK
        assert rel_l2(V, cache.v[0][:, :M]) < REL_L2_BLOCK
        vla.vla_kv_destroy(kv)
    finally:
        m.close()


def test_7b_block_512_tokens_every_row_and_repeatable(vla_lib):
    """One 7B block at 512 tokens (the gate/up GEMM's 344 tiles take two rounds and 40 tiles
    of a third on 152 SMs), every output row against the oracle, and a second run must give
    the same bits."""
    import torch
    vla = vla_lib
    s = synth.B7
    M = 512
    m = Model(s, 1, 5, M)
    try:
        xb = synth.hidden_states(M, s.hidden, 5)
        x = to_dev(xb)
        cache = oracle.KVCache([0], s.n_kv_heads, s.head_dim, M)
        ref = oracle.prefix_forward(oracle.bf16_to_f64(xb), m.weights64(), 0, 1, cache, s)
        kv = vla.vla_kv_create(m.handle, 0, 1, M)
        y = torch.empty_like(x)
        outs = []
        for _ in range(2):
            vla.vla_kv_set_length(kv, 0)
            vla.vla_prefix_prefill(m.handle, x, M, 0, 1, kv, y)
            sync()
            assert vla.vla_last_async_error(m.handle) == 0
            outs.append(y.clone())
        assert torch.equal(outs[0].view(torch.int16), outs[1].view(torch.int16))
        got = from_dev(outs[0])
        assert rel_l2(got, ref) < REL_L2_BLOCK
        row_err = np.linalg.norm(got - ref, axis=1) / np.linalg.norm(ref, axis=1)
        assert row_err.max() < 2 * REL_L2_BLOCK
        vla.vla_kv_destroy(kv)
    finally:
        m.close()


def test_prefill_continues_context_and_random_gains(vla_lib):
    """Two prefills on one cache (positions 0..99 then 100..136) with non-unit RMSNorm gains."""
    import torch
    vla = vla_lib
    s = synth.TINY
    L, max_ctx = 2, 160
    m = Model(s, L, 7, max_ctx, gain="random")
    try:
        xb = synth.hidden_states(137, s.hidden, 7)
        cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)
        r1 = oracle.prefix_forward(oracle.bf16_to_f64(xb[:100]), m.weights64(), 0, L, cache, s)
        r2 = oracle.prefix_forward(oracle.bf16_to_f64(xb[100:]), m.weights64(), 0, L, cache, s)
        kv = vla.vla_kv_create(m.handle, 0, L, max_ctx)
        y1 = torch.empty((100, s.hidden), dtype=torch.bfloat16, device="cuda")
        y2 = torch.empty((37, s.hidden), dtype=torch.bfloat16, device="cuda")
        vla.vla_prefix_prefill(m.handle, to_dev(xb[:100]), 100, 0, L, kv, y1)
        vla.vla_prefix_prefill(m.handle, to_dev(xb[100:]), 37, 0, L, kv, y2)
        sync()
        assert rel_l2(from_dev(y1), r1) < REL_L2_BLOCK
        assert rel_l2(from_dev(y2), r2) < REL_L2_BLOCK
        assert vla.vla_kv_length(kv) == 137
        vla.vla_kv_destroy(kv)
    finally:
        m.close()


def test_decode_steps_tiny(vla_lib):
    import torch
    vla = vla_lib
    s = synth.TINY
    L, max_ctx, M, steps = 2, 96, 64, 8
    m = Model(s, L, 3, max_ctx)
    try:
        xb = synth.hidden_states(M, s.hidden, 3)
        cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)
        oracle.prefix_forward(oracle.bf16_to_f64(xb), m.weights64(), 0, L, cache, s)
        kv = vla.vla_kv_create(m.handle, 0, L, max_ctx)
        y = torch.empty((M, s.hidden), dtype=torch.bfloat16, device="cuda")
        vla.vla_prefix_prefill(m.handle, to_dev(xb), M, 0, L, kv, y)
        out = torch.empty((1, s.hidden), dtype=torch.bfloat16, device="cuda")
        for t in range(steps):
            xt = synth.decode_hidden(t, s.hidden, 3)
            ref = oracle.decode_step(oracle.bf16_to_f64(xt), m.weights64(), 0, L, cache, s)
            vla.vla_prefix_decode(m.handle, to_dev(xt), 0, L, kv, out)
            sync()
            assert rel_l2(from_dev(out), ref) < REL_L2_BLOCK, t
        assert vla.vla_kv_length(kv) == M + steps
        assert vla.vla_last_async_error(m.handle) == 0
        vla.vla_kv_destroy(kv)
    finally:
        m.close()


def test_decode_7b_two_blocks_random_context(vla_lib):
    """Decode against a cache pre-filled with random K/V at positions [0, 2304)."""
    import torch
    vla = vla_lib
    s = synth.B7
    L, ctx0, steps, max_ctx = 2, 2304, 3, 2368
    m = Model(s, L, 0, max_ctx)
    try:
        cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)
        kv = vla.vla_kv_create(m.handle, 0, L, max_ctx)
        for l in range(L):
            kb, vb = synth.random_kv(ctx0, s, 0, l)
            cache.fill(l, oracle.bf16_to_f64(kb), oracle.bf16_to_f64(vb))
            kt, vt = kv_planes(vla, kv, l, s, max_ctx)
            kt[:, :ctx0].copy_(to_dev(kb))
            vt[:, :ctx0].copy_(to_dev(vb))
        sync()
        vla.vla_kv_set_length(kv, ctx0)
        out = torch.empty((1, s.hidden), dtype=torch.bfloat16, device="cuda")
        for t in range(steps):
            xt = synth.decode_hidden(t, s.hidden, 0)
            ref = oracle.decode_step(oracle.bf16_to_f64(xt), m.weights64(), 0, L, cache, s)
            vla.vla_prefix_decode(m.handle, to_dev(xt), 0, L, kv, out)
            sync()
            got = from_dev(out)
            assert rel_l2(got, ref) < REL_L2_BLOCK, t
            assert cos_sim(got, ref) > COS_FINAL
        assert vla.vla_last_async_error(m.handle) == 0
        vla.vla_kv_destroy(kv)
    finally:
        m.close()


@pytest.mark.parametrize("shape", [
    # 2 query heads per KV head, head_dim 64, FFN 700 (zero-padded to the gate/up unit)
    synth.ModelShape(hidden=256, n_heads=8, n_kv_heads=4, head_dim=64, ffn=700),
    # 8 query heads per KV head, head_dim 128, FFN 520
    synth.ModelShape(hidden=512, n_heads=16, n_kv_heads=2, head_dim=128, ffn=520),
], ids=["gqa2_dh64", "gqa8_dh128"])
def test_other_head_groupings_prefill_and_decode(vla_lib, shape):
    """The other supported query-per-KV-head groupings: two blocks over 29 tokens (block by
    block against the oracle, with the written cache), then three decode steps."""
    import torch
    vla = vla_lib
    s, L, M, max_ctx = shape, 2, 29, 40
    m = Model(s, L, 13, max_ctx, gain="random")
    try:
        xb = synth.hidden_states(M, s.hidden, 13)
        cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)
        per_block = []
        ref = oracle.prefix_forward(oracle.bf16_to_f64(xb), m.weights64(), 0, L, cache, s, per_block=per_block)
        kv = vla.vla_kv_create(m.handle, 0, L, max_ctx)
        x = to_dev(xb)
        h = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, x, M, 0, 1, kv, h)
        y = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, h, M, 1, L, kv, y)
        sync()
        assert vla.vla_last_async_error(m.handle) == 0
        assert rel_l2(from_dev(h), per_block[0]) < REL_L2_BLOCK
        assert rel_l2(from_dev(y), ref) < REL_L2_BLOCK
        assert cos_sim(from_dev(y), ref) > COS_FINAL
        for l in range(L):
            K, V = _kv_planes(vla, kv, l, s, max_ctx, M)
            assert rel_l2(K, cache.k[l][:, :M]) < REL_L2_BLOCK
            assert rel_l2(V, cache.v[l][:, :M]) < REL_L2_BLOCK
        out = torch.empty((1, s.hidden), dtype=torch.bfloat16, device="cuda")
        for t in range(3):
            xt = synth.decode_hidden(t, s.hidden, 13)
            rt = oracle.decode_step(oracle.bf16_to_f64(xt), m.weights64(), 0, L, cache, s)
            vla.vla_prefix_decode(m.handle, to_dev(xt), 0, L, kv, out)
            sync()
            assert rel_l2(from_dev(out), rt) < REL_L2_BLOCK, t
        assert vla.vla_kv_length(kv) == M + 3
        assert vla.vla_last_async_error(m.handle) == 0
        vla.vla_kv_destroy(kv)
    finally:
        m.close()
