"""Batched decode (vla_prefix_decode_batch): several independent sequences, each in its own KV
cache at its own position, stepped together with the weights streamed once. Every row must
equal the single-sequence decode of that sequence bit for bit, and match the oracle."""
import numpy as np
import pytest

import oracle
import synth
from helpers import sync, COS_FINAL, REL_L2_BLOCK, Model, cos_sim, from_dev, kv_planes, rel_l2, to_dev

pytestmark = pytest.mark.gpu


def _fill_random_context(vla, kv, s, L, max_ctx, n, seed):
    bits = []
    for l in range(L):
        kb, vb = synth.random_kv(n, s, seed, l)
        kt, vt = kv_planes(vla, kv, l, s, max_ctx)
        kt[:, :n].copy_(to_dev(kb))
        vt[:, :n].copy_(to_dev(vb))
        bits.append((kb, vb))
    sync()
    vla.vla_kv_set_length(kv, n)
    return bits


@pytest.mark.parametrize("shape_name,L,max_ctx,ctxs", [
    ("TINY", 2, 160, [5, 37, 100]),
    ("B7", 2, 2368, [1, 700, 1500, 2304]),
])
def test_batched_decode_equals_single_sequence_decode(vla_lib, shape_name, L, max_ctx, ctxs):
    import torch
    vla = vla_lib
    s = getattr(synth, shape_name)
    B = len(ctxs)
    m = Model(s, L, 9, max_ctx)
    try:
        batch_kv = [vla.vla_kv_create(m.handle, 0, L, max_ctx) for _ in range(B)]
        single_kv = [vla.vla_kv_create(m.handle, 0, L, max_ctx) for _ in range(B)]
        ctx_bits = []
        for b, n in enumerate(ctxs):
            ctx_bits.append(_fill_random_context(vla, batch_kv[b], s, L, max_ctx, n, 20 + b))
            _fill_random_context(vla, single_kv[b], s, L, max_ctx, n, 20 + b)
        cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)  # sequence B-1
        for l in range(L):
            cache.fill(l, oracle.bf16_to_f64(ctx_bits[-1][l][0]), oracle.bf16_to_f64(ctx_bits[-1][l][1]))
        y = torch.empty((B, s.hidden), dtype=torch.bfloat16, device="cuda")
        y1 = torch.empty((1, s.hidden), dtype=torch.bfloat16, device="cuda")
        for t in range(3):
            xb = np.concatenate([synth.decode_hidden(t, s.hidden, 100 + b) for b in range(B)], axis=0)
            x = to_dev(xb)
            vla.vla_prefix_decode_batch(m.handle, x, 0, L, batch_kv, y)
            rows = []
            for b in range(B):
                vla.vla_prefix_decode(m.handle, x[b:b + 1], 0, L, single_kv[b], y1)
                sync()
                rows.append(y1.clone())
            sync()
            for b in range(B):
                assert torch.equal(y[b:b + 1].view(torch.int16), rows[b].view(torch.int16)), (t, b)
            ref = oracle.decode_step(oracle.bf16_to_f64(xb[-1:]), m.weights64(), 0, L, cache, s)
            got = from_dev(y[B - 1:B])
            assert rel_l2(got, ref) < REL_L2_BLOCK, t
            assert cos_sim(got, ref) > COS_FINAL, t
        for b in range(B):
            assert vla.vla_kv_length(batch_kv[b]) == ctxs[b] + 3
        assert vla.vla_last_async_error(m.handle) == 0
        for kv in batch_kv + single_kv:
            vla.vla_kv_destroy(kv)
    finally:
        m.close()


def test_batched_decode_argument_errors(vla_lib):
    import torch
    vla = vla_lib
    s = synth.TINY
    m = Model(s, 1, 4, 64)
    try:
        a = vla.vla_kv_create(m.handle, 0, 1, 64)
        b = vla.vla_kv_create(m.handle, 0, 1, 32)
        x = torch.zeros((5, s.hidden), dtype=torch.bfloat16, device="cuda")
        y = torch.empty_like(x)

        def status(*args):
            with pytest.raises(vla.VlaError) as ei:
                vla.vla_prefix_decode_batch(m.handle, *args)
            return ei.value.name

        assert status(x, 0, 1, [a, a], y) == "VLA_ERR_INVALID_ARG"  # one token per cache
        assert status(x, 0, 1, [a, b], y) == "VLA_ERR_SHAPE"        # different max_ctx
        kvs5 = [vla.vla_kv_create(m.handle, 0, 1, 64) for _ in range(5)]
        assert status(x, 0, 1, kvs5, y) == "VLA_ERR_SHAPE"          # more than 4 sequences
        for kv in [a, b] + kvs5:
            vla.vla_kv_destroy(kv)
    finally:
        m.close()
