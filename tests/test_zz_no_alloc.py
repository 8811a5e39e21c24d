"""The allocation-free decode attention, against the oracle and the regular entry point.

vla_op_attention_decode_noalloc is for callers that may not allocate device memory while
they run (a real-time control loop with a memory budget fixed at start-up, or a host
framework whose allocator owns the GPU memory): its scratch space is a fixed array inside
the library. Every call reuses that array, so each case below is a run of calls in a row
with different data and context lengths, each checked on its own: against the float64
oracle's attention for one query at position ctx - 1, and against vla_op_attention_prefill
(one query, pos0 = ctx - 1) within the same tolerance.

The context lengths cover a long context, a ragged one, one that leaves the last key
splits empty (65 keys over 38 splits of 2 keys for 8 KV heads on 152 SMs) and a single key.
The split count is never cut down by the array's size on a 152-SM GPU: splits * n_heads *
(head_dim + 2) stays below 330,000 of the array's 524,288 floats for every supported head
grouping, so only the rejection of a head count whose one split cannot fit is tested.

Collected last on purpose (file name), so a failure here does not hide the other tests.
"""
import numpy as np
import pytest

import oracle
import synth
from helpers import REL_L2_BLOCK, from_dev, rel_l2, sync, to_dev

pytestmark = pytest.mark.gpu

MAX_CTX = 2368
CONTEXTS = (2305, 977, 65, 1)


def _case(vla, H, Hkv, dh, ctx, seed):
    import torch
    q = synth.normal_bf16((1, H * dh), seed, 11, 1.0)
    kp = synth.normal_bf16((Hkv, MAX_CTX, dh), seed, 12, 1.0)
    vp = synth.normal_bf16((Hkv, MAX_CTX, dh), seed, 13, 1.0)
    Q, K, V = to_dev(q), to_dev(kp), to_dev(vp)
    reg = torch.empty((1, H * dh), dtype=torch.bfloat16, device="cuda")
    got = torch.empty((H * dh,), dtype=torch.bfloat16, device="cuda")
    vla.vla_op_attention_prefill(Q, K, V, 1, H, Hkv, dh, MAX_CTX, ctx - 1, reg)
    vla.vla_op_attention_decode_noalloc(Q, K, V, ctx, H, Hkv, dh, MAX_CTX, got)
    sync()
    ref = oracle.causal_gqa_attention(oracle.bf16_to_f64(q).reshape(1, H, dh),
                                      oracle.bf16_to_f64(kp)[:, :ctx], oracle.bf16_to_f64(vp)[:, :ctx],
                                      np.array([ctx - 1]), Hkv).reshape(H * dh)
    return from_dev(got), from_dev(reg)[0], ref


@pytest.mark.parametrize("dh", [64, 128])
@pytest.mark.parametrize("H,Hkv", [(8, 8), (16, 8), (32, 8), (64, 8)])
def test_noalloc_decode_attention_against_oracle_and_regular_entry_point(vla_lib, H, Hkv, dh):
    for i, ctx in enumerate(CONTEXTS):
        got, reg, ref = _case(vla_lib, H, Hkv, dh, ctx, seed=1 + i)
        assert np.isfinite(got).all(), ctx
        assert rel_l2(got, ref) < REL_L2_BLOCK, ctx
        assert rel_l2(got, reg) < REL_L2_BLOCK, ctx
        if ctx == 1:  # one key: the output is its value row, rounded to bf16 once
            np.testing.assert_array_equal(got, ref)


def test_noalloc_rejects_bad_arguments(vla_lib):
    import torch
    lib = vla_lib.load()
    buf = torch.zeros(8 * 128 * 64, dtype=torch.bfloat16, device="cuda")
    p = buf.data_ptr()
    # ctx past max_ctx, unsupported head_dim, and a head count whose one split exceeds the array
    assert lib.vla_op_attention_decode_noalloc(p, p, p, 65, 4, 4, 64, 64, p, None) == 1
    assert lib.vla_op_attention_decode_noalloc(p, p, p, 8, 4, 4, 96, 64, p, None) == 9
    assert lib.vla_op_attention_decode_noalloc(p, p, p, 8, 8192, 8192, 64, 64, p, None) == 2
