"""The allocation-free decode attention against the regular attention entry point.

vla_op_attention_decode_noalloc is for callers that may not allocate device memory while
they run (a real-time control loop with a memory budget fixed at start-up, or a host
framework whose allocator owns the GPU memory): its scratch space is a fixed array inside
the library. Its result must match vla_op_attention_prefill for a single query at the last
position, call after call, since every call reuses the same array.

Collected last on purpose (file name), so a failure here does not hide the other tests.
"""
import numpy as np
import pytest

import synth
from helpers import from_dev, rel_l2, sync, to_dev

pytestmark = pytest.mark.gpu


def _case(vla, H, Hkv, dh, ctx, max_ctx, seed):
    import torch
    q = synth.normal_bf16((1, H * dh), seed, 11, 1.0)
    kp = synth.normal_bf16((Hkv, max_ctx, dh), seed, 12, 1.0)
    vp = synth.normal_bf16((Hkv, max_ctx, dh), seed, 13, 1.0)
    Q, K, V = to_dev(q), to_dev(kp), to_dev(vp)
    ref = torch.empty((1, H * dh), dtype=torch.bfloat16, device="cuda")
    got = torch.empty((H * dh,), dtype=torch.bfloat16, device="cuda")
    vla.vla_op_attention_prefill(Q, K, V, 1, H, Hkv, dh, max_ctx, ctx - 1, ref)
    vla.vla_op_attention_decode_noalloc(Q, K, V, ctx, H, Hkv, dh, max_ctx, got)
    sync()
    return from_dev(got), from_dev(ref)[0]


@pytest.mark.parametrize("H,Hkv,dh", [(32, 8, 128), (4, 4, 64)])
def test_noalloc_decode_attention_matches_regular_entry_point(vla_lib, H, Hkv, dh):
    max_ctx = 2368
    # two calls in a row on the shared scratch array, with different data and lengths
    for seed, ctx in ((1, 2305), (2, 977)):
        got, ref = _case(vla_lib, H, Hkv, dh, ctx, max_ctx, seed)
        assert np.isfinite(got).all()
        assert rel_l2(got, ref) < 1e-2, (seed, ctx)


def test_noalloc_rejects_bad_arguments(vla_lib):
    import torch
    lib = vla_lib.load()
    buf = torch.zeros(8 * 128 * 64, dtype=torch.bfloat16, device="cuda")
    p = buf.data_ptr()
    # ctx past max_ctx, unsupported head_dim, and a head count whose one split exceeds the array
    assert lib.vla_op_attention_decode_noalloc(p, p, p, 65, 4, 4, 64, 64, p, None) == 1
    assert lib.vla_op_attention_decode_noalloc(p, p, p, 8, 4, 4, 96, 64, p, None) == 9
    assert lib.vla_op_attention_decode_noalloc(p, p, p, 8, 8192, 8192, 64, 64, p, None) == 2
