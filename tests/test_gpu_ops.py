"""Kernel-level parity: the tcgen05 GEMM and the prefill attention kernel against the
float64 definitions (oracle attention; matmul of the exact bf16 inputs)."""
import numpy as np
import pytest

import oracle
import synth
from helpers import sync, from_dev, rel_l2, to_dev

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("M,N,K", [
    (64, 256, 256),        # one tile
    (200, 768, 688),       # ragged M, K tail (688 = 10.75 x 64)
    (65, 1376, 256),       # ragged N (1376 = 5 x 256 + 96)
    (1, 512, 4096),        # a single row
    (1024, 6144, 4096),    # 7B QKV projection
    (2304, 4096, 11008),   # 7B down projection at 2304 tokens
])
def test_gemm_matches_definition(vla_lib, M, N, K):
    import torch
    a = synth.normal_bf16((M, K), 1, 100 + M, 1.0)
    b = synth.normal_bf16((N, K), 1, 200 + N, 0.02)
    A, B = to_dev(a), to_dev(b)
    C = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    vla_lib.vla_op_gemm_bf16(A, B, M, N, K, C)
    sync()
    got = from_dev(C)
    rows = np.arange(M) if M <= 256 else np.random.default_rng(0).choice(M, 256, replace=False)
    ref = oracle.bf16_to_f64(a[rows]) @ oracle.bf16_to_f64(b).T
    g = got[rows]
    # bf16 output rounding (2^-8 relative) plus fp32 accumulation-order error
    tol = 2.0 ** -8 * np.abs(ref) + 1e-4 * np.sqrt(np.mean(ref ** 2))
    bad = np.abs(g - ref) > tol
    assert not bad.any(), f"{bad.sum()} mismatches, max err {np.abs(g - ref).max()}"


@pytest.mark.parametrize("M,H,Hkv,dh,pos0", [
    (64, 4, 4, 64, 0),
    (200, 32, 8, 128, 0),     # ragged M, GQA group 4
    (130, 8, 2, 128, 77),     # continuing context
    (1, 4, 1, 64, 5),         # one query, MQA
    (96, 8, 4, 64, 3),        # GQA group 2
    (150, 16, 2, 128, 9),     # GQA group 8, ragged M, continuing context
    (1024, 32, 8, 128, 0),    # 7B shape
    (64, 320, 8, 64, 0),      # more one-block query tiles than SMs: consecutive tiny units per CTA
    (100, 160, 16, 128, 300), # long continuing context, four key blocks per ragged query tile
])
def test_attention_prefill_matches_oracle(vla_lib, M, H, Hkv, dh, pos0):
    import torch
    max_ctx = pos0 + M + 13
    q = synth.normal_bf16((M, H, dh), 2, 1, 1.0)
    kp = synth.normal_bf16((Hkv, max_ctx, dh), 2, 2, 1.0)
    vp = synth.normal_bf16((Hkv, max_ctx, dh), 2, 3, 1.0)
    # positions past the context hold garbage that must not leak into the result
    kp[:, pos0 + M:] = 0x7FC0  # NaN
    vp[:, pos0 + M:] = 0x7FC0
    out = torch.empty((M, H * dh), dtype=torch.bfloat16, device="cuda")
    Q, Kc, Vc = to_dev(q), to_dev(kp), to_dev(vp)
    vla_lib.vla_op_attention_prefill(Q, Kc, Vc, M, H, Hkv, dh, max_ctx, pos0, out)
    sync()
    got = from_dev(out).reshape(M, H, dh)
    ctx = pos0 + M
    ref = oracle.causal_gqa_attention(oracle.bf16_to_f64(q), oracle.bf16_to_f64(kp[:, :ctx]),
                                      oracle.bf16_to_f64(vp[:, :ctx]), pos0 + np.arange(M), Hkv)
    assert np.isfinite(got).all()
    assert rel_l2(got, ref) < 1e-2
    # per row: the probabilities are bf16 in the P.V product -> a few 2^-9 relative
    row_err = np.linalg.norm((got - ref).reshape(M, -1), axis=1) / np.linalg.norm(ref.reshape(M, -1), axis=1)
    assert row_err.max() < 2e-2

