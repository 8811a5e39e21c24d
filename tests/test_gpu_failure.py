"""Failure detection on the GPU without a fault: a kernel whose bounded wait runs out reports
VLA_ERR_TIMEOUT through vla_last_async_error and leaves the context usable.

vla_prefix_inject_stall makes the next launch of one projection GEMM withhold one k-block of
its first tile, with its waits bounded at ~1 ms instead of ~1 s: the MMA issuer's wait on that
stage runs out, the CTA records the timeout, lets its copies in flight land, retires its
MMAs, releases tensor memory and exits. The test then checks that the same object, on the
same stream, computes the reference result again (bit for bit)."""
import time

import pytest

import synth
from helpers import Model, sync, to_dev

pytestmark = pytest.mark.gpu

TIMEOUT = 8  # VLA_ERR_TIMEOUT


@pytest.mark.parametrize("stage,shape,M", [
    ("gemm_down", "TINY", 64), ("gemm_qkv", "TINY", 64), ("gemm_o", "TINY", 64), ("gemm_gateup", "TINY", 64),
    # 7B shapes at 384 tokens: hundreds of tiles, so CTAs that withheld a stage of their first
    # tile also hold later tiles whose loads are in flight when the wait runs out
    ("gemm_gateup", "B7", 384), ("gemm_qkv", "B7", 384),
])
def test_stalled_gemm_reports_timeout_and_the_object_recovers(vla_lib, stage, shape, M):
    import torch
    vla = vla_lib
    s, L = getattr(synth, shape), 2
    m = Model(s, L, 0, M)
    try:
        kv = vla.vla_kv_create(m.handle, 0, L, M)
        x = to_dev(synth.hidden_states(M, s.hidden, 0))
        ref = torch.empty_like(x)
        out = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, x, M, 0, L, kv, ref)
        sync()
        assert vla.vla_last_async_error(m.handle) == 0
        for _ in range(2):  # twice: the object recovers every time
            vla.vla_kv_reset(kv)
            vla.vla_prefix_inject_stall(m.handle, stage, 2_000_000)  # ~1 ms at the GB300's clock
            t0 = time.time()
            vla.vla_prefix_prefill(m.handle, x, M, 0, L, kv, out)
            sync(30)
            waited = time.time() - t0
            assert vla.vla_last_async_error(m.handle) == TIMEOUT
            assert waited < 5.0, waited  # the short bound, not the default ~1 s per wait chain
            vla.vla_kv_reset(kv)
            vla.vla_prefix_prefill(m.handle, x, M, 0, L, kv, out)
            sync()
            assert vla.vla_last_async_error(m.handle) == 0
            assert torch.equal(out.view(torch.int16), ref.view(torch.int16))
        vla.vla_kv_destroy(kv)
    finally:
        m.close()


def test_inject_stall_argument_checks(vla_lib):
    vla = vla_lib
    m = Model(synth.TINY, 1, 0, 64)
    try:
        lib = vla.load()
        assert lib.vla_prefix_inject_stall(m.handle, 2, 2_000_000) == 9      # attention: not a GEMM stage
        assert lib.vla_prefix_inject_stall(m.handle, 5, 10) == 1             # budget below 1e5 cycles
        assert lib.vla_prefix_inject_stall(m.handle, 5, 3_000_000_000) == 1  # above the default bound
        assert lib.vla_prefix_inject_stall(None, 5, 2_000_000) == 1
        assert lib.vla_prefix_inject_stall(m.handle, -1, 0) == 0             # cancel
    finally:
        m.close()
