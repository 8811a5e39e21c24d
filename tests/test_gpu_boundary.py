"""The boundary hand-off of Eq. 6 / Eq. 11 on the GPU: the GPU range [0, k) writes h^(k), a
side stream copies it into page-locked host memory while the main stream continues, and
the split point may change from frame to frame (same KV cache, no reallocation). Also the
argument checks of the C ABI against a live prefix object."""
import ctypes

import numpy as np
import pytest

import synth
from helpers import sync, Model, to_dev

pytestmark = pytest.mark.gpu


def _bits(t):
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy()


def test_frames_with_overlapped_boundary_copies_and_per_frame_split(vla_lib):
    """Four 3072-token frames (6 x 448 visual + 384 text rows) through an 8-block 7B-class
    stack, double-buffered: frame f's boundary copy overlaps frame f's suffix range and
    frame f+1's prefix (checked on event timestamps). Each frame uses its own split point;
    the host copy of h^(k) and the range output equal single-stream reference runs bit for
    bit."""
    import torch
    vla = vla_lib
    s, L, M = synth.B7, 8, 3072
    ks = [2, 4, 6, 4]
    m = Model(s, L, 0, M)
    try:
        main = torch.cuda.current_stream()
        side = torch.cuda.Stream()
        kvs = [vla.vla_kv_create(m.handle, 0, L, M) for _ in range(2)]
        hdev = [torch.empty((M, s.hidden), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
        ydev = [torch.empty_like(hdev[0]) for _ in range(2)]
        pinned = [torch.empty((M, s.hidden), dtype=torch.bfloat16, pin_memory=True) for _ in range(2)]
        ready = [torch.cuda.Event() for _ in range(2)]
        done = [torch.cuda.Event() for _ in range(2)]
        for e in done:
            e.record(side)  # creates the event handle the library records into
        xs = [to_dev(synth.hidden_states(M, s.hidden, f, 2688, 1.0)) for f in range(4)]
        # references: one stream, fresh caches, no overlap
        kv_ref = vla.vla_kv_create(m.handle, 0, L, M)
        h_ref, y_ref = [], []
        for f in range(4):
            h = torch.empty_like(hdev[0])
            y = torch.empty_like(hdev[0])
            vla.vla_kv_reset(kv_ref)
            vla.vla_prefix_prefill(m.handle, xs[f], M, 0, ks[f], kv_ref, h)
            vla.vla_kv_reset(kv_ref)
            vla.vla_prefix_prefill(m.handle, xs[f], M, 0, L, kv_ref, y)
            h_ref.append(h)
            y_ref.append(y)
        sync(120)
        ref_h = [_bits(h) for h in h_ref]
        ref_y = [_bits(y) for y in y_ref]

        def check(f):
            b = f % 2
            done[b].synchronize()
            np.testing.assert_array_equal(pinned[b].view(torch.int16).numpy(), ref_h[f])

        ev = [{n: torch.cuda.Event(enable_timing=True) for n in ("copy0", "copy1", "suffix0", "suffix1")}
              for _ in range(4)]
        for f in range(4):
            b = f % 2
            if f >= 2:
                check(f - 2)  # buffer b's previous copy has landed and is verified before reuse
            vla.vla_kv_reset(kvs[b], main)
            vla.vla_prefix_prefill(m.handle, xs[f], M, 0, ks[f], kvs[b], hdev[b], main)
            ready[b].record(main)
            side.wait_event(ready[b])
            ev[f]["copy0"].record(side)
            vla.vla_boundary_to_host(hdev[b], M, s.hidden, pinned[b], side, None, done[b])
            ev[f]["copy1"].record(side)
            ev[f]["suffix0"].record(main)
            vla.vla_prefix_prefill(m.handle, hdev[b], M, ks[f], L, kvs[b], ydev[b], main)
            ev[f]["suffix1"].record(main)
            main.wait_event(done[b])  # hdev[b] is rewritten two frames later
            if f >= 2:
                sync(120)
                np.testing.assert_array_equal(_bits(ydev[b]), ref_y[f])
        check(2)
        check(3)
        sync(120)
        np.testing.assert_array_equal(_bits(ydev[1]), ref_y[3])
        # each frame's boundary copy ran while its suffix range was running (event timestamps:
        # the copy started before the suffix ended and finished after the suffix started)
        for f in range(4):
            assert ev[f]["copy0"].elapsed_time(ev[f]["suffix1"]) > 0, f
            assert ev[f]["suffix0"].elapsed_time(ev[f]["copy1"]) > 0, f
        assert vla.vla_last_async_error(m.handle) == 0
        for kv in kvs + [kv_ref]:
            vla.vla_kv_destroy(kv)
    finally:
        m.close()


def test_abi_errors_on_a_live_prefix(vla_lib):
    import torch
    vla = vla_lib
    s = synth.TINY
    L, max_ctx = 3, 32
    m = Model(s, L, 2, max_ctx)
    other = Model(s, 1, 3, max_ctx)
    try:
        x = to_dev(synth.hidden_states(16, s.hidden, 2))
        y = torch.empty_like(x)
        kv = vla.vla_kv_create(m.handle, 0, 2, max_ctx)  # covers layers [0, 2) only

        def status(fn, *a):
            with pytest.raises(vla.VlaError) as ei:
                fn(*a)
            return ei.value.name

        assert status(vla.vla_prefix_prefill, m.handle, x, 16, 0, 3, kv, y) == "VLA_ERR_RANGE"  # beyond the cache
        assert status(vla.vla_prefix_prefill, m.handle, x, 16, 2, 1, kv, y) == "VLA_ERR_RANGE"  # reversed
        assert status(vla.vla_prefix_prefill, m.handle, x, 16, 0, 4, kv, y) == "VLA_ERR_RANGE"  # beyond the model
        assert status(vla.vla_kv_create, m.handle, 0, 4, max_ctx) in ("VLA_ERR_RANGE", "VLA_ERR_INVALID_ARG")
        kv_other = vla.vla_kv_create(other.handle, 0, 1, max_ctx)
        assert status(vla.vla_prefix_prefill, m.handle, x, 16, 0, 1, kv_other, y) == "VLA_ERR_INVALID_ARG"
        # layer 0 advanced alone: a range starting at different lengths is refused
        vla.vla_prefix_prefill(m.handle, x, 16, 0, 1, kv, y)
        assert status(vla.vla_prefix_prefill, m.handle, x, 16, 0, 2, kv, y) == "VLA_ERR_RANGE"
        vla.vla_prefix_prefill(m.handle, y, 16, 1, 2, kv, y)  # in place; layer 1 catches up
        assert vla.vla_kv_length(kv) == 16
        # 16 + 17 > 32 positions
        x17 = to_dev(synth.hidden_states(17, s.hidden, 2))
        assert status(vla.vla_prefix_prefill, m.handle, x17, 17, 0, 2, kv, torch.empty_like(x17)) == "VLA_ERR_KV_FULL"
        # decode fills the cache to the last position, then refuses
        one = torch.empty((1, s.hidden), dtype=torch.bfloat16, device="cuda")
        for t in range(16):
            vla.vla_prefix_decode(m.handle, to_dev(synth.decode_hidden(t, s.hidden, 2)), 0, 2, kv, one)
        assert vla.vla_kv_length(kv) == 32
        assert status(vla.vla_prefix_decode, m.handle, one, 0, 2, kv, one) == "VLA_ERR_KV_FULL"
        # unaligned device pointers
        raw = torch.empty(16 * s.hidden + 8, dtype=torch.bfloat16, device="cuda")
        assert status(vla.vla_prefix_prefill, m.handle, raw.data_ptr() + 2, 16, 0, 2, kv, y) == "VLA_ERR_INVALID_ARG"
        # pageable host memory is refused for the boundary copy; pinned memory is accepted
        pageable = np.zeros((16, s.hidden), dtype=np.uint16)
        assert status(vla.vla_boundary_to_host, y, 16, s.hidden, pageable.ctypes.data) == "VLA_ERR_NOT_PINNED"
        pin = torch.empty((16, s.hidden), dtype=torch.bfloat16, pin_memory=True)
        vla.vla_boundary_to_host(y, 16, s.hidden, pin)
        sync()
        np.testing.assert_array_equal(pin.view(torch.int16).numpy(), _bits(y))
        # an empty range is a copy, needs no cache, and leaves lengths alone
        z = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, x, 16, 2, 2, None, z)
        sync()
        assert torch.equal(z.view(torch.int16), x.view(torch.int16))
        vla.vla_kv_reset(kv)
        sync()
        assert vla.vla_kv_length(kv) == 0
        assert vla.vla_last_async_error(m.handle) == 0
        assert ctypes.c_int(vla.vla_kv_layer_length(kv, 5)).value == -1
        vla.vla_kv_destroy(kv)
        vla.vla_kv_destroy(kv_other)
    finally:
        m.close()
        other.close()


@pytest.mark.parametrize("shape_name,L,M", [("TINY", 2, 64), ("B7", 2, 256)])
def test_prefill_to_host_fused_boundary_store(vla_lib, shape_name, L, M):
    """The last block's epilogue stores h^(L) into page-locked host memory as well: the host
    copy, the device output and a plain prefill agree bit for bit; split ranges and the empty
    range deliver the range's output; pageable memory is refused."""
    import torch
    vla = vla_lib
    s = getattr(synth, shape_name)
    m = Model(s, L, 5, M)
    try:
        x = to_dev(synth.hidden_states(M, s.hidden, 5))
        kv = vla.vla_kv_create(m.handle, 0, L, M)
        y_ref = torch.empty_like(x)
        vla.vla_prefix_prefill(m.handle, x, M, 0, L, kv, y_ref)
        host = torch.empty((M, s.hidden), dtype=torch.bfloat16, pin_memory=True)
        host.view(torch.int16).fill_(-1)
        y = torch.empty_like(x)
        vla.vla_kv_reset(kv)
        vla.vla_prefix_prefill_to_host(m.handle, x, M, 0, L, kv, y, host)
        sync()
        np.testing.assert_array_equal(_bits(y), _bits(y_ref))
        np.testing.assert_array_equal(host.view(torch.int16).numpy(), _bits(y_ref))
        # [0, 1) then [1, L) with the boundary of each range delivered to the host
        h1 = torch.empty((M, s.hidden), dtype=torch.bfloat16, pin_memory=True)
        mid = torch.empty_like(x)
        vla.vla_kv_reset(kv)
        vla.vla_prefix_prefill_to_host(m.handle, x, M, 0, 1, kv, mid, h1)
        vla.vla_prefix_prefill_to_host(m.handle, mid, M, 1, L, kv, y, host)
        sync()
        np.testing.assert_array_equal(h1.view(torch.int16).numpy(), _bits(mid))
        np.testing.assert_array_equal(host.view(torch.int16).numpy(), _bits(y_ref))
        # empty range: the input itself
        vla.vla_prefix_prefill_to_host(m.handle, x, M, 1, 1, None, y, host)
        sync()
        np.testing.assert_array_equal(host.view(torch.int16).numpy(), _bits(x))
        pageable = np.zeros((M, s.hidden), dtype=np.uint16)
        with pytest.raises(vla.VlaError) as ei:
            vla.vla_prefix_prefill_to_host(m.handle, x, M, 0, L, kv, y, pageable.ctypes.data)
        assert ei.value.name == "VLA_ERR_NOT_PINNED"
        assert vla.vla_last_async_error(m.handle) == 0
        vla.vla_kv_destroy(kv)
    finally:
        m.close()


def test_frame_to_device_uploads_pinned_frames_and_rejects_pageable_ones(vla_lib):
    """The frame's input hand-off: page-locked host bits arrive unchanged in the device buffer
    (on the caller's stream, ordered with work recorded after it); a pageable source is
    refused with NOT_PINNED and leaves the buffer alone; zero tokens copy nothing."""
    import torch
    lib = vla_lib.load()
    M, D = 300, 256
    bits = synth.hidden_states(M, D, 3)
    host = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).pin_memory()
    dev = torch.zeros((M, D), dtype=torch.bfloat16, device="cuda")
    s = torch.cuda.Stream()
    vla_lib.vla_frame_to_device(host, M, D, dev, s)
    done = torch.cuda.Event()
    done.record(s)
    done.synchronize()
    np.testing.assert_array_equal(_bits(dev), np.asarray(bits).view(np.int16).reshape(M, D))
    pageable = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    dev2 = torch.zeros((M, D), dtype=torch.bfloat16, device="cuda")
    assert lib.vla_frame_to_device(ctypes.c_void_p(pageable.data_ptr()), M, D, ctypes.c_void_p(dev2.data_ptr()),
                                   None) == 5  # VLA_ERR_NOT_PINNED
    assert lib.vla_frame_to_device(ctypes.c_void_p(host.data_ptr()), 0, D, ctypes.c_void_p(dev2.data_ptr()),
                                   None) == 0
    sync()
    assert not dev2.view(torch.int16).any()
