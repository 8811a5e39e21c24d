"""The CPU-executed suffix B_{p+1..N}^cpu of Eq. 6 (include/vla_cpu.h), on the host cores:
parity with the float64 oracle block by block (prefill and decode, with and without GQA,
random RMSNorm gains), the partition identity, causal invariance, chunked prefill, and
independence from the thread count, all bit for bit where the arithmetic is the same; plus
the host-side argument checks. Runs without a GPU."""
import ctypes
import os
import shutil

import numpy as np
import pytest

import oracle
import synth
from helpers import COS_FINAL, REL_L2_BLOCK, cos_sim, rel_l2

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="nvcc not available")


@pytest.fixture(scope="module")
def vla():
    import paper_2608_14586_gb300 as v
    v.build()
    v.load()
    return v


def _cfg(vla, s, max_ctx):
    return vla.VlaConfig(hidden=s.hidden, n_heads=s.n_heads, n_kv_heads=s.n_kv_heads, head_dim=s.head_dim,
                         ffn=s.ffn, rms_eps=s.rms_eps, rope_base=s.rope_base, max_ctx=max_ctx)


def _f64(bits):
    return oracle.bf16_to_f64(bits)


class CpuModel:
    def __init__(self, vla, s, L, seed, max_ctx, gain="ones", n_threads=0, layer_begin=0):
        self.vla, self.s = vla, s
        self.bits = [synth.layer_weights(s, seed, l, gain=gain) for l in range(L)]
        self.h = vla.vla_cpu_model_create(_cfg(vla, s, max_ctx), self.bits[layer_begin:], layer_begin, n_threads)
        self.w64 = [oracle.LayerWeights.from_bf16(b) for b in self.bits]

    def run(self, x, lb, le, kv):
        y = np.empty_like(x)
        self.vla.vla_cpu_prefill(self.h, x, x.shape[0], lb, le, kv, y)
        return y

    def kv_planes(self, kv, layer, max_ctx, n):
        kp, vp = self.vla.vla_cpu_kv_data(kv, layer)
        cnt = self.s.n_kv_heads * max_ctx * self.s.head_dim
        shp = (self.s.n_kv_heads, max_ctx, self.s.head_dim)
        k = np.ctypeslib.as_array((ctypes.c_uint16 * cnt).from_address(kp)).reshape(shp)
        v = np.ctypeslib.as_array((ctypes.c_uint16 * cnt).from_address(vp)).reshape(shp)
        return _f64(k[:, :n].copy()), _f64(v[:, :n].copy())

    def close(self):
        self.vla.vla_cpu_model_destroy(self.h)


@pytest.mark.parametrize("gain", ["ones", "random"])
def test_tiny_blocks_prefill_and_decode_match_oracle(vla, gain):
    s, L, M, max_ctx = synth.TINY, 2, 64, 80
    m = CpuModel(vla, s, L, 3, max_ctx, gain=gain, n_threads=4)
    try:
        xb = synth.hidden_states(M, s.hidden, 3)
        cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)
        per_block = []
        ref = oracle.prefix_forward(_f64(xb), m.w64, 0, L, cache, s, per_block=per_block)
        kv = vla.vla_cpu_kv_create(m.h, 0, L, max_ctx)
        h = m.run(xb, 0, 1, kv)  # block by block: each block's output against the oracle's
        assert rel_l2(_f64(h), per_block[0]) < REL_L2_BLOCK
        y = m.run(h, 1, 2, kv)
        assert rel_l2(_f64(y), ref) < REL_L2_BLOCK
        assert cos_sim(_f64(y), ref) > COS_FINAL
        for l in range(L):
            k, v = m.kv_planes(kv, l, max_ctx, M)
            assert rel_l2(k, cache.k[l][:, :M]) < REL_L2_BLOCK
            assert rel_l2(v, cache.v[l][:, :M]) < REL_L2_BLOCK
        assert vla.vla_cpu_kv_length(kv) == M
        for t in range(3):  # decode steps: one token at position M + t
            xt = synth.decode_hidden(t, s.hidden, 3)
            yt = m.run(xt, 0, L, kv)
            rt = oracle.decode_step(_f64(xt), m.w64, 0, L, cache, s)
            assert rel_l2(_f64(yt), rt) < REL_L2_BLOCK
            assert cos_sim(_f64(yt), rt) > COS_FINAL
        assert vla.vla_cpu_kv_length(kv) == M + 3
        vla.vla_cpu_kv_destroy(kv)
    finally:
        m.close()


def test_gqa_7b_block_ragged_tokens_match_oracle(vla):
    """The 7B block shape (32 query heads over 8 KV heads, head_dim 128, FFN 11008 padded to
    the 64-unit gate/up tile): 53 tokens, a ragged count for every tile size, after a
    pre-filled context of 40 positions."""
    s, M, p0 = synth.B7, 53, 40
    max_ctx = p0 + M
    m = CpuModel(vla, s, 1, 11, max_ctx, gain="random")
    try:
        kb, vb = synth.random_kv(p0, s, 11, 0)
        kv = _cache_with_context(vla, m, s, max_ctx, kb, vb)
        xb = synth.hidden_states(M, s.hidden, 11, 20, 2.0)
        rows = [0, 1, 5, 17, 30, 47, 52]
        ref, k_new, v_new = oracle.block_forward_rows(_f64(xb), m.w64[0], s, rows, p0=p0, ctx_k=_f64(kb),
                                                      ctx_v=_f64(vb))
        y = m.run(xb, 0, 1, kv)
        got = _f64(y[rows])
        for i in range(len(rows)):
            assert rel_l2(got[i], ref[i]) < REL_L2_BLOCK, rows[i]
        assert cos_sim(got, ref) > COS_FINAL
        k, v = m.kv_planes(kv, 0, max_ctx, max_ctx)
        assert rel_l2(k[:, p0:], k_new) < REL_L2_BLOCK
        assert rel_l2(v[:, p0:], v_new) < REL_L2_BLOCK
        assert vla.vla_cpu_kv_length(kv) == max_ctx
        vla.vla_cpu_kv_destroy(kv)
    finally:
        m.close()


@pytest.mark.parametrize("shape", [
    # 2 query heads per KV head, head_dim 64, FFN 700 (padded to 704: a partial gate/up unit)
    synth.ModelShape(hidden=256, n_heads=8, n_kv_heads=4, head_dim=64, ffn=700),
    # 8 query heads per KV head, head_dim 128, FFN 520 (padded to 576)
    synth.ModelShape(hidden=512, n_heads=16, n_kv_heads=2, head_dim=128, ffn=520),
], ids=["gqa2_dh64", "gqa8_dh128"])
def test_other_head_groupings_match_oracle(vla, shape):
    """The other supported query-per-KV-head groupings and an FFN width that is not a
    multiple of the gate/up unit: two blocks over 29 tokens, then two decode steps."""
    s, L, M, max_ctx = shape, 2, 29, 40
    m = CpuModel(vla, s, L, 13, max_ctx, gain="random", n_threads=3)
    try:
        xb = synth.hidden_states(M, s.hidden, 13)
        cache = oracle.KVCache(range(L), s.n_kv_heads, s.head_dim, max_ctx)
        per_block = []
        ref = oracle.prefix_forward(_f64(xb), m.w64, 0, L, cache, s, per_block=per_block)
        kv = vla.vla_cpu_kv_create(m.h, 0, L, max_ctx)
        h = m.run(xb, 0, 1, kv)
        assert rel_l2(_f64(h), per_block[0]) < REL_L2_BLOCK
        y = m.run(h, 1, L, kv)
        assert rel_l2(_f64(y), ref) < REL_L2_BLOCK
        assert cos_sim(_f64(y), ref) > COS_FINAL
        for l in range(L):
            k, v = m.kv_planes(kv, l, max_ctx, M)
            assert rel_l2(k, cache.k[l][:, :M]) < REL_L2_BLOCK
            assert rel_l2(v, cache.v[l][:, :M]) < REL_L2_BLOCK
        for t in range(2):
            xt = synth.decode_hidden(t, s.hidden, 13)
            yt = m.run(xt, 0, L, kv)
            rt = oracle.decode_step(_f64(xt), m.w64, 0, L, cache, s)
            assert rel_l2(_f64(yt), rt) < REL_L2_BLOCK
        assert vla.vla_cpu_kv_length(kv) == M + 2
        vla.vla_cpu_kv_destroy(kv)
    finally:
        m.close()


def _cache_with_context(vla, m, s, max_ctx, kb, vb):
    """A host cache whose positions [0, p0) hold the given K/V bits: a p0-token prefill sets
    the length, then its K/V rows are overwritten with the given ones."""
    p0 = kb.shape[1]
    kv = vla.vla_cpu_kv_create(m.h, 0, 1, max_ctx)
    m.run(np.zeros((p0, s.hidden), dtype=np.uint16), 0, 1, kv)
    kp, vp = vla.vla_cpu_kv_data(kv, 0)
    cnt = s.n_kv_heads * max_ctx * s.head_dim
    K = np.ctypeslib.as_array((ctypes.c_uint16 * cnt).from_address(kp)).reshape(s.n_kv_heads, max_ctx, -1)
    V = np.ctypeslib.as_array((ctypes.c_uint16 * cnt).from_address(vp)).reshape(s.n_kv_heads, max_ctx, -1)
    K[:, :p0] = kb
    V[:, :p0] = vb
    assert vla.vla_cpu_kv_length(kv) == p0
    return kv


def test_partition_identity_in_place_and_thread_count(vla):
    """[0, 3) equals [0, 1) then [1, 3) (Eq. 6), in place as well, and 1 thread equals 3."""
    s, L, M, max_ctx = synth.TINY, 3, 57, 64
    m1 = CpuModel(vla, s, L, 5, max_ctx, n_threads=1)
    m3 = CpuModel(vla, s, L, 5, max_ctx, n_threads=3)
    try:
        assert vla.vla_cpu_model_threads(m1.h) == 1 and vla.vla_cpu_model_threads(m3.h) == 3
        xb = synth.hidden_states(M, s.hidden, 5)
        kv_a = vla.vla_cpu_kv_create(m3.h, 0, L, max_ctx)
        y_full = m3.run(xb, 0, L, kv_a)
        kv_b = vla.vla_cpu_kv_create(m3.h, 0, L, max_ctx)
        buf = xb.copy()
        vla.vla_cpu_prefill(m3.h, buf, M, 0, 1, kv_b, buf)  # in place
        vla.vla_cpu_prefill(m3.h, buf, M, 1, L, kv_b, buf)
        np.testing.assert_array_equal(buf, y_full)
        kv_c = vla.vla_cpu_kv_create(m1.h, 0, L, max_ctx)
        np.testing.assert_array_equal(m1.run(xb, 0, L, kv_c), y_full)
        for kv in (kv_a, kv_b):
            vla.vla_cpu_kv_destroy(kv)
        vla.vla_cpu_kv_destroy(kv_c)
    finally:
        m1.close()
        m3.close()


def test_causal_invariance_and_chunked_prefill(vla):
    """Rows of a prefix of the frame do not depend on later tokens, and a frame prefilled in
    chunks (each at p0 = the previous chunks' length) equals one call, bit for bit, also
    through the weight-streaming path of calls of at most 4 tokens (decode steps)."""
    s, L, M, M1, max_ctx = synth.TINY, 2, 64, 37, 64
    m = CpuModel(vla, s, L, 8, max_ctx, n_threads=4)
    try:
        xb = synth.hidden_states(M, s.hidden, 8)
        kv = vla.vla_cpu_kv_create(m.h, 0, L, max_ctx)
        y = m.run(xb, 0, L, kv)
        vla.vla_cpu_kv_reset(kv)
        assert vla.vla_cpu_kv_length(kv) == 0
        y1 = m.run(xb[:M1].copy(), 0, L, kv)
        np.testing.assert_array_equal(y1, y[:M1])
        y2 = m.run(xb[M1:].copy(), 0, L, kv)
        np.testing.assert_array_equal(y2, y[M1:])
        vla.vla_cpu_kv_reset(kv)
        m.run(xb[:M1].copy(), 0, L, kv)
        for a, b in ((M1, M1 + 3), (M1 + 3, M1 + 4), (M1 + 4, M)):
            np.testing.assert_array_equal(m.run(xb[a:b].copy(), 0, L, kv), y[a:b])
        vla.vla_cpu_kv_destroy(kv)
    finally:
        m.close()


def test_model_over_a_suffix_range_and_argument_errors(vla):
    s, max_ctx = synth.TINY, 32
    lib = vla.load()
    m = CpuModel(vla, s, 3, 2, max_ctx, layer_begin=1)  # blocks [1, 3) only
    try:
        cfg, lb, le = vla.vla_cpu_model_info(m.h)
        assert (lb, le, cfg.hidden, cfg.max_ctx) == (1, 3, s.hidden, max_ctx)
        x = synth.hidden_states(16, s.hidden, 2)
        y = np.empty_like(x)

        def status(fn, *a):
            with pytest.raises(vla.VlaError) as ei:
                fn(*a)
            return ei.value.name

        assert status(vla.vla_cpu_kv_create, m.h, 0, 2, max_ctx) == "VLA_ERR_RANGE"     # block 0 not held
        assert status(vla.vla_cpu_kv_create, m.h, 1, 3, max_ctx + 1) == "VLA_ERR_SHAPE"
        kv = vla.vla_cpu_kv_create(m.h, 1, 3, max_ctx)
        assert status(vla.vla_cpu_prefill, m.h, x, 16, 0, 2, kv, y) == "VLA_ERR_RANGE"
        assert status(vla.vla_cpu_prefill, m.h, x, 16, 2, 1, kv, y) == "VLA_ERR_RANGE"
        assert status(vla.vla_cpu_prefill, m.h, x, 33, 1, 3, kv, y) == "VLA_ERR_SHAPE"
        vla.vla_cpu_prefill(m.h, x, 16, 1, 2, kv, y)                                  # block 1 alone
        assert status(vla.vla_cpu_prefill, m.h, x, 16, 1, 3, kv, y) == "VLA_ERR_RANGE"  # unequal lengths
        vla.vla_cpu_prefill(m.h, y, 16, 2, 3, kv, y)
        assert vla.vla_cpu_kv_length(kv) == 16
        x17 = synth.hidden_states(17, s.hidden, 2)
        assert status(vla.vla_cpu_prefill, m.h, x17, 17, 1, 3, kv, np.empty_like(x17)) == "VLA_ERR_KV_FULL"
        z = np.empty_like(x)
        vla.vla_cpu_prefill(m.h, x, 16, 2, 2, None, z)  # empty range: a copy, no cache needed
        np.testing.assert_array_equal(z, x)
        out = ctypes.c_void_p(7)
        assert lib.vla_cpu_model_create(None, None, 0, 1, 0, ctypes.byref(out)) == 1 and out.value is None
        assert lib.vla_cpu_prefill(None, None, 1, 0, 1, None, None) == 1
        assert lib.vla_cpu_model_destroy(None) == 0 and lib.vla_cpu_kv_destroy(None) == 0
        assert lib.vla_cpu_kv_length(None) == -1 and lib.vla_cpu_model_threads(None) == -1
        assert lib.vla_pipeline_create(None, None, 1, 1, ctypes.byref(out)) == 1
        assert lib.vla_pipeline_destroy(None) == 0 and lib.vla_pipeline_in_flight(None) == -1
        assert lib.vla_pipeline_collect(None, None, None, 0, None) == 1
        assert lib.vla_status_str(10) == b"all pipeline slots in flight"
        w1 = [synth.layer_weights(s, 2, 0)]
        for bad in (dict(head_dim=96),                     # head_dim other than 64 / 128
                    dict(n_heads=6, n_kv_heads=4),         # query heads not a multiple of KV heads
                    dict(n_heads=12, n_kv_heads=4),        # 3 query heads per KV head
                    dict(hidden=320)):                     # hidden not a multiple of 256
            c = _cfg(vla, s, max_ctx)
            for k, v in bad.items():
                setattr(c, k, v)
            assert status(vla.vla_cpu_model_create, c, w1, 0) == "VLA_ERR_UNSUPPORTED", bad
        c = _cfg(vla, s, max_ctx)
        c.rope_base = 1.0
        assert status(vla.vla_cpu_model_create, c, w1, 0) == "VLA_ERR_INVALID_ARG"
        vla.vla_cpu_kv_destroy(kv)
    finally:
        m.close()
