"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each test fixes one part of the oracle with a closed form, a hand-worked example
(``tests/golden``), an invariant or brute force, chosen so that a plausible slip (a dropped
term, a wrong sign or index, a transposed operand, a swapped gate/up) fails at least one.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from oracle import KVCache, LayerWeights

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


class Shape:
    def __init__(self, hidden, n_heads, n_kv_heads, head_dim, ffn, rms_eps=1e-6, rope_base=10000.0):
        self.hidden, self.n_heads, self.n_kv_heads = hidden, n_heads, n_kv_heads
        self.head_dim, self.ffn, self.rms_eps, self.rope_base = head_dim, ffn, rms_eps, rope_base


def _rand_layer(rng, s: Shape, std=0.3, gains=False):
    D, H, Hkv, dh, F = s.hidden, s.n_heads, s.n_kv_heads, s.head_dim, s.ffn
    g = (lambda: 1.0 + 0.2 * rng.standard_normal(D)) if gains else (lambda: np.ones(D))
    return LayerWeights(w_q=std * rng.standard_normal((H * dh, D)), w_k=std * rng.standard_normal((Hkv * dh, D)),
                        w_v=std * rng.standard_normal((Hkv * dh, D)), w_o=std * rng.standard_normal((D, H * dh)),
                        w_gate=std * rng.standard_normal((F, D)), w_up=std * rng.standard_normal((F, D)),
                        w_down=std * rng.standard_normal((D, F)), g_attn=g(), g_mlp=g())


# --------------------------------------------------------------------------------------
# bf16 encoding
# --------------------------------------------------------------------------------------
def test_bf16_decode_known_patterns():
    bits = np.array([0x3F80, 0xC000, 0x3F81, 0x0000, 0x4049, 0xBE80], dtype=np.uint16)
    exp = [1.0, -2.0, 1.0 + 2.0 ** -7, 0.0, 3.140625, -0.25]
    assert oracle.bf16_to_f64(bits).tolist() == exp


def test_bf16_round_ties_to_even():
    x = np.array([1.0 + 2.0 ** -8,        # halfway 0x3F80 / 0x3F81 -> even 0x3F80
                  1.0 + 3 * 2.0 ** -8,    # halfway 0x3F81 / 0x3F82 -> even 0x3F82
                  1.0 + 2.0 ** -8 + 2.0 ** -30,  # just above halfway -> up
                  -3.0, 0.0, 2.0 ** -100])
    assert oracle.to_bf16_bits(x).tolist() == [0x3F80, 0x3F82, 0x3F81, 0xC040, 0x0000, 0x0D80]


# --------------------------------------------------------------------------------------
# RMSNorm
# --------------------------------------------------------------------------------------
def test_rmsnorm_unit_rms_and_gain():
    rng = np.random.default_rng(1)
    x = 3.0 * rng.standard_normal((7, 64))
    u = oracle.rms_norm(x, np.ones(64), 1e-6)
    np.testing.assert_allclose(np.sqrt(np.mean(u * u, axis=1)), 1.0, rtol=1e-6)
    g = rng.standard_normal(64)
    np.testing.assert_allclose(oracle.rms_norm(x, g, 1e-6), u * g, rtol=1e-13)
    # scale invariance (per row)
    np.testing.assert_allclose(oracle.rms_norm(5.0 * x, np.ones(64), 1e-6), u, rtol=1e-6)


def test_rmsnorm_eps_inside_sqrt_closed_form():
    # constant row c: out = c / sqrt(c^2 + eps); c = 1e-3, eps = 1e-6 -> 1/sqrt(2)
    x = np.full((1, 16), 1e-3)
    u = oracle.rms_norm(x, np.ones(16), 1e-6)
    np.testing.assert_allclose(u, 1.0 / math.sqrt(2.0), rtol=1e-14)
    assert np.all(oracle.rms_norm(np.zeros((2, 8)), np.ones(8), 1e-6) == 0.0)


# --------------------------------------------------------------------------------------
# Rotary embedding
# --------------------------------------------------------------------------------------
def test_rope_closed_form_rotate_half():
    # d_h = 8, base 10^4: theta_j = 10^4^(-2j/8) = 10^-j. Unit vector e_j at position p
    # moves to cos(p theta_j) e_j + sin(p theta_j) e_{j+4}; e_{j+4} to -sin e_j + cos e_{j+4}.
    p = 3
    for j in range(4):
        th = 10.0 ** (-j)
        e = np.zeros((1, 1, 8)); e[0, 0, j] = 1.0
        r = oracle.apply_rope(e, np.array([p]), 10000.0)[0, 0]
        exp = np.zeros(8); exp[j] = math.cos(p * th); exp[j + 4] = math.sin(p * th)
        np.testing.assert_allclose(r, exp, atol=1e-15)
        e = np.zeros((1, 1, 8)); e[0, 0, j + 4] = 1.0
        r = oracle.apply_rope(e, np.array([p]), 10000.0)[0, 0]
        exp = np.zeros(8); exp[j] = -math.sin(p * th); exp[j + 4] = math.cos(p * th)
        np.testing.assert_allclose(r, exp, atol=1e-15)


def test_rope_identity_norm_and_relative_position():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((5, 3, 128))
    np.testing.assert_array_equal(oracle.apply_rope(x, np.zeros(5, dtype=int), 1e4), x)
    pos = np.array([0, 1, 7, 100, 3000])
    r = oracle.apply_rope(x, pos, 1e4)
    n0 = x[..., :64] ** 2 + x[..., 64:] ** 2
    n1 = r[..., :64] ** 2 + r[..., 64:] ** 2
    np.testing.assert_allclose(n1, n0, rtol=1e-12)
    q = rng.standard_normal((1, 1, 128)); k = rng.standard_normal((1, 1, 128))
    def score(m, n):
        return float(np.sum(oracle.apply_rope(q, np.array([m]), 1e4) * oracle.apply_rope(k, np.array([n]), 1e4)))
    assert score(10, 4) == pytest.approx(score(1006, 1000), rel=1e-10)
    assert score(10, 4) != pytest.approx(score(10, 5), rel=1e-3)


# --------------------------------------------------------------------------------------
# Attention
# --------------------------------------------------------------------------------------
def _brute_attention(q, k, v, q_pos, n_kv):
    """Scalar loops: o[i,h,:] = sum_j w_j v[g,j,:] with w the masked softmax."""
    M, H, dh = q.shape
    out = np.zeros_like(q)
    for i in range(M):
        for h in range(H):
            g = h // (H // n_kv)
            scores = []
            for j in range(int(q_pos[i]) + 1):
                s = 0.0
                for d in range(dh):
                    s += q[i, h, d] * k[g, j, d]
                scores.append(s / math.sqrt(dh))
            mx = max(scores)
            ex = [math.exp(s - mx) for s in scores]
            tot = sum(ex)
            for j, e in enumerate(ex):
                for d in range(dh):
                    out[i, h, d] += e / tot * v[g, j, d]
    return out


def test_attention_golden_two_tokens():
    with open(os.path.join(GOLDEN, "attention_2tok.json")) as f:
        g = json.load(f)
    q, k, v = np.array(g["q"]), np.array(g["k"]), np.array(g["v"])
    o = oracle.causal_gqa_attention(q, k, v, np.array(g["q_pos"]), 1)
    np.testing.assert_allclose(o, np.array(g["expected_o"]), atol=1e-14)
    w = oracle.attention_weights(q, k, np.array(g["q_pos"]), 1)
    np.testing.assert_allclose(w[0, 1], g["expected_w_row1"], atol=1e-15)


@pytest.mark.parametrize("H,Hkv,p0", [(4, 2, 0), (4, 4, 0), (4, 1, 0), (6, 2, 3)])
def test_attention_brute_force(H, Hkv, p0):
    rng = np.random.default_rng(3 + H + Hkv + p0)
    M, dh = 5, 4
    ctx = p0 + M
    q = rng.standard_normal((M, H, dh)); k = rng.standard_normal((Hkv, ctx, dh)); v = rng.standard_normal((Hkv, ctx, dh))
    pos = p0 + np.arange(M)
    np.testing.assert_allclose(oracle.causal_gqa_attention(q, k, v, pos, Hkv),
                               _brute_attention(q, k, v, pos, Hkv), rtol=1e-12, atol=1e-13)


def test_attention_rows_sum_to_one_and_mask():
    rng = np.random.default_rng(4)
    M, H, Hkv, dh = 9, 8, 2, 16
    q = 4 * rng.standard_normal((M, H, dh)); k = rng.standard_normal((Hkv, M, dh))
    w = oracle.attention_weights(q, k, np.arange(M), Hkv)
    np.testing.assert_allclose(w.sum(axis=2), 1.0, rtol=1e-14)
    assert np.all(w[:, np.triu_indices(M, 1)[0], np.triu_indices(M, 1)[1]] == 0.0)


def test_attention_gqa_equals_mha_with_repeated_kv():
    rng = np.random.default_rng(5)
    M, H, Hkv, dh = 6, 8, 2, 8
    q = rng.standard_normal((M, H, dh)); k = rng.standard_normal((Hkv, M, dh)); v = rng.standard_normal((Hkv, M, dh))
    pos = np.arange(M)
    krep = np.repeat(k, H // Hkv, axis=0); vrep = np.repeat(v, H // Hkv, axis=0)
    np.testing.assert_allclose(oracle.causal_gqa_attention(q, k, v, pos, Hkv),
                               oracle.causal_gqa_attention(q, krep, vrep, pos, H), rtol=1e-14)


def test_attention_constant_keys_give_running_mean():
    rng = np.random.default_rng(6)
    M, dh = 7, 4
    q = rng.standard_normal((M, 1, dh)); k = np.tile(rng.standard_normal((1, 1, dh)), (1, M, 1))
    v = rng.standard_normal((1, M, dh))
    o = oracle.causal_gqa_attention(q, k, v, np.arange(M), 1)
    run = np.cumsum(v[0], axis=0) / np.arange(1, M + 1)[:, None]
    np.testing.assert_allclose(o[:, 0], run, rtol=1e-13)


# --------------------------------------------------------------------------------------
# SwiGLU
# --------------------------------------------------------------------------------------
def test_silu_closed_forms():
    z = np.array([0.0, 1.0, -1.0, 40.0, -40.0])
    e = math.e
    exp = [0.0, e / (1 + e), -1 / (1 + e), 40.0, -40.0 * math.exp(-40.0) / (1 + math.exp(-40.0))]
    np.testing.assert_allclose(oracle.silu(z), exp, rtol=1e-14, atol=1e-300)
    np.testing.assert_allclose(oracle.swiglu(np.array([1.0]), np.array([3.0])), [3 * e / (1 + e)], rtol=1e-15)


# --------------------------------------------------------------------------------------
# Whole block: special cases with closed forms
# --------------------------------------------------------------------------------------
def _perm(n, shift):
    """Matrix P with (x @ P.T)[i] = x[(i + shift) % n], i.e. P[i, (i+shift) % n] = 1."""
    p = np.zeros((n, n))
    p[np.arange(n), (np.arange(n) + shift) % n] = 1.0
    return p


def test_block_zero_projections_is_identity():
    s = Shape(16, 2, 1, 8, 24)
    rng = np.random.default_rng(7)
    w = _rand_layer(rng, s)
    w.w_o[:] = 0.0
    w.w_down[:] = 0.0
    x = rng.standard_normal((5, 16))
    cache = KVCache([0], 1, 8, 16)
    np.testing.assert_array_equal(oracle.block_forward(x, w, cache, 0, s), x)
    assert cache.length[0] == 5


def test_block_attention_path_closed_form():
    # W_q = W_k = 0: scores are all 0, so row i averages v over positions 0..i.
    # H = H_kv = 2, d_h = 4, D = 8; W_v = P_1 (shift), W_o = P_3, W_down = 0.
    # The rotary embedding does not touch v, so y_i = x_i + roll(mean_{j<=i} roll(u_j, 1), 3).
    s = Shape(8, 2, 2, 4, 8)
    rng = np.random.default_rng(8)
    w = _rand_layer(rng, s, gains=True)
    w.w_q[:] = 0.0; w.w_k[:] = 0.0
    w.w_v = _perm(8, 1); w.w_o = _perm(8, 3); w.w_down[:] = 0.0
    x = rng.standard_normal((6, 8))
    u = x / np.sqrt(np.mean(x ** 2, axis=1, keepdims=True) + 1e-6) * w.g_attn
    vrows = np.roll(u, -1, axis=1)  # vrows[:, i] = u[:, i+1]
    run = np.cumsum(vrows, axis=0) / np.arange(1, 7)[:, None]
    exp = x + np.roll(run, -3, axis=1)
    y = oracle.block_forward(x, w, KVCache([0], 2, 4, 8), 0, s)
    np.testing.assert_allclose(y, exp, rtol=1e-12, atol=1e-12)


def test_block_mlp_path_closed_form():
    # Attention contributes 0 (W_o = 0). W_gate = c*I, W_up = P_2, W_down = P_5 (F = D):
    # m = silu(c u) * roll(u, -2); y = x + roll(m, -5).
    s = Shape(8, 2, 2, 4, 8)
    rng = np.random.default_rng(9)
    w = _rand_layer(rng, s, gains=True)
    w.w_o[:] = 0.0
    c = 1.7
    w.w_gate = c * np.eye(8); w.w_up = _perm(8, 2); w.w_down = _perm(8, 5)
    x = rng.standard_normal((4, 8))
    u = x / np.sqrt(np.mean(x ** 2, axis=1, keepdims=True) + 1e-6) * w.g_mlp
    m = (c * u) / (1.0 + np.exp(-c * u)) * np.roll(u, -2, axis=1)
    exp = x + np.roll(m, -5, axis=1)
    y = oracle.block_forward(x, w, KVCache([0], 2, 4, 8), 0, s)
    np.testing.assert_allclose(y, exp, rtol=1e-12, atol=1e-12)


def test_block_scores_depend_on_relative_position():
    # Identical rows -> identical unrotated q, k; after the rotary embedding the score
    # q_i . k_j depends on i - j only (and does vary with it).
    s = Shape(32, 2, 1, 16, 48)
    rng = np.random.default_rng(10)
    w = _rand_layer(rng, s)
    x = np.tile(rng.standard_normal((1, 32)), (6, 1))
    taps = {}
    oracle.block_forward(x, w, KVCache([0], 1, 16, 8), 0, s, taps=taps)
    q, k = taps["q"][:, 0], taps["k"][:, 0]
    for i in range(5):
        for j in range(i + 1):
            assert q[i] @ k[j] == pytest.approx(q[i + 1] @ k[j + 1], rel=1e-9, abs=1e-12)
    assert abs(q[3] @ k[0] - q[3] @ k[3]) > 1e-3


def test_block_kv_cache_holds_rotated_keys_and_values():
    s = Shape(16, 4, 2, 4, 24)
    rng = np.random.default_rng(11)
    w = _rand_layer(rng, s)
    x = rng.standard_normal((3, 16))
    cache = KVCache([0], 2, 4, 8)
    taps = {}
    oracle.block_forward(x, w, cache, 0, s, taps=taps)
    u = oracle.rms_norm(x, w.g_attn, 1e-6)
    vexp = (u @ w.w_v.T).reshape(3, 2, 4)
    np.testing.assert_allclose(cache.v[0][:, :3], vexp.transpose(1, 0, 2), rtol=1e-13)
    kun = (u @ w.w_k.T).reshape(3, 2, 4)
    # the rotation keeps each (j, j + 2) pair's norm; position 0 is unrotated
    np.testing.assert_allclose(cache.k[0][:, 0], kun[0], rtol=1e-13)
    kc = cache.k[0][:, :3].transpose(1, 0, 2)
    np.testing.assert_allclose(kc[..., :2] ** 2 + kc[..., 2:] ** 2, kun[..., :2] ** 2 + kun[..., 2:] ** 2, rtol=1e-12)
    assert np.all(cache.k[0][:, 3:] == 0.0)


# --------------------------------------------------------------------------------------
# Prefix-level invariants (Eq. 5, Eq. 6)
# --------------------------------------------------------------------------------------
def _stack(seed, s, L):
    rng = np.random.default_rng(seed)
    return [_rand_layer(rng, s, std=0.15, gains=True) for _ in range(L)]


def test_partition_identity_bit_exact():
    s = Shape(32, 4, 2, 8, 40)
    ws = _stack(12, s, 3)
    x = np.random.default_rng(13).standard_normal((7, 32))
    c_full = KVCache(range(3), 2, 8, 16)
    full = oracle.prefix_forward(x, ws, 0, 3, c_full, s)
    for k in (0, 1, 2, 3):
        c = KVCache(range(3), 2, 8, 16)
        h = oracle.prefix_forward(x, ws, 0, k, c, s)
        h = oracle.boundary_transfer(h)
        y = oracle.prefix_forward(h, ws, k, 3, c, s)
        np.testing.assert_array_equal(y, full)
        for l in range(3):
            np.testing.assert_array_equal(c.k[l], c_full.k[l])
            np.testing.assert_array_equal(c.v[l], c_full.v[l])


def test_block_rows_equals_full_block_at_those_rows():
    """The sampled-row evaluation used for full-size parity is the full block restricted to
    some query rows: same outputs at those rows and the same cache entries, with and without
    context before p0."""
    s = Shape(32, 4, 2, 8, 40)
    w = _stack(21, s, 1)[0]
    x = np.random.default_rng(22).standard_normal((11, 32))
    rows = [0, 3, 4, 10]
    c = KVCache([0], 2, 8, 32)
    full = oracle.block_forward(x, w, c, 0, s)
    y, k, v = oracle.block_forward_rows(x, w, s, rows)
    np.testing.assert_allclose(y, full[rows], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(k, c.k[0][:, :11], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(v, c.v[0][:, :11], rtol=1e-12, atol=1e-12)
    x2 = np.random.default_rng(23).standard_normal((5, 32))
    full2 = oracle.block_forward(x2, w, c, 0, s)  # positions 11..15 after the first call
    y2, k2, _ = oracle.block_forward_rows(x2, w, s, [1, 4], p0=11, ctx_k=c.k[0], ctx_v=c.v[0])
    np.testing.assert_allclose(y2, full2[[1, 4]], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(k2, c.k[0][:, 11:16], rtol=1e-12, atol=1e-12)


def test_empty_range_returns_input():
    s = Shape(16, 2, 1, 8, 24)
    x = np.random.default_rng(14).standard_normal((3, 16))
    y = oracle.prefix_forward(x, _stack(15, s, 1), 1, 1, KVCache([0], 1, 8, 8), s)
    np.testing.assert_array_equal(y, x)


def test_causal_invariance_appending_tokens():
    s = Shape(32, 4, 2, 8, 40)
    ws = _stack(16, s, 2)
    x = np.random.default_rng(17).standard_normal((9, 32))
    a = oracle.prefix_forward(x[:5], ws, 0, 2, KVCache(range(2), 2, 8, 16), s)
    cb = KVCache(range(2), 2, 8, 16)
    b = oracle.prefix_forward(x, ws, 0, 2, cb, s)
    np.testing.assert_allclose(b[:5], a, rtol=1e-12, atol=1e-12)


def test_prefill_then_decode_equals_longer_prefill():
    s = Shape(32, 4, 2, 8, 40)
    ws = _stack(18, s, 2)
    x = np.random.default_rng(19).standard_normal((6, 32))
    full = oracle.prefix_forward(x, ws, 0, 2, KVCache(range(2), 2, 8, 16), s)
    c = KVCache(range(2), 2, 8, 16)
    oracle.prefix_forward(x[:4], ws, 0, 2, c, s)
    y4 = oracle.decode_step(x[4:5], ws, 0, 2, c, s)
    y5 = oracle.decode_step(x[5:6], ws, 0, 2, c, s)
    np.testing.assert_allclose(y4[0], full[4], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(y5[0], full[5], rtol=1e-11, atol=1e-12)
    assert c.length == {0: 6, 1: 6}


def test_kv_fill_seeds_context_like_a_prefill():
    """A cache seeded by fill() with a prefill's own keys and values continues exactly like
    the cache that prefill wrote: a decode step after it equals the longer prefill's row."""
    s = Shape(32, 4, 2, 8, 40)
    ws = _stack(24, s, 2)
    x = np.random.default_rng(25).standard_normal((6, 32))
    full = oracle.prefix_forward(x, ws, 0, 2, KVCache(range(2), 2, 8, 16), s)
    c = KVCache(range(2), 2, 8, 16)
    oracle.prefix_forward(x[:5], ws, 0, 2, c, s)
    seeded = KVCache(range(2), 2, 8, 16)
    for l in range(2):
        seeded.fill(l, c.k[l][:, :5].copy(), c.v[l][:, :5].copy())
    assert seeded.length == {0: 5, 1: 5}
    y = oracle.decode_step(x[5:6], ws, 0, 2, seeded, s)
    np.testing.assert_allclose(y[0], full[5], rtol=1e-11, atol=1e-12)


def test_kv_fill_closed_form_uniform_attention():
    # W_q = W_k = 0 and every seeded key 0: the decode query at position n attends uniformly
    # to the n seeded positions and its own. Seeded values v_j = (j + 1) * e_{(j mod d_h)} in
    # KV head 0 and 0 in head 1; W_v = 0, so the new value is 0. With W_o = I and W_down = 0,
    # y = x + concat(o_head0, o_head0, o_head1...) where o for query heads 0, 1 (KV head 0)
    # is sum_j v_j / (n + 1), and 0 for query heads 2, 3 (KV head 1).
    s = Shape(32, 4, 2, 8, 40)
    rng = np.random.default_rng(26)
    w = _rand_layer(rng, s)
    w.w_q[:] = 0.0; w.w_k[:] = 0.0; w.w_v[:] = 0.0
    w.w_o = np.eye(32); w.w_down[:] = 0.0
    n = 11
    kseed = np.zeros((2, n, 8))
    vseed = np.zeros((2, n, 8))
    for j in range(n):
        vseed[0, j, j % 8] = j + 1.0
    cache = KVCache([0], 2, 8, 16)
    cache.fill(0, kseed, vseed)
    x = rng.standard_normal((1, 32))
    y = oracle.decode_step(x, [w], 0, 1, cache, s)
    o0 = np.zeros(8)
    for j in range(n):
        o0[j % 8] += (j + 1.0) / (n + 1)
    exp = x[0] + np.concatenate([o0, o0, np.zeros(16)])
    np.testing.assert_allclose(y[0], exp, rtol=1e-12, atol=1e-12)
    assert cache.length[0] == n + 1
    np.testing.assert_array_equal(cache.v[0][:, :n], vseed)


def test_kv_full_raises():
    s = Shape(16, 2, 1, 8, 24)
    with pytest.raises(ValueError):
        oracle.block_forward(np.zeros((5, 16)), _stack(20, s, 1)[0], KVCache([0], 1, 8, 4), 0, s)


def test_boundary_bytes_eq11_golden():
    with open(os.path.join(GOLDEN, "boundary_bytes.json")) as f:
        g = json.load(f)
    for c in g["cases"]:
        assert oracle.boundary_bytes(c["B"], c["L_p"], c["D"], c["b"]) == c["bytes"]
