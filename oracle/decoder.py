"""Float64 reference of the GPU-resident LLM prefix (test infrastructure only).

Notation follows the paper where it has notation: blocks B_1..B_N, partition point p,
boundary hidden state h^(p) (Eq. 5), the partitioned model F_p (Eq. 6) and the boundary
size S_hid = B * L_p * D * b (Eq. 11). Inside a block (which the paper leaves undefined,
Sec. IV-B) the symbols are D (hidden), H (query heads), H_kv (key/value heads), d_h (head
dim), F (feed-forward width), M (tokens in the call), p0 (first position of the call).

Readings of points the paper leaves open (each listed in the design notes):
  * RMSNorm: x / sqrt(mean(x^2) + eps) * gain, eps inside the square root.
  * Rotary embedding: rotate-half pairing (j, j + d_h/2), theta_j = base^(-2j/d_h),
    positions counted from 0 at the first token of the frame, angles in float64.
  * Attention: strictly causal over the whole multimodal sequence, scale 1/sqrt(d_h),
    query head h reads key/value head floor(h / (H / H_kv)).
  * MLP: SwiGLU, m = silu(u W_gate^T) * (u W_up^T), silu(z) = z / (1 + e^-z).
  * Block output is the residual stream (no final norm: the head belongs to the suffix).
No stage is blocked, fused or reordered; numpy's matmul is the only library step.
"""
from __future__ import annotations

import dataclasses

import numpy as np


# ---------------------------------------------------------------------------------------
# bf16 <-> float64 (input/output encoding; bf16 = top 16 bits of an IEEE binary32)
# ---------------------------------------------------------------------------------------
def bf16_to_f64(bits) -> np.ndarray:
    """Exact float64 value of bf16 bit patterns (uint16)."""
    b = np.asarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def to_bf16_bits(x) -> np.ndarray:
    """Round float64 values to the nearest bf16 (ties to even) and return the bit patterns.

    bf16 keeps 8 significant bits: with x = m * 2^e, 0.5 <= |m| < 1, the rounded value is
    rint(m * 2^8) * 2^(e-8) (numpy's rint rounds ties to even). Finite, normal range only.
    """
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)
    y = np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)
    return (y.astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


# ---------------------------------------------------------------------------------------
# Block stages
# ---------------------------------------------------------------------------------------
def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """Pre-norm of the block (the "normalization" stage named in Sec. IV-B).

    u_i = x_i / sqrt(mean_d(x_id^2) + eps) * gain, over the last axis.
    """
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * gain


def rope_cos_sin(positions: np.ndarray, head_dim: int, base: float):
    """cos / sin of the rotary angles pos * theta_j, theta_j = base^(-2j/d_h), j < d_h/2."""
    half = head_dim // 2
    j = np.arange(half, dtype=np.float64)
    theta = np.power(float(base), -2.0 * j / head_dim)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * theta[None, :]
    return np.cos(ang), np.sin(ang)


def apply_rope(x: np.ndarray, positions: np.ndarray, base: float) -> np.ndarray:
    """Rotate-half rotary embedding of x [M, n_heads, d_h] at positions [M].

    The pair (a, b) = (x[..., j], x[..., j + d_h/2]) becomes
    (a cos - b sin, b cos + a sin) with angle positions * theta_j.
    """
    dh = x.shape[-1]
    half = dh // 2
    c, s = rope_cos_sin(positions, dh, base)
    c = c[:, None, :]
    s = s[:, None, :]
    a = x[..., :half]
    b = x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def attention_weights(q: np.ndarray, k: np.ndarray, q_pos: np.ndarray, n_kv_heads: int):
    """Softmax weights of causal grouped-query attention.

    q [M, H, d_h]; k [H_kv, ctx, d_h] (cache positions 0..ctx-1); q_pos [M] absolute
    positions of the queries. Returns w [H, M, ctx] with w[h, i, j] = 0 for j > q_pos[i].
    """
    M, H, dh = q.shape
    ctx = k.shape[1]
    group = H // n_kv_heads
    w = np.zeros((H, M, ctx), dtype=np.float64)
    mask = np.arange(ctx)[None, :] > np.asarray(q_pos)[:, None]
    for h in range(H):
        g = h // group
        s = (q[:, h, :] @ k[g].T) / np.sqrt(dh)
        s = np.where(mask, -np.inf, s)
        s = s - np.max(s, axis=1, keepdims=True)
        e = np.exp(s)
        w[h] = e / np.sum(e, axis=1, keepdims=True)
    return w


def causal_gqa_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, q_pos: np.ndarray,
                         n_kv_heads: int) -> np.ndarray:
    """o[i, h] = sum_{j <= q_pos[i]} softmax_j(q_ih . k_gj / sqrt(d_h)) v_gj, g = h // (H/H_kv).

    q [M, H, d_h]; k, v [H_kv, ctx, d_h]. Returns o [M, H, d_h].
    """
    M, H, dh = q.shape
    group = H // n_kv_heads
    w = attention_weights(q, k, q_pos, n_kv_heads)
    o = np.empty((M, H, dh), dtype=np.float64)
    for h in range(H):
        o[:, h, :] = w[h] @ v[h // group]
    return o


def silu(z: np.ndarray) -> np.ndarray:
    """silu(z) = z / (1 + e^-z)."""
    return z / (1.0 + np.exp(-z))


def swiglu(g: np.ndarray, u: np.ndarray) -> np.ndarray:
    """Gated feed-forward activation silu(g) * u."""
    return silu(g) * u


# ---------------------------------------------------------------------------------------
# Weights and KV cache
# ---------------------------------------------------------------------------------------
@dataclasses.dataclass
class LayerWeights:
    """One block's parameters in float64, each matrix [out, in]."""
    w_q: np.ndarray
    w_k: np.ndarray
    w_v: np.ndarray
    w_o: np.ndarray
    w_gate: np.ndarray
    w_up: np.ndarray
    w_down: np.ndarray
    g_attn: np.ndarray
    g_mlp: np.ndarray

    @staticmethod
    def from_bf16(bits: dict) -> "LayerWeights":
        return LayerWeights(**{f.name: bf16_to_f64(bits[f.name]) for f in dataclasses.fields(LayerWeights)})


class KVCache:
    """Per-layer key/value store, K[l] and V[l] of shape [H_kv, max_ctx, d_h], float64.

    Keys are stored after the rotary embedding. ``length[l]`` is the number of valid
    positions of layer l.
    """

    def __init__(self, layers, n_kv_heads: int, head_dim: int, max_ctx: int):
        self.layers = list(layers)
        self.max_ctx = max_ctx
        self.k = {l: np.zeros((n_kv_heads, max_ctx, head_dim)) for l in self.layers}
        self.v = {l: np.zeros((n_kv_heads, max_ctx, head_dim)) for l in self.layers}
        self.length = {l: 0 for l in self.layers}

    def fill(self, layer: int, k: np.ndarray, v: np.ndarray):
        """Set positions [0, n) of a layer from arrays [H_kv, n, d_h] (pre-filled context)."""
        n = k.shape[1]
        self.k[layer][:, :n] = k
        self.v[layer][:, :n] = v
        self.length[layer] = n


# ---------------------------------------------------------------------------------------
# Block, prefix range, decode step, boundary
# ---------------------------------------------------------------------------------------
def block_forward(x: np.ndarray, w: LayerWeights, cache: KVCache, layer: int, shape,
                  taps: dict | None = None) -> np.ndarray:
    """One decoder block B_l on x [M, D] starting at position p0 = cache.length[layer].

    Writes the block's post-rotary keys and its values at positions [p0, p0 + M) of the
    layer's cache and returns the block's output residual stream [M, D].
    """
    M, D = x.shape
    H, Hkv, dh = shape.n_heads, shape.n_kv_heads, shape.head_dim
    p0 = cache.length[layer]
    if p0 + M > cache.max_ctx:
        raise ValueError("KV cache full")
    pos = p0 + np.arange(M)

    # attention half: pre-norm, projections, rotary embedding, cache write, attention
    r = x
    u = rms_norm(x, w.g_attn, shape.rms_eps)
    q = (u @ w.w_q.T).reshape(M, H, dh)
    k = (u @ w.w_k.T).reshape(M, Hkv, dh)
    v = (u @ w.w_v.T).reshape(M, Hkv, dh)
    q = apply_rope(q, pos, shape.rope_base)
    k = apply_rope(k, pos, shape.rope_base)
    cache.k[layer][:, p0:p0 + M] = k.transpose(1, 0, 2)
    cache.v[layer][:, p0:p0 + M] = v.transpose(1, 0, 2)
    cache.length[layer] = p0 + M
    ctx = p0 + M
    o = causal_gqa_attention(q, cache.k[layer][:, :ctx], cache.v[layer][:, :ctx], pos, Hkv)
    x = r + o.reshape(M, H * dh) @ w.w_o.T

    # feed-forward half: pre-norm, SwiGLU, down projection, residual
    r = x
    u2 = rms_norm(x, w.g_mlp, shape.rms_eps)
    m = swiglu(u2 @ w.w_gate.T, u2 @ w.w_up.T)
    y = r + m @ w.w_down.T
    if taps is not None:
        taps.update(q=q, k=k, v=v, attn=o.reshape(M, H * dh), x_mid=x, m=m, y=y)
    return y


def block_forward_rows(x: np.ndarray, w: LayerWeights, shape, rows, p0: int = 0,
                       ctx_k: np.ndarray | None = None, ctx_v: np.ndarray | None = None):
    """Block B_l on x [M, D] at positions p0.., evaluated only at the query rows ``rows``.

    Same stages as block_forward: every row's key and value are formed (attention needs
    them), but the query, attention output, projections and feed-forward are computed only
    for the selected rows. ``ctx_k`` / ``ctx_v`` [H_kv, p0, d_h] hold the cached positions
    before p0 (post-rotary keys). Returns (y [len(rows), D], k [H_kv, M, d_h], v [H_kv, M, d_h])
    where k, v are this call's cache entries.
    """
    M, D = x.shape
    H, Hkv, dh = shape.n_heads, shape.n_kv_heads, shape.head_dim
    rows = np.asarray(rows, dtype=np.int64)
    pos = p0 + np.arange(M)
    u = rms_norm(x, w.g_attn, shape.rms_eps)
    k = apply_rope((u @ w.w_k.T).reshape(M, Hkv, dh), pos, shape.rope_base).transpose(1, 0, 2)
    v = (u @ w.w_v.T).reshape(M, Hkv, dh).transpose(1, 0, 2)
    if p0 > 0:
        k_all = np.concatenate([ctx_k[:, :p0], k], axis=1)
        v_all = np.concatenate([ctx_v[:, :p0], v], axis=1)
    else:
        k_all, v_all = k, v
    q = apply_rope((u[rows] @ w.w_q.T).reshape(len(rows), H, dh), pos[rows], shape.rope_base)
    o = causal_gqa_attention(q, k_all, v_all, pos[rows], Hkv)
    xm = x[rows] + o.reshape(len(rows), H * dh) @ w.w_o.T
    u2 = rms_norm(xm, w.g_mlp, shape.rms_eps)
    y = xm + swiglu(u2 @ w.w_gate.T, u2 @ w.w_up.T) @ w.w_down.T
    return y, k, v


def prefix_forward(x: np.ndarray, weights, layer_begin: int, layer_end: int, cache: KVCache,
                   shape, per_block: list | None = None) -> np.ndarray:
    """Blocks [layer_begin, layer_end) applied in order (Eq. 5 for layer_begin = 0).

    ``weights[l]`` is block l's LayerWeights (a mapping or list indexed by absolute layer).
    Returns the boundary hidden state h^(layer_end). An empty range returns x unchanged.
    ``per_block`` (optional) receives each block's output in order.
    """
    h = x
    for l in range(layer_begin, layer_end):
        h = block_forward(h, weights[l], cache, l, shape)
        if per_block is not None:
            per_block.append(h)
    return h


def decode_step(x1: np.ndarray, weights, layer_begin: int, layer_end: int, cache: KVCache,
                shape) -> np.ndarray:
    """One autoregressive step: the prefix range on a single token x1 [1, D] at
    position p0 = cache length, appending one key/value position per layer."""
    if x1.shape[0] != 1:
        raise ValueError("decode takes one token")
    return prefix_forward(x1, weights, layer_begin, layer_end, cache, shape)


def boundary_transfer(h: np.ndarray) -> np.ndarray:
    """T(.) of Eq. 6: moves h^(p) across devices; the values are unchanged."""
    return np.array(h, copy=True)


def boundary_bytes(batch: int, seq_len: int, hidden: int, elem_bytes: int) -> int:
    """S_hid(p) = B * L_p * D * b of Eq. 11: bytes of the one tensor handed off per frame."""
    return batch * seq_len * hidden * elem_bytes
