"""Seeded synthetic inputs for the LLM-prefix workloads.

This module is the only code shared by the CUDA path (its tests and benchmark) and the CPU
oracle. It holds none of the method's arithmetic: it draws bf16 bit patterns (``uint16``
arrays) from a counter-based normal generator (``synth_gen.c``) and arranges them into the
weight / hidden-state / KV-cache shapes of the workloads below. Both sides receive the same
bits; each side does its own bf16 decoding.

The paper (Sec. V) evaluates on Bench2Drive frames through Orion/MindDrive. Neither the
frames nor the weights exist here, so every workload is synthetic with the shapes of a
7B-class LLaMA-style backbone: weights ~ N(0, 0.02), RMSNorm gains 1.0, visual tokens
~ 2*N(0,1) (where the workload says so) followed by text tokens ~ N(0,1).
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth_gen.c")
_LIB_PATH = os.path.join(_HERE, "libsynth_gen.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile ``synth_gen.c`` into ``libsynth_gen.so`` next to it (gcc, OpenMP)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.synth_normal_bf16.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64,
                                              ctypes.c_uint64, ctypes.c_double, ctypes.c_int64]
            lib.synth_normal_bf16.restype = None
            lib.synth_fill_bf16.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_double]
            lib.synth_fill_bf16.restype = None
            _lib = lib
    return _lib


def normal_bf16(shape, seed: int, stream: int, std: float = 1.0, offset: int = 0) -> np.ndarray:
    """bf16 bits of ``std * N(0,1)`` for element indices ``[offset, offset+prod(shape))``."""
    out = np.empty(shape, dtype=np.uint16)
    n = out.size
    if n:
        _load().synth_normal_bf16(out.ctypes.data, n, seed & (2**64 - 1), stream & (2**64 - 1),
                                  float(std), offset)
    return out


def fill_bf16(shape, value: float) -> np.ndarray:
    out = np.empty(shape, dtype=np.uint16)
    if out.size:
        _load().synth_fill_bf16(out.ctypes.data, out.size, float(value))
    return out


# --------------------------------------------------------------------------------------
# Model shapes
# --------------------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class ModelShape:
    hidden: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    rms_eps: float = 1e-6
    rope_base: float = 10000.0


TINY = ModelShape(hidden=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688)
B7 = ModelShape(hidden=4096, n_heads=32, n_kv_heads=8, head_dim=128, ffn=11008)

# stream ids: one per tensor kind so that every tensor is an independent draw
_STREAM = {"w_q": 1, "w_k": 2, "w_v": 3, "w_o": 4, "w_gate": 5, "w_up": 6, "w_down": 7,
           "hidden": 16, "kv_k": 17, "kv_v": 18, "decode_hidden": 19}

WEIGHT_STD = 0.02


def layer_weights(shape: ModelShape, seed: int, layer: int, gain: str = "ones") -> dict:
    """bf16 bits of one decoder block's weights, each ``[out, in]`` row-major.

    ``gain``: "ones" (RMSNorm gains exactly 1.0, the workloads' recipe) or "random"
    (gains 1 + 0.1 N(0,1), used by tests that exercise gain handling).
    """
    D, H, Hkv, dh, F = shape.hidden, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn
    dims = {"w_q": (H * dh, D), "w_k": (Hkv * dh, D), "w_v": (Hkv * dh, D), "w_o": (D, H * dh),
            "w_gate": (F, D), "w_up": (F, D), "w_down": (D, F)}
    w = {}
    for name, shp in dims.items():
        w[name] = normal_bf16(shp, seed, (layer << 8) | _STREAM[name], WEIGHT_STD)
    if gain == "ones":
        w["g_attn"] = fill_bf16((D,), 1.0)
        w["g_mlp"] = fill_bf16((D,), 1.0)
    elif gain == "random":
        g1 = normal_bf16((D,), seed, (layer << 8) | 32, 0.1)
        g2 = normal_bf16((D,), seed, (layer << 8) | 33, 0.1)
        w["g_attn"] = _add_one_bf16(g1)
        w["g_mlp"] = _add_one_bf16(g2)
    else:
        raise ValueError(gain)
    return w


def _add_one_bf16(bits: np.ndarray) -> np.ndarray:
    """bf16 bits of 1 + x for bf16 bits x (input preparation for random gains)."""
    f = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float32) + np.float32(1.0)
    u = f.view(np.uint32)
    u = u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return (u >> np.uint32(16)).astype(np.uint16)


def hidden_states(n_tokens: int, hidden: int, seed: int, visual_tokens: int = 0,
                  visual_scale: float = 1.0, stream: str = "hidden") -> np.ndarray:
    """bf16 bits of a frame's input hidden states ``[n_tokens, hidden]``.

    Rows ``[0, visual_tokens)`` are ``visual_scale * N(0,1)`` (the encoder's visual tokens),
    the remaining rows ``N(0,1)`` (text / query tokens).
    """
    out = np.empty((n_tokens, hidden), dtype=np.uint16)
    s = _STREAM[stream]
    nv = min(visual_tokens, n_tokens)
    if nv:
        out[:nv] = normal_bf16((nv, hidden), seed, s, visual_scale, 0)
    if n_tokens > nv:
        out[nv:] = normal_bf16((n_tokens - nv, hidden), seed, s, 1.0, nv * hidden)
    return out


def decode_hidden(step: int, hidden: int, seed: int) -> np.ndarray:
    """bf16 bits of the ``[1, hidden]`` input of decode step ``step`` (independent draws)."""
    return normal_bf16((1, hidden), seed, (_STREAM["decode_hidden"] << 20) | step, 1.0)


def random_kv(n_ctx: int, shape: ModelShape, seed: int, layer: int):
    """bf16 bits of a pre-filled KV cache slice: K, V each ``[n_kv_heads, n_ctx, head_dim]``."""
    shp = (shape.n_kv_heads, n_ctx, shape.head_dim)
    k = normal_bf16(shp, seed, (layer << 8) | _STREAM["kv_k"], 1.0)
    v = normal_bf16(shp, seed, (layer << 8) | _STREAM["kv_v"], 1.0)
    return k, v


# --------------------------------------------------------------------------------------
# Workloads (shape, token mix, depth) named by what they are
# --------------------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    shape: ModelShape
    n_layers: int            # blocks that exist in the model
    prefix_layers: int       # blocks run on the GPU ([0, k))
    n_tokens: int            # prefill tokens per frame
    visual_tokens: int
    visual_scale: float
    decode_steps: int = 0
    prefill_ctx: int = 0     # KV positions pre-filled with random K/V before decode
    frames: int = 1
    seed: int = 0


WORKLOADS = {
    "tiny_2blk_64tok": Workload("tiny_2blk_64tok", TINY, 2, 1, 64, 0, 1.0),
    "7b_block_1024tok": Workload("7b_block_1024tok", B7, 1, 1, 1024, 768, 2.0),
    "7b_prefix16_2304tok": Workload("7b_prefix16_2304tok", B7, 32, 16, 2304, 1920, 1.0),
    "7b_decode16_ctx2304": Workload("7b_decode16_ctx2304", B7, 32, 16, 0, 0, 1.0,
                                    decode_steps=64, prefill_ctx=2304),
    "7b_pipeline32_3072tok": Workload("7b_pipeline32_3072tok", B7, 32, 16, 3072, 2688, 1.0,
                                      frames=4),
}
