"""Shared test plumbing: bf16 transfer between numpy bits and torch device tensors, error
metrics, and model set-up on both sides (GPU library and CPU oracle) from the same seeded
synthetic bits."""
from __future__ import annotations

import numpy as np

import oracle
import synth

# Floating-point bars (bf16 operands and storage, fp32 accumulation):
REL_L2_BLOCK = 1e-2    # per-block relative L2 error against the float64 oracle
COS_FINAL = 0.999      # cosine similarity of the final boundary hidden state


def sync(seconds: float = 60.0):
    """Wait for the current stream with a deadline instead of blocking in the driver, so a
    stalled kernel fails the test (and ends the process) rather than holding the GPU."""
    import time

    import torch
    s = torch.cuda.current_stream()
    t0 = time.time()
    while not s.query():
        if time.time() - t0 > seconds:
            # end the process: its CUDA context (and the stalled work) goes with it
            import os
            import traceback
            msg = f"GPU work did not finish within {seconds} s; exiting\n" + "".join(traceback.format_stack())
            out = os.environ.get("VLA_ARTIFACT_DIR",
                                 os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "artifacts"))
            os.makedirs(out, exist_ok=True)
            with open(os.path.join(out, "watchdog.txt"), "a") as f:
                f.write(msg)
            os._exit(3)
        time.sleep(0.0005)
    torch.cuda.synchronize()


def rel_l2(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def cos_sim(a, b) -> float:
    a = np.asarray(a, dtype=np.float64).ravel()
    b = np.asarray(b, dtype=np.float64).ravel()
    return float(a @ b / (np.linalg.norm(a) * np.linalg.norm(b)))


def to_dev(bits: np.ndarray):
    """uint16 bf16 bits -> torch.bfloat16 CUDA tensor (same bits)."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.cuda()


def from_dev(t) -> np.ndarray:
    """torch.bfloat16 tensor -> float64 numpy (exact)."""
    import torch
    bits = t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return oracle.bf16_to_f64(bits)


class _CudaArray:
    def __init__(self, ptr: int, numel: int):
        self.__cuda_array_interface__ = {"data": (int(ptr), False), "shape": (int(numel),), "typestr": "<i2",
                                         "strides": None, "version": 3}


def dev_view(ptr: int, numel: int):
    """torch.bfloat16 CUDA tensor viewing ``numel`` bf16 elements at a raw device pointer."""
    import torch
    return torch.as_tensor(_CudaArray(ptr, numel), device="cuda").view(torch.bfloat16)


def kv_planes(vla, kv, layer, shape, max_ctx):
    """(K, V) torch views [Hkv, max_ctx, dh] of one layer of a library KV cache."""
    kp, vp = vla.vla_kv_data(kv, layer)
    n = shape.n_kv_heads * max_ctx * shape.head_dim
    shp = (shape.n_kv_heads, max_ctx, shape.head_dim)
    return dev_view(kp, n).view(shp), dev_view(vp, n).view(shp)


def vla_cfg(shape, max_ctx: int):
    import paper_2608_14586_gb300 as vla
    return vla.VlaConfig(hidden=shape.hidden, n_heads=shape.n_heads, n_kv_heads=shape.n_kv_heads,
                         head_dim=shape.head_dim, ffn=shape.ffn, rms_eps=shape.rms_eps,
                         rope_base=shape.rope_base, max_ctx=max_ctx)


class Model:
    """One synthetic model on both sides: bf16 bits, device tensors, library handle, oracle
    float64 weights (converted lazily per layer)."""

    def __init__(self, shape, n_layers: int, seed: int, max_ctx: int, gain: str = "ones"):
        import paper_2608_14586_gb300 as vla
        self.shape = shape
        self.n_layers = n_layers
        self.bits = [synth.layer_weights(shape, seed, l, gain=gain) for l in range(n_layers)]
        dev = [{k: to_dev(v) for k, v in b.items()} for b in self.bits]
        self.handle = vla.vla_prefix_create(vla_cfg(shape, max_ctx), dev)
        del dev  # the library keeps its own repacked copies
        self._w64 = {}

    def w64(self, l: int) -> oracle.LayerWeights:
        if l not in self._w64:
            self._w64[l] = oracle.LayerWeights.from_bf16(self.bits[l])
        return self._w64[l]

    def drop_w64(self):
        self._w64.clear()

    def weights64(self):
        return _LazyWeights(self)

    def close(self):
        import paper_2608_14586_gb300 as vla
        vla.vla_prefix_destroy(self.handle)


class _LazyWeights:
    def __init__(self, m: Model):
        self.m = m

    def __getitem__(self, l):
        return self.m.w64(l)
