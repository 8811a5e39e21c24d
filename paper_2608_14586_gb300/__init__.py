"""GB300 LLM-prefix library: Python binding of the C ABI in ``include/vla_prefix.h``,
``include/vla_ops.h`` and ``include/vla_cpu.h`` (CPU suffix and cross-frame pipeline).

Argument marshalling only: every stage of the prefix forward runs in the CUDA kernels of
``libvla_prefix.so`` (built in-tree from ``csrc/`` by ``build()``). Tensors are passed as
device pointers (torch tensors are accepted for convenience: their ``data_ptr()`` is used),
streams as ``torch.cuda.Stream`` or raw ``cudaStream_t`` integers. There is no CPU fallback:
``load()`` raises if the library has not been built.
"""
from __future__ import annotations

import ctypes
import os

from ._build import LIB as LIB_PATH
from ._build import build as _build_lib

__all__ = [
    "build", "load", "VlaError", "VlaConfig", "VlaLayerWeights",
    "vla_prefix_create", "vla_prefix_destroy", "vla_kv_create", "vla_kv_destroy", "vla_kv_reset",
    "vla_kv_length", "vla_kv_layer_length", "vla_kv_data", "vla_kv_decode_plan", "vla_kv_set_length", "vla_prefix_prefill",
    "vla_prefix_prefill_to_host", "vla_prefix_decode", "vla_prefix_decode_batch", "vla_boundary_to_host", "vla_frame_to_device", "vla_last_async_error", "vla_status_str",
    "vla_last_launch_count", "vla_op_gemm_bf16", "vla_op_attention_prefill", "vla_prefix_set_timing",
    "vla_prefix_stage_times", "vla_prefix_inject_stall", "vla_op_attention_decode_noalloc", "vla_prefix_info", "STATUS", "STAGES",
    "VlaFrameTimes", "vla_cpu_model_create", "vla_cpu_model_destroy", "vla_cpu_model_threads", "vla_cpu_model_info",
    "vla_cpu_kv_create", "vla_cpu_kv_destroy", "vla_cpu_kv_reset", "vla_cpu_kv_length", "vla_cpu_kv_data",
    "vla_cpu_prefill", "vla_pipeline_create", "vla_pipeline_submit", "vla_pipeline_collect",
    "vla_pipeline_in_flight", "vla_pipeline_destroy", "VlaSchedConfig", "VlaSchedState", "vla_scheduler_create",
    "vla_scheduler_observe", "vla_scheduler_next", "vla_scheduler_estimates", "vla_scheduler_destroy",
]

# stage ids of vla_prefix_stage_times (VLA_STAGE_* in vla_prefix.h)
STAGES = ("rowstat", "gemm_qkv", "attn_prefill", "gemm_o", "gemm_gateup", "gemm_down", "kv_len",
          "dec_qkv", "dec_attn", "dec_o", "dec_gateup", "dec_down")

STATUS = {0: "VLA_OK", 1: "VLA_ERR_INVALID_ARG", 2: "VLA_ERR_SHAPE", 3: "VLA_ERR_RANGE", 4: "VLA_ERR_KV_FULL",
          5: "VLA_ERR_NOT_PINNED", 6: "VLA_ERR_OOM", 7: "VLA_ERR_CUDA", 8: "VLA_ERR_TIMEOUT",
          9: "VLA_ERR_UNSUPPORTED", 10: "VLA_ERR_BUSY"}


class VlaError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        self.name = STATUS.get(status, str(status))
        super().__init__(f"{where}: {self.name} ({_lib.vla_status_str(status).decode() if _lib else status})")


class VlaConfig(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_int), ("n_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("ffn", ctypes.c_int), ("rms_eps", ctypes.c_float),
                ("rope_base", ctypes.c_float), ("max_ctx", ctypes.c_int)]


_WNAMES = ("w_q", "w_k", "w_v", "w_o", "w_gate", "w_up", "w_down", "g_attn", "g_mlp")


class VlaLayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in _WNAMES]


class VlaFrameTimes(ctypes.Structure):
    """Per-frame stage times of the pipeline (vla_frame_times): T_G, T_X, T_C of Eq. 8-10."""
    _fields_ = [("t_gpu_ms", ctypes.c_double), ("t_xfer_ms", ctypes.c_double), ("t_cpu_ms", ctypes.c_double),
                ("t_submit_s", ctypes.c_double), ("t_start_s", ctypes.c_double), ("t_ready_s", ctypes.c_double),
                ("t_done_s", ctypes.c_double),
                ("split", ctypes.c_int), ("n_tokens", ctypes.c_int)]

    def as_dict(self) -> dict:
        return {n: getattr(self, n) for n, _ in self._fields_}


class VlaSchedConfig(ctypes.Structure):
    """Zones and controller settings of the split scheduler (vla_sched_config)."""
    _fields_ = [("n_layers", ctypes.c_int), ("k_min", ctypes.c_int), ("k_max", ctypes.c_int),
                ("k_init", ctypes.c_int), ("max_step", ctypes.c_int), ("alpha", ctypes.c_double),
                ("backlog_limit", ctypes.c_int)]


class VlaSchedState(ctypes.Structure):
    """Runtime state z_t = [u_gpu, u_cpu, q_t] of Eq. 15 (vla_sched_state)."""
    _fields_ = [("u_gpu", ctypes.c_double), ("u_cpu", ctypes.c_double), ("backlog", ctypes.c_int)]


_lib = None


def build(force: bool = False) -> str:
    """Compile the CUDA library (nvcc, sm_103a) in-tree; returns its path."""
    return _build_lib(force=force)


def load():
    """Load ``libvla_prefix.so``; raises if it has not been built (no fallback exists)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: run paper_2608_14586_gb300.build() (needs nvcc)")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, V = ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p
    sig = {
        "vla_prefix_create": ([ctypes.POINTER(VlaConfig), ctypes.POINTER(VlaLayerWeights), I,
                               ctypes.POINTER(P)], I),
        "vla_prefix_destroy": ([P], I),
        "vla_kv_create": ([P, I, I, I, ctypes.POINTER(P)], I),
        "vla_kv_destroy": ([P], I),
        "vla_kv_decode_plan": ([P, ctypes.POINTER(I), ctypes.POINTER(I), ctypes.POINTER(I)], I),
        "vla_kv_reset": ([P, V], I),
        "vla_kv_length": ([P], I),
        "vla_kv_layer_length": ([P, I], I),
        "vla_kv_data": ([P, I, ctypes.POINTER(P), ctypes.POINTER(P)], I),
        "vla_kv_set_length": ([P, I, V], I),
        "vla_prefix_prefill": ([P, V, I, I, I, P, V, V], I),
        "vla_prefix_decode": ([P, V, I, I, P, V, V], I),
        "vla_prefix_prefill_to_host": ([P, V, I, I, I, P, V, V, V], I),
        "vla_prefix_decode_batch": ([P, V, I, I, I, ctypes.POINTER(P), V, V], I),
        "vla_boundary_to_host": ([V, I, I, V, V, V, V], I),
        "vla_frame_to_device": ([V, I, I, V, V], I),
        "vla_last_async_error": ([P], I),
        "vla_status_str": ([I], ctypes.c_char_p),
        "vla_last_launch_count": ([P], I),
        "vla_op_gemm_bf16": ([V, V, I, I, I, V, V], I),
        "vla_op_attention_prefill": ([V, V, V, I, I, I, I, I, I, V, V], I),
        "vla_prefix_set_timing": ([P, ctypes.c_uint], I),
        "vla_prefix_inject_stall": ([P, I, ctypes.c_longlong], I),
        "vla_op_attention_decode_noalloc": ([V, V, V, I, I, I, I, I, V, V], I),
        "vla_prefix_stage_times": ([P, ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_int), I], I),
        "vla_prefix_info": ([P, ctypes.POINTER(VlaConfig), ctypes.POINTER(I)], I),
        "vla_cpu_model_create": ([ctypes.POINTER(VlaConfig), ctypes.POINTER(VlaLayerWeights), I, I, I,
                                  ctypes.POINTER(P)], I),
        "vla_cpu_model_destroy": ([P], I),
        "vla_cpu_model_threads": ([P], I),
        "vla_cpu_model_info": ([P, ctypes.POINTER(VlaConfig), ctypes.POINTER(I), ctypes.POINTER(I)], I),
        "vla_cpu_kv_create": ([P, I, I, I, ctypes.POINTER(P)], I),
        "vla_cpu_kv_destroy": ([P], I),
        "vla_cpu_kv_reset": ([P], I),
        "vla_cpu_kv_length": ([P], I),
        "vla_cpu_kv_data": ([P, I, ctypes.POINTER(P), ctypes.POINTER(P)], I),
        "vla_cpu_prefill": ([P, V, I, I, I, P, V], I),
        "vla_pipeline_create": ([P, P, I, I, ctypes.POINTER(P)], I),
        "vla_pipeline_submit": ([P, ctypes.c_int64, V, I, I, V], I),
        "vla_pipeline_collect": ([P, ctypes.POINTER(ctypes.c_int64), V, I, ctypes.POINTER(VlaFrameTimes)], I),
        "vla_pipeline_in_flight": ([P], I),
        "vla_pipeline_destroy": ([P], I),
        "vla_scheduler_create": ([ctypes.POINTER(VlaSchedConfig), ctypes.POINTER(P)], I),
        "vla_scheduler_observe": ([P, ctypes.POINTER(VlaFrameTimes)], I),
        "vla_scheduler_next": ([P, ctypes.POINTER(VlaSchedState)], I),
        "vla_scheduler_estimates": ([P, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double),
                                     ctypes.POINTER(ctypes.c_double)], I),
        "vla_scheduler_destroy": ([P], I),
    }
    for name, (args, res) in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    _lib = lib
    return lib


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "__array_interface__"):  # numpy array in host memory
        return x.__array_interface__["data"][0]
    if hasattr(x, "value"):
        return x.value
    raise TypeError(f"cannot take a device pointer of {type(x)}")


def _stream(s) -> int | None:
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    if hasattr(s, "cuda_stream"):
        return s.cuda_stream
    raise TypeError(f"not a stream: {type(s)}")


def _event(e) -> int | None:
    if e is None:
        return None
    if isinstance(e, int):
        return e
    if hasattr(e, "cuda_event"):
        return e.cuda_event
    raise TypeError(f"not an event: {type(e)}")


def _check(st: int, where: str):
    if st != 0:
        raise VlaError(st, where)


def vla_status_str(status: int) -> str:
    return load().vla_status_str(status).decode()


def vla_prefix_create(cfg: VlaConfig, layers) -> ctypes.c_void_p:
    """``layers``: sequence of mappings name -> device tensor / pointer (see VlaLayerWeights)."""
    lib = load()
    arr = (VlaLayerWeights * len(layers))()
    for i, w in enumerate(layers):
        for n in _WNAMES:
            setattr(arr[i], n, _ptr(w[n]))
    out = ctypes.c_void_p()
    _check(lib.vla_prefix_create(ctypes.byref(cfg), arr, len(layers), ctypes.byref(out)), "vla_prefix_create")
    return out


def vla_prefix_destroy(p):
    _check(load().vla_prefix_destroy(p), "vla_prefix_destroy")


def vla_kv_create(p, layer_begin: int, layer_end: int, max_ctx: int) -> ctypes.c_void_p:
    out = ctypes.c_void_p()
    _check(load().vla_kv_create(p, layer_begin, layer_end, max_ctx, ctypes.byref(out)), "vla_kv_create")
    return out


def vla_kv_destroy(kv):
    _check(load().vla_kv_destroy(kv), "vla_kv_destroy")


def vla_kv_reset(kv, stream=None):
    _check(load().vla_kv_reset(kv, _stream(stream)), "vla_kv_reset")


def vla_kv_length(kv) -> int:
    return load().vla_kv_length(kv)


def vla_kv_layer_length(kv, layer: int) -> int:
    return load().vla_kv_layer_length(kv, layer)


def vla_kv_decode_plan(kv) -> dict:
    """The cache's decode-attention launch plan: tensor_cores, cluster_size, keys_per_cta."""
    tc, cs, keys = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check(load().vla_kv_decode_plan(kv, ctypes.byref(tc), ctypes.byref(cs), ctypes.byref(keys)),
           "vla_kv_decode_plan")
    return {"tensor_cores": tc.value, "cluster_size": cs.value, "keys_per_cta": keys.value}


def vla_kv_data(kv, layer: int):
    k, v = ctypes.c_void_p(), ctypes.c_void_p()
    _check(load().vla_kv_data(kv, layer, ctypes.byref(k), ctypes.byref(v)), "vla_kv_data")
    return k.value, v.value


def vla_kv_set_length(kv, length: int, stream=None):
    _check(load().vla_kv_set_length(kv, length, _stream(stream)), "vla_kv_set_length")


def vla_prefix_prefill(p, hidden_in, n_tokens: int, layer_begin: int, layer_end: int, kv, hidden_out,
                       stream=None):
    _check(load().vla_prefix_prefill(p, _ptr(hidden_in), n_tokens, layer_begin, layer_end, kv, _ptr(hidden_out),
                                     _stream(stream)), "vla_prefix_prefill")


def vla_prefix_prefill_to_host(p, hidden_in, n_tokens: int, layer_begin: int, layer_end: int, kv, hidden_out,
                               pinned_dst, stream=None):
    """Prefill whose last block also stores h^(layer_end) into page-locked host memory."""
    _check(load().vla_prefix_prefill_to_host(p, _ptr(hidden_in), n_tokens, layer_begin, layer_end, kv,
                                             _ptr(hidden_out), _ptr(pinned_dst), _stream(stream)),
           "vla_prefix_prefill_to_host")


def vla_prefix_decode(p, hidden_in, layer_begin: int, layer_end: int, kv, hidden_out, stream=None):
    _check(load().vla_prefix_decode(p, _ptr(hidden_in), layer_begin, layer_end, kv, _ptr(hidden_out),
                                    _stream(stream)), "vla_prefix_decode")


def vla_prefix_decode_batch(p, hidden_in, layer_begin: int, layer_end: int, kvs, hidden_out, stream=None):
    """One decode step for len(kvs) sequences; hidden_in / hidden_out are [batch, hidden]."""
    arr = (ctypes.c_void_p * len(kvs))(*[k.value if hasattr(k, "value") else k for k in kvs])
    _check(load().vla_prefix_decode_batch(p, _ptr(hidden_in), len(kvs), layer_begin, layer_end, arr,
                                          _ptr(hidden_out), _stream(stream)), "vla_prefix_decode_batch")


def vla_boundary_to_host(hidden_out, n_tokens: int, hidden: int, pinned_dst, side_stream=None, ready=None,
                         done=None):
    _check(load().vla_boundary_to_host(_ptr(hidden_out), n_tokens, hidden, _ptr(pinned_dst), _stream(side_stream),
                                       _event(ready), _event(done)), "vla_boundary_to_host")


def vla_frame_to_device(pinned_src, n_tokens: int, hidden: int, hidden_in, stream=None):
    _check(load().vla_frame_to_device(_ptr(pinned_src), n_tokens, hidden, _ptr(hidden_in), _stream(stream)),
           "vla_frame_to_device")


def vla_last_async_error(p) -> int:
    return load().vla_last_async_error(p)


def vla_last_launch_count(p) -> int:
    return load().vla_last_launch_count(p)


def vla_prefix_inject_stall(p, stage, wait_budget_cycles: int):
    """Arms the failure-detection test fault on the next prefill launch of a GEMM stage (a
    name of STAGES or its id; -1 / None cancels)."""
    sid = -1 if stage is None or stage == -1 else (STAGES.index(stage) if isinstance(stage, str) else int(stage))
    _check(load().vla_prefix_inject_stall(p, sid, int(wait_budget_cycles)), "vla_prefix_inject_stall")


def vla_op_gemm_bf16(A, B, M: int, N: int, K: int, C, stream=None):
    _check(load().vla_op_gemm_bf16(_ptr(A), _ptr(B), M, N, K, _ptr(C), _stream(stream)), "vla_op_gemm_bf16")


def vla_op_attention_prefill(q, k_plane, v_plane, n_tokens: int, n_heads: int, n_kv_heads: int, head_dim: int,
                             max_ctx: int, pos0: int, out, stream=None):
    _check(load().vla_op_attention_prefill(_ptr(q), _ptr(k_plane), _ptr(v_plane), n_tokens, n_heads, n_kv_heads,
                                           head_dim, max_ctx, pos0, _ptr(out), _stream(stream)),
           "vla_op_attention_prefill")


def vla_prefix_set_timing(p, stages=()):
    """Time the kernels of the named stages (an iterable of STAGES names, or "all"); () = off."""
    if stages == "all":
        stages = STAGES
    mask = 0
    for name in stages:
        mask |= 1 << STAGES.index(name)
    _check(load().vla_prefix_set_timing(p, mask), "vla_prefix_set_timing")


def vla_prefix_stage_times(p) -> dict:
    """{stage name: (milliseconds, launches)} accumulated since the last read."""
    n = len(STAGES)
    ms = (ctypes.c_float * n)()
    cnt = (ctypes.c_int * n)()
    _check(load().vla_prefix_stage_times(p, ms, cnt, n), "vla_prefix_stage_times")
    return {STAGES[i]: (float(ms[i]), int(cnt[i])) for i in range(n)}


def vla_op_attention_decode_noalloc(q, k_plane, v_plane, ctx: int, n_heads: int, n_kv_heads: int, head_dim: int,
                                    max_ctx: int, out, stream=None):
    """Decode attention whose scratch is a fixed array inside the library (no allocation)."""
    _check(load().vla_op_attention_decode_noalloc(_ptr(q), _ptr(k_plane), _ptr(v_plane), ctx, n_heads, n_kv_heads,
                                                  head_dim, max_ctx, _ptr(out), _stream(stream)),
           "vla_op_attention_decode_noalloc")


def vla_prefix_info(p) -> tuple:
    """(VlaConfig, layer_count) of a prefix object."""
    cfg, n = VlaConfig(), ctypes.c_int()
    _check(load().vla_prefix_info(p, ctypes.byref(cfg), ctypes.byref(n)), "vla_prefix_info")
    return cfg, n.value


# ---------------------------------------------------------------------------------------
# CPU suffix and cross-frame pipeline (include/vla_cpu.h)
# ---------------------------------------------------------------------------------------
def vla_cpu_model_create(cfg: VlaConfig, layers, layer_begin: int, n_threads: int = 0) -> ctypes.c_void_p:
    """CPU copy of blocks [layer_begin, layer_begin + len(layers)); ``layers`` holds HOST
    arrays (numpy uint16 bf16 bit patterns or CPU torch tensors) by weight name."""
    lib = load()
    arr = (VlaLayerWeights * len(layers))()
    keep = []
    for i, w in enumerate(layers):
        for n in _WNAMES:
            a = w[n]
            if hasattr(a, "__array_interface__") and not a.flags["C_CONTIGUOUS"]:
                import numpy as np
                a = np.ascontiguousarray(a)
            keep.append(a)
            setattr(arr[i], n, _ptr(a))
    out = ctypes.c_void_p()
    _check(lib.vla_cpu_model_create(ctypes.byref(cfg), arr, layer_begin, layer_begin + len(layers), n_threads,
                                    ctypes.byref(out)), "vla_cpu_model_create")
    return out


def vla_cpu_model_destroy(m):
    _check(load().vla_cpu_model_destroy(m), "vla_cpu_model_destroy")


def vla_cpu_model_threads(m) -> int:
    return load().vla_cpu_model_threads(m)


def vla_cpu_model_info(m) -> tuple:
    """(VlaConfig, layer_begin, layer_end) of a CPU model."""
    cfg, a, b = VlaConfig(), ctypes.c_int(), ctypes.c_int()
    _check(load().vla_cpu_model_info(m, ctypes.byref(cfg), ctypes.byref(a), ctypes.byref(b)), "vla_cpu_model_info")
    return cfg, a.value, b.value


def vla_cpu_kv_create(m, layer_begin: int, layer_end: int, max_ctx: int) -> ctypes.c_void_p:
    out = ctypes.c_void_p()
    _check(load().vla_cpu_kv_create(m, layer_begin, layer_end, max_ctx, ctypes.byref(out)), "vla_cpu_kv_create")
    return out


def vla_cpu_kv_destroy(kv):
    _check(load().vla_cpu_kv_destroy(kv), "vla_cpu_kv_destroy")


def vla_cpu_kv_reset(kv):
    _check(load().vla_cpu_kv_reset(kv), "vla_cpu_kv_reset")


def vla_cpu_kv_length(kv) -> int:
    return load().vla_cpu_kv_length(kv)


def vla_cpu_kv_data(kv, layer: int):
    """Host addresses of a layer's K and V planes [n_kv_heads][max_ctx][head_dim] bf16."""
    k, v = ctypes.c_void_p(), ctypes.c_void_p()
    _check(load().vla_cpu_kv_data(kv, layer, ctypes.byref(k), ctypes.byref(v)), "vla_cpu_kv_data")
    return k.value, v.value


def vla_cpu_prefill(m, hidden_in, n_tokens: int, layer_begin: int, layer_end: int, kv, hidden_out):
    """Blocks [layer_begin, layer_end) on the host; hidden_in / hidden_out are host arrays."""
    _check(load().vla_cpu_prefill(m, _ptr(hidden_in), n_tokens, layer_begin, layer_end, kv, _ptr(hidden_out)),
           "vla_cpu_prefill")


def vla_pipeline_create(gpu, cpu, max_tokens: int, depth: int = 2) -> ctypes.c_void_p:
    out = ctypes.c_void_p()
    _check(load().vla_pipeline_create(gpu, cpu, max_tokens, depth, ctypes.byref(out)), "vla_pipeline_create")
    return out


def vla_pipeline_submit(pl, frame_id: int, hidden_in, n_tokens: int, split: int, stream=None):
    _check(load().vla_pipeline_submit(pl, frame_id, _ptr(hidden_in), n_tokens, split, _stream(stream)),
           "vla_pipeline_submit")


def vla_pipeline_collect(pl, hidden_out=None, timeout_ms: int = -1) -> tuple:
    """(frame_id, VlaFrameTimes) of the oldest frame once done; h^(N) copied into hidden_out."""
    fid, t = ctypes.c_int64(), VlaFrameTimes()
    _check(load().vla_pipeline_collect(pl, ctypes.byref(fid), _ptr(hidden_out), timeout_ms, ctypes.byref(t)),
           "vla_pipeline_collect")
    return fid.value, t


def vla_pipeline_in_flight(pl) -> int:
    return load().vla_pipeline_in_flight(pl)


def vla_pipeline_destroy(pl):
    _check(load().vla_pipeline_destroy(pl), "vla_pipeline_destroy")


def vla_scheduler_create(n_layers: int, k_min: int, k_max: int, k_init: int, max_step: int = 1,
                         alpha: float = 0.5, backlog_limit: int = 2) -> ctypes.c_void_p:
    """Split-point controller Phi over the dynamic zone [k_min, k_max] (Sec. IV-D)."""
    cfg = VlaSchedConfig(n_layers=n_layers, k_min=k_min, k_max=k_max, k_init=k_init, max_step=max_step,
                         alpha=alpha, backlog_limit=backlog_limit)
    out = ctypes.c_void_p()
    _check(load().vla_scheduler_create(ctypes.byref(cfg), ctypes.byref(out)), "vla_scheduler_create")
    return out


def vla_scheduler_observe(s, times: VlaFrameTimes):
    _check(load().vla_scheduler_observe(s, ctypes.byref(times)), "vla_scheduler_observe")


def vla_scheduler_next(s, u_gpu: float = 0.0, u_cpu: float = 0.0, backlog: int = 0) -> int:
    z = VlaSchedState(u_gpu=u_gpu, u_cpu=u_cpu, backlog=backlog)
    return load().vla_scheduler_next(s, ctypes.byref(z))


def vla_scheduler_estimates(s) -> tuple:
    """(ms per GPU block, ms per CPU block, ms per transfer); -1 where never observed."""
    g, c, x = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    _check(load().vla_scheduler_estimates(s, ctypes.byref(g), ctypes.byref(c), ctypes.byref(x)),
           "vla_scheduler_estimates")
    return g.value, c.value, x.value


def vla_scheduler_destroy(s):
    _check(load().vla_scheduler_destroy(s), "vla_scheduler_destroy")
