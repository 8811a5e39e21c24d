"""The C-ABI library builds for sm_103a, loads without a GPU, exports every function that
include/*.h declares, and rejects bad arguments on the host before touching CUDA."""
import ctypes
import glob
import os
import re
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        txt = open(h).read()
        txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
        for m in re.finditer(r"^\s*(?:const\s+)?(?:vla_status|int|char\s*\*|void)\s*\*?\s*(vla_\w+)\s*\(", txt,
                             flags=re.M):
            names.add(m.group(1))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    import paper_2608_14586_gb300 as vla
    vla.build()
    return vla.load()


def test_header_declares_the_boundary():
    names = _declared_functions()
    for required in ("vla_prefix_create", "vla_prefix_destroy", "vla_kv_create", "vla_prefix_prefill",
                     "vla_prefix_decode", "vla_boundary_to_host", "vla_last_async_error", "vla_status_str"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    names = _declared_functions()
    assert len(names) >= 15
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_host_side_argument_errors(lib):
    import paper_2608_14586_gb300 as vla
    assert lib.vla_status_str(4) == b"kv cache full"
    assert lib.vla_status_str(0) == b"ok"
    out = ctypes.c_void_p(123)
    assert lib.vla_prefix_create(None, None, 1, ctypes.byref(out)) == 1 and out.value is None
    assert lib.vla_prefix_create(None, None, 1, None) == 1
    assert lib.vla_prefix_destroy(None) == 0
    assert lib.vla_kv_destroy(None) == 0
    assert lib.vla_kv_length(None) == -1
    assert lib.vla_kv_layer_length(None, 0) == -1
    assert lib.vla_last_launch_count(None) == 0
    assert lib.vla_prefix_prefill(None, None, 1, 0, 1, None, None, None) == 1
    assert lib.vla_prefix_decode(None, None, 0, 1, None, None, None) == 1
    assert lib.vla_prefix_prefill_to_host(None, None, 1, 0, 1, None, None, None, None) == 1
    assert lib.vla_prefix_decode_batch(None, None, 2, 0, 1, None, None, None) == 1
    assert lib.vla_boundary_to_host(None, 1, 1, None, None, None, None) == 1
    assert lib.vla_frame_to_device(None, 1, 1, None, None) == 1
    assert lib.vla_op_gemm_bf16(None, None, 1, 1, 1, None, None) == 1
    assert lib.vla_last_async_error(None) == 1
    # unsupported shapes are refused before any allocation (head_dim 96)
    cfg = vla.VlaConfig(hidden=256, n_heads=4, n_kv_heads=4, head_dim=96, ffn=688, rms_eps=1e-6,
                        rope_base=1e4, max_ctx=64)
    w = (vla.VlaLayerWeights * 1)()
    for n, _ in vla.VlaLayerWeights._fields_:
        setattr(w[0], n, 16)
    assert lib.vla_prefix_create(ctypes.byref(cfg), w, 1, ctypes.byref(out)) == 9
    cfg.head_dim, cfg.n_kv_heads = 64, 3  # 4 % 3 != 0
    assert lib.vla_prefix_create(ctypes.byref(cfg), w, 1, ctypes.byref(out)) == 9
    cfg.n_kv_heads, cfg.max_ctx = 4, 0
    assert lib.vla_prefix_create(ctypes.byref(cfg), w, 1, ctypes.byref(out)) == 1


def test_binding_names_match_the_header():
    import paper_2608_14586_gb300 as vla
    for n in _declared_functions():
        assert n in vla.__all__, n


def test_headers_are_plain_c_and_the_c_example_compiles():
    """Every public header compiles as C (not only C++), and the C usage example
    (tests/c_example/boundary_example.c) matches the declared signatures."""
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    cuda_inc = "/usr/local/cuda/include"
    if not os.path.exists(os.path.join(cuda_inc, "cuda_runtime.h")):
        pytest.skip("CUDA headers not found")
    for h in sorted(glob.glob(os.path.join(ROOT, "include", "*.h"))):
        r = subprocess.run([cc, "-std=c11", "-fsyntax-only", "-Wall", "-Werror", "-x", "c", h,
                            "-I", os.path.join(ROOT, "include"), "-I", cuda_inc], capture_output=True, text=True)
        assert r.returncode == 0, (h, r.stderr)
    example = os.path.join(ROOT, "tests", "c_example", "boundary_example.c")
    r = subprocess.run([cc, "-std=c11", "-fsyntax-only", "-Wall", "-Werror", example,
                        "-I", os.path.join(ROOT, "include"), "-I", cuda_inc], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
