"""The CPU suffix's four-lane exp (``csrc/cpu_math.h``) against float64 exp: relative error
within 2 ulp of fp32 over a dense sweep of the normal range, the range ends, and the
special values the softmax and SiLU can pass it. Compiled with the library's own host
flags. Runs without a GPU."""
import os
import shutil
import subprocess
import tempfile

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_14586_gb300", "csrc")

DRIVER = r"""
#include "cpu_math.h"
#include <cstdio>
#include <cstdlib>
int main(int argc, char** argv) {
    FILE* in = std::fopen(argv[1], "rb");
    FILE* out = std::fopen(argv[2], "wb");
    const long n = std::atol(argv[3]);
    for (long i = 0; i < n; i += 4) {
        vla_cpu::v4f x;
        if (std::fread(&x, sizeof(float), 4, in) != 4) return 1;
        const vla_cpu::v4f y = vla_cpu::exp4(x);
        std::fwrite(&y, sizeof(float), 4, out);
    }
    std::fclose(in);
    std::fclose(out);
    return 0;
}
"""


def _cxx():
    for c in (os.environ.get("CXX"), shutil.which("g++"), shutil.which("c++")):
        if c and os.path.exists(c):
            return c
    return None


@pytest.mark.skipif(_cxx() is None, reason="no host C++ compiler")
def test_exp4_error_bound_and_special_values():
    from paper_2608_14586_gb300._build import CXX_FLAGS
    base = os.environ.get("VLA_ARTIFACT_DIR", os.path.join(ROOT, "artifacts"))
    os.makedirs(base, exist_ok=True)
    work = tempfile.mkdtemp(prefix="cpu_math_", dir=base)
    try:
        src = os.path.join(work, "drv.cpp")
        exe = os.path.join(work, "drv")
        with open(src, "w") as f:
            f.write(DRIVER)
        flags = [a for a in CXX_FLAGS if a not in ("-fPIC",)]
        subprocess.check_call([_cxx(), *flags, "-I", CSRC, src, "-o", exe])
        lo, hi = np.float32(-87.3365479), np.float32(88.7228394)
        sweep = np.linspace(lo, np.float32(88.72), 2_000_000, dtype=np.float32)
        special = np.array([0.0, -0.0, 1.0, -1.0, 0.5, -0.5, lo, -87.34, -100.0, -1e30, -np.inf,
                            88.73, 1e30, np.inf, 1e-30, -1e-30, 20.0, -20.0], dtype=np.float32)
        x = np.concatenate([sweep, special])
        x = np.concatenate([x, np.zeros((-len(x)) % 4, dtype=np.float32)])
        fin, fout = os.path.join(work, "x.bin"), os.path.join(work, "y.bin")
        x.tofile(fin)
        subprocess.check_call([exe, fin, fout, str(len(x))])
        y = np.fromfile(fout, dtype=np.float32)
    finally:
        shutil.rmtree(work, ignore_errors=True)
    with np.errstate(over="ignore"):
        ref = np.exp(x.astype(np.float64))
    normal = (x >= lo) & (x <= np.float32(88.72))
    rel = np.abs(y[normal].astype(np.float64) - ref[normal]) / ref[normal]
    assert rel.max() <= 2 * 2.0 ** -23, rel.max()  # 2 ulp of fp32
    got = dict(zip(x[len(sweep):].tolist(), y[len(sweep):].tolist()))
    assert got[0.0] == 1.0 and got[-0.0] == 1.0
    for v in (-87.34, -100.0, -1e30, -np.inf):      # below the normal range: flushed to 0
        assert got[float(np.float32(v))] == 0.0, v
    for v in (88.73, 1e30, np.inf):                  # above the largest finite result
        assert got[float(np.float32(v))] == np.inf, v
    assert np.isfinite(y[normal]).all() and (y[normal] > 0).all()
