"""Mutation check of the oracle's pins: each plausible slip below is planted in a copy of the
oracle (source text of ``oracle/decoder.py``, on the CPU), and the pin tests of
``tests/test_oracle_pins.py`` are run against that copy in a fresh interpreter. Every mutant
must fail at least one pin; the unmodified copy must pass them all. This is what backs the
claim that the pins tie each part of the oracle to something other than itself (closed
forms, hand-worked examples, invariants, brute force)."""
import concurrent.futures
import os
import shutil
import subprocess
import sys
import tempfile

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (name, text in oracle/decoder.py, replacement); the text must occur exactly once.
MUTANTS = [
    # bf16 encoding
    ("bf16 decode shift", "<< np.uint32(16)).view(np.float32)", "<< np.uint32(15)).view(np.float32)"),
    ("bf16 rounding truncates", "np.rint(np.ldexp(m, 8))", "np.trunc(np.ldexp(m, 8))"),
    # RMSNorm (Sec. IV-B normalisation stage)
    ("eps outside the root", "x / np.sqrt(ms + eps) * gain", "x / (np.sqrt(ms) + eps) * gain"),
    ("norm gain dropped", "x / np.sqrt(ms + eps) * gain", "x / np.sqrt(ms + eps)"),
    ("sum instead of mean", "ms = np.mean(x * x, axis=-1, keepdims=True)",
     "ms = np.sum(x * x, axis=-1, keepdims=True)"),
    # rotary embedding
    ("rope rotation sign", "[a * c - b * s, b * c + a * s]", "[a * c + b * s, b * c - a * s]"),
    ("rope interleaved pairing", "    a = x[..., :half]\n    b = x[..., half:]",
     "    a = x[..., 0::2]\n    b = x[..., 1::2]"),
    ("rope theta exponent", "theta = np.power(float(base), -2.0 * j / head_dim)",
     "theta = np.power(float(base), -1.0 * j / head_dim)"),
    ("rope missing on q", "    q = apply_rope(q, pos, shape.rope_base)\n", ""),
    ("rope missing on k", "    k = apply_rope(k, pos, shape.rope_base)\n", ""),
    ("positions off by one", "        raise ValueError(\"KV cache full\")\n    pos = p0 + np.arange(M)",
     "        raise ValueError(\"KV cache full\")\n    pos = p0 + 1 + np.arange(M)"),
    # attention
    ("gqa head mapping", "        g = h // group\n", "        g = h % n_kv_heads\n"),
    ("gqa value head mapping", "o[:, h, :] = w[h] @ v[h // group]", "o[:, h, :] = w[h] @ v[h % n_kv_heads]"),
    ("score scale", "(q[:, h, :] @ k[g].T) / np.sqrt(dh)", "(q[:, h, :] @ k[g].T) / dh"),
    ("mask lets the next key in", "mask = np.arange(ctx)[None, :] > np.asarray(q_pos)[:, None]",
     "mask = np.arange(ctx)[None, :] > np.asarray(q_pos)[:, None] + 1"),
    ("softmax not normalised", "w[h] = e / np.sum(e, axis=1, keepdims=True)", "w[h] = e"),
    ("value cache holds keys", "cache.v[layer][:, p0:p0 + M] = v.transpose(1, 0, 2)",
     "cache.v[layer][:, p0:p0 + M] = k.transpose(1, 0, 2)"),
    # block structure
    ("attention residual dropped", "x = r + o.reshape(M, H * dh) @ w.w_o.T", "x = o.reshape(M, H * dh) @ w.w_o.T"),
    ("mlp residual dropped", "y = r + m @ w.w_down.T", "y = m @ w.w_down.T"),
    ("gate and up swapped", "m = swiglu(u2 @ w.w_gate.T, u2 @ w.w_up.T)",
     "m = swiglu(u2 @ w.w_up.T, u2 @ w.w_gate.T)"),
    ("down projection transposed", "y = r + m @ w.w_down.T", "y = r + m @ w.w_down"),
    ("mlp norm gain of attention", "u2 = rms_norm(x, w.g_mlp, shape.rms_eps)",
     "u2 = rms_norm(x, w.g_attn, shape.rms_eps)"),
    ("mlp norm of the block input", "u2 = rms_norm(x, w.g_mlp, shape.rms_eps)",
     "u2 = rms_norm(r - o.reshape(M, H * dh) @ w.w_o.T, w.g_mlp, shape.rms_eps)"),
    ("silu sign", "return z / (1.0 + np.exp(-z))", "return z / (1.0 + np.exp(z))"),
    # sampled-row evaluation used for full-size parity
    ("rows: residual dropped", "xm = x[rows] + o.reshape(len(rows), H * dh) @ w.w_o.T",
     "xm = o.reshape(len(rows), H * dh) @ w.w_o.T"),
    ("rows: context keys ignored", "k_all = np.concatenate([ctx_k[:, :p0], k], axis=1)",
     "k_all = np.concatenate([np.zeros_like(ctx_k[:, :p0]), k], axis=1)"),
    # seeding a cache with a given context
    ("fill swaps the planes", "self.k[layer][:, :n] = k\n        self.v[layer][:, :n] = v",
     "self.k[layer][:, :n] = v\n        self.v[layer][:, :n] = k"),
    ("fill length off by one", "self.length[layer] = n\n", "self.length[layer] = n - 1\n"),
    ("fill reads the head axis as length", "n = k.shape[1]", "n = k.shape[0]"),
    # layer range and boundary
    ("range reuses the first block's weights", "h = block_forward(h, weights[l], cache, l, shape)",
     "h = block_forward(h, weights[layer_begin], cache, l, shape)"),
    ("boundary bytes without the batch", "return batch * seq_len * hidden * elem_bytes",
     "return seq_len * hidden * elem_bytes"),
]


def _make_copy(dst: str, mutant):
    os.makedirs(os.path.join(dst, "tests"))
    shutil.copytree(os.path.join(ROOT, "oracle"), os.path.join(dst, "oracle"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), os.path.join(dst, "tests", "golden"))
    shutil.copy(os.path.join(ROOT, "tests", "test_oracle_pins.py"), os.path.join(dst, "tests"))
    if mutant is not None:
        _, old, new = mutant
        path = os.path.join(dst, "oracle", "decoder.py")
        with open(path) as f:
            src = f.read()
        assert src.count(old) == 1, f"mutation site not unique or missing: {old!r}"
        with open(path, "w") as f:
            f.write(src.replace(old, new))


def _run_pins(dst: str) -> int:
    env = dict(os.environ)
    env["PYTHONPATH"] = dst
    env["PYTHONDONTWRITEBYTECODE"] = "1"
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        os.path.join("tests", "test_oracle_pins.py")],
                       cwd=dst, env=env, capture_output=True, text=True, timeout=300)
    return r.returncode


def test_every_planted_slip_fails_a_pin():
    # the copies live under the repository's (ignored) artifact folder and are removed after
    base = os.environ.get("VLA_ARTIFACT_DIR", os.path.join(ROOT, "artifacts"))
    os.makedirs(base, exist_ok=True)
    work = tempfile.mkdtemp(prefix="oracle_mutants_", dir=base)
    try:
        dirs = {"unmodified": os.path.join(work, "unmodified")}
        _make_copy(dirs["unmodified"], None)
        for i, mt in enumerate(MUTANTS):
            d = os.path.join(work, f"m{i:02d}")
            _make_copy(d, mt)
            dirs[mt[0]] = d
        with concurrent.futures.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 2)) as ex:
            rc = dict(zip(dirs, ex.map(_run_pins, dirs.values())))
    finally:
        shutil.rmtree(work, ignore_errors=True)
    assert rc["unmodified"] == 0, "the pins fail on an unmodified copy of the oracle"
    survived = [name for name, code in rc.items() if name != "unmodified" and code != 1]
    assert not survived, f"slips no pin catches (pytest exit codes {[rc[n] for n in survived]}): {survived}"
