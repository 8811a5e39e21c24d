"""Multi-process plumbing of bench.py on CPU (gloo, world size 2): the path shards as
independent replicas, so the only cross-rank traffic is the barrier around the timed region
and the max-reduction of the measured time; the reference arm runs on rank 0 alone."""
import os
import socket
import subprocess
import sys
import textwrap

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _run_ranks(code: str, world: int = 2, timeout: float = 120.0, args=()):
    port = _free_port()
    procs = []
    for r in range(world):
        env = dict(os.environ, WORLD_SIZE=str(world), RANK=str(r), LOCAL_RANK=str(r), MASTER_ADDR="127.0.0.1",
                   MASTER_PORT=str(port), PYTHONPATH=ROOT)
        procs.append(subprocess.Popen([sys.executable, "-c", code, *args], env=env, cwd=ROOT, stdout=subprocess.PIPE,
                                      stderr=subprocess.PIPE, text=True))
    outs = []
    for p in procs:
        try:
            out, err = p.communicate(timeout=timeout)
        except subprocess.TimeoutExpired:
            for q in procs:
                q.kill()
            raise
        outs.append((p.returncode, out, err))
    return outs


def test_barrier_and_max_over_ranks():
    code = textwrap.dedent("""
        import bench
        d = bench.Dist()
        d.init("gloo")
        d.barrier()
        t = d.max(10.0 + d.rank)          # per-rank times 10 and 11 -> every rank sees 11
        d.barrier()
        print("RESULT", d.rank, d.world, t)
        d.close()
    """)
    outs = _run_ranks(code)
    for r, (rc, out, err) in enumerate(outs):
        assert rc == 0, err
        assert f"RESULT {r} 2 11.0" in out, out


def test_reference_arm_prints_on_rank_zero_only():
    """Rank 1 of the reference arm exits 0 without work or output; rank 0 prints the line.
    Rank 0's oracle run is stubbed here (the full reference arm runs it in the bench)."""
    code = textwrap.dedent("""
        import json, sys
        import bench
        bench.oracle_prefill_time = lambda n, seed=0: (0.5, 1)
        sys.argv = ["bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3"]
        bench.main()
    """)
    outs = _run_ranks(code)
    (rc0, out0, err0), (rc1, out1, err1) = outs
    assert rc0 == 0 and rc1 == 0, (err0, err1)
    assert out1.strip() == ""
    import json
    line = json.loads(out0.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    # one block over the whole 2304-token frame in 0.5 s per step, taken x16 for the 16-block
    # prefix; the reported step time is the measured sample step
    assert abs(line["value"] - 2304 / (0.5 * 16)) < 1e-9
    assert abs(line["ms_per_step"] - 500.0) < 1e-9
