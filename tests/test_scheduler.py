"""The split-point controller Phi of Sec. IV-D (Eq. 15-17) as stated in include/vla_cpu.h:
cost estimates from observed frames, the Eq. 13 interval it minimises over the dynamic zone,
the per-frame step limit, the utilisation scaling, the backlog rule and the zone bounds.
Host logic only; runs without a GPU."""
import os
import shutil

import pytest

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="nvcc not available")


@pytest.fixture(scope="module")
def vla():
    import paper_2608_14586_gb300 as v
    v.build()
    v.load()
    return v


def _frame(vla, split, g_ms, c_ms, x_ms, N):
    """Stage times of a frame at `split` with g ms per GPU block and c ms per CPU block."""
    return vla.VlaFrameTimes(t_gpu_ms=split * g_ms, t_xfer_ms=x_ms, t_cpu_ms=(N - split) * c_ms, split=split,
                             n_tokens=1)


def _interval(p, g, c, x, N):
    return max(p * g, x + (N - p) * c)


def test_moves_toward_the_eq13_optimum_by_at_most_max_step(vla):
    N, g, c, x = 32, 1.0, 10.0, 0.1
    s = vla.vla_scheduler_create(N, 16, 32, 24, max_step=2, alpha=1.0)
    try:
        assert vla.vla_scheduler_next(s) == 24  # nothing observed yet: stays
        vla.vla_scheduler_observe(s, _frame(vla, 24, g, c, x, N))
        est = vla.vla_scheduler_estimates(s)
        assert est == pytest.approx((g, c, x))
        best = min(range(16, 33), key=lambda p: _interval(p, g, c, x, N))
        assert best == 30  # brute force over the zone
        seq = [vla.vla_scheduler_next(s) for _ in range(5)]
        assert seq == [26, 28, 30, 30, 30]
    finally:
        vla.vla_scheduler_destroy(s)


def test_gpu_load_moves_the_boundary_to_the_cpu_and_zone_bounds_hold(vla):
    N = 32
    s = vla.vla_scheduler_create(N, 20, 30, 30, max_step=4, alpha=1.0)
    try:
        vla.vla_scheduler_observe(s, _frame(vla, 30, 1.0, 10.0, 0.0, N))
        # 90% of the GPU taken by other work: g' = 10 = c, balance at p = 16, clamped to k_min
        assert [vla.vla_scheduler_next(s, u_gpu=0.9) for _ in range(4)] == [26, 22, 20, 20]
        # load gone: back toward the GPU side; p = 29 and 30 tie at 30 ms, the nearer one wins
        assert [vla.vla_scheduler_next(s) for _ in range(4)] == [24, 28, 29, 29]
        assert [vla.vla_scheduler_next(s, u_cpu=0.5) for _ in range(2)] == [30, 30]  # never past k_max
    finally:
        vla.vla_scheduler_destroy(s)


def test_moving_average_and_sides_without_blocks(vla):
    N = 8
    s = vla.vla_scheduler_create(N, 0, 8, 8, alpha=0.5)
    try:
        vla.vla_scheduler_observe(s, _frame(vla, 8, 2.0, 99.0, 0.2, N))  # no CPU blocks: c unknown
        g, c, x = vla.vla_scheduler_estimates(s)
        assert g == pytest.approx(2.0) and c == -1.0 and x == pytest.approx(0.2)
        assert vla.vla_scheduler_next(s, backlog=5) == 8  # cannot tell which side is slower
        vla.vla_scheduler_observe(s, _frame(vla, 4, 4.0, 6.0, 0.4, N))
        g, c, x = vla.vla_scheduler_estimates(s)
        assert g == pytest.approx(3.0) and c == pytest.approx(6.0) and x == pytest.approx(0.3)
    finally:
        vla.vla_scheduler_destroy(s)


def test_backlog_moves_off_the_slower_stage_when_the_prediction_is_flat(vla):
    N = 4
    s = vla.vla_scheduler_create(N, 1, 3, 2, alpha=1.0, backlog_limit=2)
    try:
        vla.vla_scheduler_observe(s, _frame(vla, 2, 1.0, 1.5, 0.0, N))
        # intervals 4.5, 3, 3 over p = 1..3: p = 2 ties with 3 and is nearer, no move without backlog
        assert vla.vla_scheduler_next(s, backlog=1) == 2
        # with backlog: at p = 2 the CPU stage (3 ms) is slower than the GPU stage (2 ms)
        assert vla.vla_scheduler_next(s, backlog=2) == 3
    finally:
        vla.vla_scheduler_destroy(s)


def test_invalid_configs(vla):
    lib = vla.load()
    for args in ((32, 10, 5, 7), (32, 0, 33, 3), (32, 4, 8, 9), (0, 0, 0, 0)):
        with pytest.raises(vla.VlaError) as ei:
            vla.vla_scheduler_create(*args)
        assert ei.value.name == "VLA_ERR_INVALID_ARG"
    with pytest.raises(vla.VlaError):
        vla.vla_scheduler_create(8, 0, 8, 4, max_step=0)
    with pytest.raises(vla.VlaError):
        vla.vla_scheduler_create(8, 0, 8, 4, alpha=0.0)
    assert lib.vla_scheduler_next(None, None) == -1
    assert lib.vla_scheduler_destroy(None) == 0


def test_closed_loop_tracks_the_eq13_optimum_as_costs_change(vla):
    """Frames simulated from true per-block costs that change mid-run (the GPU slows 8x at
    frame 20, as under a co-tenant the controller is not told about, then recovers at frame
    45), with 5% multiplicative noise on every stage time. Φ only sees the observed times.
    After each change it reaches the split that minimises Eq. 13 for the new costs within a
    bounded number of frames, stays within one block of it, never leaves the zone and never
    moves more than max_step blocks per frame."""
    import random
    rng = random.Random(7)
    N, k_min, k_max, step = 32, 12, 32, 2
    x = 0.2
    phases = [(0, 1.0, 24.0), (20, 8.0, 24.0), (45, 1.0, 24.0)]  # (first frame, g, c) in ms per block

    def truth(t):
        return [(g, c) for f, g, c in phases if f <= t][-1]

    def best(g, c):
        return min(range(k_min, k_max + 1), key=lambda p: (_interval(p, g, c, x, N), -p))

    s = vla.vla_scheduler_create(N, k_min, k_max, 24, max_step=step, alpha=0.5)
    try:
        k, trace = 24, []
        for t in range(70):
            g, c = truth(t)
            noise = lambda: 1.0 + rng.uniform(-0.05, 0.05)  # noqa: E731
            f = vla.VlaFrameTimes(t_gpu_ms=k * g * noise(), t_xfer_ms=x * noise(),
                                  t_cpu_ms=(N - k) * c * noise(), split=k, n_tokens=1)
            vla.vla_scheduler_observe(s, f)
            k_next = vla.vla_scheduler_next(s)
            assert k_min <= k_next <= k_max and abs(k_next - k) <= step
            k = k_next
            trace.append(k)
        assert [best(g, c) for _, g, c in phases] == [31, 24, 31]
        for start, g, c in phases:
            opt = best(g, c)
            settle = start + 8  # optima 31, 24, 31: 7 blocks at 2 per frame, plus the averages' lag
            end = next((f for f, _, _ in phases if f > start), 70)
            assert all(abs(p - opt) <= 1 for p in trace[settle:end]), (start, opt, trace[start:end])
    finally:
        vla.vla_scheduler_destroy(s)
