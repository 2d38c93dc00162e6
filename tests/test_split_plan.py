"""The sequence split of the tensor-core schedule (Eq. chunk_boundary_main applied
across segments), through gtr_gla_split_plan: host arithmetic, so it runs
without a GPU.  The plans below are the segment lengths a GB300 sweep measured
fastest or within 4 % of it (graph-replayed calls, interleaved rounds); the
invariants hold for any shape: the last segment is not empty, a split fits one
wave of the SMs, and sequences that already fill half the SMs, or have at most
5 chunks, are never split."""
import math

import numpy as np
import pytest

from paper_2609_26590_gb300 import build as gbuild

GB300_SMS = 152


@pytest.fixture(scope="module")
def gla():
    gbuild.build()
    from paper_2609_26590_gb300 import gla as g
    g.load()
    return g


# (B, H, grid_h, grid_w, Dk, Dv) -> (segments, chunks per segment) on 152 SMs; the
# times are graph-replayed calls of a GB300 sweep over every segment length
MEASURED = [
    ((1, 6, 40, 40, 64, 64), (13, 2)),      # 25 chunks: length 2 fastest (15.3 us; 16.6 at 3, 36.5 whole)
    ((1, 2, 128, 128, 64, 64), (64, 4)),    # 256 chunks over 2 sequences: the shortest length one wave
                                            # allows (26.9 us; 26.5 at 5, 30.1 at 8)
    ((1, 1, 128, 128, 128, 128), (64, 4)),  # two key halves, two value slices: 2 units (49.2 us; 47.5 at 5)
    ((1, 4, 80, 80, 32, 64), (34, 3)),      # 100 chunks: length 3 (20.7 us, as length 2; 22.5 at 5)
    ((1, 6, 44, 44, 64, 64), (16, 2)),      # 31 chunks (prime): length 2 (16.9 us; 17.9 at 3)
    ((1, 2, 24, 24, 64, 64), (5, 2)),       # 9 chunks: length 2 (14.5 us; 16.9 whole)
    ((2, 8, 128, 128, 128, 128), (4, 64)),  # 32 units: at most 4 segments fit one wave
    ((1, 1, 16, 20, 64, 64), (1, 5)),       # 5 chunks: whole (11.4 us against 13.4 split)
    ((32, 12, 40, 40, 64, 64), (1, 25)),    # 384 units fill the device: unsplit
    ((8, 16, 80, 80, 64, 64), (1, 100)),    # 128 units > half the SMs: unsplit
]


def model_cost(L, nseg):
    return 15 * L + nseg


@pytest.mark.parametrize("shape,plan", MEASURED, ids=[f"{s[0]}x{s[1]}-{s[2]}x{s[3]}-d{s[4]}_{s[5]}"
                                                      for s, _ in MEASURED])
def test_plan_matches_measured_choice(gla, shape, plan):
    assert gla.split_plan(*shape, GB300_SMS) == plan


def test_plan_invariants_random_shapes(gla):
    rng = np.random.Generator(np.random.PCG64(2609))
    for _ in range(400):
        B, H = int(rng.integers(1, 5)), int(rng.integers(1, 13))
        gh, gw = int(rng.integers(1, 140)), int(rng.integers(1, 140))
        Dk, Dv = 8 * int(rng.integers(1, 17)), 8 * int(rng.integers(1, 17))
        n_sm = int(rng.choice([8, 32, 132, 148, 152]))
        nseg, L = gla.split_plan(B, H, gh, gw, Dk, Dv, n_sm)
        N = math.ceil(gh * gw / 64)
        units = B * H * math.ceil(Dv / 64)
        if nseg == 1:
            assert L == N
            continue
        assert 2 <= L < N
        assert nseg == math.ceil(N / L)
        assert (nseg - 1) * L < N <= nseg * L          # the last segment holds a real chunk
        assert units * nseg <= n_sm                     # one wave
        assert 2 * units <= n_sm                        # only launches that leave SMs idle split
        assert N > 5                                    # short sequences stay whole


def test_plan_is_optimal_under_its_cost_model(gla):
    # brute force over every admissible length on small problems: short sequences and
    # launches that fill half the SMs stay whole; otherwise the length minimising the
    # model over the lengths one wave allows (the first such length on ties)
    for N in range(1, 80):
        for units in (1, 2, 3, 6, 19, 40, 76, 77):
            H, gh, gw = units, N, 64          # grid_w = 64: exactly N chunks per sequence
            nseg, L = gla.split_plan(1, H, gh, gw, 64, 64, GB300_SMS)
            cost = {}
            if 2 * units <= GB300_SMS and N > 5:
                for l in range(2, N):
                    d = math.ceil(N / l)
                    if units * d <= GB300_SMS:
                        cost[l] = model_cost(l, d)
            if not cost:
                assert (nseg, L) == (1, N), (N, units, nseg, L)
                continue
            best = min(cost.values())
            best_l = min(l for l, c in cost.items() if c == best)
            assert (nseg, L) == (math.ceil(N / best_l), best_l), (N, units, nseg, L)


def test_plan_rejects_invalid_arguments(gla):
    import ctypes
    lib = gla.load()
    a, b = ctypes.c_int(-7), ctypes.c_int(-7)
    assert lib.gtr_gla_split_plan(1, 1, 8, 8, 64, 64, 0, ctypes.byref(a), ctypes.byref(b)) == 1
    assert lib.gtr_gla_split_plan(1, 1, 0, 8, 64, 64, 152, ctypes.byref(a), ctypes.byref(b)) == 1
    assert lib.gtr_gla_split_plan(1, 1, 8, 8, 64, 300, 152, ctypes.byref(a), ctypes.byref(b)) == 1
    assert lib.gtr_gla_split_plan(1, 1, 8, 8, 64, 64, 152, None, ctypes.byref(b)) == 1
    assert a.value == -7 and b.value == -7
    assert gla.split_plan(0, 3, 8, 8, 64, 64, 152) == (1, 1)


# (B, H, grid_h, grid_w, Dk, Dv) -> balanced on 152 SMs
BALANCE = [
    ((32, 12, 40, 40, 64, 64), True),       # 384 units: round-robin's 3 waves are 1.19x an even split
    ((24, 12, 40, 40, 64, 64), False),      # 288 units: 2 waves against 1.89 (measured 0.98x balanced)
    ((38, 12, 40, 40, 64, 64), False),      # 456 units: exactly 3 waves
    ((16, 12, 80, 80, 64, 64), True),       # 192 units: 2 waves against 1.26 (measured 1.23x faster)
    ((1, 160, 8, 16, 64, 64), True),        # 160 units: 8 SMs would take a second one
    ((8, 16, 80, 80, 64, 64), False),       # 128 units: one wave already
    ((2, 150, 8, 8, 64, 64), False),        # 300 units: the last wave only 1 % short
    ((32, 12, 40, 40, 128, 128), False),    # two key halves: ranges hand over one half only
    ((32, 12, 40, 40, 32, 128), True),      # one (padded) key half, two value slices: 768 units, 1.19
    ((5, 32, 40, 40, 32, 128), True),       # 320 units: 3 waves against 2.1
    ((1, 6, 40, 40, 64, 64), False),        # split instead
]


@pytest.mark.parametrize("shape,bal", BALANCE, ids=[f"{s[0]}x{s[1]}-{s[2]}x{s[3]}-d{s[4]}_{s[5]}"
                                                    for s, _ in BALANCE])
def test_balanced_plan(gla, shape, bal):
    assert gla.balanced_plan(*shape, GB300_SMS) == bal


def test_balanced_plan_invariants(gla):
    """Balanced only for one key half, more units than SMs, no split, and round-robin
    waves at least 1.1 times an even split's share."""
    rng = np.random.default_rng(5)
    for _ in range(400):
        B, H = int(rng.integers(1, 40)), int(rng.integers(1, 40))
        gh, gw = int(rng.integers(1, 90)), int(rng.integers(1, 90))
        Dk, Dv = 8 * int(rng.integers(1, 17)), 8 * int(rng.integers(1, 17))
        n_sm = int(rng.integers(1, 200))
        units = B * H * math.ceil(Dv / 64)
        bal = gla.balanced_plan(B, H, gh, gw, Dk, Dv, n_sm)
        nseg, _ = gla.split_plan(B, H, gh, gw, Dk, Dv, n_sm)
        expect = Dk <= 64 and units > n_sm and nseg == 1 and math.ceil(units / n_sm) * n_sm * 10 >= units * 11
        assert bal == expect, (B, H, gh, gw, Dk, Dv, n_sm)
    assert not gla.balanced_plan(16, 12, 80, 80, 64, 64, 0)
