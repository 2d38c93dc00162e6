"""The balanced schedule's decode (Eq. chunk_boundary_main carried across CTAs),
through gtr_gla_balanced_walk: the host runs the kernel's own range and position
code, so this runs without a GPU.  Whatever the sizes, the CTAs' walks must cover
every (unit, chunk) exactly once, each CTA's share must be within one chunk of
an even split, each unit's chunks must run in order within a CTA, and a unit cut
between two CTAs must continue at the chunk where the earlier CTA's head run
stopped, from that CTA's hand-off."""
import numpy as np
import pytest

from paper_2609_26590_gb300 import build as gbuild


@pytest.fixture(scope="module")
def gla():
    gbuild.build()
    from paper_2609_26590_gb300 import gla as g
    g.load()
    return g


def check_schedule(gla, n_units, n_chunks, grid):
    walks = [gla.balanced_walk(n_units, n_chunks, grid, cta) for cta in range(grid)]
    seen = np.zeros((n_units, n_chunks), dtype=np.int64)
    sizes = []
    for cta, (entries, head) in enumerate(walks):
        sizes.append(len(entries))
        for unit, chunk, _, _ in entries:
            seen[unit, chunk] += 1
        # runs of one unit, consecutive chunks; a run starts (start = 1) at chunk 0 or at
        # the hand-in, which only the last run may have
        runs = []
        for i, (unit, chunk, start, hin) in enumerate(entries):
            if i == 0 or unit != entries[i - 1][0]:
                runs.append([unit, chunk, chunk, hin])
                assert start == 1, (n_units, n_chunks, grid, cta, i)
                assert hin == (1 if chunk != 0 else 0), (n_units, n_chunks, grid, cta, i)
            else:
                assert chunk == entries[i - 1][1] + 1 and start == 0 and hin == 0, (n_units, n_chunks, grid, cta, i)
                runs[-1][2] = chunk
        # the head run (from chunk 0, cut before the unit's end) comes first, the tail run last
        assert 0 <= head < n_chunks
        if head > 0:
            assert runs[0][1] == 0 and runs[0][2] == head - 1 and runs[0][3] == 0
        for r in runs[(1 if head > 0 else 0):-1] if len(runs) > 1 else []:
            assert r[1] == 0 and r[2] == n_chunks - 1, (n_units, n_chunks, grid, cta, r)  # whole units
        if not (head > 0 and len(runs) == 1):
            assert runs[-1][2] == n_chunks - 1  # the last run ends its unit (tail or whole unit)
        hin_runs = [r for r in runs if r[3] == 1]
        assert len(hin_runs) <= 1 and (not hin_runs or hin_runs[0] is runs[-1])
        if hin_runs:
            # continues the unit the previous CTA's head run started, where it stopped
            prev_entries, prev_head = walks[cta - 1]
            assert cta > 0 and prev_head > 0
            assert hin_runs[0][0] == prev_entries[0][0] and hin_runs[0][1] == prev_head
            assert hin_runs[0][2] == n_chunks - 1
        elif cta > 0:
            assert walks[cta - 1][1] == 0  # no hand-off was made for this CTA
    assert (seen == 1).all(), (n_units, n_chunks, grid)
    assert max(sizes) - min(sizes) <= 1 and sum(sizes) == n_units * n_chunks
    assert walks[0][1] == 0 or grid > 1
    assert walks[-1][1] == 0  # the last range ends at the last unit's end: nothing to hand over


@pytest.mark.parametrize("n_units,n_chunks,grid", [
    (384, 25, 152),      # the batched 40 x 40 workload: 63-64 chunks a CTA
    (192, 100, 152),     # B = 16, 80 x 80
    (160, 2, 152),       # 2-chunk sequences, ranges of 2-3 chunks
    (153, 7, 152),       # one unit more than CTAs
    (152, 9, 152),       # exactly one unit each: no hand-offs
    (5, 1, 3),
    (1, 13, 1),
])
def test_balanced_walk_cases(gla, n_units, n_chunks, grid):
    check_schedule(gla, n_units, n_chunks, grid)


def test_balanced_walk_random(gla):
    rng = np.random.default_rng(17)
    for _ in range(150):
        n_units = int(rng.integers(1, 400))
        n_chunks = int(rng.integers(1, 60))
        grid = int(rng.integers(1, min(n_units, 200) + 1))
        check_schedule(gla, n_units, n_chunks, grid)


def test_balanced_walk_rejects_invalid(gla):
    lib = gla.load()
    import ctypes
    h = ctypes.c_int(0)
    buf = (ctypes.c_int * 8)()
    assert lib.gtr_gla_balanced_walk(0, 5, 1, 0, buf, 2, ctypes.byref(h)) == -1
    assert lib.gtr_gla_balanced_walk(4, 0, 1, 0, buf, 2, ctypes.byref(h)) == -1
    assert lib.gtr_gla_balanced_walk(4, 5, 5, 0, buf, 2, ctypes.byref(h)) == -1   # ranges shorter than a unit
    assert lib.gtr_gla_balanced_walk(4, 5, 2, 2, buf, 2, ctypes.byref(h)) == -1   # cta out of range
    assert lib.gtr_gla_balanced_walk(4, 5, 2, 0, None, 2, ctypes.byref(h)) == -1
    assert lib.gtr_gla_balanced_walk(4, 5, 2, 0, buf, 2, None) == -1
    assert lib.gtr_gla_balanced_walk(1 << 20, 1 << 12, 2, 0, buf, 2, ctypes.byref(h)) == -1  # index overflow
    assert lib.gtr_gla_balanced_walk(4, 5, 2, 0, None, 0, ctypes.byref(h)) == 10  # count only
