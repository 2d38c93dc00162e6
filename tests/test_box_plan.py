"""The scan-order gather of the tensor-core schedule (Sec. 3.1, directional scanning:
left-to-right, right-to-left, top-to-bottom, bottom-to-top) checked on the host
through gtr_gla_chunk_boxes, which runs the kernel producer's own box enumeration.
For every chunk of every grid, in every order, including the all-zero padding
chunks of a split's last segment: the boxes cover the chunk's 64 tile rows
exactly once, each box holds the tokens of the chunk's scan positions in scan
order, and a box with rows outside the sequence loads only zeros (it lies wholly
outside the tensor).  Column-order chunks inside the sequence load as one im2col
walk instead (gtr_gla_chunk_walk): its start and traversal give the same rows.
No GPU is used."""
import math

import numpy as np

import pytest

from paper_2609_26590_gb300 import build as gbuild
from paper_2609_26590_gb300 import workloads as wl

C = 64
HEIGHTS = set(range(1, 8)) | {8 * j for j in range(1, 9)}   # the tensor maps' box heights


@pytest.fixture(scope="module")
def gla():
    gbuild.build()
    from paper_2609_26590_gb300 import gla as g
    g.load()
    return g


def scan_token(order, gh, gw, s):
    """Spatial token (row-major) at scan position s of a gh x gw grid, or None outside."""
    T = gh * gw
    if s < 0 or s >= T:
        return None
    if order == wl.ROW_FWD:
        return s
    if order == wl.ROW_REV:
        return T - 1 - s
    y, x = s % gh, s // gh                    # column-major walk
    if order == wl.COL_FWD:
        return y * gw + x
    return (gh - 1 - y) * gw + (gw - 1 - x)   # COL_REV: the column-major walk reversed


def check_chunk(gla, gh, gw, order, c):
    T = gh * gw
    boxes = gla.chunk_boxes(gh, gw, order, c)
    assert boxes, (gh, gw, order, c)
    # tile row r of a chunk holds walk position w0 + r, w0 = 64 c (forward) or T - 64 (c + 1)
    # (reverse orders walk the forward walk backwards, so tile rows run in walk order)
    rev = order in (wl.ROW_REV, wl.COL_REV)
    w0 = T - C * (c + 1) if rev else C * c
    covered = [0] * C
    for rows, r0, c2, c3 in boxes:
        assert rows in HEIGHTS
        assert 0 <= r0 and r0 + rows <= C
        for i in range(rows):
            covered[r0 + i] += 1
            w = w0 + r0 + i                     # walk position of this tile row
            if order in (wl.ROW_FWD, wl.ROW_REV):
                assert c3 == 0
                tok = c2 + i                    # token coordinate; out of [0, T) reads zeros
                expect = w if 0 <= w < T else None
                assert (tok if 0 <= tok < T else None) == expect, (gh, gw, order, c, r0, i)
            else:
                if c2 >= gw:                    # a zero box: only rows outside the sequence
                    assert c2 == gw and not (0 <= w < T), (gh, gw, order, c, r0, i)
                else:
                    assert 0 <= c3 and c3 + rows <= gh, ("box crosses a column", gh, gw, order, c)
                    assert 0 <= w < T
                    # forward column walk: position w -> column w // gh, row w % gh
                    assert (c2, c3 + i) == (w // gh, w % gh), (gh, gw, order, c, r0, i)
    assert covered == [1] * C, (gh, gw, order, c, covered)
    # the reversed walks read the forward walk's tokens backwards: the same tokens as the
    # oracle's scan order at the mirrored scan positions
    if rev:
        for r in range(C):
            w = w0 + r
            s = T - 1 - w                       # scan position of walk position w
            if 0 <= w < T:
                fwd = wl.ROW_FWD if order == wl.ROW_REV else wl.COL_FWD
                assert scan_token(order, gh, gw, s) == scan_token(fwd, gh, gw, w)


@pytest.mark.parametrize("order", wl.ALL_ORDERS, ids=wl.ORDER_NAMES)
def test_every_chunk_of_many_grids(gla, order):
    grids = [(gh, gw) for gh in range(1, 70) for gw in (1, 2, 3, 5, 7, 8, 13, 44)]
    grids += [(40, 40), (44, 44), (80, 80), (128, 128), (36, 36), (40, 36), (7, 11)]
    for gh, gw in grids:
        N = math.ceil(gh * gw / C)
        for c in range(N + 3):                  # three padding chunks past the end
            check_chunk(gla, gh, gw, order, c)


@pytest.mark.parametrize("order", wl.ALL_ORDERS, ids=wl.ORDER_NAMES)
def test_walk_loads(gla, order):
    # a chunk loads as one im2col walk exactly when it is a column-order chunk wholly inside the
    # sequence; the walk starts at the grid position of the chunk's first walk position and its
    # 64 pixels (down the column, then on into the next ones) are the rows its boxes would load
    grids = [(gh, gw) for gh in (1, 2, 3, 7, 8, 25, 40, 44, 63, 64, 65, 80) for gw in (1, 3, 13, 40, 44)]
    for gh, gw in grids:
        T = gh * gw
        N = math.ceil(T / C)
        rev = order in (wl.ROW_REV, wl.COL_REV)
        for c in range(N + 2):
            w0 = T - C * (c + 1) if rev else C * c
            walk = gla.chunk_walk(gh, gw, order, c)
            inside = 0 <= w0 and w0 + C <= T
            if order in (wl.ROW_FWD, wl.ROW_REV) or not inside:
                assert walk is None, (gh, gw, order, c)
                continue
            assert walk == (w0 // gh, w0 % gh), (gh, gw, order, c, walk)
            x, y = walk
            pixels = []
            for _ in range(C):                  # the im2col traversal: rows fastest, then columns
                pixels.append((x, y))
                y += 1
                if y == gh:
                    x, y = x + 1, 0
            boxes = gla.chunk_boxes(gh, gw, order, c)
            rows = {}
            for nrows, r0, c2, c3 in boxes:
                for i in range(nrows):
                    rows[r0 + i] = (c2, c3 + i)
            assert [rows[r] for r in range(C)] == pixels, (gh, gw, order, c)


def test_walk_start_division_large_grids(gla):
    # the walk start is the grid position (w0 // grid_h, w0 % grid_h), computed with a
    # multiply-high division by grid_h (Granlund-Montgomery): checked here for many divisors,
    # powers of two and their neighbours, and walk positions up to the largest sequences
    rng = np.random.default_rng(31)
    divisors = [1, 2, 3, 5, 7, 63, 64, 65, 127, 128, 129, 255, 256, 257, 1000, 4095, 4096, 4097,
                32767, 32768, 32769, 65535, 65536, 65537, 1 << 20, (1 << 20) + 1, (1 << 24) - 1]
    divisors += [int(d) for d in rng.integers(1, 1 << 20, size=60)]
    for gh in divisors:
        gw = max(1, (1 << 30) // gh)
        T = gh * gw
        N = T // C
        cs = {0, 1, N - 1, N // 2} | {int(c) for c in rng.integers(0, N, size=40)}
        for c in sorted(cs):
            w0 = C * c
            if w0 + C > T:
                continue
            assert gla.chunk_walk(gh, gw, wl.COL_FWD, c) == (w0 // gh, w0 % gh), (gh, gw, c)
            wr = T - C * (c + 1)
            assert gla.chunk_walk(gh, gw, wl.COL_REV, c) == (wr // gh, wr % gh), (gh, gw, c)


def test_padding_chunks_load_only_zeros(gla):
    for gh, gw in [(44, 44), (40, 40), (5, 7), (64, 1)]:
        T = gh * gw
        N = math.ceil(T / C)
        for order in wl.ALL_ORDERS:
            for c in range(N, N + 4):
                for rows, r0, c2, c3 in gla.chunk_boxes(gh, gw, order, c):
                    if order in (wl.ROW_FWD, wl.ROW_REV):
                        assert c2 + rows <= 0 or c2 >= T
                    else:
                        assert c2 == gw


def test_rejects_invalid_arguments(gla):
    import ctypes
    lib = gla.load()
    buf = (ctypes.c_int * 8)()
    assert lib.gtr_gla_chunk_boxes(0, 4, 0, 0, buf, 2) == -1
    assert lib.gtr_gla_chunk_boxes(4, 4, 7, 0, buf, 2) == -1
    assert lib.gtr_gla_chunk_boxes(4, 4, 0, -1, buf, 2) == -1
    assert lib.gtr_gla_chunk_boxes(4, 4, 0, 0, None, 2) == -1
    assert lib.gtr_gla_chunk_boxes(4, 4, 2, 0, None, 0) >= 1     # count only
    x, y = ctypes.c_int(), ctypes.c_int()
    assert lib.gtr_gla_chunk_walk(0, 4, 2, 0, ctypes.byref(x), ctypes.byref(y)) == -1
    assert lib.gtr_gla_chunk_walk(4, 4, 9, 0, ctypes.byref(x), ctypes.byref(y)) == -1
    assert lib.gtr_gla_chunk_walk(4, 4, 2, -1, ctypes.byref(x), ctypes.byref(y)) == -1
    assert lib.gtr_gla_chunk_walk(4, 4, 2, 0, None, ctypes.byref(y)) == -1
    assert lib.gtr_gla_chunk_walk(16, 16, 2, 1, ctypes.byref(x), ctypes.byref(y)) == 1
    assert (x.value, y.value) == (4, 0)
