"""The scratch bound stated for gtr_gla_fwd_noalloc in include/gtr_gla.h: over SM
counts up to 160 and every head size the tensor-core schedule takes (multiples of
8 up to 128), the workspace the split or balanced schedule would need, computed
from the library's own host-side plans (gtr_gla_split_plan,
gtr_gla_balanced_plan), never exceeds the stated per-SM bound, and so stays within
GTR_GLA_NOALLOC_SCRATCH_BYTES.  Host arithmetic only."""
import os
import re

import pytest

from paper_2609_26590_gb300 import build as gbuild

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "gtr_gla.h")


def scratch_limit():
    m = re.search(r"#define\s+GTR_GLA_NOALLOC_SCRATCH_BYTES\s+\((\d+)u\s*<<\s*(\d+)\)", open(HEADER).read())
    assert m
    return int(m.group(1)) << int(m.group(2))


def pad64(d):
    return (d + 63) // 64 * 64


@pytest.fixture(scope="module")
def gla_mod():
    gbuild.build()
    from paper_2609_26590_gb300 import gla
    gla.load()
    return gla


def need_bytes(gla, B, H, gh, gw, Dk, Dv, n_sm):
    nseg, _ = gla.split_plan(B, H, gh, gw, Dk, Dv, n_sm)
    if nseg > 1:
        return B * H * (nseg - 1) * (pad64(Dk) * pad64(Dv) + pad64(Dk)) * 4
    if gla.balanced_plan(B, H, gh, gw, Dk, Dv, n_sm):
        return n_sm * (64 * 64 * 4 + 8)
    return 0


def test_noalloc_scratch_bound(gla_mod):
    limit = scratch_limit()
    dims = list(range(8, 129, 8))
    grids = [(8, 8), (44, 44), (80, 80), (128, 128)]
    worst = 0
    for n_sm in (1, 3, 16, 100, 148, 152, 160):
        per_sm_bound = n_sm * 33280
        assert per_sm_bound <= limit
        for Dk in dims:
            for Dv in dims:
                nv = pad64(Dv) // 64
                for bh in sorted({1, 2, 3, max(1, n_sm // (2 * nv)), max(1, n_sm // (4 * nv)), n_sm + 1,
                                  3 * n_sm // 2 + 1}):
                    for gh, gw in grids:
                        need = need_bytes(gla_mod, bh, 1, gh, gw, Dk, Dv, n_sm)
                        assert need <= per_sm_bound, (n_sm, Dk, Dv, bh, gh, gw, need)
                        worst = max(worst, need)
    assert 0 < worst <= limit
