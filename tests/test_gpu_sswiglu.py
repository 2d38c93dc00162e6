"""Spatial SwiGLU between its projections (Sec. 3.1, Eq. spatial_swiglu),
gtr_sswiglu_dwconv against the fp64 oracle element by element: small grids that
span several row tiles and a ragged last tile, channel counts that leave a
partial 128-byte slice, both input layouts (the two halves of one [B, T, 2F]
projection output, and separate tensors), no bias, the widest supported grid,
and sampled (image, channel) slices of the full-size workloads.

Bar: the output is accumulated in fp32 from exactly the stored inputs and
rounded once, the same bar as the mixer's (16-bit: rel L2 <= 2e-3, max-abs <=
1e-2 max|z|; fp32: rel L2 <= 1e-5)."""
import numpy as np
import pytest
import torch

import oracle
from gla_testutil import assert_within_bar, to_torch
from paper_2609_26590_gb300 import build as gbuild
from paper_2609_26590_gb300 import gla
from paper_2609_26590_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

TORCH_DT = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}


@pytest.fixture(scope="module", autouse=True)
def _built():
    gbuild.build()
    gla.load()


def _np(t):
    if t.dtype == torch.bfloat16:
        return t.float().cpu().numpy().astype(np.float64)
    return t.cpu().numpy().astype(np.float64)


def _run(inp, B, gh, gw, F, dtype, layout="concat", bias=True):
    h = to_torch(inp["h"], dtype)
    if layout == "concat":
        gate, value = h[:, :, :F], h[:, :, F:]
    else:  # separate contiguous tensors
        gate, value = h[:, :, :F].contiguous(), h[:, :, F:].contiguous()
        assert gate.stride(1) == F
    w = torch.from_numpy(inp["weight"]).cuda()
    b = torch.from_numpy(inp["bias"]).cuda() if (bias and inp["bias"] is not None) else None
    out = gla.sswiglu_dwconv(gate, value, w, b, gh, gw)
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    return out


def _ref(inp, F, dtype, gh, gw, bias=True):
    h = wl.storage_to_f64(inp["h"], dtype)
    return oracle.sswiglu_dwconv(h[:, :, :F], h[:, :, F:], inp["weight"], inp["bias"] if bias else None, gh, gw)


# (B, grid_h, grid_w, F, dtype)
CASES = [
    (1, 1, 1, 64, "bf16"),      # one token: the centre tap only
    (1, 1, 7, 64, "f16"),       # one row
    (2, 7, 1, 64, "bf16"),      # one column
    (1, 5, 6, 8, "f16"),        # F = 8: one channel group of the slice
    (3, 13, 9, 24, "bf16"),     # partial slice (24 of 64 channels)
    (1, 40, 40, 136, "f16"),    # 3 row tiles (ragged last), 3 slices (the last partial)
    (2, 9, 11, 64, "f32"),      # fp32: 32-channel slices
    (1, 6, 5, 12, "f32"),       # fp32, partial slice
    (1, 20, 128, 64, "bf16"),   # wide grid: 4 rows per tile
    (1, 3, 254, 16, "f16"),     # the widest grid the box takes
]


@pytest.mark.parametrize("case", CASES, ids=[f"{c[0]}x{c[1]}x{c[2]}-F{c[3]}-{c[4]}" for c in CASES])
def test_matches_oracle(case):
    B, gh, gw, F, dtype = case
    inp = wl.sswiglu_inputs(B, gh, gw, F, dtype, seed=6000 + CASES.index(case))
    out = _run(inp, B, gh, gw, F, dtype)
    assert_within_bar(_np(out), _ref(inp, F, dtype, gh, gw), dtype, f"sswiglu {case}")


@pytest.mark.parametrize("dtype", ["f16", "bf16", "f32"])
def test_separate_inputs_no_bias(dtype):
    B, gh, gw, F = 2, 11, 17, 72 if dtype != "f32" else 36
    inp = wl.sswiglu_inputs(B, gh, gw, F, dtype, seed=6100, with_bias=False)
    out = _run(inp, B, gh, gw, F, dtype, layout="separate", bias=False)
    assert_within_bar(_np(out), _ref(inp, F, dtype, gh, gw, bias=False), dtype, "separate, no bias")
    # the same inputs as halves of one tensor give the same bits
    out2 = _run(inp, B, gh, gw, F, dtype, layout="concat", bias=False)
    assert torch.equal(out, out2)


def test_rejects_bad_arguments():
    inp = wl.sswiglu_inputs(1, 4, 4, 16, "f16", seed=1)
    h = to_torch(inp["h"], "f16")
    w = torch.from_numpy(inp["weight"]).cuda()
    with pytest.raises(ValueError):
        gla.sswiglu_dwconv(h[:, :, :16], h[:, :, 16:], w, None, 4, 5)          # T != grid_h * grid_w
    with pytest.raises(gla.GLAError):
        gla.sswiglu_dwconv(h[:, :, :12], h[:, :, 16:28], w[:12], None, 4, 4)   # F = 12: not a multiple of 8
    big = torch.zeros((1, 2 * 256, 32), dtype=torch.float16, device="cuda")
    wb = torch.zeros((16, 3, 3), dtype=torch.float32, device="cuda")
    with pytest.raises(gla.GLAError) as ei:
        gla.sswiglu_dwconv(big[:, :, :16], big[:, :, 16:], wb, None, 2, 256)  # grid wider than the box
    assert ei.value.status == 2


@pytest.mark.parametrize("wid", [1, 2, 3])
def test_full_size_workload_sampled(wid):
    """Full-size launch (the configuration bench.py --op sswiglu times), checked on the
    first and last image and a spread of channels."""
    sw = wl.SWIGLU_WORKLOADS[wid]
    inp = wl.sswiglu_inputs(sw.B, sw.grid_h, sw.grid_w, sw.F, sw.dtype, seed=2609 + wid)
    out = _np(_run(inp, sw.B, sw.grid_h, sw.grid_w, sw.F, sw.dtype))
    F = sw.F
    bsel = sorted({0, sw.B - 1})
    fsel = np.unique(np.linspace(0, F - 1, 40).astype(int))
    h = wl.storage_to_f64(inp["h"][bsel], sw.dtype)
    ref = oracle.sswiglu_dwconv(h[:, :, fsel], h[:, :, F + fsel], inp["weight"][fsel], inp["bias"][fsel],
                                sw.grid_h, sw.grid_w)
    assert_within_bar(out[bsel][:, :, fsel], ref, sw.dtype, f"{sw.name} sampled")
