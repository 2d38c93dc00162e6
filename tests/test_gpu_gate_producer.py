"""The mixer with the retention gate computed in the kernel (Sec. 3.1, the key-wise gate
from its rank-16 projection): gtr_gla_fwd_lowrank_gate against the fp64 oracle's
gate_producer followed by its recurrence, element by element on o and the final state, at
the mixer's bar.  Covers both 16-bit types, all four scan orders, a ragged grid, the
paper's mild gates (tau = 16) and strongly decaying ones (tau = 1, whose chunks take the
tf32 score path), Dk below 64 (zero-padded key channels), Dv = 128 (two value slices) and
more sequences than SMs (a CTA walks several heads, so the W2 block changes between
units)."""
import numpy as np
import pytest
import torch

import oracle
from gla_testutil import assert_within_bar, inputs_f64, to_torch
from paper_2609_26590_gb300 import gla
from paper_2609_26590_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

# (B, H, grid_h, grid_w, Dk, Dv, dtype, order, tau, z_mean)
CASES = [
    (2, 3, 20, 23, 64, 64, "bf16", wl.ROW_FWD, 16.0, 0.0),
    (2, 3, 20, 23, 64, 64, "bf16", wl.ROW_REV, 16.0, 0.0),
    (2, 3, 20, 23, 64, 64, "f16", wl.COL_FWD, 16.0, 0.0),
    (2, 3, 20, 23, 64, 64, "f16", wl.COL_REV, 16.0, 0.0),
    (1, 4, 16, 16, 64, 64, "f16", wl.ROW_FWD, 1.0, -1.0),
    (1, 4, 16, 16, 64, 64, "bf16", wl.COL_REV, 1.0, -1.0),
    (1, 2, 40, 40, 32, 64, "f16", wl.COL_REV, 16.0, 0.0),
    (1, 2, 24, 24, 64, 128, "bf16", wl.ROW_REV, 16.0, 0.0),
    (16, 12, 16, 20, 64, 64, "bf16", wl.COL_FWD, 16.0, 0.0),
]


def _run(B, H, gh, gw, Dk, Dv, dtype, order, tau, zm, seed):
    T = gh * gw
    inp = wl.make_inputs(B, H, gh, gw, Dk, Dv, dtype, seed=seed)
    gp = wl.gate_producer_inputs(B, H, T, Dk, dtype, seed=seed + 1, z_mean=zm)
    t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v")}
    a = to_torch(gp["a"], dtype)
    w2 = to_torch(gp["w2"], dtype)
    bias = torch.from_numpy(gp["bias"]).cuda()
    out = torch.full_like(t["v"], float("nan"))
    fs = torch.full((B, H, Dk, Dv), float("nan"), dtype=torch.float32, device="cuda")
    gla.forward_lowrank_gate(t["q"], t["k"], t["v"], a, w2, bias, tau, gh, gw, order, out=out, final_state=fs)
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    assert gla.last_schedule() == ("tc", "tc")
    f = inputs_f64(inp, dtype)
    g64 = oracle.gate_producer(wl.storage_to_f64(gp["a"], dtype), wl.storage_to_f64(gp["w2"], dtype),
                               gp["bias"].astype(np.float64), tau)
    ref_o, ref_s = oracle.recurrence(f["q"], f["k"], f["v"], g64, gh, gw, order)
    return out, fs, ref_o, ref_s


@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(str(x) for x in c[:6]) + f"-{c[6]}-o{c[7]}-tau{c[8]:g}")
def test_gate_producer_matches_oracle(case):
    gla.load()
    B, H, gh, gw, Dk, Dv, dtype, order, tau, zm = case
    out, fs, ref_o, ref_s = _run(B, H, gh, gw, Dk, Dv, dtype, order, tau, zm, seed=7300 + CASES.index(case))
    assert_within_bar(out.float().cpu().numpy().astype(np.float64), ref_o, dtype, "out")
    assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, dtype, "final_state")


def test_gate_producer_rejects_unsupported_shapes():
    gla.load()
    B, H, gh, gw, D = 1, 2, 16, 16, 64
    t = torch.zeros((B, gh * gw, H, D), dtype=torch.float16, device="cuda")
    a = torch.zeros((B, gh * gw, 16), dtype=torch.float16, device="cuda")
    w2 = torch.zeros((H, 16, D), dtype=torch.float16, device="cuda")
    bias = torch.zeros((H, D), dtype=torch.float32, device="cuda")
    with pytest.raises(gla.GLAError) as ei:   # T = 192: fewer than four chunks
        tt = torch.zeros((B, 192, H, D), dtype=torch.float16, device="cuda")
        gla.forward_lowrank_gate(tt, tt, tt, a[:, :192], w2, bias, 16.0, 12, 16)
    assert ei.value.status == 2
    with pytest.raises(gla.GLAError) as ei:   # rank 8
        gla.forward_lowrank_gate(t, t, t, a[:, :, :8].contiguous(), w2[:, :8].contiguous(), bias, 16.0, gh, gw)
    assert ei.value.status == 2
    with pytest.raises(gla.GLAError) as ei:   # tau = 0
        gla.forward_lowrank_gate(t, t, t, a, w2, bias, 0.0, gh, gw)
    assert ei.value.status == 1
