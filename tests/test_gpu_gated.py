"""The mixer followed by its output gate (Sec. 3.1; App. C.3 fuses it into the
kernel's stores) against the fp64 oracle: u = SiLU(r) * RMSNorm(o) per head with
o the oracle's recurrence.

Bars for 16-bit u: where the tensor-core schedule applies the gate in its stores
(Dk, Dv <= 64, few sequences: 2 B H <= SMs) u is rounded once, from the fp32 outputs, and
is held to the mixer's bar (rel L2 <= 2e-3, max-abs <= 1e-2 max|u|).  Elsewhere a
second kernel applies the gate to the stored (rounded) o, so u carries two
roundings, and the gate multiplies each output by SiLU(r) w / rms, so an output
error at the mixer's bar can grow relative to max|u| where that factor is largest:
rel L2 <= 4e-3 and max-abs <= 4e-2 max|u|.  fp32: rel L2 <= 1e-5."""
import numpy as np
import pytest
import torch

import oracle
from gla_testutil import assert_within_bar, errors, inputs_f64, to_torch
from paper_2609_26590_gb300 import build as gbuild
from paper_2609_26590_gb300 import gla
from paper_2609_26590_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

TORCH_DT = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}

# (B, H, grid_h, grid_w, Dk, Dv, dtype, tau, z_mean)
CASES = [
    (2, 3, 16, 12, 64, 64, "bf16", 16.0, 0.0),     # fp16 score mode
    (1, 2, 48, 40, 64, 64, "f16", 1.0, -1.0),      # strong decay: tf32 score mode, split sequences
    (1, 3, 16, 12, 128, 64, "bf16", 16.0, 0.0),    # two key halves
    (37, 9, 16, 12, 64, 64, "bf16", 16.0, 0.0),    # many sequences per CTA
    (1, 2, 12, 12, 64, 64, "f32", 16.0, 0.0),     # fp32: CUDA cores + gate kernel
    (1, 2, 16, 8, 64, 128, "bf16", 16.0, 0.0),    # Dv = 128: two value slices, gate kernel
    (2, 2, 9, 13, 32, 32, "f16", 16.0, 0.0),      # Dk = Dv = 32, ragged
]


@pytest.fixture(scope="module", autouse=True)
def _built():
    gbuild.build()
    gla.load()


def _gate_inputs(B, H, T, Dv, dtype, seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    r = wl.round_to_storage(rng.standard_normal((B, T, H, Dv)) * 1.5, dtype)
    w = (1.0 + 0.2 * rng.standard_normal(Dv)).astype(np.float32)
    return r, w


@pytest.mark.parametrize("case", CASES, ids=[f"{c[0]}x{c[1]}-{c[2]}x{c[3]}-d{c[4]}_{c[5]}-{c[6]}"
                                             for c in CASES])
def test_gated_output_all_orders(case):
    B, H, gh, gw, Dk, Dv, dtype, tau, zm = case
    T = gh * gw
    inp = wl.make_inputs(B, H, gh, gw, Dk, Dv, dtype, seed=9000 + CASES.index(case), tau=tau, z_mean=zm)
    r, w = _gate_inputs(B, H, T, Dv, dtype, seed=9500 + CASES.index(case))
    eps = 1e-5
    f = inputs_f64(inp, dtype)
    r64 = wl.storage_to_f64(r, dtype)
    t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v", "g")}
    tr = to_torch(r, dtype)
    tw = torch.from_numpy(w).cuda()
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    fused = dtype != "f32" and Dk <= 64 and Dv <= 64 and 2 * B * H <= n_sm
    scale = 1.0 if (dtype == "f32" or fused) else 2.0
    for order in wl.ALL_ORDERS:
        ref_o, ref_s = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], gh, gw, order)
        ref_u = oracle.gated_output(ref_o, r64, w.astype(np.float64), eps)
        out = torch.full_like(t["v"], float("nan"))
        u, fs = gla.forward_gated(t["q"], t["k"], t["v"], t["g"], tr, tw, eps, gh, gw, order, out=out)
        torch.cuda.synchronize()
        assert gla.sync_status() == 0
        got = u.float().cpu().numpy().astype(np.float64)
        e = errors(got, ref_u)
        assert e["finite"], e
        bar_l2 = 1e-5 if dtype == "f32" else 2e-3 * scale
        assert e["rel_l2"] <= bar_l2, f"order {order}: {e}"
        if dtype != "f32":
            assert e["max_abs"] <= (1e-2 if fused else 4e-2) * e["max_ref"], f"order {order}: {e}"
        assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, dtype, f"state {order}")


def test_gated_matches_forward_then_gate():
    """The gated call = the plain forward followed by the gate on its stored o."""
    B, H, gh, gw, D, dtype = 3, 4, 16, 16, 64, "bf16"
    inp = wl.make_inputs(B, H, gh, gw, D, D, dtype, seed=9900)
    r, w = _gate_inputs(B, H, gh * gw, D, dtype, seed=9901)
    t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v", "g")}
    o, _ = gla.forward(t["q"], t["k"], t["v"], t["g"], gh, gw, wl.COL_REV)
    u, _ = gla.forward_gated(t["q"], t["k"], t["v"], t["g"], to_torch(r, dtype), torch.from_numpy(w).cuda(),
                             1e-6, gh, gw, wl.COL_REV)
    torch.cuda.synchronize()
    # the reference starts from the stored (rounded) o: two roundings apart, twice the bar
    ref = oracle.gated_output(o.float().cpu().numpy(), wl.storage_to_f64(r, dtype), w, 1e-6)
    e = errors(u.float().cpu().numpy().astype(np.float64), ref)
    assert e["finite"] and e["rel_l2"] <= 4e-3 and e["max_abs"] <= 4e-2 * e["max_ref"], e


def test_gated_ws_matches_and_captures_split():
    """gtr_gla_fwd_gated_ws: the caller's workspace gives the same split schedule as the
    internal one (identical bits), a short workspace is refused before any launch, and
    the call captured into a CUDA graph keeps the split and reproduces the bits."""
    B, H, gh, gw, D, dtype = 1, 6, 40, 40, 64, "f16"      # 25 chunks per sequence: split
    T = gh * gw
    need = gla.workspace_bytes(B, H, gh, gw, D, D, TORCH_DT[dtype])
    assert need > 0, "this shape should split its sequences"
    inp = wl.make_inputs(B, H, gh, gw, D, D, dtype, seed=9701)
    r, w = _gate_inputs(B, H, T, D, dtype, seed=9702)
    t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v", "g")}
    tr, tw = to_torch(r, dtype), torch.from_numpy(w).cuda()
    ref, ref_fs = gla.forward_gated(t["q"], t["k"], t["v"], t["g"], tr, tw, 1e-5, gh, gw, wl.COL_REV)
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    out, fs = gla.forward_gated(t["q"], t["k"], t["v"], t["g"], tr, tw, 1e-5, gh, gw, wl.COL_REV,
                                workspace=ws)
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    assert torch.equal(out, ref) and torch.equal(fs, ref_fs)
    with pytest.raises(gla.GLAError) as ei:
        gla.forward_gated(t["q"], t["k"], t["v"], t["g"], tr, tw, 1e-5, gh, gw, wl.COL_REV,
                          workspace=ws[: need - 256])
    assert ei.value.status == 3                             # GTR_ERR_WORKSPACE
    out2 = torch.full_like(out, float("nan"))
    fs2 = torch.full_like(fs, float("nan"))
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            gla.forward_gated(t["q"], t["k"], t["v"], t["g"], tr, tw, 1e-5, gh, gw, wl.COL_REV, out=out2,
                              final_state=fs2, stream=s, workspace=ws)
    torch.cuda.current_stream().wait_stream(s)
    g.replay()
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    assert torch.equal(out2, ref) and torch.equal(fs2, ref_fs)
