"""GPU parity: the CUDA path (through the C ABI) against the fp64 CPU oracle on
the same seeded inputs, element by element, at the five workloads' full sizes
(every scan order) and at small ragged shapes, plus edge cases, determinism,
CUDA-graph capture, the host-memory entry point and guard bands."""
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


@pytest.fixture(scope="module", autouse=True)
def _built():
    gbuild.build()
    gla.load()


class _Cache:
    """Inputs and oracle results of one workload at a time (the big ones take GBs)."""
    wid = None
    inp = None
    f64 = None
    ref = {}

    @classmethod
    def get(cls, wid):
        if cls.wid != wid:
            cls.wid, cls.ref = wid, {}
            w = wl.WORKLOADS[wid]
            cls.inp = wl.workload_inputs(w)
            cls.f64 = inputs_f64(cls.inp, w.dtype)
        return cls.inp, cls.f64

    @classmethod
    def oracle(cls, wid, order):
        if order not in cls.ref:
            w = wl.WORKLOADS[wid]
            _, f = cls.get(wid)
            cls.ref[order] = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], w.grid_h, w.grid_w,
                                               order)
        return cls.ref[order]


def _run(inp, dtype, gh, gw, order, schedule="auto", final_state=True):
    t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v", "g")}
    out, fs = gla.forward(t["q"], t["k"], t["v"], t["g"], gh, gw, order,
                          final_state=final_state, schedule=schedule)
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    return out, fs


def _np(t):
    return t.float().cpu().numpy().astype(np.float64)


WORKLOAD_CASES = [(w.wid, o, s) for w in wl.WORKLOADS.values() for o in w.orders
                  for s in ("auto", "simt")]


@pytest.mark.parametrize("wid,order,schedule", WORKLOAD_CASES,
                         ids=[f"w{w}-{wl.ORDER_NAMES[o]}-{s}" for w, o, s in WORKLOAD_CASES])
def test_workload_full_size(wid, order, schedule):
    w = wl.WORKLOADS[wid]
    inp, _ = _Cache.get(wid)
    ref_o, ref_s = _Cache.oracle(wid, order)
    out, fs = _run(inp, w.dtype, w.grid_h, w.grid_w, order, schedule)
    assert_within_bar(_np(out), ref_o, w.dtype, f"out w{wid} {schedule}")
    assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, w.dtype, f"state w{wid}")


# (B, H, grid_h, grid_w, Dk, Dv, dtype, tau, z_mean) -- several chunks, ragged tails,
# fewer tokens than a chunk, non-square grids, Dk != Dv, strong decay.
SMALL = [
    (2, 3, 9, 13, 64, 64, "f16", 16.0, 0.0),
    (1, 2, 5, 5, 64, 64, "bf16", 16.0, 0.0),
    (2, 2, 16, 24, 64, 64, "bf16", 1.0, -1.0),
    (1, 3, 40, 8, 64, 64, "f16", 1.0, -1.0),
    (1, 1, 1, 1, 64, 64, "f32", 16.0, 0.0),
    (1, 2, 3, 100, 128, 128, "bf16", 16.0, 0.0),
    (2, 1, 8, 16, 128, 128, "f16", 1.0, -1.0),
    (1, 2, 16, 16, 32, 64, "f16", 16.0, 0.0),
    (1, 2, 12, 12, 64, 32, "f32", 16.0, 0.0),
    (2, 2, 24, 16, 64, 64, "f16", 1.0, -3.0),
    (1, 2, 8, 8, 64, 64, "bf16", 16.0, 0.0),
    (1, 2, 8, 13, 64, 64, "bf16", 16.0, 0.0),
    (2, 1, 16, 9, 64, 64, "f16", 1.0, -1.0),
    (3, 2, 8, 24, 64, 64, "f16", 16.0, 0.0),
    (1, 1, 48, 40, 64, 64, "bf16", 1.0, -1.0),
    (2, 2, 8, 24, 64, 128, "f16", 16.0, 0.0),
    (1, 3, 16, 12, 128, 64, "bf16", 1.0, -1.0),
    (1, 2, 24, 8, 128, 128, "f16", 1.0, -3.0),
    (1, 6, 44, 44, 64, 64, "f16", 16.0, 0.0),     # 704^2 input at stride 16 (1936 tokens): ragged columns
    (2, 2, 7, 11, 64, 64, "bf16", 1.0, -1.0),      # odd grid: every column segment has a remainder box
    (2, 2, 16, 16, 32, 64, "bf16", 1.0, -1.0),     # the paper's dk = 32, dv = 64: zero-padded key half
    (1, 3, 12, 10, 96, 40, "bf16", 16.0, 0.0),     # padded second key half and value slice
]


@pytest.mark.parametrize("case", SMALL, ids=[f"{c[0]}x{c[1]}-{c[2]}x{c[3]}-d{c[4]}_{c[5]}-{c[6]}"
                                             for c in SMALL])
@pytest.mark.parametrize("schedule", ["auto", "simt", "tc"])
def test_small_shapes_all_orders(case, schedule):
    B, H, gh, gw, Dk, Dv, dtype, tau, zm = case
    if schedule == "tc" and not gla.tc_supported(B, H, gh, gw, Dk, Dv, 0, TORCH_DT[dtype]):
        pytest.skip("tensor-core schedule does not take this shape")
    inp = wl.make_inputs(B, H, gh, gw, Dk, Dv, dtype, seed=1000 + SMALL.index(case), tau=tau,
                         z_mean=zm)
    f = inputs_f64(inp, dtype)
    for order in wl.ALL_ORDERS:
        ref_o, ref_s = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], gh, gw, order)
        out, fs = _run(inp, dtype, gh, gw, order, schedule)
        assert_within_bar(_np(out), ref_o, dtype, f"out order {order}")
        assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, dtype, f"state {order}")


# More (b, h) sequences than a GB300 has SMs, so that every persistent CTA of the
# tensor-core schedule walks two or three sequences back to back through one
# pipeline (state reset, final state and output positions per sequence).
STREAM = [
    (37, 9, 16, 12, 64, 64, "bf16", 16.0, 0.0),    # 333 sequences of 3 full chunks
    (41, 8, 8, 13, 64, 64, "f16", 1.0, -1.0),      # 328 sequences of 104 tokens (ragged), strong decay
    (23, 15, 24, 16, 64, 64, "bf16", 1.0, -3.0),   # 345 sequences, decays beyond the fp16 split range
    (20, 9, 16, 8, 128, 128, "bf16", 16.0, 0.0),   # 360 work units: two value slices per sequence
]


@pytest.mark.parametrize("case", STREAM, ids=[f"{c[0]}x{c[1]}-{c[2]}x{c[3]}-d{c[4]}_{c[5]}-{c[6]}"
                                              for c in STREAM])
def test_many_sequences_per_cta(case):
    B, H, gh, gw, Dk, Dv, dtype, tau, zm = case
    assert gla.tc_supported(B, H, gh, gw, Dk, Dv, 0, TORCH_DT[dtype])
    inp = wl.make_inputs(B, H, gh, gw, Dk, Dv, dtype, seed=3000 + STREAM.index(case), tau=tau,
                         z_mean=zm)
    f = inputs_f64(inp, dtype)
    for order in wl.ALL_ORDERS:
        ref_o, ref_s = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], gh, gw, order)
        out, fs = _run(inp, dtype, gh, gw, order, "tc")
        assert_within_bar(_np(out), ref_o, dtype, f"out order {order}")
        assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, dtype, f"state {order}")


# Few, long sequences: the tensor-core schedule splits each into segments of equal
# length but the last (a summary pass, then every segment from the fold of the earlier
# summaries).  When the chunk count is not a multiple of the length, the last segment
# runs past the sequence over all-zero padding chunks, in every scan order.
SPLIT = [
    (1, 2, 64, 64, 64, 64, "bf16", 16.0, 0.0, 0.0),     # 64 chunks, segments of 4
    (1, 1, 48, 40, 64, 64, "f16", 1.0, -1.0, 0.0),      # strong decay: tf32 scores; 30 chunks, 2 padding
    (1, 1, 32, 32, 128, 128, "bf16", 16.0, 0.0, 0.0),   # two key halves, two value slices
    (1, 1, 64, 16, 128, 64, "f16", 16.0, 0.0, 0.02),    # Dk != Dv, some gamma = 0 gates (exact path)
    (1, 2, 64, 40, 32, 64, "bf16", 16.0, 0.0, 0.0),     # padded key half: summaries keep the padded layout
    (1, 6, 40, 40, 64, 64, "f16", 16.0, 0.0, 0.0),      # 25 chunks: 3 padding chunks in the last segment
    (1, 6, 44, 44, 64, 64, "bf16", 16.0, 0.0, 0.0),     # 31 chunks, the last one ragged (16 tokens)
    (1, 3, 40, 36, 32, 64, "bf16", 16.0, 0.0, 0.0),     # Dk = 32, Dv = 64; 23 chunks
    (1, 1, 36, 36, 128, 128, "f16", 16.0, 0.0, 0.0),    # two key halves over padding chunks; 21 chunks
]


@pytest.mark.parametrize("case", SPLIT, ids=[f"{c[0]}x{c[1]}-{c[2]}x{c[3]}-d{c[4]}_{c[5]}-{c[6]}"
                                             for c in SPLIT])
def test_split_sequences(case):
    B, H, gh, gw, Dk, Dv, dtype, tau, zm, frac_zero = case
    ws_bytes = gla.workspace_bytes(B, H, gh, gw, Dk, Dv, TORCH_DT[dtype])
    assert ws_bytes > 0, "the schedule should split these sequences"
    inp = wl.make_inputs(B, H, gh, gw, Dk, Dv, dtype, seed=4000 + SPLIT.index(case), tau=tau,
                         z_mean=zm)
    if frac_zero > 0:
        rng = np.random.Generator(np.random.PCG64(77))
        g = wl.storage_to_f64(inp["g"], dtype)
        g[rng.random(g.shape) < frac_zero] = -np.inf
        inp["g"] = wl.round_to_storage(g, dtype)
    f = inputs_f64(inp, dtype)
    t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v", "g")}
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    for order in wl.ALL_ORDERS:
        ref_o, ref_s = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], gh, gw, order)
        out, fs = _run(inp, dtype, gh, gw, order, "tc")  # internal workspace
        assert_within_bar(_np(out), ref_o, dtype, f"out order {order}")
        assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, dtype, f"state {order}")
        out2 = torch.empty_like(t["v"])
        fs2 = torch.empty_like(fs)
        gla.forward_ws(t["q"], t["k"], t["v"], t["g"], gh, gw, order, out2, fs2, ws)
        torch.cuda.synchronize()
        assert gla.sync_status() == 0
        assert torch.equal(out2, out) and torch.equal(fs2, fs)  # same schedule, same bits


@pytest.mark.parametrize("dtype", ["f16", "bf16", "f32"])
@pytest.mark.parametrize("gate", ["one", "zero"])
def test_gate_extremes(dtype, gate):
    """gamma = 1 (g = 0: causal linear attention) and gamma = 0 (g = -inf:
    o_t = (q_t . k_t) v_t) on every schedule that takes the shape."""
    B, H, gh, gw, D = 2, 2, 16, 12, 64
    inp = wl.make_inputs(B, H, gh, gw, D, D, dtype, seed=5)
    g = np.zeros((B, gh * gw, H, D)) if gate == "one" else np.full((B, gh * gw, H, D), -np.inf)
    inp["g"] = wl.round_to_storage(g, dtype)
    f = inputs_f64(inp, dtype)
    for schedule in ("auto", "simt"):
        for order in wl.ALL_ORDERS:
            ref_o, ref_s = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], gh, gw, order)
            out, fs = _run(inp, dtype, gh, gw, order, schedule)
            assert_within_bar(_np(out), ref_o, dtype, f"{gate} {schedule} {order}")
            assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, dtype, "state")


def test_no_final_state_and_empty_batch():
    inp = wl.make_inputs(1, 2, 8, 8, 64, 64, "f16", seed=3)
    f = inputs_f64(inp, "f16")
    out, fs = _run(inp, "f16", 8, 8, wl.COL_FWD, final_state=None)
    assert fs is None
    ref_o, _ = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], 8, 8, wl.COL_FWD)
    assert_within_bar(_np(out), ref_o, "f16")
    z = torch.empty((0, 64, 2, 64), dtype=torch.float16, device="cuda")
    o, s = gla.forward(z, z, z, z, 8, 8, 0)
    assert o.shape == z.shape and s.shape == (0, 2, 64, 64)


@pytest.mark.parametrize("wid", [1, 3])
def test_deterministic(wid):
    w = wl.WORKLOADS[wid]
    inp, _ = _Cache.get(wid)
    a, sa = _run(inp, w.dtype, w.grid_h, w.grid_w, wl.COL_REV)
    b, sb = _run(inp, w.dtype, w.grid_h, w.grid_w, wl.COL_REV)
    assert torch.equal(a, b) and torch.equal(sa, sb)


def test_guard_bands_and_full_coverage():
    """Outputs pre-filled with NaN inside a sentinel-padded allocation: every
    output element is written, nothing outside is touched."""
    B, H, gh, gw, D = 2, 3, 9, 13, 64
    inp = wl.make_inputs(B, H, gh, gw, D, D, "bf16", seed=9)
    t = {n: to_torch(inp[n], "bf16") for n in ("q", "k", "v", "g")}
    n_out = B * gh * gw * H * D
    pad = 4096
    buf = torch.full((n_out + 2 * pad,), 1024.0, dtype=torch.bfloat16, device="cuda")
    buf[pad:pad + n_out] = float("nan")
    out = buf[pad:pad + n_out].view(B, gh * gw, H, D)
    fbuf = torch.full((B * H * D * D + 2 * pad,), -777.0, device="cuda")
    fbuf[pad:pad + B * H * D * D] = float("nan")
    fs = fbuf[pad:pad + B * H * D * D].view(B, H, D, D)
    for order in wl.ALL_ORDERS:
        gla.forward(t["q"], t["k"], t["v"], t["g"], gh, gw, order, out=out, final_state=fs)
        torch.cuda.synchronize()
        assert not torch.isnan(out).any() and not torch.isnan(fs).any()
        assert (buf[:pad] == 1024.0).all() and (buf[pad + n_out:] == 1024.0).all()
        assert (fbuf[:pad] == -777.0).all() and (fbuf[pad + B * H * D * D:] == -777.0).all()


def test_cuda_graph_capture():
    """Replaying a captured graph equals eager execution.  With a caller-owned
    workspace both run the same schedule (here the split one: two kernels), bit for
    bit.  gtr_gla_fwd does not use its internal workspace under capture and runs
    the sequences unsplit there: that result is held to the oracle's bar."""
    w = wl.WORKLOADS[1]
    inp, _ = _Cache.get(1)
    ref_o, ref_s = _Cache.oracle(1, wl.ROW_REV)
    t = {n: to_torch(inp[n], w.dtype) for n in ("q", "k", "v", "g")}
    ws_bytes = gla.workspace_bytes(w.B, w.H, w.grid_h, w.grid_w, w.Dk, w.Dv, TORCH_DT[w.dtype])
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda") if ws_bytes else None
    out = torch.empty_like(t["v"])
    fs = torch.empty((w.B, w.H, w.Dk, w.Dv), device="cuda")
    gla.forward_ws(t["q"], t["k"], t["v"], t["g"], w.grid_h, w.grid_w, wl.ROW_REV, out, fs, ws)
    torch.cuda.synchronize()
    ref, ref_fs = out.clone(), fs.clone()
    out.zero_()
    fs.zero_()
    out2 = torch.empty_like(t["v"])
    fs2 = torch.empty_like(fs)
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            gla.forward_ws(t["q"], t["k"], t["v"], t["g"], w.grid_h, w.grid_w, wl.ROW_REV, out, fs, ws,
                           stream=s)
            gla.forward(t["q"], t["k"], t["v"], t["g"], w.grid_h, w.grid_w, wl.ROW_REV, out=out2,
                        final_state=fs2, stream=s)
    g.replay()
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    assert torch.equal(out, ref) and torch.equal(fs, ref_fs)
    assert_within_bar(_np(out2), ref_o, w.dtype, "captured gtr_gla_fwd")
    assert_within_bar(fs2.cpu().numpy().astype(np.float64), ref_s, w.dtype, "captured state")


def test_host_memory_entry_point():
    w = wl.WORKLOADS[1]
    inp, f = _Cache.get(1)
    host = {n: to_torch(inp[n], w.dtype, device="cpu").pin_memory() for n in ("q", "k", "v", "g")}
    out = torch.empty(host["v"].shape, dtype=host["v"].dtype).pin_memory()
    fs = torch.empty((w.B, w.H, w.Dk, w.Dv)).pin_memory()
    nbytes = gla.host_buffer_bytes(w.B, w.H, w.grid_h, w.grid_w, w.Dk, w.Dv, host["q"].dtype)
    dev = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    gla.forward_host(host["q"], host["k"], host["v"], host["g"], w.grid_h, w.grid_w, wl.COL_FWD,
                     out, fs, dev)
    torch.cuda.synchronize()
    ref_o, ref_s = _Cache.oracle(1, wl.COL_FWD)
    assert_within_bar(out.float().numpy().astype(np.float64), ref_o, w.dtype, "host out")
    assert_within_bar(fs.numpy().astype(np.float64), ref_s, w.dtype, "host state")


def test_explicit_schedule_rejects_unsupported():
    inp = wl.make_inputs(1, 1, 4, 4, 64, 64, "f32", seed=1)
    t = {n: to_torch(inp[n], "f32") for n in ("q", "k", "v", "g")}
    with pytest.raises(gla.GLAError) as ei:
        gla.forward(t["q"], t["k"], t["v"], t["g"], 4, 4, 0, schedule="tc")
    assert ei.value.status == 2


def test_workspace_matches_split_plan():
    """The workspace the schedule asks for is that of the plan gtr_gla_split_plan and
    gtr_gla_balanced_plan report for this device's SM count: (segments - 1) per
    sequence of padded (Dk x Dv + Dk) floats for a split, one 64 x 64 fp32 state and
    one 64-bit flag per SM for balanced ranges, else nothing."""
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    pad = lambda d: (d + 63) // 64 * 64
    for B, H, gh, gw, Dk, Dv in [(1, 6, 40, 40, 64, 64), (1, 6, 44, 44, 64, 64), (2, 8, 128, 128, 128, 128),
                                 (32, 12, 40, 40, 64, 64), (1, 3, 40, 36, 32, 64), (1, 1, 16, 20, 64, 64),
                                 (8, 16, 80, 80, 64, 64), (1, 160, 8, 16, 64, 64)]:
        nseg, seg_len = gla.split_plan(B, H, gh, gw, Dk, Dv, n_sm)
        bal = gla.balanced_plan(B, H, gh, gw, Dk, Dv, n_sm)
        assert not (bal and nseg > 1)
        if nseg > 1:
            expect = B * H * (nseg - 1) * (pad(Dk) * pad(Dv) + pad(Dk)) * 4
        else:
            expect = n_sm * (64 * 64 * 4 + 8) if bal else 0
        for dt in (torch.float16, torch.bfloat16):
            assert gla.workspace_bytes(B, H, gh, gw, Dk, Dv, dt) == expect, (B, H, gh, gw, Dk, Dv, nseg, seg_len, bal)


# More (sequence, value slice) units than SMs, not a multiple of them: the tensor-core
# schedule gives every CTA an equal contiguous range of chunks, and a unit cut by a range
# boundary continues on the next CTA from the state handed over through the workspace
# (its end state after the head of the range before).  H is set from the device's SM
# count so that the units exceed it by a few; (Dv, dtype, grid_h, grid_w, extra units).
BALANCED = [(64, "bf16", 8, 16, 8), (64, "f16", 24, 8, 40), (128, "bf16", 16, 12, 10), (32, "f16", 5, 13, 3)]


@pytest.mark.parametrize("case", BALANCED, ids=[f"dv{c[0]}_{c[1]}-{c[2]}x{c[3]}+{c[4]}" for c in BALANCED])
def test_balanced_ranges(case):
    Dv, dtype, gh, gw, extra = case
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    nv = (Dv + 63) // 64
    H = (n_sm + extra + nv - 1) // nv
    B, Dk = 1, 64
    assert gla.balanced_plan(B, H, gh, gw, Dk, Dv, n_sm), "the schedule should balance these units"
    ws_bytes = gla.workspace_bytes(B, H, gh, gw, Dk, Dv, TORCH_DT[dtype])
    assert ws_bytes == n_sm * (64 * 64 * 4 + 8)
    inp = wl.make_inputs(B, H, gh, gw, Dk, Dv, dtype, seed=7100 + BALANCED.index(case))
    f = inputs_f64(inp, dtype)
    t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v", "g")}
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    for order in wl.ALL_ORDERS:
        ref_o, ref_s = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], gh, gw, order)
        out, fs = _run(inp, dtype, gh, gw, order, "tc")  # internal workspace
        assert_within_bar(_np(out), ref_o, dtype, f"out order {order}")
        assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, dtype, f"state {order}")
        for rep in range(2):  # a caller workspace twice: flags of the call before are not taken
            out2, fs2 = torch.empty_like(t["v"]), torch.empty_like(fs)
            gla.forward_ws(t["q"], t["k"], t["v"], t["g"], gh, gw, order, out2, fs2, ws)
            torch.cuda.synchronize()
            assert gla.sync_status() == 0
            assert torch.equal(out2, out) and torch.equal(fs2, fs)  # same schedule, same bits
    # one captured launch replayed: each replay hands its states over afresh
    order = wl.COL_REV
    out_ref, fs_ref = _run(inp, dtype, gh, gw, order, "tc")
    out3, fs3 = torch.empty_like(t["v"]), torch.empty_like(fs_ref)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(g, stream=side):
            gla.forward_ws(t["q"], t["k"], t["v"], t["g"], gh, gw, order, out3, fs3, ws, stream=side)
    torch.cuda.current_stream().wait_stream(side)
    for rep in range(3):
        out3.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert gla.sync_status() == 0
        assert torch.equal(out3, out_ref) and torch.equal(fs3, fs_ref)
