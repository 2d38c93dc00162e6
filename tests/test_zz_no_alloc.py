"""gtr_gla_fwd_noalloc, the entry point for callers that cannot allocate device
memory on the call path, keeps the split and balanced schedules' scratch in the
library's fixed array.  Checked here through the C ABI:

* on two calls in a row (the second runs over what the first left in the shared
  array) its results are bit-identical to gtr_gla_fwd_ws with a caller-owned
  workspace, which runs the same schedule, and both meet the mixer's bar against
  the fp64 oracle;
* once a call of each shape has run (the one-time address lookup and kernel
  loading), further calls leave the device's free memory unchanged;
* an empty batch returns GTR_OK with null pointers and launches nothing.

The file's name makes pytest collect it last, after every other test has used the
library; it also passes alone in a fresh process."""
import os
import re

import numpy as np
import pytest
import torch

import oracle
from gla_testutil import assert_within_bar, inputs_f64, to_torch
from paper_2609_26590_gb300 import build as gbuild
from paper_2609_26590_gb300 import gla
from paper_2609_26590_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

TORCH_DT = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}
HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "gtr_gla.h")

# (B, H, grid_h, grid_w, Dk, Dv, dtype, order): both calls split their sequences,
# so both use the scratch array; the second needs fewer summaries than the first
# wrote and reads a different layout of them.
CALLS = [(1, 2, 64, 64, 64, 64, "bf16", wl.ROW_FWD),
         (1, 1, 32, 32, 128, 128, "f16", wl.COL_REV)]


def scratch_limit():
    m = re.search(r"#define\s+GTR_GLA_NOALLOC_SCRATCH_BYTES\s+\((\d+)u\s*<<\s*(\d+)\)",
                  open(HEADER).read())
    assert m, "GTR_GLA_NOALLOC_SCRATCH_BYTES not found"
    return int(m.group(1)) << int(m.group(2))


def test_noalloc_matches_ws_bitwise_and_oracle_on_consecutive_calls():
    gbuild.build()
    gla.load()
    limit = scratch_limit()
    runs = []
    for i, (B, H, gh, gw, Dk, Dv, dtype, order) in enumerate(CALLS):
        need = gla.workspace_bytes(B, H, gh, gw, Dk, Dv, TORCH_DT[dtype])
        assert 0 < need <= limit, (need, limit)
        inp = wl.make_inputs(B, H, gh, gw, Dk, Dv, dtype, seed=9100 + i)
        t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v", "g")}
        out = torch.full_like(t["v"], float("nan"))
        fs = torch.full((B, H, Dk, Dv), float("nan"), dtype=torch.float32, device="cuda")
        runs.append((inp, t, out, fs))
    # one call of each shape first: it looks up the array's address and lets the
    # driver load each kernel (module loading may take device memory once)
    for (B, H, gh, gw, Dk, Dv, dtype, order), (inp, t, out, fs) in zip(CALLS, runs):
        gla.forward_noalloc(t["q"], t["k"], t["v"], t["g"], gh, gw, order, out, fs)
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    for _, _, out, fs in runs:
        out.fill_(float("nan"))
        fs.fill_(float("nan"))
    torch.cuda.synchronize()
    free_before = torch.cuda.mem_get_info()[0]
    # the two calls back to back on one stream: the second runs over what the first
    # left in the shared array; neither may change the device's free memory
    for (B, H, gh, gw, Dk, Dv, dtype, order), (inp, t, out, fs) in zip(CALLS, runs):
        gla.forward_noalloc(t["q"], t["k"], t["v"], t["g"], gh, gw, order, out, fs)
        assert gla.last_schedule()[0] == "tc_split"
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    assert torch.cuda.mem_get_info()[0] == free_before
    for (B, H, gh, gw, Dk, Dv, dtype, order), (inp, t, out, fs) in zip(CALLS, runs):
        need = gla.workspace_bytes(B, H, gh, gw, Dk, Dv, TORCH_DT[dtype])
        ws = torch.empty(need, dtype=torch.uint8, device="cuda")
        ref_out, ref_fs = torch.empty_like(out), torch.empty_like(fs)
        gla.forward_ws(t["q"], t["k"], t["v"], t["g"], gh, gw, order, ref_out, ref_fs, ws)
        torch.cuda.synchronize()
        assert gla.sync_status() == 0
        # same schedule, same arithmetic: the same bits
        assert torch.equal(out, ref_out)
        assert torch.equal(fs, ref_fs)
        f = inputs_f64(inp, dtype)
        o64, s64 = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], gh, gw, order)
        for got, what in ((out, "noalloc"), (ref_out, "ws")):
            assert_within_bar(got.float().cpu().numpy().astype(np.float64), o64, dtype, f"{what} out")
        for got, what in ((fs, "noalloc"), (ref_fs, "ws")):
            assert_within_bar(got.cpu().numpy().astype(np.float64), s64, dtype, f"{what} state")


def test_noalloc_empty_batch_launches_nothing():
    lib = gla.load()
    free0 = torch.cuda.mem_get_info()[0]
    st = lib.gtr_gla_fwd_noalloc(None, None, None, None, 0, 4, 40, 40, 64, 64, 0, 2, None, None, None)
    assert st == 0
    assert gla.last_schedule() == ("none", "none")
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
