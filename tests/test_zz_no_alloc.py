"""gtr_gla_fwd_noalloc, the entry point that allocates no device memory and keeps
the split schedule's segment summaries in the library's fixed scratch array,
against gtr_gla_fwd on the same inputs.  Consecutive calls share that array, so
the second call runs over what the first left there.  The file's name makes
pytest collect it last, after every other test has used the library."""
import os
import re

import numpy as np
import pytest
import torch

from gla_testutil import assert_within_bar, to_torch
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


def test_noalloc_matches_fwd_on_consecutive_calls():
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
        runs.append((t, out, fs))
    # the two no-allocation calls back to back on one stream
    for (B, H, gh, gw, Dk, Dv, dtype, order), (t, out, fs) in zip(CALLS, runs):
        gla.forward_noalloc(t["q"], t["k"], t["v"], t["g"], gh, gw, order, out, fs)
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    for (B, H, gh, gw, Dk, Dv, dtype, order), (t, out, fs) in zip(CALLS, runs):
        ref_o, ref_s = gla.forward(t["q"], t["k"], t["v"], t["g"], gh, gw, order)
        torch.cuda.synchronize()
        assert gla.sync_status() == 0
        assert_within_bar(out.float().cpu().numpy().astype(np.float64),
                          ref_o.float().cpu().numpy().astype(np.float64), dtype, "out")
        assert_within_bar(fs.cpu().numpy().astype(np.float64),
                          ref_s.cpu().numpy().astype(np.float64), dtype, "state")
