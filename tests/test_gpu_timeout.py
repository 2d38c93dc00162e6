"""Failure detection without a GPU fault.  With the test hook
GTR_GLA_TEST_DROP_LOAD=1 the tensor-core kernel's producer in CTA 0 withholds
the load of its first chunk: the data never arrives, the bounded waits give up
after their limit (1 s), every warp role unwinds (copies drained, MMAs
completed, TMEM freed) and gtr_gla_sync_status reports GTR_ERR_TIMEOUT.  The
status word is cleared by that read and the context stays usable."""
import os

import numpy as np
import pytest
import torch

import oracle
from gla_testutil import assert_within_bar, inputs_f64, to_torch
from paper_2609_26590_gb300 import build as gbuild
from paper_2609_26590_gb300 import gla
from paper_2609_26590_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

GTR_ERR_TIMEOUT = 5


def test_bounded_wait_reports_timeout_and_context_survives():
    gbuild.build()
    gla.load()
    B, H, gh, gw, D, dtype = 1, 2, 8, 8, 64, "bf16"   # one chunk per sequence: a single launch
    assert gla.tc_supported(B, H, gh, gw, D, D, 0, torch.bfloat16)
    assert gla.workspace_bytes(B, H, gh, gw, D, D, torch.bfloat16) == 0
    inp = wl.make_inputs(B, H, gh, gw, D, D, dtype, seed=8100)
    t = {n: to_torch(inp[n], dtype) for n in ("q", "k", "v", "g")}
    assert gla.sync_status() == 0
    os.environ["GTR_GLA_TEST_DROP_LOAD"] = "1"
    try:
        gla.forward(t["q"], t["k"], t["v"], t["g"], gh, gw, wl.ROW_FWD, schedule="tc")
        status = gla.sync_status()
    finally:
        del os.environ["GTR_GLA_TEST_DROP_LOAD"]
    assert status == GTR_ERR_TIMEOUT
    assert gla.sync_status() == 0        # reading the word cleared it
    f = inputs_f64(inp, dtype)
    ref_o, ref_s = oracle.recurrence(f["q"], f["k"], f["v"], f["g"], gh, gw, wl.ROW_FWD)
    out, fs = gla.forward(t["q"], t["k"], t["v"], t["g"], gh, gw, wl.ROW_FWD, schedule="tc")
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    assert_within_bar(out.float().cpu().numpy().astype(np.float64), ref_o, dtype, "out after timeout")
    assert_within_bar(fs.cpu().numpy().astype(np.float64), ref_s, dtype, "state after timeout")
