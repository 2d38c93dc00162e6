"""gtr_gla_last_schedule reports which schedule a forward call launched and which one
it planned: the internal-workspace entry point outside stream capture splits a
batch-1 sequence, and under capture it runs unsplit and says so (the two results
agree within the mixer's bar)."""
import numpy as np
import pytest
import torch

from gla_testutil import assert_within_bar, to_torch
from paper_2609_26590_gb300 import gla
from paper_2609_26590_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def test_last_schedule_split_and_under_capture():
    gla.load()
    B, H, gh, gw, D, dt = 1, 2, 64, 64, 64, "bf16"
    inp = wl.make_inputs(B, H, gh, gw, D, D, dt, seed=515)
    t = {n: to_torch(inp[n], dt) for n in ("q", "k", "v", "g")}
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    assert gla.split_plan(B, H, gh, gw, D, D, n_sm)[0] > 1
    out, fs = gla.forward(t["q"], t["k"], t["v"], t["g"], gh, gw, wl.COL_FWD)
    assert gla.last_schedule() == ("tc_split", "tc_split")
    torch.cuda.synchronize()
    assert gla.sync_status() == 0

    out2 = torch.empty_like(out)
    fs2 = torch.empty_like(fs)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            gla.forward(t["q"], t["k"], t["v"], t["g"], gh, gw, wl.COL_FWD, out=out2, final_state=fs2)
    assert gla.last_schedule() == ("tc", "tc_split")
    torch.cuda.current_stream().wait_stream(s)
    g.replay()
    torch.cuda.synchronize()
    assert gla.sync_status() == 0
    assert_within_bar(out2.float().cpu().numpy().astype(np.float64),
                      out.float().cpu().numpy().astype(np.float64), dt, "out")
    assert_within_bar(fs2.cpu().numpy().astype(np.float64), fs.cpu().numpy().astype(np.float64), dt, "state")

    # the fp32 path has a single schedule
    t32 = {n: t[n].float() for n in t}
    gla.forward(t32["q"], t32["k"], t32["v"], t32["g"], gh, gw, wl.ROW_FWD)
    assert gla.last_schedule() == ("simt", "simt")
    torch.cuda.synchronize()
