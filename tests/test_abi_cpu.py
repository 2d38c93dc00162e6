"""The C-ABI library builds, loads and exports every symbol include/gtr_gla.h
declares; host-only entry points (argument validation, support queries,
sizes, status strings) behave as documented.  No compute is launched, so
these run without a GPU."""
import ctypes
import os
import re

import pytest

from paper_2609_26590_gb300 import build as gbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include"))
           if f.endswith(".h")]


@pytest.fixture(scope="module")
def lib():
    path = gbuild.build()
    from paper_2609_26590_gb300 import gla
    return gla.load(path)


def declared_functions():
    names = set()
    for h in HEADERS:
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        src = re.sub(r"//[^\n]*", "", src)
        for m in re.finditer(r"\b(gtr_[a-z0-9_]+)\s*\(", src):
            names.add(m.group(1))
    return sorted(names)


def test_header_declares_entry_points():
    names = declared_functions()
    for must in ("gtr_gla_fwd", "gtr_gla_fwd_sched", "gtr_gla_fwd_host", "gtr_gla_sync_status",
                 "gtr_status_string", "gtr_gla_workspace_bytes", "gtr_gla_fwd_ws"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    raw = ctypes.CDLL(gbuild.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(raw, n)]
    assert not missing, missing


def test_status_strings_and_version(lib):
    for s in range(6):
        assert lib.gtr_status_string(s)
    assert lib.gtr_status_string(99) == b"unknown status"
    assert lib.gtr_version() >= 100


def _fwd(lib, q=16, k=16, v=16, g=16, out=16, fs=None, B=1, H=1, gh=8, gw=8, Dk=64, Dv=64,
         order=0, dtype=1, sched=0):
    return lib.gtr_gla_fwd_sched(q, k, v, g, B, H, gh, gw, Dk, Dv, order, dtype, out, fs, sched,
                                 None)


def test_validation_rejects_before_launch(lib):
    # null / misaligned pointers, bad sizes and enums never reach the GPU
    assert _fwd(lib, q=None) == 1
    assert _fwd(lib, out=None) == 1
    assert _fwd(lib, k=24) == 1              # not 16-byte aligned
    assert _fwd(lib, fs=8) == 1
    assert _fwd(lib, Dk=0) == 1
    assert _fwd(lib, Dv=129) == 1
    assert _fwd(lib, gh=0) == 1
    assert _fwd(lib, B=-1) == 1
    assert _fwd(lib, order=4) == 1
    assert _fwd(lib, dtype=3) == 1
    assert _fwd(lib, sched=7) == 1
    # output overlapping an input
    assert lib.gtr_gla_fwd_sched(4096, 1 << 20, 2 << 20, 3 << 20, 1, 1, 8, 8, 64, 64, 0, 1,
                                 4096 + 64, None, 0, None) == 1
    # empty batch: valid, nothing to launch
    assert _fwd(lib, B=0, q=1 << 20, k=2 << 20, v=3 << 20, g=4 << 20, out=5 << 20) == 0


def test_last_schedule_after_an_empty_call(lib):
    # an empty call launches nothing and says so; NULL outputs are allowed
    assert _fwd(lib, B=0, q=1 << 20, k=2 << 20, v=3 << 20, g=4 << 20, out=5 << 20) == 0
    ran, planned = ctypes.c_int(-1), ctypes.c_int(-1)
    assert lib.gtr_gla_last_schedule(ctypes.byref(ran), ctypes.byref(planned)) == 0
    assert (ran.value, planned.value) == (0, 0)
    assert lib.gtr_gla_last_schedule(None, None) == 0


def test_host_buffer_bytes(lib):
    n = lib.gtr_gla_host_buffer_bytes(2, 3, 4, 5, 64, 32, 1, 1)
    T = 20
    rnd = lambda x: (x + 255) // 256 * 256
    assert n == 3 * rnd(2 * T * 3 * 64 * 2) + 2 * rnd(2 * T * 3 * 32 * 2) + rnd(2 * 3 * 64 * 32 * 4)
    assert lib.gtr_gla_host_buffer_bytes(1, 1, 0, 5, 64, 64, 1, 1) == 0
    # host entry point: missing device buffer
    assert lib.gtr_gla_fwd_host(16, 16, 16, 16, 1, 1, 8, 8, 64, 64, 0, 1, 16, None, None, 0,
                                None) == 3


def test_tc_support_query_is_host_only(lib):
    assert lib.gtr_gla_tc_supported(1, 1, 8, 8, 64, 64, 0, 0) == 0    # fp32 never on tensor cores
    assert lib.gtr_gla_tc_supported(1, 1, 8, 8, 0, 64, 0, 1) == 0     # invalid shape


def test_workspace_entry_point_validates_before_any_launch(lib):
    # invalid shapes ask for no workspace; a misaligned workspace is rejected
    assert lib.gtr_gla_workspace_bytes(1, 1, 0, 8, 64, 64, 1) == 0
    assert lib.gtr_gla_workspace_bytes(1, 1, 8, 8, 64, 64, 7) == 0
    assert lib.gtr_gla_fwd_ws(16, 16, 16, 16, 1, 1, 8, 8, 64, 64, 0, 1, 16, None, 8, 0, None) == 1
    # an empty batch needs neither inputs nor a workspace
    assert lib.gtr_gla_fwd_ws(None, None, None, None, 0, 4, 8, 8, 64, 64, 0, 1, None, None, None,
                              0, None) == 0


def test_noalloc_entry_point_validates_before_any_launch(lib):
    # bad arguments are rejected before the scratch array is looked up
    assert lib.gtr_gla_fwd_noalloc(None, 16, 16, 16, 1, 1, 8, 8, 64, 64, 0, 1, 16, None,
                                   None) == 1
    assert lib.gtr_gla_fwd_noalloc(16, 16, 16, 16, 1, 1, 8, 8, 64, 64, 5, 1, 16, None,
                                   None) == 1
    # an empty batch launches nothing and needs no device
    assert lib.gtr_gla_fwd_noalloc(None, None, None, None, 0, 4, 8, 8, 64, 64, 0, 1, None, None,
                                   None) == 0


def test_gated_entry_point_validates_before_any_launch(lib):
    fwd = lib.gtr_gla_fwd_gated
    ok = dict(q=16, k=16, v=16, g=16, gate=1 << 24, w=1 << 25, eps=1e-6)

    def call(**kw):
        a = dict(ok, **kw)
        return fwd(a["q"], a["k"], a["v"], a["g"], a["gate"], a["w"], a["eps"], 1, 1, 8, 8, 64, 64,
                   0, 1, 1 << 26, None, None)
    assert call(gate=None) == 1
    assert call(w=None) == 1
    assert call(gate=(1 << 24) + 8) == 1          # not 16-byte aligned
    assert call(eps=-1.0) == 1
    assert call(eps=float("nan")) == 1
    assert call(gate=(1 << 26) + 64) == 1         # overlaps the output
    # an empty batch launches nothing
    assert fwd(None, None, None, None, None, None, 1e-6, 0, 2, 8, 8, 64, 64, 0, 1, None, None, None) == 0


def test_gated_ws_entry_point_validates_before_any_launch(lib):
    fwd = lib.gtr_gla_fwd_gated_ws
    ok = dict(q=16, k=16, v=16, g=16, gate=1 << 24, w=1 << 25, eps=1e-6)

    def call(**kw):
        a = dict(ok, **kw)
        return fwd(a["q"], a["k"], a["v"], a["g"], a["gate"], a["w"], a["eps"], 1, 1, 8, 8, 64, 64,
                   0, 1, 1 << 26, None, None, 0, None)
    assert call(gate=None) == 1
    assert call(w=None) == 1
    assert call(gate=(1 << 24) + 8) == 1          # not 16-byte aligned
    assert call(eps=-1.0) == 1
    assert call(gate=(1 << 26) + 64) == 1         # overlaps the output
    assert fwd(None, None, None, None, None, None, 1e-6, 0, 2, 8, 8, 64, 64, 0, 1, None, None, None, 0,
               None) == 0


def test_sswiglu_entry_point_validates_before_any_launch(lib):
    fwd = lib.gtr_sswiglu_dwconv
    fwd.restype = ctypes.c_int
    fwd.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_longlong, ctypes.c_void_p, ctypes.c_void_p] + \
        [ctypes.c_int] * 5 + [ctypes.c_void_p, ctypes.c_void_p]
    g, v, w, o = 1 << 24, (1 << 24) + 128, 1 << 25, 1 << 26

    def call(gate=g, value=v, stride=128, weight=w, B=1, gh=4, gw=4, F=64, dtype=1, out=o):
        return fwd(gate, value, stride, weight, None, B, gh, gw, F, dtype, out, None)
    assert call(F=12) == 1                 # not a multiple of 8 elements
    assert call(stride=60) == 1            # token stride below F
    assert call(stride=68) == 1            # token stride not a multiple of 16 bytes
    assert call(gate=g + 8) == 1           # not 16-byte aligned
    assert call(weight=None) == 1
    assert call(gh=0) == 1
    assert call(dtype=7) == 1
    assert call(out=g + 1024) == 1         # the output overlaps the inputs
    assert call(B=0, gate=None, value=None, weight=None, out=None) == 0   # empty batch: nothing to do


def test_lowrank_gate_validation_rejects_before_launch(lib):
    # gtr_gla_fwd_lowrank_gate(q, k, v, a_low, w2, bias, tau, rank, B, H, gh, gw, Dk, Dv, order, dtype,
    #                          out, final_state, stream): bad arguments never reach the GPU
    q, k, v, out = 1 << 20, 2 << 20, 3 << 20, 4 << 20
    a, w2, bias = 5 << 20, 6 << 20, 7 << 20

    def call(a=a, w2=w2, bias=bias, tau=16.0, rank=16, B=1, Dk=64, q=q):
        return lib.gtr_gla_fwd_lowrank_gate(q, k, v, a, w2, bias, tau, rank, B, 2, 16, 16, Dk, 64, 0, 1,
                                            out, None, None)

    assert call(tau=0.0) == 1
    assert call(tau=-1.0) == 1
    assert call(tau=float("nan")) == 1
    assert call(rank=0) == 1
    assert call(a=None) == 1
    assert call(w2=None) == 1
    assert call(bias=None) == 1
    assert call(bias=bias + 4) == 1          # the bias must be 16-byte aligned
    assert call(a=a + 8) == 1
    assert call(q=None) == 1
    # an empty batch is valid and launches nothing
    assert call(B=0) == 0
    ran, planned = ctypes.c_int(-1), ctypes.c_int(-1)
    assert lib.gtr_gla_last_schedule(ctypes.byref(ran), ctypes.byref(planned)) == 0
    assert (ran.value, planned.value) == (0, 0)
