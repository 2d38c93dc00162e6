"""Thin ctypes binding over the C ABI in ``include/gtr_gla.h``.

Argument marshalling only: every step of the forward runs in the library's
CUDA kernels.  PyTorch supplies device memory and the current CUDA stream.
There is no CPU fallback: if the library is not built, importing the entry
points raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional, Tuple

import torch

from . import build as _build

ROW_FWD, ROW_REV, COL_FWD, COL_REV = 0, 1, 2, 3
SCHEDULES = {"auto": 0, "simt": 1, "tc": 2}
STATUS = {0: "GTR_OK", 1: "GTR_ERR_INVALID_ARG", 2: "GTR_ERR_UNSUPPORTED", 3: "GTR_ERR_WORKSPACE",
          4: "GTR_ERR_CUDA", 5: "GTR_ERR_TIMEOUT"}
_DTYPES = {torch.float32: 0, torch.float16: 1, torch.bfloat16: 2}

_lock = threading.Lock()
_lib = None


class GLAError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {STATUS.get(status, status)}")


def lib_path() -> str:
    return _build.LIB_PATH


def load(path: Optional[str] = None):
    """Load the CUDA library (built by ``__graft_entry__.build()``)."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or _build.LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"CUDA library not built: {p} (run __graft_entry__.build())")
        lib = ctypes.CDLL(p)
        vp, ci, st = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        lib.gtr_gla_fwd.restype = ci
        lib.gtr_gla_fwd.argtypes = [vp] * 4 + [ci] * 8 + [vp, vp, vp]
        lib.gtr_gla_fwd_sched.restype = ci
        lib.gtr_gla_fwd_sched.argtypes = [vp] * 4 + [ci] * 8 + [vp, vp, ci, vp]
        lib.gtr_gla_tc_supported.restype = ci
        lib.gtr_gla_tc_supported.argtypes = [ci] * 8
        lib.gtr_gla_workspace_bytes.restype = st
        lib.gtr_gla_workspace_bytes.argtypes = [ci] * 7
        lib.gtr_sswiglu_dwconv.restype = ci
        lib.gtr_sswiglu_dwconv.argtypes = [vp, vp, ctypes.c_longlong, vp, vp] + [ci] * 5 + [vp, vp]
        lib.gtr_gla_chunk_boxes.restype = ci
        lib.gtr_gla_chunk_boxes.argtypes = [ci] * 4 + [ctypes.POINTER(ci), ci]
        lib.gtr_gla_chunk_walk.restype = ci
        lib.gtr_gla_chunk_walk.argtypes = [ci] * 4 + [ctypes.POINTER(ci)] * 2
        lib.gtr_gla_balanced_walk.restype = ci
        lib.gtr_gla_balanced_walk.argtypes = [ci] * 4 + [ctypes.POINTER(ci), ci, ctypes.POINTER(ci)]
        lib.gtr_gla_split_plan.restype = ci
        lib.gtr_gla_split_plan.argtypes = [ci] * 7 + [ctypes.POINTER(ci)] * 2
        lib.gtr_gla_balanced_plan.restype = ci
        lib.gtr_gla_balanced_plan.argtypes = [ci] * 7
        lib.gtr_gla_fwd_ws.restype = ci
        lib.gtr_gla_fwd_ws.argtypes = [vp] * 4 + [ci] * 8 + [vp, vp, vp, st, vp]
        lib.gtr_gla_fwd_gated.restype = ci
        lib.gtr_gla_fwd_gated.argtypes = [vp] * 6 + [ctypes.c_float] + [ci] * 8 + [vp, vp, vp]
        lib.gtr_gla_fwd_gated_ws.restype = ci
        lib.gtr_gla_fwd_gated_ws.argtypes = [vp] * 6 + [ctypes.c_float] + [ci] * 8 + [vp, vp, vp, st, vp]
        lib.gtr_gla_fwd_noalloc.restype = ci
        lib.gtr_gla_fwd_noalloc.argtypes = [vp] * 4 + [ci] * 8 + [vp, vp, vp]
        lib.gtr_gla_host_buffer_bytes.restype = st
        lib.gtr_gla_host_buffer_bytes.argtypes = [ci] * 8
        lib.gtr_gla_fwd_host.restype = ci
        lib.gtr_gla_fwd_host.argtypes = [vp] * 4 + [ci] * 8 + [vp, vp, vp, st, vp]
        lib.gtr_gla_sync_status.restype = ci
        lib.gtr_gla_sync_status.argtypes = [vp]
        lib.gtr_status_string.restype = ctypes.c_char_p
        lib.gtr_status_string.argtypes = [ci]
        lib.gtr_last_cuda_error.restype = ci
        lib.gtr_last_cuda_error.argtypes = []
        lib.gtr_version.restype = ci
        lib.gtr_version.argtypes = []
        lib.gtr_gla_fwd_lowrank_gate.restype = ci
        lib.gtr_gla_fwd_lowrank_gate.argtypes = [vp] * 6 + [ctypes.c_float] + [ci] * 9 + [vp, vp, vp]
        lib.gtr_gla_last_schedule.restype = ci
        lib.gtr_gla_last_schedule.argtypes = [ctypes.POINTER(ci)] * 2
        if path is None:
            _lib = lib
        return lib


def _stream_ptr(stream) -> int:
    s = torch.cuda.current_stream() if stream is None else stream
    return int(s.cuda_stream)


def _dims(q, v, grid_h, grid_w):
    if q.dim() != 4 or v.dim() != 4:
        raise ValueError("q/k/log_gate must be [B,T,H,Dk] and v [B,T,H,Dv]")
    B, T, H, Dk = q.shape
    if T != grid_h * grid_w:
        raise ValueError(f"T={T} != grid_h*grid_w={grid_h * grid_w}")
    return B, H, Dk, v.shape[3]


def _check(status: int, what: str, lib) -> None:
    if status != 0:
        msg = what
        if status == 4:
            msg += f" (cudaError {lib.gtr_last_cuda_error()})"
        raise GLAError(status, msg)


def tc_supported(B, H, grid_h, grid_w, Dk, Dv, order, dtype: torch.dtype) -> bool:
    return bool(load().gtr_gla_tc_supported(B, H, grid_h, grid_w, Dk, Dv, order, _DTYPES[dtype]))


def forward(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, log_gate: torch.Tensor,
            grid_h: int, grid_w: int, order: int = ROW_FWD, out: Optional[torch.Tensor] = None,
            final_state=True, schedule: str = "auto",
            stream: Optional[torch.cuda.Stream] = None) -> Tuple[torch.Tensor, Optional[torch.Tensor]]:
    """Chunkwise GLA forward through ``gtr_gla_fwd_sched``.

    q, k, log_gate: [B, T, H, Dk]; v: [B, T, H, Dv]; contiguous CUDA tensors of
    one dtype (float32 / float16 / bfloat16), T = grid_h * grid_w in spatial
    row-major order.  ``final_state``: True (allocate), None/False (skip) or a
    preallocated [B, H, Dk, Dv] float32 tensor.  Returns (out, final_state).
    """
    lib = load()
    for name, t in (("q", q), ("k", k), ("v", v), ("log_gate", log_gate)):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA tensor")
        if t.dtype != q.dtype:
            raise ValueError("all inputs must share one dtype")
    if q.dtype not in _DTYPES:
        raise ValueError(f"unsupported dtype {q.dtype}")
    B, H, Dk, Dv = _dims(q, v, grid_h, grid_w)
    if out is None:
        out = torch.empty(v.shape, dtype=v.dtype, device=v.device)
    fs = None
    if final_state is True:
        fs = torch.empty((B, H, Dk, Dv), dtype=torch.float32, device=q.device)
    elif isinstance(final_state, torch.Tensor):
        fs = final_state
    status = lib.gtr_gla_fwd_sched(
        q.data_ptr(), k.data_ptr(), v.data_ptr(), log_gate.data_ptr(), B, H, grid_h, grid_w,
        Dk, Dv, order, _DTYPES[q.dtype], out.data_ptr(), fs.data_ptr() if fs is not None else None,
        SCHEDULES[schedule], _stream_ptr(stream))
    _check(status, "gtr_gla_fwd", lib)
    return out, fs


def workspace_bytes(B, H, grid_h, grid_w, Dk, Dv, dtype: torch.dtype) -> int:
    """Device workspace ``forward_ws`` needs for these arguments (0: none)."""
    return int(load().gtr_gla_workspace_bytes(B, H, grid_h, grid_w, Dk, Dv, _DTYPES[dtype]))


def split_plan(B: int, H: int, grid_h: int, grid_w: int, Dk: int, Dv: int, n_sm: int) -> Tuple[int, int]:
    """(segments per sequence, chunks per segment) of the tensor-core schedule on a
    device with ``n_sm`` SMs, through ``gtr_gla_split_plan`` (host arithmetic only)."""
    lib = load()
    nseg, seg_len = ctypes.c_int(0), ctypes.c_int(0)
    status = lib.gtr_gla_split_plan(B, H, grid_h, grid_w, Dk, Dv, n_sm, ctypes.byref(nseg),
                                    ctypes.byref(seg_len))
    _check(status, "gtr_gla_split_plan", lib)
    return nseg.value, seg_len.value


def balanced_plan(B: int, H: int, grid_h: int, grid_w: int, Dk: int, Dv: int, n_sm: int) -> bool:
    """Whether the tensor-core schedule gives every CTA an equal contiguous range of
    chunks on a device with ``n_sm`` SMs, through ``gtr_gla_balanced_plan`` (host
    arithmetic only)."""
    return bool(load().gtr_gla_balanced_plan(B, H, grid_h, grid_w, Dk, Dv, n_sm))


def sswiglu_dwconv(gate: torch.Tensor, value: torch.Tensor, weight: torch.Tensor, bias: Optional[torch.Tensor],
                   grid_h: int, grid_w: int, out: Optional[torch.Tensor] = None,
                   stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """Spatial SwiGLU between its projections through ``gtr_sswiglu_dwconv``:
    out = SiLU(gate) * DWConv3x3(value) on the grid.  gate, value: [B, T, F] CUDA
    tensors of one dtype whose last dimension is contiguous and whose token
    stride is shared (e.g. the two halves of one [B, T, 2F] tensor); weight:
    [F, 3, 3] float32, bias: [F] float32 or None (CUDA).  Returns out [B, T, F]."""
    lib = load()
    if gate.dim() != 3 or gate.shape != value.shape or gate.dtype != value.dtype:
        raise ValueError("gate and value must be [B, T, F] tensors of one dtype")
    if gate.dtype not in _DTYPES:
        raise ValueError(f"unsupported dtype {gate.dtype}")
    B, T, F = gate.shape
    if T != grid_h * grid_w:
        raise ValueError("T must equal grid_h * grid_w")
    if gate.stride(2) != 1 or value.stride(2) != 1 or gate.stride(1) != value.stride(1) or \
            gate.stride(0) != T * gate.stride(1) or value.stride(0) != T * value.stride(1):
        raise ValueError("gate and value need contiguous channels and one shared token stride")
    if not gate.is_cuda or not value.is_cuda or not weight.is_cuda:
        raise ValueError("inputs must be CUDA tensors")
    if weight.dtype != torch.float32 or not weight.is_contiguous() or tuple(weight.shape) != (F, 3, 3):
        raise ValueError("weight must be a contiguous [F, 3, 3] float32 tensor")
    if bias is not None and (bias.dtype != torch.float32 or not bias.is_contiguous() or tuple(bias.shape) != (F,)):
        raise ValueError("bias must be a contiguous [F] float32 tensor")
    if out is None:
        out = torch.empty((B, T, F), dtype=gate.dtype, device=gate.device)
    status = lib.gtr_sswiglu_dwconv(gate.data_ptr(), value.data_ptr(), gate.stride(1), weight.data_ptr(),
                                    bias.data_ptr() if bias is not None else None, B, grid_h, grid_w, F,
                                    _DTYPES[gate.dtype], out.data_ptr(), _stream_ptr(stream))
    _check(status, "gtr_sswiglu_dwconv", lib)
    return out


def chunk_boxes(grid_h: int, grid_w: int, order: int, c: int):
    """The TMA boxes (rows, tile row, coordinate 2, coordinate 3) the tensor-core
    producer loads for chunk c, through ``gtr_gla_chunk_boxes`` (host only)."""
    lib = load()
    cap = 80  # a chunk has at most 64 column segments plus 4 zero-fill boxes
    buf = (ctypes.c_int * (4 * cap))()
    n = lib.gtr_gla_chunk_boxes(grid_h, grid_w, order, c, buf, cap)
    if n < 0 or n > cap:
        raise ValueError(f"gtr_gla_chunk_boxes returned {n}")
    return [tuple(buf[4 * i:4 * i + 4]) for i in range(n)]


def chunk_walk(grid_h: int, grid_w: int, order: int, c: int):
    """(x, y) grid position where the producer's single im2col walk load of chunk c
    starts, or None when the chunk loads as boxes, through ``gtr_gla_chunk_walk``
    (host only)."""
    lib = load()
    x, y = ctypes.c_int(-1), ctypes.c_int(-1)
    r = lib.gtr_gla_chunk_walk(grid_h, grid_w, order, c, ctypes.byref(x), ctypes.byref(y))
    if r < 0:
        raise ValueError(f"gtr_gla_chunk_walk returned {r}")
    return (x.value, y.value) if r == 1 else None


def balanced_walk(n_units: int, n_chunks: int, grid: int, cta: int):
    """(entries, head) of CTA ``cta`` of the balanced schedule, through
    ``gtr_gla_balanced_walk`` (host only): entries are (unit, chunk, start, hand_in)
    tuples in the CTA's order, head the length of its head run."""
    lib = load()
    head = ctypes.c_int(-1)
    n = lib.gtr_gla_balanced_walk(n_units, n_chunks, grid, cta, None, 0, ctypes.byref(head))
    if n < 0:
        raise ValueError(f"gtr_gla_balanced_walk returned {n}")
    buf = (ctypes.c_int * (4 * max(n, 1)))()
    lib.gtr_gla_balanced_walk(n_units, n_chunks, grid, cta, buf, n, ctypes.byref(head))
    return [tuple(buf[4 * i:4 * i + 4]) for i in range(n)], head.value


def forward_ws(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, log_gate: torch.Tensor,
               grid_h: int, grid_w: int, order: int, out: torch.Tensor,
               final_state: Optional[torch.Tensor], workspace: Optional[torch.Tensor],
               stream: Optional[torch.cuda.Stream] = None) -> None:
    """Forward through ``gtr_gla_fwd_ws`` with a caller-owned device workspace (a
    CUDA uint8 tensor of at least workspace_bytes(), or None when that is 0)."""
    lib = load()
    B, H, Dk, Dv = _dims(q, v, grid_h, grid_w)
    status = lib.gtr_gla_fwd_ws(
        q.data_ptr(), k.data_ptr(), v.data_ptr(), log_gate.data_ptr(), B, H, grid_h, grid_w, Dk,
        Dv, order, _DTYPES[q.dtype], out.data_ptr(),
        final_state.data_ptr() if final_state is not None else None,
        workspace.data_ptr() if workspace is not None else None,
        workspace.numel() * workspace.element_size() if workspace is not None else 0,
        _stream_ptr(stream))
    _check(status, "gtr_gla_fwd_ws", lib)


def forward_gated(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, log_gate: torch.Tensor,
                  gate: torch.Tensor, norm_weight: torch.Tensor, eps: float, grid_h: int, grid_w: int,
                  order: int = ROW_FWD, out: Optional[torch.Tensor] = None, final_state=True,
                  stream: Optional[torch.cuda.Stream] = None,
                  workspace: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, Optional[torch.Tensor]]:
    """Mixer plus output gate through ``gtr_gla_fwd_gated``: returns
    (u = SiLU(gate) * RMSNorm(o) per head, final_state).  gate: like v;
    norm_weight: Dv float32 values on the device.  With ``workspace`` (a CUDA
    uint8 tensor of at least workspace_bytes()) the call goes through
    ``gtr_gla_fwd_gated_ws``: no allocation, safe to capture into a CUDA graph."""
    lib = load()
    B, H, Dk, Dv = _dims(q, v, grid_h, grid_w)
    if out is None:
        out = torch.empty(v.shape, dtype=v.dtype, device=v.device)
    fs = None
    if final_state is True:
        fs = torch.empty((B, H, Dk, Dv), dtype=torch.float32, device=q.device)
    elif isinstance(final_state, torch.Tensor):
        fs = final_state
    args = (q.data_ptr(), k.data_ptr(), v.data_ptr(), log_gate.data_ptr(), gate.data_ptr(),
            norm_weight.data_ptr(), float(eps), B, H, grid_h, grid_w, Dk, Dv, order, _DTYPES[q.dtype],
            out.data_ptr(), fs.data_ptr() if fs is not None else None)
    if workspace is None:
        status = lib.gtr_gla_fwd_gated(*args, _stream_ptr(stream))
        _check(status, "gtr_gla_fwd_gated", lib)
    else:
        status = lib.gtr_gla_fwd_gated_ws(*args, workspace.data_ptr(),
                                          workspace.numel() * workspace.element_size(), _stream_ptr(stream))
        _check(status, "gtr_gla_fwd_gated_ws", lib)
    return out, fs


def forward_noalloc(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, log_gate: torch.Tensor,
                    grid_h: int, grid_w: int, order: int, out: torch.Tensor,
                    final_state: Optional[torch.Tensor],
                    stream: Optional[torch.cuda.Stream] = None) -> None:
    """Forward through ``gtr_gla_fwd_noalloc``: no device memory is allocated;
    split-schedule summaries go to the library's fixed scratch array, which all
    calls on a device share (calls that overlap on the GPU race)."""
    lib = load()
    B, H, Dk, Dv = _dims(q, v, grid_h, grid_w)
    status = lib.gtr_gla_fwd_noalloc(
        q.data_ptr(), k.data_ptr(), v.data_ptr(), log_gate.data_ptr(), B, H, grid_h, grid_w, Dk,
        Dv, order, _DTYPES[q.dtype], out.data_ptr(),
        final_state.data_ptr() if final_state is not None else None, _stream_ptr(stream))
    _check(status, "gtr_gla_fwd_noalloc", lib)


def host_buffer_bytes(B, H, grid_h, grid_w, Dk, Dv, dtype: torch.dtype, with_final_state=True):
    return int(load().gtr_gla_host_buffer_bytes(B, H, grid_h, grid_w, Dk, Dv, _DTYPES[dtype],
                                                int(bool(with_final_state))))


def forward_host(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, log_gate: torch.Tensor,
                 grid_h: int, grid_w: int, order: int, out: torch.Tensor,
                 final_state: Optional[torch.Tensor], dev_buffer: torch.Tensor,
                 stream: Optional[torch.cuda.Stream] = None) -> None:
    """End-to-end forward from host tensors through ``gtr_gla_fwd_host``: the
    library copies the inputs into ``dev_buffer`` (a CUDA uint8 tensor of
    host_buffer_bytes()), runs the forward and copies ``out`` / ``final_state``
    back, all enqueued on the stream.  Synchronise before reading results."""
    lib = load()
    B, H, Dk, Dv = _dims(q, v, grid_h, grid_w)
    for t in (q, k, v, log_gate, out):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError("host tensors must be contiguous CPU tensors")
    status = lib.gtr_gla_fwd_host(
        q.data_ptr(), k.data_ptr(), v.data_ptr(), log_gate.data_ptr(), B, H, grid_h, grid_w, Dk,
        Dv, order, _DTYPES[q.dtype], out.data_ptr(),
        final_state.data_ptr() if final_state is not None else None, dev_buffer.data_ptr(),
        dev_buffer.numel() * dev_buffer.element_size(), _stream_ptr(stream))
    _check(status, "gtr_gla_fwd_host", lib)


def forward_lowrank_gate(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, a_low: torch.Tensor,
                         w2: torch.Tensor, gate_bias: torch.Tensor, tau: float, grid_h: int, grid_w: int,
                         order: int = ROW_FWD, out: Optional[torch.Tensor] = None, final_state=True,
                         stream: Optional[torch.cuda.Stream] = None) -> Tuple[torch.Tensor, Optional[torch.Tensor]]:
    """Mixer with the retention gate computed in the kernel, through ``gtr_gla_fwd_lowrank_gate``:
    g = logsigmoid(a_low W2 + b) / tau.  a_low: [B, T, r] (same dtype as q); w2: [H, r, Dk];
    gate_bias: [H, Dk] float32; all contiguous CUDA tensors.  Returns (out, final_state)."""
    lib = load()
    B, H, Dk, Dv = _dims(q, v, grid_h, grid_w)
    if a_low.dim() != 3 or a_low.shape[:2] != q.shape[:2] or w2.dim() != 3 or tuple(w2.shape[::2]) != (H, Dk):
        raise ValueError("a_low must be [B, T, r] and w2 [H, r, Dk]")
    if tuple(gate_bias.shape) != (H, Dk) or gate_bias.dtype != torch.float32:
        raise ValueError("gate_bias must be a [H, Dk] float32 tensor")
    for name, t in (("q", q), ("k", k), ("v", v), ("a_low", a_low), ("w2", w2), ("gate_bias", gate_bias)):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA tensor")
    rank = a_low.shape[2]
    if out is None:
        out = torch.empty(v.shape, dtype=v.dtype, device=v.device)
    fs = None
    if final_state is True:
        fs = torch.empty((B, H, Dk, Dv), dtype=torch.float32, device=q.device)
    elif isinstance(final_state, torch.Tensor):
        fs = final_state
    status = lib.gtr_gla_fwd_lowrank_gate(
        q.data_ptr(), k.data_ptr(), v.data_ptr(), a_low.data_ptr(), w2.data_ptr(), gate_bias.data_ptr(),
        float(tau), rank, B, H, grid_h, grid_w, Dk, Dv, order, _DTYPES[q.dtype], out.data_ptr(),
        fs.data_ptr() if fs is not None else None, _stream_ptr(stream))
    _check(status, "gtr_gla_fwd_lowrank_gate", lib)
    return out, fs


RAN = {0: "none", 1: "simt", 2: "tc", 3: "tc_split", 4: "tc_balanced"}


def last_schedule() -> Tuple[str, str]:
    """(schedule launched, schedule planned) of this thread's last successful forward
    call, through ``gtr_gla_last_schedule``; they differ when the split or balanced
    schedule was dropped for lack of workspace."""
    lib = load()
    ran, planned = ctypes.c_int(-1), ctypes.c_int(-1)
    _check(lib.gtr_gla_last_schedule(ctypes.byref(ran), ctypes.byref(planned)), "gtr_gla_last_schedule", lib)
    return RAN[ran.value], RAN[planned.value]


def sync_status(stream: Optional[torch.cuda.Stream] = None) -> int:
    """Synchronise the stream and return/clear the device status word."""
    return int(load().gtr_gla_sync_status(_stream_ptr(stream)))
