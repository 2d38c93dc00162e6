"""fp64 CPU oracle for the GTR token mixer -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The CUDA
path never imports it and shares no code with it.

What it computes (paper "GTR: Gated Token Recurrence for Efficient Dense
Prediction"):

* :func:`recurrence` -- Sec. 3.1, "Key-only gated recurrence":
  ``S_t = Diag(exp(g_t)) S_{t-1} + k_t^T v_t``, ``S_0 = 0``, ``o_t = q_t S_t``,
  run along one of the four scan orders of Sec. 3.1, "Directional scanning",
  outputs written back at each token's spatial position.  This is the
  definition the chunkwise operator must reproduce (Sec. 3.3: the chunked
  schedule "changes only the execution schedule").
* :func:`chunkwise` -- Sec. 3.3, Eq. (chunk_boundary_main) and the chunk-output
  formula after it, with a free chunk size; a second restatement used to pin
  the chunk equations against the recurrence.
* :func:`scan_tokens` -- the scan permutation alone (position -> spatial token).
* :func:`gated_output` -- Sec. 3.1, the output gate applied to the mixer's
  output: ``u_t = SiLU(r_t) * RMSNorm(o_t)`` (the epilogue the paper's deployed
  kernel fuses, App. C.3).
* :func:`gate_producer` -- Sec. 3.1, the key-wise retention gate from its
  low-rank projection: ``g = log gamma = logsigmoid(x W1 W2 + b) / tau`` (the
  log-decay the mixer consumes), from ``a = x W1``.
* :func:`sswiglu_dwconv` -- Sec. 3.1, "Spatial SwiGLU", Eq. (spatial_swiglu):
  the part between its two projections, ``SiLU(X W_g) * DWConv3x3(X W_v)``
  on the patch grid (the part the deployed S-SwiGLU kernel fuses, Sec. 4).

Pins: tests/test_oracle_pins.py checks the functions against hand-worked
example (tests/golden/), brute-force quadratic forms, closed forms (gate 1 =
causal linear attention, gate 0 = (q.k) v, T = 1) and invariants (reversal,
grid transpose, linearity, chunk-size invariance).

Inputs are numpy arrays of any float dtype; they are widened to float64 here
(the values the CUDA path reads, rounded to its storage dtype, are exactly
representable in float64).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

ROW_FWD, ROW_REV, COL_FWD, COL_REV = 0, 1, 2, 3
ORDER_NAMES = {ROW_FWD: "row_fwd", ROW_REV: "row_rev", COL_FWD: "col_fwd", COL_REV: "col_rev"}

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gla_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libgla_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle with gcc (OpenMP, no fp contraction); return the .so path."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
           "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            dp = ctypes.POINTER(ctypes.c_double)
            ip = ctypes.POINTER(ctypes.c_int)
            lib.gla_oracle_recurrence.restype = ctypes.c_int
            lib.gla_oracle_recurrence.argtypes = [dp, dp, dp, dp] + [ctypes.c_int] * 7 + [
                ip, ip, ctypes.c_int, dp, dp, ctypes.c_int]
            lib.gla_oracle_chunkwise.restype = ctypes.c_int
            lib.gla_oracle_chunkwise.argtypes = [dp, dp, dp, dp] + [ctypes.c_int] * 8 + [
                dp, dp, ctypes.c_int]
            lib.gla_oracle_scan_token.restype = ctypes.c_long
            lib.gla_oracle_scan_token.argtypes = [ctypes.c_int, ctypes.c_long, ctypes.c_long,
                                                  ctypes.c_long]
            lib.gla_oracle_max_threads.restype = ctypes.c_int
            lib.gla_oracle_max_threads.argtypes = []
            _lib = lib
    return _lib


class using_library:
    """Context manager that points this module at another build of the oracle
    source (used by the mutation test, which compiles deliberately broken
    copies of gla_oracle.c and checks that the pins reject them)."""

    def __init__(self, so_path: str):
        self.so_path = so_path
        self.prev = None

    def __enter__(self):
        global _lib
        _load()
        with _lock:
            self.prev = _lib
            _lib = None
        saved = globals()["build"]
        globals()["build"] = lambda force=False: self.so_path
        try:
            _load()
        finally:
            globals()["build"] = saved
        return self

    def __exit__(self, *exc):
        global _lib
        with _lock:
            _lib = self.prev
        return False


def _f64(a: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _shapes(q, k, v, g, grid_h, grid_w):
    if q.ndim != 4 or k.shape != q.shape or g.shape != q.shape or v.ndim != 4:
        raise ValueError("q, k, g must be [B, T, H, Dk] and v [B, T, H, Dv]")
    B, T, H, Dk = q.shape
    if v.shape[:3] != (B, T, H):
        raise ValueError("v must share B, T, H with q")
    if T != grid_h * grid_w:
        raise ValueError(f"T={T} != grid_h*grid_w={grid_h * grid_w}")
    return B, T, H, Dk, v.shape[3]


def max_threads() -> int:
    """OpenMP threads the oracle uses by default on this host."""
    return int(_load().gla_oracle_max_threads())


def scan_tokens(order: int, grid_h: int, grid_w: int) -> np.ndarray:
    """Spatial token visited at each scan position (Sec. 3.1 'Directional scanning')."""
    lib = _load()
    T = grid_h * grid_w
    return np.array([lib.gla_oracle_scan_token(order, grid_h, grid_w, s) for s in range(T)],
                    dtype=np.int64)


def recurrence(q, k, v, g, grid_h: int, grid_w: int, order: int = ROW_FWD,
               pairs=None, n_threads: int = 0):
    """Sequential fp64 token recurrence (Sec. 3.1).

    Returns ``(out [B,T,H,Dv], final_state [B,H,Dk,Dv])`` in float64.  With
    ``pairs`` (a sequence of (b, h)) only those heads are computed; the other
    entries of both outputs are NaN.
    """
    q, k, v, g = _f64(q), _f64(k), _f64(v), _f64(g)
    B, T, H, Dk, Dv = _shapes(q, k, v, g, grid_h, grid_w)
    fill = np.nan if pairs is not None else 0.0
    out = np.full((B, T, H, Dv), fill, dtype=np.float64)
    fs = np.full((B, H, Dk, Dv), fill, dtype=np.float64)
    lib = _load()
    if pairs is not None:
        pb = np.ascontiguousarray([p[0] for p in pairs], dtype=np.int32)
        ph = np.ascontiguousarray([p[1] for p in pairs], dtype=np.int32)
        if np.any(pb < 0) or np.any(pb >= B) or np.any(ph < 0) or np.any(ph >= H):
            raise ValueError("pair out of range")
        ipt = ctypes.POINTER(ctypes.c_int)
        rc = lib.gla_oracle_recurrence(_ptr(q), _ptr(k), _ptr(v), _ptr(g), B, H, grid_h, grid_w,
                                       Dk, Dv, order, pb.ctypes.data_as(ipt),
                                       ph.ctypes.data_as(ipt), len(pb), _ptr(out), _ptr(fs),
                                       n_threads)
    else:
        rc = lib.gla_oracle_recurrence(_ptr(q), _ptr(k), _ptr(v), _ptr(g), B, H, grid_h, grid_w,
                                       Dk, Dv, order, None, None, 0, _ptr(out), _ptr(fs),
                                       n_threads)
    if rc != 0:
        raise RuntimeError(f"gla_oracle_recurrence failed ({rc})")
    return out, fs


def chunkwise(q, k, v, g, grid_h: int, grid_w: int, order: int = ROW_FWD, chunk: int = 64,
              n_threads: int = 0):
    """fp64 chunkwise schedule (Sec. 3.3, Eq. chunk_boundary_main) with chunk size ``chunk``."""
    q, k, v, g = _f64(q), _f64(k), _f64(v), _f64(g)
    B, T, H, Dk, Dv = _shapes(q, k, v, g, grid_h, grid_w)
    out = np.zeros((B, T, H, Dv), dtype=np.float64)
    fs = np.zeros((B, H, Dk, Dv), dtype=np.float64)
    rc = _load().gla_oracle_chunkwise(_ptr(q), _ptr(k), _ptr(v), _ptr(g), B, H, grid_h, grid_w,
                                      Dk, Dv, order, chunk, _ptr(out), _ptr(fs), n_threads)
    if rc != 0:
        raise RuntimeError(f"gla_oracle_chunkwise failed ({rc})")
    return out, fs


def gated_output(o, r_pre, weight, eps: float) -> np.ndarray:
    """Output gate of Sec. 3.1: ``u_t = SiLU(r_t) * RMSNorm(o_t)``.

    ``r_pre`` is the gate's pre-activation ``x_t W_r`` (the paper writes
    ``r_t = SiLU(x_t W_r)``; the fused epilogue of App. C.3 applies the SiLU).
    RMSNorm (Zhang and Sennrich, 2019) runs over each head's Dv outputs,
    ``o_j / sqrt(mean_j o_j^2 + eps) * weight_j``, with one weight vector of
    length Dv shared by the heads.  o, r_pre: [B, T, H, Dv]; weight: [Dv].
    Plain fp64 numpy, written out from the definitions.
    """
    o = np.asarray(o, dtype=np.float64)
    r = np.asarray(r_pre, dtype=np.float64)
    w = np.asarray(weight, dtype=np.float64)
    if o.shape != r.shape or w.shape != (o.shape[-1],):
        raise ValueError("o, r_pre must share a shape and weight must have Dv entries")
    rms = np.sqrt(np.mean(o * o, axis=-1, keepdims=True) + float(eps))
    with np.errstate(over="ignore"):
        silu = r / (1.0 + np.exp(-r))   # r * sigmoid(r); exp overflow gives -0 for r << 0
    return silu * (o / rms) * w


def sswiglu_dwconv(gate_pre, value_pre, weight, bias, grid_h: int, grid_w: int) -> np.ndarray:
    """Sec. 3.1, Eq. (spatial_swiglu), between the projections:
    ``Z = SiLU(X W_g) * DWConv3x3(X W_v)``.

    gate_pre = X W_g and value_pre = X W_v: [B, T, F] with T = grid_h * grid_w
    tokens in spatial row-major order.  The value branch is read as the
    grid_h x grid_w image of F channels and convolved per channel with its own
    3 x 3 kernel: ``weight[f, i, j]`` multiplies the value at row offset i - 1
    and column offset j - 1 (a cross-correlation, as a depthwise 2-D
    convolution layer computes it), with zeros outside the grid, plus
    ``bias[f]`` (None: no bias).  Plain fp64 numpy: nine shifted, weighted
    copies of the zero-padded image summed, then the SiLU gate.
    """
    g = np.asarray(gate_pre, dtype=np.float64)
    v = np.asarray(value_pre, dtype=np.float64)
    w = np.asarray(weight, dtype=np.float64)
    if g.shape != v.shape or g.ndim != 3 or g.shape[1] != grid_h * grid_w:
        raise ValueError("gate_pre and value_pre must be [B, grid_h*grid_w, F]")
    B, T, F = v.shape
    if w.shape != (F, 3, 3):
        raise ValueError("weight must be [F, 3, 3]")
    img = v.reshape(B, grid_h, grid_w, F)
    pad = np.zeros((B, grid_h + 2, grid_w + 2, F))
    pad[:, 1:grid_h + 1, 1:grid_w + 1, :] = img
    conv = np.zeros((B, grid_h, grid_w, F))
    for i in range(3):
        for j in range(3):
            conv += w[:, i, j] * pad[:, i:i + grid_h, j:j + grid_w, :]
    if bias is not None:
        conv += np.asarray(bias, dtype=np.float64)
    with np.errstate(over="ignore"):
        silu = g / (1.0 + np.exp(-g))
    return silu * conv.reshape(B, T, F)


def gate_producer(a_low, w2, bias, tau: float) -> np.ndarray:
    """Sec. 3.1, the retention gate: ``gamma_t = sigmoid(x_t W1 W2 + b)^(1/tau)``,
    so the log-decay the mixer consumes is ``g_t = logsigmoid(x_t W1 W2 + b) / tau``.

    a_low = x W1: [B, T, r] (the rank-r projection, r = 16 in the paper); w2:
    [H, r, Dk] (the second factor, one block of key channels per head); bias:
    [H, Dk]; tau > 0 (16 in the paper).  Returns g: [B, T, H, Dk] in float64.
    logsigmoid(z) = -log(1 + e^{-z}), evaluated as min(z, 0) - log1p(e^{-|z|})
    so that neither sign of z overflows.
    """
    a = np.asarray(a_low, dtype=np.float64)
    w = np.asarray(w2, dtype=np.float64)
    b = np.asarray(bias, dtype=np.float64)
    if a.ndim != 3 or w.ndim != 3 or w.shape[1] != a.shape[2] or b.shape != (w.shape[0], w.shape[2]):
        raise ValueError("a_low [B, T, r], w2 [H, r, Dk], bias [H, Dk]")
    if not tau > 0:
        raise ValueError("tau must be positive")
    z = np.einsum("btr,hrd->bthd", a, w) + b
    return (np.minimum(z, 0.0) - np.log1p(np.exp(-np.abs(z)))) / float(tau)
