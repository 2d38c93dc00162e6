"""Seeded synthetic inputs shaped like the GTR dense-prediction workloads.

This module is the one piece shared by the CUDA path's tests/benchmarks and the
CPU oracle: it draws random numbers and rounds them to a storage dtype.  It
holds none of the mixer's arithmetic.

Workloads (stride-16 patch grids of the paper's input resolutions, Sec. 3 and
Table "gtr_architecture": head width 64; 16.4K tokens is the paper's longest
operator benchmark, Sec. 3.3):

====  ======  ==========  ===============  =====  ====================================
 id   dtype   B x H        grid (T)        Dk=Dv  log-gate g
====  ======  ==========  ===============  =====  ====================================
 0    f32     1 x 2        16x16 (256)      64    logsigmoid(z)/16, z ~ N(0,1)
 1    f16     1 x 6        40x40 (1600)     64    logsigmoid(z)/16, z ~ N(0,1)
 2    bf16    32 x 12      40x40 (1600)     64    as 1, plus 10% of (h, channel) g = 0
 3    f16     8 x 16       80x80 (6400)     64    logsigmoid(z), z ~ N(-1,1)
 4    bf16    2 x 8      128x128 (16384)   128    logsigmoid(z)/16, z ~ N(0,1)
====  ======  ==========  ===============  =====  ====================================

q, k, v ~ N(0, 1) with k scaled by 1/sqrt(Dk) before rounding; every value is
rounded (round-to-nearest-even) to the storage dtype, and both the GPU path and
the oracle read exactly those rounded values.  Seeds are 1234 + workload id.
The paper's datasets are not used: these inputs stand in for its images.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Optional, Tuple

import numpy as np

ROW_FWD, ROW_REV, COL_FWD, COL_REV = 0, 1, 2, 3
ALL_ORDERS = (ROW_FWD, ROW_REV, COL_FWD, COL_REV)
ORDER_NAMES = ("row_fwd", "row_rev", "col_fwd", "col_rev")

DTYPES = ("f32", "f16", "bf16")
ELEM_SIZE = {"f32": 4, "f16": 2, "bf16": 2}


@dataclasses.dataclass(frozen=True)
class Workload:
    wid: int
    name: str
    dtype: str
    B: int
    H: int
    grid_h: int
    grid_w: int
    Dk: int
    Dv: int
    tau: float = 16.0          # g = logsigmoid(z) / tau
    z_mean: float = 0.0        # z ~ N(z_mean, 1)
    frac_nodecay: float = 0.0  # fraction of (h, key channel) pairs with g = 0
    orders: Tuple[int, ...] = ALL_ORDERS
    final_state: bool = True
    seed: Optional[int] = None

    @property
    def T(self) -> int:
        return self.grid_h * self.grid_w

    @property
    def token_heads(self) -> int:
        return self.B * self.T * self.H

    def algorithmic_bytes(self, final_state: Optional[bool] = None) -> int:
        """Bytes a perfect single pass moves: q, k, g, v read once, o written once,
        plus the fp32 final state when it is returned."""
        es = ELEM_SIZE[self.dtype]
        fs = self.final_state if final_state is None else final_state
        n = self.token_heads * es * (3 * self.Dk + 2 * self.Dv)
        if fs:
            n += self.B * self.H * self.Dk * self.Dv * 4
        return n

    def algorithmic_flops(self, chunk: int = 64) -> float:
        """Useful FLOPs of the chunkwise forward per call: summary + readout
        (4 Dk Dv), the causal intra-chunk triangle ((C+1)(Dk+Dv)) and the state
        update (2 Dk Dv / C), per token-head."""
        C = chunk
        per = 4 * self.Dk * self.Dv + (C + 1) * (self.Dk + self.Dv) + 2 * self.Dk * self.Dv / C
        return float(self.token_heads) * per


WORKLOADS: Dict[int, Workload] = {
    0: Workload(0, "tiny_fp32_16x16", "f32", 1, 2, 16, 16, 64, 64, orders=(ROW_FWD,)),
    1: Workload(1, "gtr_s_640_40x40", "f16", 1, 6, 40, 40, 64, 64),
    2: Workload(2, "batched_40x40_h12", "bf16", 32, 12, 40, 40, 64, 64, frac_nodecay=0.10),
    3: Workload(3, "highres_1280_80x80", "f16", 8, 16, 80, 80, 64, 64, tau=1.0, z_mean=-1.0),
    4: Workload(4, "vhr_2048_128x128_d128", "bf16", 2, 8, 128, 128, 128, 128),
}


def round_to_storage(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round float64 values to the storage dtype (RNE).  bf16 is returned as its
    uint16 bit pattern (numpy has no bfloat16)."""
    if dtype == "f32":
        return x.astype(np.float32)
    if dtype == "f16":
        return x.astype(np.float16)
    if dtype == "bf16":
        u = x.astype(np.float32).view(np.uint32)
        bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
        return ((u + bias) >> np.uint32(16)).astype(np.uint16)
    raise ValueError(f"unknown dtype {dtype!r}")


def storage_to_f64(a: np.ndarray, dtype: str) -> np.ndarray:
    """Widen storage values (see round_to_storage) to float64, exactly."""
    if dtype == "bf16":
        return (a.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def _logsigmoid(z: np.ndarray) -> np.ndarray:
    # log(1 / (1 + exp(-z))) evaluated without overflow for either sign of z
    return np.minimum(z, 0.0) - np.log1p(np.exp(-np.abs(z)))


def make_inputs(B: int, H: int, grid_h: int, grid_w: int, Dk: int, Dv: int, dtype: str,
                seed: int, tau: float = 16.0, z_mean: float = 0.0,
                frac_nodecay: float = 0.0) -> Dict[str, np.ndarray]:
    """Seeded q, k, v, g in [B, T, H, D] spatial row-major layout, storage dtype."""
    rng = np.random.Generator(np.random.PCG64(seed))
    T = grid_h * grid_w
    out = {}
    out["q"] = round_to_storage(rng.standard_normal((B, T, H, Dk)), dtype)
    out["k"] = round_to_storage(rng.standard_normal((B, T, H, Dk)) / np.sqrt(Dk), dtype)
    out["v"] = round_to_storage(rng.standard_normal((B, T, H, Dv)), dtype)
    z = rng.standard_normal((B, T, H, Dk)) + z_mean
    g = _logsigmoid(z) / tau
    del z
    if frac_nodecay > 0.0:
        n_pairs = H * Dk
        n_sel = int(round(frac_nodecay * n_pairs))
        sel = rng.permutation(n_pairs)[:n_sel]
        mask = np.zeros(n_pairs, dtype=bool)
        mask[sel] = True
        g[:, :, mask.reshape(H, Dk)] = 0.0
    out["g"] = round_to_storage(g, dtype)
    return out


GATE_RANK = 16   # rank r of the gate's low-rank projection (Sec. 3.1)


def gate_producer_inputs(B: int, H: int, T: int, Dk: int, dtype: str, seed: int,
                         z_mean: float = 0.0, rank: int = GATE_RANK,
                         bias_std: float = 0.25) -> Dict[str, np.ndarray]:
    """Seeded inputs of the in-kernel retention gate: the projection a = x W1 [B, T, rank]
    ~ N(0, 1), the second factor W2 [H, rank, Dk] ~ N(0, 1/rank) (so a W2 ~ N(0, 1)), both in
    the storage dtype, and the bias [H, Dk] ~ z_mean + N(0, bias_std^2) in float32 (bias_std
    = 0: the gate pre-activation is N(z_mean, 1) per token and channel, as in the workloads)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    a = round_to_storage(rng.standard_normal((B, T, rank)), dtype)
    w2 = round_to_storage(rng.standard_normal((H, rank, Dk)) / np.sqrt(rank), dtype)
    bias = (z_mean + bias_std * rng.standard_normal((H, Dk))).astype(np.float32)
    return {"a": a, "w2": w2, "bias": bias}


def workload_inputs(w: Workload, B: Optional[int] = None, seed: Optional[int] = None):
    """Inputs of workload ``w`` (optionally with a smaller batch, same distributions)."""
    s = (1234 + w.wid) if seed is None else seed
    return make_inputs(w.B if B is None else B, w.H, w.grid_h, w.grid_w, w.Dk, w.Dv, w.dtype,
                       s, tau=w.tau, z_mean=w.z_mean, frac_nodecay=w.frac_nodecay)


# ---------------------------------------------------------------- Spatial SwiGLU (Sec. 3.1)
#
# Inputs of the step between the two projections of Eq. (spatial_swiglu): the
# projection output X [W_g | W_v] as one [B, T, 2F] tensor (gate channels first),
# the depthwise 3 x 3 taps [F, 3, 3] and the bias [F] (fp32).  F is the model
# width times the S-SwiGLU expansion ratio (App. B.3: widths 192 / 384, ratio 4,
# 6 for GTR-X).  Seeds are 2609 + id.
#
# ====  ======  ====  ===============  =====  =====================================
#  id   dtype    B     grid (T)         F      model
# ====  ======  ====  ===============  =====  =====================================
#  0    f32      1     8x12 (96)          64   small correctness case
#  1    f16      1     40x40 (1600)      768   GTR-S at 640^2
#  2    bf16    32     40x40 (1600)     1536   GTR-L at 640^2, batch 32
#  3    f16      8     80x80 (6400)     2304   GTR-X at 1280^2, batch 8
# ====  ======  ====  ===============  =====  =====================================
#
# gate and value pre-activations ~ N(0, 1), taps ~ N(0, 1/9), bias ~ N(0, 0.1^2),
# all rounded to the storage dtype (taps and bias to fp32).

@dataclasses.dataclass(frozen=True)
class SwigluWorkload:
    wid: int
    name: str
    dtype: str
    B: int
    grid_h: int
    grid_w: int
    F: int

    @property
    def T(self) -> int:
        return self.grid_h * self.grid_w

    def algorithmic_bytes(self) -> int:
        """Gate and value read once, the output written once, plus the taps and bias."""
        return self.B * self.T * 3 * self.F * ELEM_SIZE[self.dtype] + self.F * 10 * 4


SWIGLU_WORKLOADS: Dict[int, SwigluWorkload] = {
    0: SwigluWorkload(0, "sswiglu_tiny_8x12", "f32", 1, 8, 12, 64),
    1: SwigluWorkload(1, "sswiglu_gtr_s_640", "f16", 1, 40, 40, 768),
    2: SwigluWorkload(2, "sswiglu_gtr_l_640_b32", "bf16", 32, 40, 40, 1536),
    3: SwigluWorkload(3, "sswiglu_gtr_x_1280_b8", "f16", 8, 80, 80, 2304),
}


def sswiglu_inputs(B: int, grid_h: int, grid_w: int, F: int, dtype: str, seed: int,
                   with_bias: bool = True) -> Dict[str, np.ndarray]:
    """Seeded [B, T, 2F] projection output (gate channels, then value channels) in
    the storage dtype, fp32 taps [F, 3, 3] and bias [F] (None without bias)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    T = grid_h * grid_w
    h = round_to_storage(rng.standard_normal((B, T, 2 * F)), dtype)
    w = (rng.standard_normal((F, 3, 3)) / 3.0).astype(np.float32)
    b = (0.1 * rng.standard_normal(F)).astype(np.float32) if with_bias else None
    return {"h": h, "weight": w, "bias": b}
