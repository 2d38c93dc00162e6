"""Helpers shared by the test files: input conversion and the acceptance bar."""
import numpy as np

from paper_2609_26590_gb300 import workloads as wl

# Acceptance bar on o and final_state against the fp64 oracle.
REL_L2_16BIT = 2e-3        # fp16 / bf16 inputs: relative L2 error
MAX_ABS_16BIT = 1e-2       # fp16 / bf16 inputs: max-abs error / max |oracle|
REL_L2_F32 = 1e-5          # fp32 inputs: relative L2 error


def to_torch(a: np.ndarray, dtype: str, device="cuda"):
    import torch
    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a))
    return t.to(device) if device != "cpu" else t


def inputs_f64(inp, dtype):
    return {n: wl.storage_to_f64(inp[n], dtype) for n in ("q", "k", "v", "g")}


def errors(got: np.ndarray, ref: np.ndarray):
    got = np.asarray(got, dtype=np.float64)
    d = got - ref
    nref = np.linalg.norm(ref.ravel())
    rel = np.linalg.norm(d.ravel()) / max(nref, 1e-300)
    max_abs = float(np.max(np.abs(d))) if d.size else 0.0
    max_ref = float(np.max(np.abs(ref))) if ref.size else 0.0
    ngot = np.linalg.norm(got.ravel())
    cos = float(np.dot(got.ravel(), ref.ravel()) / max(ngot * nref, 1e-300))
    return {"rel_l2": float(rel), "max_abs": max_abs, "max_ref": max_ref, "cos": cos,
            "finite": bool(np.all(np.isfinite(got)))}


def assert_within_bar(got, ref, dtype, what=""):
    e = errors(got, ref)
    assert e["finite"], f"{what}: non-finite values {e}"
    if dtype == "f32":
        assert e["rel_l2"] <= REL_L2_F32, f"{what}: {e}"
    else:
        assert e["rel_l2"] <= REL_L2_16BIT, f"{what}: {e}"
        assert e["max_abs"] <= MAX_ABS_16BIT * e["max_ref"], f"{what}: {e}"
    return e
