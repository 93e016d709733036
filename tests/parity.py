"""Shared helpers of the GPU parity tests: move seeded inputs to the device,
run the SS2D steps through the C ABI, and compare with the fp64 oracle."""
from __future__ import annotations

import numpy as np

# Tolerances fixed for the floating-point outputs of the scans:
#   fp32 storage: relative L2 error <= 1e-5 and max abs error <= 1e-4 * max|y|
#   bf16 storage: relative L2 error <= 1e-2
FP32_REL_L2 = 1e-5
FP32_MAX_ABS_FRAC = 1e-4
BF16_REL_L2 = 1e-2


def rel_l2(got, ref) -> float:
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    den = np.linalg.norm(ref)
    return float(np.linalg.norm(got - ref) / den) if den > 0 else float(np.linalg.norm(got))


def check(got, ref, dtype: str, what: str):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, f"{what}: shape {got.shape} vs {ref.shape}"
    assert np.all(np.isfinite(got)), f"{what}: non-finite values"
    e = rel_l2(got, ref)
    if dtype == "bf16":
        assert e <= BF16_REL_L2, f"{what}: rel-L2 {e:.3e} > {BF16_REL_L2}"
    else:
        m = float(np.max(np.abs(got - ref))) if got.size else 0.0
        scale = float(np.max(np.abs(ref))) if ref.size else 0.0
        assert e <= FP32_REL_L2, f"{what}: rel-L2 {e:.3e} > {FP32_REL_L2}"
        assert m <= FP32_MAX_ABS_FRAC * scale + 1e-30, f"{what}: max abs {m:.3e} > {FP32_MAX_ABS_FRAC} * {scale:.3e}"
    return e


def to_device(inp, device):
    import torch
    tdt = torch.bfloat16 if inp.wl.dtype == "bf16" else torch.float32
    out = {}
    for k, v in inp.arrays().items():
        t = torch.from_numpy(np.ascontiguousarray(v))
        if k in ("x", "draw", "Bs", "Cs"):
            t = t.to(tdt)  # bf16 workloads hold exactly representable values: exact
        out[k] = t.to(device)
    return out


def to_numpy(t):
    return t.float().cpu().numpy().astype(np.float64)
