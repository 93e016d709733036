"""GPU parity of the grouped basis (reduced channel dimension d = groups > 1:
the channel mean of Eq. 9 over each of d channel groups) through the C ABI
against the fp64 oracle, with the same bar as the mean scan."""
import numpy as np
import pytest

import oracle
import workloads
from tests.parity import check, to_device, to_numpy

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU, skipped by marker
    pytest.skip("needs a GPU", allow_module_level=True)

import paper_2412_16602_gb300 as vmb  # noqa: E402

DEV = torch.device("cuda", 0)

CASES = [
    # (B, D, N, H, W, dtype, groups)
    (1, 24, 16, 12, 14, "f32", 2),
    (1, 24, 16, 12, 14, "f32", 3),
    (2, 12, 5, 7, 9, "f32", 4),       # padded states, odd L
    (1, 48, 16, 56, 56, "f32", 8),    # L = 3136: many chunks per sequence
    (2, 16, 16, 16, 16, "bf16", 4),
    (1, 6, 8, 9, 10, "f32", 6),       # one channel per group: the full scan
]


def run(inp, groups, flags=vmb.VMB_FLAG_SOFTPLUS):
    g = to_device(inp, DEV)
    wl = inp.wl
    xs = vmb.vmb_cross_scan(g["x"])
    y, yb = vmb.vmb_mean_scan_grouped_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H,
                                          wl.W, groups, want_ybar=True, flags=flags)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    return g, xs, y, yb


@pytest.mark.parametrize("case", CASES, ids=[f"B{c[0]}_D{c[1]}_N{c[2]}_{c[3]}x{c[4]}_{c[5]}_G{c[6]}" for c in CASES])
def test_grouped_parity(case):
    B, D, N, H, W, dt, G = case
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=500 + D + G)
    inp = workloads.make_inputs(wl, params="random")
    _, xs, y, yb = run(inp, G)
    u = oracle.cross_scan(inp.x)
    y_ref, yb_ref = oracle.mean_scan_grouped(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias, G)
    check(to_numpy(y), y_ref, dt, "grouped y")
    check(to_numpy(yb), yb_ref, "f32" if dt == "f32" else "bf16", "grouped ybar")
    if G == D:
        check(to_numpy(y), oracle.selective_scan(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias), dt,
              "one channel per group = full scan")


@pytest.mark.parametrize("flags", [vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_SKIP_MEAN,
                                   vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_B_ZOH], ids=["skip_mean", "zoh"])
def test_grouped_flags(flags):
    wl = workloads.small_case(B=1, D=20, N=16, H=10, W=12, seed=520)
    inp = workloads.make_inputs(wl, params="random")
    _, _, y, yb = run(inp, 4, flags=flags)
    u = oracle.cross_scan(inp.x)
    kw = dict(skip_mode=1 if flags & vmb.VMB_FLAG_SKIP_MEAN else 0, b_mode=1 if flags & vmb.VMB_FLAG_B_ZOH else 0)
    y_ref, yb_ref = oracle.mean_scan_grouped(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias, 4, **kw)
    check(to_numpy(y), y_ref, "f32", "grouped y")
    check(to_numpy(yb), yb_ref, "f32", "grouped ybar")


def test_one_group_is_the_mean_scan_bit_for_bit():
    wl = workloads.small_case(B=2, D=32, N=16, H=14, W=14, seed=530)
    inp = workloads.make_inputs(wl, params="random")
    g, xs, y, yb = run(inp, 1)
    ym, ybm = vmb.vmb_mean_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W,
                                    want_ybar=True)
    torch.cuda.synchronize()
    assert torch.equal(y, ym)
    assert torch.equal(yb[:, :, 0], ybm)


def test_grouped_rejects_non_divisor():
    wl = workloads.small_case(B=1, D=10, N=4, H=4, W=4, seed=531)
    g = to_device(workloads.make_inputs(wl, params="random"), DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    with pytest.raises(ValueError):
        vmb.vmb_mean_scan_grouped_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], 4, 4, 3)
