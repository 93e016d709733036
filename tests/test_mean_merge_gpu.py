"""The channel-mean path with the broadcast fused into the cross-merge
(vmb_mean_scan_merge_fwd), and the whole scan side of the block from the map
(vmb_ss2d_mean_fwd: no materialised cross-scan either), against the fp64
oracle's unfused chain, and bit for bit against the library's own unfused
calls for fp32 storage."""
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

SHAPES = [
    # (B, D, N, H, W, dtype)
    (1, 192, 16, 14, 14, "f32"),   # the small SS2D workload
    (2, 40, 16, 9, 11, "f32"),     # odd L: element-wise merge path
    (1, 70, 16, 32, 40, "f32"),    # several L-chunks
    (3, 33, 5, 7, 7, "f32"),       # padded states, L = 49
    (2, 64, 1, 12, 16, "f32"),     # N = 1
    (1, 300, 16, 8, 8, "f32"),     # D > 256: two channel-table groups, several channel blocks
    (1, 48, 3, 5, 13, "bf16"),     # bf16, odd L
    (2, 96, 16, 16, 16, "bf16"),   # bf16 vector path
]


def _run(inp, flags=vmb.VMB_FLAG_SOFTPLUS):
    g = to_device(inp, DEV)
    wl = inp.wl
    xs = vmb.vmb_cross_scan(g["x"])
    out, ybar = vmb.vmb_mean_scan_merge_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], g["x"],
                                            wl.H, wl.W, flags=flags)
    ym, yb_plain = vmb.vmb_mean_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W,
                                         want_ybar=True, flags=flags)
    om = vmb.vmb_cross_merge(ym, wl.H, wl.W)
    og, ybg = vmb.vmb_ss2d_mean_fwd(g["x"], g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], flags=flags)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    # gathered from the map: the same values and operations as the fused pair
    assert torch.equal(og, out) and torch.equal(ybg, ybar), "the gathered path must match the fused pair bit for bit"
    return out, ybar, om, yb_plain


@pytest.mark.parametrize("shape", SHAPES, ids=[f"B{s[0]}_D{s[1]}_N{s[2]}_{s[3]}x{s[4]}_{s[5]}" for s in SHAPES])
def test_fused_mean_merge_matches_oracle(shape):
    B, D, N, H, W, dt = shape
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=700 + D + N)
    inp = workloads.make_inputs(wl, params="random")
    out, ybar, om, yb_plain = _run(inp)
    _, _, ybar_ref, out_ref = oracle.ss2d_mean(inp)
    check(to_numpy(out), out_ref, dt, "fused mean out")
    check(to_numpy(ybar), ybar_ref, "f32" if dt == "f32" else "bf16", "fused ybar")
    # ybar is the same quantity the unfused scan reports
    assert torch.equal(ybar, yb_plain)
    if dt == "f32":
        # the same fp32 operations in the same order as the unfused pair
        assert torch.equal(out, om), "fused and unfused fp32 results must be bit-identical"


def test_fused_mean_merge_skip_mean_mode():
    wl = workloads.small_case(B=2, D=40, N=16, H=12, W=10, seed=731)
    inp = workloads.make_inputs(wl, params="random")
    flags = vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_SKIP_MEAN
    out, _, om, _ = _run(inp, flags=flags)
    _, _, _, out_ref = oracle.ss2d_mean(inp, skip_mode=oracle.SKIP_MEAN)
    check(to_numpy(out), out_ref, "f32", "fused mean out (mean skip)")
    assert torch.equal(out, om)


def test_fused_mean_merge_zoh():
    wl = workloads.small_case(B=1, D=24, N=8, H=9, W=9, seed=732)
    inp = workloads.make_inputs(wl, params="random")
    flags = vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_B_ZOH
    out, _, om, _ = _run(inp, flags=flags)
    _, _, _, out_ref = oracle.ss2d_mean(inp, b_mode=1)
    check(to_numpy(out), out_ref, "f32", "fused mean out (ZOH)")
    assert torch.equal(out, om)


def test_fused_mean_merge_misaligned_map():
    """x and out one element off a 16-byte boundary: the element-wise merge path."""
    wl = workloads.small_case(B=1, D=16, N=16, H=8, W=8, seed=733)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xbuf = torch.empty(g["x"].numel() + 1, device=DEV)
    x = xbuf[1:].view_as(g["x"])
    x.copy_(g["x"])
    obuf = torch.empty_like(xbuf)
    out = obuf[1:].view_as(g["x"])
    xs = vmb.vmb_cross_scan(x)
    vmb.vmb_mean_scan_merge_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], x, 8, 8, out=out)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    _, _, _, out_ref = oracle.ss2d_mean(inp)
    check(to_numpy(out), out_ref, "f32", "fused mean out (misaligned)")


def test_kernel_count_query():
    """The chunked full scan of a batch-1 56x56 map launches three kernels, the
    mean scan one; an empty problem none."""
    assert vmb.vmb_scan_kernel_count(vmb.VMB_PATH_FULL, 1, 4, 192, 16, 56, 56) == 3
    assert vmb.vmb_scan_kernel_count(vmb.VMB_PATH_MEAN, 1, 4, 192, 16, 56, 56) == 1
    assert vmb.vmb_scan_kernel_count(vmb.VMB_PATH_FULL, 128, 4, 256, 16, 56, 56) == 1
    assert vmb.vmb_scan_kernel_count(vmb.VMB_PATH_FULL, 0, 4, 192, 16, 56, 56) == 0
