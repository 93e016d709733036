"""The full-channel scan side of an SS2D block from the map (vmb_ss2d_full_fwd:
the selective scan reads each direction's steps from the map or its transpose,
no materialised cross-scan) against the fp64 oracle, and bit for bit against
the library's own three calls (cross-scan, full scan, cross-merge) run with
the same plan.  Forcing the warp-specialised tile shape exercises the
gathering kernel on small maps (reversed directions read mirrored boxes,
including one that starts before step 0); the planner's own choice on small
maps, 13 states and rows that are not 16-byte multiples exercise the
cross-scan-into-y fallback with the scan in place."""
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
    (1, 64, 16, 16, 24, "f32"),    # L = 384
    (2, 72, 16, 12, 10, "f32"),    # H != W; a tile with three consumer warps
    (1, 40, 16, 9, 12, "f32"),     # L = 108: the last stage half full, its mirrored box starts at step -4
    (1, 48, 16, 16, 16, "bf16"),   # bf16 rows of 16-byte multiples
    (1, 256, 16, 56, 56, "f32"),   # 392 stages, two channel tiles
    (1, 32, 16, 7, 7, "f32"),      # L = 49: rows not 16-byte multiples -> cross-scan into y, scan in place
    (2, 24, 13, 8, 8, "f32"),      # 13 states: B/C rows past N read as zero
    (1, 24, 5, 8, 8, "f32"),       # 5 states (padded to 8): not the warp-specialised kernel
]


def _three_calls(g, wl):
    xs = vmb.vmb_cross_scan(g["x"])
    y = vmb.vmb_selective_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W)
    return vmb.vmb_cross_merge(y, wl.H, wl.W), y


@pytest.mark.parametrize("forced", [True, False], ids=["gathering", "planner"])
@pytest.mark.parametrize("shape", SHAPES, ids=[f"B{s[0]}_D{s[1]}_N{s[2]}_{s[3]}x{s[4]}_{s[5]}" for s in SHAPES])
def test_full_path_from_the_map(shape, forced, force_plan):
    B, D, N, H, W, dt = shape
    if forced:
        force_plan.full("19")
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=1200 + D + N)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    out, y = vmb.vmb_ss2d_full_fwd(g["x"], g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"])
    out2, y2 = vmb.vmb_ss2d_full_fwd(g["x"], g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"])
    ref_out, ref_y = _three_calls(g, wl)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    assert torch.equal(y, ref_y), "y must be the scan of the cross-scanned map, bit for bit"
    assert torch.equal(out, ref_out), "out must be the merge of the three calls, bit for bit"
    assert torch.equal(out, out2) and torch.equal(y, y2), "deterministic"
    _, y_ref, out_ref = oracle.ss2d_full(inp)
    check(to_numpy(y), y_ref, dt, "full y from the map")
    check(to_numpy(out), out_ref, dt, "full out from the map")


def test_full_path_from_the_map_at_the_benchmark_size():
    """The benchmark workload (batch 128, D 256, N 16, 56x56, fp32), planner's
    choice: bit-identical to the three calls (whose parity the full-size
    sampled tests check against the oracle)."""
    wl = workloads.WORKLOADS["batch128_d256_n16_56x56_sigma0.05_f32"]
    g = workloads.make_device_inputs(wl, DEV, params="random")
    out, y = vmb.vmb_ss2d_full_fwd(g["x"], g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"])
    ref_out, ref_y = _three_calls(g, wl)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    assert torch.equal(y, ref_y)
    assert torch.equal(out, ref_out)
