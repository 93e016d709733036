"""The Delta branch of Eq. 6 kept low-rank through the scan: the selection
functions writing the rank-R intermediate z (vmb_selection_lowrank_fwd) and the
full and channel-mean scans forming the raw Deltas Wup z themselves
(vmb_selective_scan_lowrank_fwd, vmb_mean_scan_lowrank_fwd),
against the fp64 oracle's selection -> scan chain, and in fp32 bit for bit
against the library's selection -> raw Deltas -> scan.  Forcing the
warp-specialised tile shape exercises the fused expansion on small problems;
the planner's own choice there, 5 states and rows that are not 16-byte
multiples exercise the expand-into-y fallback (for the mean scan: ranks above
8 and the ZOH form)."""
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
    # (B, D, N, R, H, W, dtype)
    (1, 64, 16, 6, 16, 24, "f32"),    # VMamba-T's rank 6
    (2, 72, 16, 1, 12, 10, "f32"),    # rank 1 (the printed Broadcast_D(Linear_1(u)) with random Wup)
    (1, 40, 16, 12, 9, 12, "f32"),    # rank 12 (the 16-wide Wup rows); L = 108, a half-full last stage
    (1, 48, 16, 6, 16, 16, "bf16"),   # bf16 storage, fp32 z and raw Deltas
    (1, 32, 16, 6, 7, 7, "f32"),      # L = 49: rows not 16-byte multiples -> raw Deltas into y, scan in place
    (1, 24, 5, 4, 8, 8, "f32"),       # 5 states: not the warp-specialised kernel
]


def _weights(rng, K, D, N, R):
    s = 1.0 / np.sqrt(D)
    return (s * rng.standard_normal((K, N, D)), s * rng.standard_normal((K, N, D)), s * rng.standard_normal((K, R, D)),
            rng.standard_normal((K, D, R)))


@pytest.mark.parametrize("forced", [True, False], ids=["warp_specialised", "planner"])
@pytest.mark.parametrize("case", CASES, ids=[f"B{c[0]}_D{c[1]}_N{c[2]}_R{c[3]}_{c[4]}x{c[5]}_{c[6]}" for c in CASES])
def test_lowrank_selection_and_scan(case, forced, force_plan):
    B, D, N, R, H, W, dt = case
    if forced:
        force_plan.full("19")
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=1300 + D + R)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    u = vmb.vmb_cross_scan(g["x"])
    rng = np.random.default_rng(1301 + D + R)
    gw = [torch.from_numpy(w).float().to(DEV) for w in _weights(rng, 4, D, N, R)]
    WB, WC, Wz, Wup = gw
    z, Bs, Cs = vmb.vmb_selection_lowrank_fwd(u, WB, WC, Wz, H, W)
    y = vmb.vmb_selective_scan_lowrank_fwd(u, z, Wup, g["A"], Bs, Cs, g["Dskip"], g["bias"], H, W)
    y2 = vmb.vmb_selective_scan_lowrank_fwd(u, z, Wup, g["A"], Bs, Cs, g["Dskip"], g["bias"], H, W)
    dr, Bs_u, Cs_u = vmb.vmb_selection_fwd(u, WB, WC, Wz, Wup, H, W)
    y_u = vmb.vmb_selective_scan_fwd(u, dr, g["A"], Bs_u, Cs_u, g["Dskip"], g["bias"], H, W)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    assert torch.equal(y, y2), "deterministic"
    assert torch.equal(Bs, Bs_u) and torch.equal(Cs, Cs_u), "the low-rank selection's B and C are the selection's"
    if dt == "f32":
        assert torch.equal(y, y_u), "fp32: bit-identical to selection -> raw Deltas -> scan"
    # the oracle chain on the values the GPU saw
    un = to_numpy(u).astype(np.float64)
    Ws = [w.double().cpu().numpy() for w in gw]
    rdr, rB, rC = oracle.selection(un, *Ws)
    y_ref = oracle.selective_scan(un, rdr, inp.A, rB, rC, inp.Dskip, inp.bias)
    check(to_numpy(y), y_ref, dt, "low-rank scan y")
    # z: with Wup the first R unit vectors (D >= R), the oracle's raw Deltas of
    # channels 0 .. R-1 are z itself
    eye = np.zeros((4, D, R))
    for r in range(R):
        eye[:, r, r] = 1.0
    rz = oracle.selection(un, Ws[0], Ws[1], Ws[2], eye)[0][:, :, :R, :]
    check(to_numpy(z), rz, "f32", "low-rank selection z")


MEAN_CASES = [
    # (B, D, N, R, H, W, dtype, flags)
    (1, 64, 16, 6, 16, 24, "f32", 0),
    (2, 40, 16, 1, 9, 11, "f32", 0),     # odd L, rank 1
    (1, 300, 16, 8, 8, 8, "f32", 0),     # two channel-table groups; the largest rank held in registers
    (1, 48, 5, 6, 16, 16, "bf16", 0),    # padded states, bf16 storage, fp32 raw Deltas
    (1, 32, 16, 12, 8, 8, "f32", 0),     # rank 12: raw Deltas into y, scan in place
    (1, 24, 8, 6, 9, 9, "f32", 1),       # ZOH: raw Deltas into y, scan in place
    (2, 40, 16, 6, 12, 10, "f32", 2),    # the mean skip term
]


@pytest.mark.parametrize("case", MEAN_CASES, ids=[f"B{c[0]}_D{c[1]}_N{c[2]}_R{c[3]}_{c[4]}x{c[5]}_{c[6]}_f{c[7]}"
                                                  for c in MEAN_CASES])
def test_lowrank_mean_scan(case):
    B, D, N, R, H, W, dt, fl = case
    flags = vmb.VMB_FLAG_SOFTPLUS | (vmb.VMB_FLAG_B_ZOH if fl == 1 else 0) | (vmb.VMB_FLAG_SKIP_MEAN if fl == 2 else 0)
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=1350 + D + R)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    u = vmb.vmb_cross_scan(g["x"])
    rng = np.random.default_rng(1351 + D + R)
    gw = [torch.from_numpy(w).float().to(DEV) for w in _weights(rng, 4, D, N, R)]
    WB, WC, Wz, Wup = gw
    z, Bs, Cs = vmb.vmb_selection_lowrank_fwd(u, WB, WC, Wz, H, W)
    y, yb = vmb.vmb_mean_scan_lowrank_fwd(u, z, Wup, g["A"], Bs, Cs, g["Dskip"], g["bias"], H, W, want_ybar=True,
                                          flags=flags)
    dr, _, _ = vmb.vmb_selection_fwd(u, WB, WC, Wz, Wup, H, W)
    y_u, yb_u = vmb.vmb_mean_scan_fwd(u, dr, g["A"], Bs, Cs, g["Dskip"], g["bias"], H, W, want_ybar=True,
                                      flags=flags)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    if dt == "f32":
        assert torch.equal(y, y_u) and torch.equal(yb, yb_u), "fp32: bit-identical to raw Deltas -> mean scan"
    un = to_numpy(u).astype(np.float64)
    Ws = [w.double().cpu().numpy() for w in gw]
    rdr, rB, rC = oracle.selection(un, *Ws)
    y_ref, yb_ref = oracle.mean_scan(un, rdr, inp.A, rB, rC, inp.Dskip, inp.bias, b_mode=1 if fl == 1 else 0,
                                     skip_mode=oracle.SKIP_MEAN if fl == 2 else oracle.SKIP_PER_CHANNEL)
    check(to_numpy(y), y_ref, dt, "low-rank mean y")
    check(to_numpy(yb), yb_ref, "f32" if dt == "f32" else "bf16", "low-rank mean ybar")


def test_lowrank_scan_at_the_benchmark_size():
    """Batch 128, D 256, N 16, 56x56, fp32, rank 6, the planner's choice (the
    warp-specialised kernel): bit-identical to selection -> raw Deltas -> scan."""
    wl = workloads.WORKLOADS["batch128_d256_n16_56x56_sigma0.05_f32"]
    g = workloads.make_device_inputs(wl, DEV, params="random")
    u = vmb.vmb_cross_scan(g["x"])
    rng = np.random.default_rng(1390)
    WB, WC, Wz, Wup = [torch.from_numpy(w).float().to(DEV) for w in _weights(rng, 4, wl.D, wl.N, 6)]
    z, Bs, Cs = vmb.vmb_selection_lowrank_fwd(u, WB, WC, Wz, wl.H, wl.W)
    y = vmb.vmb_selective_scan_lowrank_fwd(u, z, Wup, g["A"], Bs, Cs, g["Dskip"], g["bias"], wl.H, wl.W)
    dr, _, _ = vmb.vmb_selection_fwd(u, WB, WC, Wz, Wup, wl.H, wl.W)
    y_u = vmb.vmb_selective_scan_fwd(u, dr, g["A"], Bs, Cs, g["Dskip"], g["bias"], wl.H, wl.W)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    assert torch.equal(y, y_u)
