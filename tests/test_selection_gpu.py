"""GPU parity of the selection functions of Eq. 6 (B, C and the raw Delta as
linear maps of the scan input) through the C ABI against the fp64 oracle, and
the selection feeding the full scan."""
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


def weights(rng, K, D, N, R, printed=False):
    s = 1.0 / np.sqrt(D)
    WB = s * rng.standard_normal((K, N, D))
    WC = s * rng.standard_normal((K, N, D))
    Wz = s * rng.standard_normal((K, R, D))
    Wup = np.ones((K, D, R)) if printed else rng.standard_normal((K, D, R))
    return WB, WC, Wz, Wup


CASES = [
    # (B, K, D, N, R, H, W, dtype, printed form)
    (1, 4, 40, 16, 6, 7, 9, "f32", False),     # L = 63 < one CTA of steps
    (2, 2, 70, 5, 1, 10, 13, "f32", True),     # two channel blocks, padded N, the printed rank-1 broadcast
    (1, 4, 200, 16, 16, 12, 11, "f32", False),  # four channel blocks, R = 16, L = 132 (two step blocks)
    (2, 4, 48, 8, 3, 9, 9, "bf16", False),
    (1, 1, 3, 1, 1, 1, 5, "f32", False),       # tiny
    (2, 4, 256, 16, 6, 56, 56, "f32", False),  # the batch-128 workload's shape at batch 2 (8 chunks, 25 step blocks)
    (1, 4, 192, 16, 6, 128, 128, "bf16", False),  # the 512^2 map's stage-1 shape, bf16
    (1, 2, 1536, 16, 16, 7, 7, "f32", False),  # stage-4 width: 48 channel chunks, R = 16
]


@pytest.mark.parametrize("case", CASES, ids=[f"B{c[0]}K{c[1]}D{c[2]}N{c[3]}R{c[4]}_{c[5]}x{c[6]}_{c[7]}"
                                             for c in CASES])
def test_selection_parity(case):
    B, K, D, N, R, H, W, dt, printed = case
    rng = np.random.default_rng(600 + D + N + R)
    u = rng.standard_normal((B, K, D, H * W))
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32
    gu = torch.from_numpy(u).to(tdt).to(DEV)
    u = gu.double().cpu().numpy()  # the values the GPU sees
    Ws = weights(rng, K, D, N, R, printed)
    gw = [torch.from_numpy(w).float().to(DEV) for w in Ws]
    Ws = [w.double().cpu().numpy() for w in gw]
    dr, Bs, Cs = vmb.vmb_selection_fwd(gu, *gw, H, W)
    torch.cuda.synchronize()
    rdr, rB, rC = oracle.selection(u, *Ws)
    check(to_numpy(dr), rdr, dt, "delta_raw")
    check(to_numpy(Bs), rB, dt, "B")
    check(to_numpy(Cs), rC, dt, "C")
    if printed:
        d = to_numpy(dr)
        assert np.array_equal(d, np.broadcast_to(d[:, :, :1], d.shape)), "rank-1 unit form must broadcast over D"


def test_selection_feeds_the_scan():
    """u -> selection (Delta raw, B, C) -> full scan, against the oracle chain."""
    wl = workloads.small_case(B=1, D=32, N=16, H=10, W=12, seed=610)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    rng = np.random.default_rng(611)
    gw = [torch.from_numpy(w).float().to(DEV) for w in weights(rng, 4, wl.D, wl.N, 6)]
    dr, Bs, Cs = vmb.vmb_selection_fwd(xs, *gw, wl.H, wl.W)
    y = vmb.vmb_selective_scan_fwd(xs, dr, g["A"], Bs, Cs, g["Dskip"], g["bias"], wl.H, wl.W)
    torch.cuda.synchronize()
    u = oracle.cross_scan(inp.x)
    rdr, rB, rC = oracle.selection(u, *[w.double().cpu().numpy() for w in gw])
    y_ref = oracle.selective_scan(u, rdr, inp.A, rB, rC, inp.Dskip, inp.bias)
    check(to_numpy(y), y_ref, "f32", "selection -> scan")
