"""GPU parity of the paper's scan-only kernel setting (Sec. 4): discretisation
into materialised operands, their channel means (Eq. 9's T), and the scan
alone, each through the C ABI against the fp64 oracle.

The operands and the scan output are fp32 whatever the storage type, so every
comparison uses the fp32 bar (rel-L2 <= 1e-5, max-abs <= 1e-4 max|ref|).  The
scan alone is fed the oracle's operands rounded to fp32, and compared with the
oracle run on exactly those values.
"""
import numpy as np
import pytest

import oracle
import workloads
from tests.parity import check, to_numpy

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU, skipped by marker
    pytest.skip("needs a GPU", allow_module_level=True)

import paper_2412_16602_gb300 as vmb  # noqa: E402

DEV = torch.device("cuda", 0)


def inputs(B, D, N, H, W, dt, seed):
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=seed)
    inp = workloads.make_inputs(wl, params="random")
    u = oracle.cross_scan(inp.x)
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32

    def dev(a, store=True):
        t = torch.from_numpy(np.ascontiguousarray(a))
        return (t.to(tdt) if store else t.float()).to(DEV)

    g = dict(u=dev(u), draw=dev(inp.draw), Bs=dev(inp.Bs), Cs=dev(inp.Cs), A=dev(inp.A, False),
             bias=dev(inp.bias, False), Dskip=dev(inp.Dskip, False))
    return inp, u, g


SHAPES = [
    # (B, D, N, H, W, dtype)
    (1, 8, 16, 5, 7, "f32"),       # L = 35: element-wise loads, ragged segments
    (2, 6, 5, 8, 8, "f32"),        # odd N (padded lanes), L = 64
    (1, 12, 1, 14, 14, "f32"),     # N = 1
    (2, 5, 8, 6, 6, "bf16"),       # N = 8, bf16 storage
    (1, 4, 3, 1, 1, "f32"),        # L = 1
    (1, 10, 16, 16, 24, "bf16"),   # L = 384, aligned rows: vector loads
]
IDS = [f"B{s[0]}_D{s[1]}_N{s[2]}_{s[3]}x{s[4]}_{s[5]}" for s in SHAPES]
FLAGS = [vmb.VMB_FLAG_SOFTPLUS, vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_B_ZOH]


@pytest.mark.parametrize("flags", FLAGS, ids=["euler", "zoh"])
@pytest.mark.parametrize("shape", SHAPES, ids=IDS)
def test_discretise_parity(shape, flags):
    B, D, N, H, W, dt = shape
    inp, u, g = inputs(B, D, N, H, W, dt, seed=300 + D + N)
    zoh = 1 if flags & vmb.VMB_FLAG_B_ZOH else 0
    dA, dBu = vmb.vmb_discretise_fwd(g["u"], g["draw"], g["A"], g["Bs"], g["bias"], H, W, flags=flags)
    dAm, dBum = vmb.vmb_discretise_mean_fwd(g["u"], g["draw"], g["A"], g["Bs"], g["bias"], H, W, flags=flags)
    torch.cuda.synchronize()
    rA, rB = oracle.discretise(u, inp.draw, inp.A, inp.Bs, inp.bias, b_mode=zoh)
    rAm, rBm = oracle.discretise_mean(u, inp.draw, inp.A, inp.Bs, inp.bias, b_mode=zoh)
    check(to_numpy(dA), rA, "f32", "dA")
    check(to_numpy(dBu), rB, "f32", "dBu")
    check(to_numpy(dAm), rAm, "f32", "dA mean")
    check(to_numpy(dBum), rBm, "f32", "dBu mean")


def test_discretise_softplus_off():
    inp, u, g = inputs(1, 6, 4, 6, 7, "f32", seed=311)
    draw = np.abs(inp.draw) * 0.05
    bias = np.abs(inp.bias)
    gd = torch.from_numpy(draw).float().to(DEV)
    gb = torch.from_numpy(bias).float().to(DEV)
    dA, dBu = vmb.vmb_discretise_fwd(g["u"], gd, g["A"], g["Bs"], gb, 6, 7, flags=0)
    rA, rB = oracle.discretise(u, draw, inp.A, inp.Bs, bias, softplus_on=False)
    check(to_numpy(dA), rA, "f32", "dA softplus off")
    check(to_numpy(dBu), rB, "f32", "dBu softplus off")


def scan_only_case(B, K, Dm, N, H, W, dt, seed, one=False):
    """Random operands in the range the discretisation produces."""
    rng = np.random.default_rng(seed)
    L = H * W
    shape = (B, K, N, L) if one else (B, K, Dm, N, L)
    dA = rng.uniform(0.3, 1.0, size=shape).astype(np.float32)
    dBu = (0.1 * rng.standard_normal(shape)).astype(np.float32)
    Cs = rng.standard_normal((B, K, N, L))
    if dt == "bf16":
        Cs = torch.from_numpy(Cs).to(torch.bfloat16).float().numpy()
    Cs = Cs.astype(np.float32)
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32
    g = (torch.from_numpy(dA).to(DEV), torch.from_numpy(dBu).to(DEV), torch.from_numpy(Cs).to(tdt).to(DEV))
    return (dA, dBu, Cs), g


ONLY_SHAPES = [
    # (B, K, Dm, N, H, W, dtype, one channel)
    (1, 4, 8, 16, 5, 7, "f32", False),     # L = 35 over 64 segments: most of them empty
    (1, 4, 96, 16, 56, 56, "f32", False),  # 384 channels, L = 3136
    (2, 4, 1, 16, 56, 56, "f32", True),    # the channel-mean operands [B, K, N, L]
    (2, 3, 7, 5, 9, 11, "f32", False),     # padded states, L = 99
    (1, 2, 33, 1, 8, 8, "f32", False),     # N = 1 (256 segments per channel), odd channel count
    (2, 2, 5, 2, 6, 10, "bf16", False),    # N = 2, bf16 C
    (1, 2, 9, 4, 16, 16, "bf16", False),   # N = 4, vector loads
    (1, 1, 3, 8, 1, 3, "f32", False),      # L = 3 < one block
]


@pytest.mark.parametrize("shape", ONLY_SHAPES, ids=[f"B{s[0]}K{s[1]}Dm{s[2]}N{s[3]}_{s[4]}x{s[5]}_{s[6]}"
                                                    for s in ONLY_SHAPES])
def test_scan_only_parity(shape):
    B, K, Dm, N, H, W, dt, one = shape
    (dA, dBu, Cs), (gA, gB, gC) = scan_only_case(B, K, Dm, N, H, W, dt, seed=400 + Dm + N + H, one=one)
    y = vmb.vmb_scan_only_fwd(gA, gB, gC, H, W)
    torch.cuda.synchronize()
    check(to_numpy(y), oracle.scan_only(dA, dBu, Cs), "f32", "scan only y")


def test_scan_only_deterministic():
    _, (gA, gB, gC) = scan_only_case(1, 4, 40, 16, 28, 28, "f32", seed=450)
    y1 = vmb.vmb_scan_only_fwd(gA, gB, gC, 28, 28)
    y2 = vmb.vmb_scan_only_fwd(gA, gB, gC, 28, 28)
    assert torch.equal(y1, y2)


@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_split_path_matches_fused_path(dt):
    """Discretise, scan alone, add the skip term: the full path's y.  Means,
    scan alone: the channel-mean path's ybar.  Both against the oracle."""
    B, D, N, H, W = 1, 24, 16, 12, 14
    inp, u, g = inputs(B, D, N, H, W, dt, seed=460)
    dA, dBu = vmb.vmb_discretise_fwd(g["u"], g["draw"], g["A"], g["Bs"], g["bias"], H, W)
    y = vmb.vmb_scan_only_fwd(dA, dBu, g["Cs"], H, W)
    y = y + g["Dskip"].view(1, 4, D, 1) * g["u"].float()
    dAm, dBum = vmb.vmb_discretise_mean_fwd(g["u"], g["draw"], g["A"], g["Bs"], g["bias"], H, W)
    yb = vmb.vmb_scan_only_fwd(dAm, dBum, g["Cs"], H, W)
    torch.cuda.synchronize()
    yf_ref = oracle.selective_scan(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias)
    _, yb_ref = oracle.mean_scan(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias)
    check(to_numpy(y), yf_ref, "f32", "split full y")
    check(to_numpy(yb), yb_ref, "f32", "split mean ybar")


def test_empty_problem_launches_nothing():
    z = torch.empty((0, 4, 8, 16, 9), dtype=torch.float32, device=DEV)
    c = torch.empty((0, 4, 16, 9), dtype=torch.float32, device=DEV)
    y = vmb.vmb_scan_only_fwd(z, z, c, 3, 3)
    assert y.shape == (0, 4, 8, 9)
