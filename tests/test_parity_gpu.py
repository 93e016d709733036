"""GPU parity: the CUDA path through the C ABI against the fp64 oracle.

Index work (cross-scan) is compared bit for bit; floating-point outputs within
rel-L2 <= 1e-5 and max-abs <= 1e-4 max|y| (fp32 storage) or rel-L2 <= 1e-2
(bf16 storage).  Shapes span several tiles and chunks and ragged tails.
"""
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


def gpu_step(inp, flags=vmb.VMB_FLAG_SOFTPLUS, mean_flags=None):
    g = to_device(inp, DEV)
    wl = inp.wl
    xs = vmb.vmb_cross_scan(g["x"])
    yf = vmb.vmb_selective_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W,
                                    flags=flags)
    ym, ybar = vmb.vmb_mean_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W,
                                     want_ybar=True, flags=flags if mean_flags is None else mean_flags)
    of = vmb.vmb_cross_merge(yf, wl.H, wl.W)
    om = vmb.vmb_cross_merge(ym, wl.H, wl.W)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    return {k: v for k, v in dict(xs=xs, yf=yf, ym=ym, ybar=ybar, of=of, om=om).items()}


SHAPES = [
    # (B, D, N, H, W, dtype)
    (1, 192, 16, 14, 14, "f32"),     # the small SS2D workload
    (2, 40, 16, 9, 11, "f32"),       # ragged channel tile, odd L = 99 (element-wise path)
    (1, 70, 16, 32, 40, "f32"),      # L = 1280: several stages and L-chunks
    (3, 33, 5, 7, 7, "f32"),         # odd N (padded states), L = 49
    (2, 64, 1, 12, 16, "f32"),       # N = 1
    (2, 24, 8, 8, 8, "f32"),         # N = 8
    (1, 48, 3, 5, 13, "bf16"),       # bf16, odd L
    (2, 96, 16, 16, 16, "bf16"),     # bf16, aligned rows
    (1, 8, 16, 64, 64, "f32"),       # few channels, long sequence: many chunks
    (1, 6, 4, 37, 29, "f32"),        # band cross-scan/merge: ragged last band, odd width (element path)
    (2, 6, 4, 32, 40, "bf16"),       # band cross-scan/merge, bf16 vector path
]


@pytest.mark.parametrize("shape", SHAPES, ids=[f"B{s[0]}_D{s[1]}_N{s[2]}_{s[3]}x{s[4]}_{s[5]}" for s in SHAPES])
def test_ss2d_parity(shape):
    B, D, N, H, W, dt = shape
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=100 + D + N)
    inp = workloads.make_inputs(wl, params="random")
    out = gpu_step(inp)
    u_ref, yf_ref, of_ref = oracle.ss2d_full(inp)
    _, ym_ref, ybar_ref, om_ref = oracle.ss2d_mean(inp)
    xs = to_numpy(out["xs"])
    assert np.array_equal(xs, u_ref), "cross-scan must be bit-exact"
    check(to_numpy(out["yf"]), yf_ref, dt, "full y")
    check(to_numpy(out["of"]), of_ref, dt, "full merged")
    check(to_numpy(out["ym"]), ym_ref, dt, "mean y")
    check(to_numpy(out["ybar"]), ybar_ref, "f32" if dt == "f32" else "bf16", "mean ybar")
    check(to_numpy(out["om"]), om_ref, dt, "mean merged")


@pytest.mark.parametrize("flags", [0, vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_B_ZOH, vmb.VMB_FLAG_B_ZOH])
def test_flag_variants(flags):
    wl = workloads.small_case(B=1, D=50, N=16, H=10, W=12, seed=5)
    inp = workloads.make_inputs(wl, params="random")
    if not flags & vmb.VMB_FLAG_SOFTPLUS:
        inp.bias[:] = np.abs(inp.bias)          # keep delta = raw + bias positive without softplus
        inp.draw[:] = np.abs(inp.draw) * 0.05
    out = gpu_step(inp, flags=flags)
    kw = dict(softplus_on=bool(flags & vmb.VMB_FLAG_SOFTPLUS), b_mode=1 if flags & vmb.VMB_FLAG_B_ZOH else 0)
    _, yf_ref, _ = oracle.ss2d_full(inp, **kw)
    _, ym_ref, ybar_ref, _ = oracle.ss2d_mean(inp, **kw)
    check(to_numpy(out["yf"]), yf_ref, "f32", "full y")
    check(to_numpy(out["ym"]), ym_ref, "f32", "mean y")


def test_skip_mean_mode():
    wl = workloads.small_case(B=2, D=30, N=4, H=6, W=8, seed=6)
    inp = workloads.make_inputs(wl, params="random")
    out = gpu_step(inp, mean_flags=vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_SKIP_MEAN)
    _, ym_ref, _, _ = oracle.ss2d_mean(inp, skip_mode=oracle.SKIP_MEAN)
    check(to_numpy(out["ym"]), ym_ref, "f32", "mean y (skip mean)")


def test_merge_exact_on_integers():
    """With integer-valued inputs every partial sum is exact: the merge is bit-exact.
    Maps of 1024 pixels or more take the band kernel (32-row fp32 bands, 16-row
    bf16 bands): 72 and 40 rows end in a short band on the vector path, 37 x 29
    on the element path."""
    rng = np.random.default_rng(9)
    for (B, D, H, W, dt) in [(2, 3, 5, 7, "f32"), (1, 4, 8, 8, "f32"), (3, 2, 1, 9, "f32"), (1, 3, 72, 40, "f32"),
                             (1, 2, 37, 29, "f32"), (2, 2, 40, 48, "bf16"), (1, 2, 56, 56, "f32")]:
        ys = rng.integers(-30, 31, size=(B, 4, D, H * W)).astype(np.float32)
        t = torch.from_numpy(ys).to(DEV)
        if dt == "bf16":
            t = t.to(torch.bfloat16)  # |sums| <= 120: exact in bf16
        got = vmb.vmb_cross_merge(t, H, W).float().cpu().numpy()
        assert np.array_equal(got.astype(np.float64), oracle.cross_merge(ys, H, W)), (H, W, dt)


def test_misaligned_views_take_element_path():
    """Tensors starting 4 bytes into an allocation are valid (element-wise path)."""
    wl = workloads.small_case(B=1, D=20, N=16, H=8, W=8, seed=8)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)

    def shifted(t):
        buf = torch.empty(t.numel() + 1, dtype=t.dtype, device=DEV)
        v = buf[1:].view(t.shape)
        v.copy_(t)
        return v

    xs = vmb.vmb_cross_scan(shifted(g["x"]), shifted(torch.empty((1, 4, 20, 64), device=DEV)))
    y = shifted(torch.empty_like(xs))
    vmb.vmb_selective_scan_fwd(xs, shifted(g["draw"]), g["A"], shifted(g["Bs"]), shifted(g["Cs"]), g["Dskip"],
                               g["bias"], 8, 8, y=y)
    _, yf_ref, _ = oracle.ss2d_full(inp)
    check(to_numpy(y), yf_ref, "f32", "full y (misaligned)")


def test_empty_problem_is_a_noop():
    x = torch.empty((0, 4, 5, 5), device=DEV)
    assert vmb.vmb_cross_scan(x).shape == (0, 4, 4, 25)


@pytest.mark.parametrize("plan", ["", "5,6"])
def test_workspace_reuse_over_many_calls(plan, force_plan):
    """The workspace stays consistent over repeated chunked calls (the default
    chunked variant and a forced look-back plan), with bit-identical results."""
    if plan:
        force_plan.full(plan)
    wl = workloads.small_case(B=1, D=16, N=16, H=40, W=40, seed=10)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    ref = None
    for _ in range(20):
        y = vmb.vmb_selective_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], 40, 40)
        ym, _ = vmb.vmb_mean_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], 40, 40)
        if ref is None:
            ref = (y.clone(), ym.clone())
        else:
            assert torch.equal(y, ref[0]) and torch.equal(ym, ref[1]), "results must be deterministic"
    assert vmb.vmb_read_status() == vmb.VMB_OK


@pytest.mark.parametrize("mean", [False, True])
def test_lookback_wait_times_out_cleanly(mean, force_plan):
    """A chunk that never publishes makes its successors' bounded waits run out:
    the call reports VMB_ERR_TIMEOUT and the context and workspace stay usable."""
    if not mean:
        force_plan.full("5,6")  # a look-back plan (the default here is the chunked variant)
    wl = workloads.small_case(B=1, D=16, N=16, H=48, W=48, seed=11)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    ws = torch.zeros(vmb.vmb_scan_workspace_bytes(1 if mean else 0, 1, 4, 16, 16, 48, 48) + 256,
                     dtype=torch.uint8, device=DEV)
    args = (xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], 48, 48)
    flags = vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_TEST_SUPPRESS_PUBLISH
    if mean:
        vmb.vmb_mean_scan_fwd(*args, flags=flags, workspace=ws)
    else:
        vmb.vmb_selective_scan_fwd(*args, flags=flags, workspace=ws)
    assert vmb.vmb_read_status(ws) == vmb.VMB_ERR_TIMEOUT
    assert vmb.vmb_read_status(ws) == vmb.VMB_OK  # cleared
    # the same workspace works again
    if mean:
        y, _ = vmb.vmb_mean_scan_fwd(*args, workspace=ws)
        _, ref, _, _ = oracle.ss2d_mean(inp)
    else:
        y = vmb.vmb_selective_scan_fwd(*args, workspace=ws)
        _, ref, _ = oracle.ss2d_full(inp)
    assert vmb.vmb_read_status(ws) == vmb.VMB_OK
    check(to_numpy(y), ref, "f32", "after timeout")


@pytest.mark.parametrize("plan", ["0", "1", "2", "3", "4", "5", "6", "7", "8", "9", "10", "11", "12", "13", "14", "15",
                                  "16", "17", "18", "19", "0,3", "3,5", "4,2", "5,4", "6,7", "7,3", "7,6"])
@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_every_tile_shape(plan, dt, force_plan):
    """Each tile shape of the full scan (and forced L-chunking) against the oracle."""
    force_plan.full(plan)
    wl = workloads.small_case(B=1, D=72, N=16, H=24, W=28, dtype=dt, seed=21)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    y = vmb.vmb_selective_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    _, ref, _ = oracle.ss2d_full(inp)
    check(to_numpy(y), ref, dt, f"full y plan {plan}")


def test_warp_specialised_stage_wait_times_out_cleanly(force_plan):
    """The warp-specialised full scan with the first stage never handed over
    (test hook): the compute warps' bounded waits and then the copy warp's run
    out, the call reports VMB_ERR_TIMEOUT, the status clears, and the same
    workspace then gives correct results."""
    force_plan.full("19")
    wl = workloads.small_case(B=1, D=64, N=16, H=16, W=16, seed=88)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    ws = torch.zeros(vmb.vmb_scan_workspace_bytes(0, 1, 4, 64, 16, 16, 16), dtype=torch.uint8, device=DEV)
    args = (xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], 16, 16)
    vmb.vmb_selective_scan_fwd(*args, flags=vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_TEST_SUPPRESS_PUBLISH, workspace=ws)
    assert vmb.vmb_read_status(ws) == vmb.VMB_ERR_TIMEOUT
    assert vmb.vmb_read_status(ws) == vmb.VMB_OK  # cleared
    y = vmb.vmb_selective_scan_fwd(*args, workspace=ws)
    assert vmb.vmb_read_status(ws) == vmb.VMB_OK
    _, ref, _ = oracle.ss2d_full(inp)
    check(to_numpy(y), ref, "f32", "after the stage wait ran out")


WS_CASES = [
    # (B, D, N, H, W, dtype)
    (1, 256, 16, 9, 12, "f32"),   # L = 108: the last 8-step stage half full; two full channel tiles
    (2, 72, 16, 16, 24, "bf16"),  # bf16 rows of 16-byte multiples; a tile with three consumer warps
    (1, 200, 13, 8, 10, "f32"),   # 13 states: B/C rows past N read as zero; a 72-channel tile
    (1, 128, 16, 56, 56, "f32"),  # 392 stages: the 4-slot ring wraps around many times
    (1, 64, 16, 7, 7, "f32"),     # L = 49: rows not 16-byte multiples -> the packed variant instead
]


@pytest.mark.parametrize("case", WS_CASES, ids=[f"B{s[0]}_D{s[1]}_N{s[2]}_{s[3]}x{s[4]}_{s[5]}" for s in WS_CASES])
def test_warp_specialised_full_scan(case, force_plan):
    """The warp-specialised full scan (tensor copies, mbarrier hand-over) against
    the oracle, deterministic, and bit-identical to the packed streaming variant
    whose arithmetic it shares."""
    B, D, N, H, W, dt = case
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=71 + D + N)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    args = (xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W)
    force_plan.full("19")
    y = vmb.vmb_selective_scan_fwd(*args)
    y2 = vmb.vmb_selective_scan_fwd(*args)
    force_plan.full("16")
    yp = vmb.vmb_selective_scan_fwd(*args)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    _, ref, _ = oracle.ss2d_full(inp)
    check(to_numpy(y), ref, dt, "warp-specialised full y")
    assert torch.equal(y, y2), "the warp-specialised scan must be deterministic"
    assert torch.equal(y, yp), "the warp-specialised scan must match the packed variant bit for bit"


CHUNKED_CASES = [
    # (B, D, N, H, W, dtype)
    (1, 72, 16, 20, 30, "f32"),   # L = 600: ragged last chunk, ragged channel tile, vector rows
    (1, 72, 16, 23, 29, "f32"),   # L = 667: element-wise rows
    (2, 40, 12, 17, 19, "bf16"),  # padded states, odd L, bf16
    (2, 64, 16, 16, 24, "bf16"),  # bf16 vector rows
    (1, 24, 16, 5, 5, "f32"),     # one chunk only: no aggregate or carry launch
]


@pytest.mark.parametrize("plan", ["8", "9", "10", "11"])
@pytest.mark.parametrize("case", CHUNKED_CASES, ids=[f"B{s[0]}_D{s[1]}_N{s[2]}_{s[3]}x{s[4]}_{s[5]}"
                                                     for s in CHUNKED_CASES])
def test_chunked_full_scan(plan, case, force_plan):
    """The three-launch chunked full scan (aggregates, carry fold, rerun) against the oracle."""
    force_plan.full(plan)
    B, D, N, H, W, dt = case
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=31 + D)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    y = vmb.vmb_selective_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W)
    y2 = vmb.vmb_selective_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    _, ref, _ = oracle.ss2d_full(inp)
    check(to_numpy(y), ref, dt, f"chunked full y plan {plan}")
    assert torch.equal(y, y2), "the chunked scan must be deterministic"


@pytest.mark.parametrize("tc", ["32", "64", "128"])
@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_every_mean_chunk_length(tc, dt, force_plan):
    """Each chunk length of the channel-mean scan against the oracle (ragged last chunk)."""
    force_plan.mean(tc)
    wl = workloads.small_case(B=2, D=70, N=16, H=19, W=21, dtype=dt, seed=22)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    y, yb = vmb.vmb_mean_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W,
                                  want_ybar=True)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    _, ref, ybar_ref, _ = oracle.ss2d_mean(inp)
    check(to_numpy(y), ref, dt, f"mean y tc {tc}")
    check(to_numpy(yb), ybar_ref, dt, f"mean ybar tc {tc}")


_ZOH_FIRST = r"""
import sys
sys.path.insert(0, sys.argv[1])
import torch
import oracle, workloads
import paper_2412_16602_gb300 as vmb
from tests.parity import check, to_device, to_numpy

dev = torch.device("cuda", 0)
wl = workloads.small_case(B=1, D=8, N=16, H=32, W=32, seed=61)
inp = workloads.make_inputs(wl, params="random")
g = to_device(inp, dev)
xs = vmb.vmb_cross_scan(g["x"])
args = (xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W)
flags = vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_B_ZOH
wsf = torch.zeros(vmb.vmb_scan_workspace_bytes(0, 1, 4, 8, 16, 32, 32), dtype=torch.uint8, device=dev)
wsm = torch.zeros(vmb.vmb_scan_workspace_bytes(1, 1, 4, 8, 16, 32, 32), dtype=torch.uint8, device=dev)
yf = vmb.vmb_selective_scan_fwd(*args, flags=flags, workspace=wsf)
ym, _ = vmb.vmb_mean_scan_fwd(*args, flags=flags, workspace=wsm)
assert vmb.vmb_read_status(wsf) == 0 and vmb.vmb_read_status(wsm) == 0
_, rf, _ = oracle.ss2d_full(inp, b_mode=1)
_, rm, _, _ = oracle.ss2d_mean(inp, b_mode=1)
check(to_numpy(yf), rf, "f32", "zoh full y")
check(to_numpy(ym), rm, "f32", "zoh mean y")
print("zoh-first ok")
"""


def test_zoh_first_call_with_exactly_sized_workspace():
    """In a fresh process (no workspace grown by earlier calls), the first scans
    use the zero-order-hold form on a workspace of exactly the size the query
    returns: on this few-row, L = 1024 map the ZOH plan is chunked while the
    Euler plan is not, so the query must cover both forms."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "-c", _ZOH_FIRST, root], cwd=root, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "zoh-first ok" in r.stdout
