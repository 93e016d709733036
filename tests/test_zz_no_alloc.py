"""vmb_selective_scan_fwd_noalloc: the full scan for callers that cannot
allocate device memory (plugins inside a framework whose memory pool owns the
device, serving loops that must not allocate once they run), whose scratch is
an array built into the library instead of a caller workspace.

Called through the C ABI (ctypes) and compared, on two calls in a row (the
second runs on whatever the first left in the shared array), with
vmb_selective_scan_fwd, which takes a caller-allocated workspace, and with the
fp64 oracle.  The file is named so that pytest collects it last.
"""
import ctypes

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
SCRATCH_BYTES = 16 << 20  # the size of the built-in array


def noalloc_fn():
    fn = vmb.lib.vmb_selective_scan_fwd_noalloc
    vp, i = ctypes.c_void_p, ctypes.c_int
    fn.argtypes = [vp] * 8 + [i] * 6 + [ctypes.c_uint, i, vp]
    fn.restype = i
    return fn


def plan_bytes(flags, B, K, D, N, H, W, dtype):
    """Workspace bytes of the full-scan plan for exactly these flags (test-only query)."""
    fn = vmb.lib.vmb_testing_plan_workspace_bytes
    fn.argtypes = [ctypes.c_int, ctypes.c_uint] + [ctypes.c_int] * 7
    fn.restype = ctypes.c_size_t
    return int(fn(vmb.VMB_PATH_FULL, flags, B, K, D, N, H, W, dtype))


def _call(fn, args, y, B, D, N, H, W, flags, dtype):
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return fn(*(ctypes.c_void_p(t.data_ptr()) for t in args), ctypes.c_void_p(y.data_ptr()),
              B, 4, D, N, H, W, flags, dtype, stream)


FLAGS = {"euler": vmb.VMB_FLAG_SOFTPLUS, "zoh": vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_B_ZOH}
SHAPES = [(1, 64, 16, 48, 48, "f32"),   # few rows, long sequence: a multi-chunk plan
          (2, 96, 16, 16, 16, "bf16"),  # one chunk
          (1, 40, 3, 9, 11, "f32")]     # padded states, element-wise rows


@pytest.mark.parametrize("form", sorted(FLAGS))
@pytest.mark.parametrize("shape", SHAPES, ids=[f"B{s[0]}_D{s[1]}_N{s[2]}_{s[3]}x{s[4]}_{s[5]}" for s in SHAPES])
def test_noalloc_matches_workspace_entry_point(shape, form):
    B, D, N, H, W, dt = shape
    flags = FLAGS[form]
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=400 + D)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    args = (xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"])
    ref = vmb.vmb_selective_scan_fwd(*args, H, W, flags=flags)
    _, oref, _ = oracle.ss2d_full(inp, b_mode=1 if flags & vmb.VMB_FLAG_B_ZOH else 0)
    fn = noalloc_fn()
    dtype = vmb.VMB_BF16 if dt == "bf16" else vmb.VMB_F32
    for call in range(2):
        y = torch.full_like(ref, float("nan"))
        st = _call(fn, args, y, B, D, N, H, W, flags, dtype)
        assert st == vmb.VMB_OK, vmb.status_string(st)
        torch.cuda.synchronize()
        check(to_numpy(y), to_numpy(ref), dt, f"noalloc call {call + 1} vs the workspace entry point")
        check(to_numpy(y), oref, dt, f"noalloc call {call + 1} vs the oracle")


def test_noalloc_single_chunk_after_multi_chunk():
    """A one-chunk call clears only the status header; after a multi-chunk call
    the array still holds that call's flags and states, which it must not read."""
    fn = noalloc_fn()
    for shape in [(1, 64, 16, 48, 48, "f32"), (2, 96, 16, 16, 16, "f32"), (1, 64, 16, 48, 48, "f32")]:
        B, D, N, H, W, dt = shape
        wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=500 + D)
        inp = workloads.make_inputs(wl, params="random")
        g = to_device(inp, DEV)
        xs = vmb.vmb_cross_scan(g["x"])
        args = (xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"])
        y = torch.full_like(xs, float("nan"))
        st = _call(fn, args, y, B, D, N, H, W, vmb.VMB_FLAG_SOFTPLUS, vmb.VMB_F32)
        assert st == vmb.VMB_OK, vmb.status_string(st)
        torch.cuda.synchronize()
        _, oref, _ = oracle.ss2d_full(inp)
        check(to_numpy(y), oref, dt, f"noalloc {shape}")


def test_noalloc_rejects_plans_beyond_the_array():
    """A problem whose plan needs more scratch than the built-in array gets
    VMB_ERR_WORKSPACE and queues nothing (the output keeps its contents).  The
    buffers are real and sized for the problem."""
    fn = noalloc_fn()
    found = None
    for flags in (vmb.VMB_FLAG_SOFTPLUS | vmb.VMB_FLAG_B_ZOH, vmb.VMB_FLAG_SOFTPLUS):
        for (B, D, N, H, W) in [(1, 1, 16, 256, 256), (1, 1, 16, 512, 512), (1, 2, 16, 512, 512)]:
            if plan_bytes(flags, B, 4, D, N, H, W, vmb.VMB_F32) > SCRATCH_BYTES:
                found = (flags, B, D, N, H, W)
                break
        if found:
            break
    if found is None:
        pytest.skip("no candidate problem needs more than 16 MiB of scratch on this device")
    flags, B, D, N, H, W = found
    L = H * W
    gen = torch.Generator(device=DEV)
    gen.manual_seed(3)
    u = torch.randn(B, 4, D, L, device=DEV, generator=gen)
    draw = torch.randn(B, 4, D, L, device=DEV, generator=gen)
    Bs = torch.randn(B, 4, N, L, device=DEV, generator=gen)
    Cs = torch.randn(B, 4, N, L, device=DEV, generator=gen)
    A = -torch.ones(4 * D, N, device=DEV)
    Dskip = torch.ones(4 * D, device=DEV)
    bias = torch.full((4 * D,), -3.0, device=DEV)
    y = torch.full_like(u, 7.0)
    torch.cuda.synchronize()
    st = _call(fn, (u, draw, A, Bs, Cs, Dskip, bias), y, B, D, N, H, W, flags, vmb.VMB_F32)
    assert st == vmb.VMB_ERR_WORKSPACE, vmb.status_string(st)
    torch.cuda.synchronize()
    assert bool(torch.all(y == 7.0)), "a rejected call must not write its output"


def test_noalloc_rejects_invalid_arguments():
    fn = noalloc_fn()
    st = fn(*([ctypes.c_void_p(0)] * 8), 1, 4, 8, 16, 4, 4, vmb.VMB_FLAG_SOFTPLUS, vmb.VMB_F32, ctypes.c_void_p(0))
    assert st == vmb.VMB_ERR_INVALID_ARG
    st = fn(*([ctypes.c_void_p(0x10000)] * 8), 1, 4, 8, 17, 4, 4, vmb.VMB_FLAG_SOFTPLUS, vmb.VMB_F32,
            ctypes.c_void_p(0))
    assert st == vmb.VMB_ERR_UNSUPPORTED
    # a misaligned pointer (valid shape): rejected before anything is queued
    buf = torch.zeros(64, device=DEV)
    p = [ctypes.c_void_p(buf.data_ptr())] * 8
    p[0] = ctypes.c_void_p(buf.data_ptr() + 2)
    st = fn(*p, 1, 4, 1, 1, 1, 1, vmb.VMB_FLAG_SOFTPLUS, vmb.VMB_F32, ctypes.c_void_p(0))
    assert st == vmb.VMB_ERR_MISALIGNED
