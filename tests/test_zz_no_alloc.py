"""vmb_selective_scan_fwd_noalloc: the full scan for callers that cannot
allocate device memory, whose scratch is an array built into the library.

Called through the C ABI (ctypes) and compared with vmb_selective_scan_fwd,
which takes a caller-allocated workspace, on two calls in a row: the second
call runs on whatever the first one left in the shared scratch array.  The
file is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest

import workloads
from tests.parity import check, to_device, to_numpy

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU, skipped by marker
    pytest.skip("needs a GPU", allow_module_level=True)

import paper_2412_16602_gb300 as vmb  # noqa: E402

DEV = torch.device("cuda", 0)


def noalloc_fn():
    fn = vmb.lib.vmb_selective_scan_fwd_noalloc
    vp, i = ctypes.c_void_p, ctypes.c_int
    fn.argtypes = [vp] * 8 + [i] * 6 + [ctypes.c_uint, i, vp]
    fn.restype = i
    return fn


@pytest.mark.parametrize("shape", [(1, 64, 16, 48, 48, "f32"), (2, 96, 16, 16, 16, "bf16"), (1, 40, 3, 9, 11, "f32")])
def test_noalloc_matches_workspace_entry_point(shape):
    B, D, N, H, W, dt = shape
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=400 + D)
    inp = workloads.make_inputs(wl)
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    args = (xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"])
    ref = vmb.vmb_selective_scan_fwd(*args, H, W)
    fn = noalloc_fn()
    dtype = vmb.VMB_BF16 if dt == "bf16" else vmb.VMB_F32
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):
        y = torch.full_like(ref, float("nan"))
        st = fn(*(ctypes.c_void_p(t.data_ptr()) for t in args), ctypes.c_void_p(y.data_ptr()),
                B, 4, D, N, H, W, vmb.VMB_FLAG_SOFTPLUS, dtype, stream)
        assert st == vmb.VMB_OK, vmb.status_string(st)
        torch.cuda.synchronize()
        check(to_numpy(y), to_numpy(ref), dt, f"noalloc call {call + 1}")


def test_noalloc_rejects_invalid_arguments():
    fn = noalloc_fn()
    st = fn(*([ctypes.c_void_p(0)] * 8), 1, 4, 8, 16, 4, 4, vmb.VMB_FLAG_SOFTPLUS, vmb.VMB_F32, ctypes.c_void_p(0))
    assert st == vmb.VMB_ERR_INVALID_ARG
    st = fn(*([ctypes.c_void_p(0x10000)] * 8), 1, 4, 8, 17, 4, 4, vmb.VMB_FLAG_SOFTPLUS, vmb.VMB_F32,
            ctypes.c_void_p(0))
    assert st == vmb.VMB_ERR_UNSUPPORTED
