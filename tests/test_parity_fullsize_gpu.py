"""Full-size parity: every benchmark workload, in the launch configuration the
benchmark times, checked against the fp64 oracle on sampled outputs.

The full scan is independent per channel row, so sampled rows (b, k, d) are
recomputed by the oracle one by one; the channel-mean scan needs every
channel of a (b, k), so sampled sequences are recomputed whole; merged maps
are checked on sampled (b, d) planes from the oracle's four direction rows.
The cross-scan is checked bit for bit on the sampled planes.
"""
import zlib

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


def _param_slice(inp, k, d_idx):
    K, D = inp.wl.K, inp.wl.D
    c = k * D + np.asarray(d_idx)
    return inp.A[c], inp.Dskip[c], inp.bias[c]


@pytest.mark.parametrize("name", sorted(workloads.WORKLOADS))
def test_fullsize_sampled(name):
    wl = workloads.WORKLOADS[name]
    inp = workloads.make_inputs(wl)
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    yf = vmb.vmb_selective_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W)
    ym, ybar = vmb.vmb_mean_scan_fwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], wl.H, wl.W,
                                     want_ybar=True)
    of = vmb.vmb_cross_merge(yf, wl.H, wl.W)
    om = vmb.vmb_cross_merge(ym, wl.H, wl.W)
    assert vmb.vmb_read_status() == vmb.VMB_OK
    torch.cuda.synchronize()
    rng = np.random.default_rng(zlib.crc32(name.encode()))
    B, D = wl.B, wl.D
    dt = wl.dtype
    # ---- sampled planes: cross-scan bit-exact, full rows of all four directions, merged plane
    for _ in range(3):
        b, d = int(rng.integers(B)), int(rng.integers(D))
        u_ref = oracle.cross_scan(inp.x[b:b + 1, d:d + 1])                        # [1, 4, 1, L]
        assert np.array_equal(to_numpy(xs[b, :, d]), u_ref[0, :, 0]), "cross-scan must be bit-exact"
        rows = []
        for k in range(4):
            A, Dsk, bias = _param_slice(inp, k, [d])
            y = oracle.selective_scan(u_ref[:, k:k + 1], inp.draw[b:b + 1, k:k + 1, d:d + 1], A,
                                      inp.Bs[b:b + 1, k:k + 1], inp.Cs[b:b + 1, k:k + 1], Dsk, bias)
            rows.append(y[0, 0, 0])
            check(to_numpy(yf[b, k, d]), y[0, 0, 0], dt, f"{name} full row b={b} k={k} d={d}")
        merged = oracle.cross_merge(np.stack(rows)[None, :, None, :], wl.H, wl.W)[0, 0]
        check(to_numpy(of[b, d]), merged, dt, f"{name} full merged b={b} d={d}")
    # ---- the channel-mean path for one batch element: all four directions, all channels
    b = int(rng.integers(B))
    u_ref = oracle.cross_scan(inp.x[b:b + 1])                                      # [1, 4, D, L]
    y_ref, yb_ref = oracle.mean_scan(u_ref, inp.draw[b:b + 1], inp.A, inp.Bs[b:b + 1], inp.Cs[b:b + 1],
                                     inp.Dskip, inp.bias)
    check(to_numpy(ybar[b]), yb_ref[0], "f32" if dt == "f32" else "bf16", f"{name} ybar b={b}")
    for k in range(4):
        dd = rng.choice(D, size=min(D, 16), replace=False)
        check(to_numpy(ym[b, k][dd]), y_ref[0, k][dd], dt, f"{name} mean rows b={b} k={k}")
    for d in rng.choice(D, size=2, replace=False):
        merged = oracle.cross_merge(y_ref[:, :, d:d + 1], wl.H, wl.W)[0, 0]
        check(to_numpy(om[b, d]), merged, dt, f"{name} mean merged b={b} d={d}")
