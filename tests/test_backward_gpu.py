"""GPU parity of the backward of the (grouped) channel-mean scan through the C
ABI against the fp64 oracle's gradients (which tests/oracle_pins.py pins to
finite differences of the forward)."""
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
    (1, 8, 4, 3, 5, "f32", 1),       # tiny, padded states
    (2, 40, 16, 9, 11, "f32", 1),    # odd L, ragged channel block
    (1, 70, 16, 32, 40, "f32", 1),   # L = 1280, several step blocks
    (2, 48, 16, 8, 8, "f32", 4),     # grouped basis: gB, gC summed over the groups
    (1, 24, 5, 7, 7, "f32", 3),      # three groups, odd N
    (1, 256, 16, 14, 14, "f32", 1),  # two channel blocks of launch 3
    (1, 48, 16, 16, 16, "bf16", 1),
    (2, 32, 8, 6, 10, "bf16", 2),
    (1, 128, 16, 8, 8, "f32", 2),    # two groups of 64 channels: whole channel blocks per group
    (1, 96, 16, 12, 12, "bf16", 2),  # groups of 48 channels: a partial channel block per group
    (1, 64, 16, 40, 40, "f32", 1),   # L = 1600: several step spans of launch 5, chunks of the scans
]


@pytest.mark.parametrize("case", CASES, ids=[f"B{c[0]}_D{c[1]}_N{c[2]}_{c[3]}x{c[4]}_{c[5]}_G{c[6]}" for c in CASES])
def test_mean_backward_matches_oracle(case):
    B, D, N, H, W, dt, G = case
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=900 + D + N + G)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    rng = np.random.default_rng(901 + D)
    gy_np = rng.standard_normal((B, 4, D, H * W)).astype(np.float32)
    if dt == "bf16":
        gy_np = workloads.round_to_bf16(gy_np)
    gy = torch.from_numpy(gy_np).to(xs.dtype).to(DEV)
    got = vmb.vmb_mean_scan_bwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], gy, H, W, groups=G)
    got2 = vmb.vmb_mean_scan_bwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"], gy, H, W, groups=G)
    torch.cuda.synchronize()
    u = oracle.cross_scan(inp.x)
    ref = oracle.mean_scan_bwd(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias, gy_np, groups=G)
    names = {"u": "u", "delta": "delta", "A": "A", "Bs": "Bs", "Cs": "Cs", "Dskip": "Dskip", "delta_bias": "bias"}
    for gname, rname in names.items():
        # the per-element gradients are stored in the input dtype; the parameter sums in fp32
        kind = dt if gname in ("u", "delta", "Bs", "Cs") else ("f32" if dt == "f32" else "bf16")
        check(to_numpy(got[gname]), ref[rname], kind, f"grad {gname}")
        assert torch.equal(got[gname], got2[gname]), f"grad {gname} must be deterministic"


@pytest.mark.parametrize("case", CASES, ids=[f"B{c[0]}_D{c[1]}_N{c[2]}_{c[3]}x{c[4]}_{c[5]}_G{c[6]}" for c in CASES])
def test_mean_backward_from_saved_means(case):
    """The training pair: vmb_mean_scan_train_fwd (y bit-identical to the
    grouped forward) keeps the group means, and the backward given them matches
    the oracle's gradients."""
    B, D, N, H, W, dt, G = case
    wl = workloads.small_case(B=B, D=D, N=N, H=H, W=W, dtype=dt, seed=940 + D + N + G)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    args = (xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"])
    y, saved, _ = vmb.vmb_mean_scan_train_fwd(*args, H, W, groups=G)
    y_ref, _ = vmb.vmb_mean_scan_grouped_fwd(*args, H, W, G)
    assert torch.equal(y, y_ref), "the training forward's y must be the grouped forward's"
    rng = np.random.default_rng(941 + D)
    gy_np = rng.standard_normal((B, 4, D, H * W)).astype(np.float32)
    if dt == "bf16":
        gy_np = workloads.round_to_bf16(gy_np)
    gy = torch.from_numpy(gy_np).to(xs.dtype).to(DEV)
    got = vmb.vmb_mean_scan_bwd(*args, gy, H, W, groups=G, saved=saved)
    torch.cuda.synchronize()
    assert vmb.vmb_read_status() == vmb.VMB_OK
    ref = oracle.mean_scan_bwd(oracle.cross_scan(inp.x), inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias, gy_np,
                               groups=G)
    names = {"u": "u", "delta": "delta", "A": "A", "Bs": "Bs", "Cs": "Cs", "Dskip": "Dskip", "delta_bias": "bias"}
    for gname, rname in names.items():
        kind = dt if gname in ("u", "delta", "Bs", "Cs") else ("f32" if dt == "f32" else "bf16")
        check(to_numpy(got[gname]), ref[rname], kind, f"grad {gname} (saved means)")


def test_mean_backward_softplus_off():
    wl = workloads.small_case(B=1, D=20, N=16, H=6, W=9, seed=931)
    inp = workloads.make_inputs(wl, params="random")
    inp.bias[:] = np.abs(inp.bias) + 0.5   # keep delta = raw + bias positive without the softplus
    inp.draw[:] = np.abs(inp.draw) * 0.05
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    gy_np = np.random.default_rng(932).standard_normal((1, 4, 20, 54)).astype(np.float32)
    got = vmb.vmb_mean_scan_bwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"],
                                torch.from_numpy(gy_np).to(DEV), 6, 9, flags=0)
    ref = oracle.mean_scan_bwd(oracle.cross_scan(inp.x), inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias, gy_np,
                               softplus_on=False)
    for gname, rname in [("u", "u"), ("delta", "delta"), ("A", "A"), ("Bs", "Bs"), ("Cs", "Cs"),
                         ("Dskip", "Dskip"), ("delta_bias", "bias")]:
        check(to_numpy(got[gname]), ref[rname], "f32", f"grad {gname} (softplus off)")


def test_mean_backward_matches_autograd_of_the_forward_on_one_sequence():
    """An independent check of the whole chain: the gradient of sum(gy * y) for
    the library's forward, taken by torch autograd of a plain fp64 restatement
    of the forward on the CPU, equals the library's backward."""
    wl = workloads.small_case(B=1, D=6, N=4, H=3, W=4, seed=933)
    inp = workloads.make_inputs(wl, params="random")
    g = to_device(inp, DEV)
    xs = vmb.vmb_cross_scan(g["x"])
    gy_np = np.random.default_rng(934).standard_normal((1, 4, 6, 12)).astype(np.float32)
    got = vmb.vmb_mean_scan_bwd(xs, g["draw"], g["A"], g["Bs"], g["Cs"], g["Dskip"], g["bias"],
                                torch.from_numpy(gy_np).to(DEV), 3, 4)
    t = {k: torch.from_numpy(np.asarray(v, dtype=np.float64)).requires_grad_(True) for k, v in
         dict(u=oracle.cross_scan(inp.x), delta=inp.draw, A=inp.A, Bs=inp.Bs, Cs=inp.Cs, Dskip=inp.Dskip,
              bias=inp.bias).items()}
    K, D, N, L = 4, 6, 4, 12
    total = 0.0
    for k in range(K):
        dl = torch.nn.functional.softplus(t["delta"][0, k] + t["bias"][k * D:(k + 1) * D, None])   # [D, L]
        Ak = t["A"][k * D:(k + 1) * D]                                                          # [D, N]
        abar = torch.exp(dl[:, :, None] * Ak[:, None, :]).mean(0)                                 # [L, N]
        s = (dl * t["u"][0, k]).mean(0)                                                          # [L]
        h = torch.zeros(N, dtype=torch.float64)
        for l in range(L):
            h = abar[l] * h + t["Bs"][0, k, :, l] * s[l]
            ybar = (t["Cs"][0, k, :, l] * h).sum()
            y = ybar + t["Dskip"][k * D:(k + 1) * D] * t["u"][0, k, :, l]
            total = total + (torch.from_numpy(gy_np[0, k, :, l]).double() * y).sum()
    total.backward()
    for gname, tname in [("u", "u"), ("delta", "delta"), ("A", "A"), ("Bs", "Bs"), ("Cs", "Cs"),
                         ("Dskip", "Dskip"), ("delta_bias", "bias")]:
        check(to_numpy(got[gname]), t[tname].grad.numpy(), "f32", f"grad {gname} vs autograd")
