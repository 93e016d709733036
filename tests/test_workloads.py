"""The seeded input recipe the parity tests and the benchmark draw from
(workloads.make_inputs): reproducible per seed; under params="random" every
channel has its own A row and skip weight (so a kernel reading another
channel's or state's parameters cannot pass a parity test), while the draws
shared with the benchmark recipe stay the same; channel_identical=True shares
everything over the channels of a direction; bf16 workloads hold values that
bf16 represents exactly.  CPU only."""
import numpy as np
import pytest

import workloads


def _small(dtype="f32", **kw):
    return workloads.small_case(B=2, D=6, N=5, H=4, W=7, dtype=dtype, seed=41, **kw)


def test_same_seed_same_inputs():
    wl = _small()
    a, b = workloads.make_inputs(wl, params="random"), workloads.make_inputs(wl, params="random")
    for k, v in a.arrays().items():
        assert np.array_equal(v, b.arrays()[k]), k
    c = workloads.make_inputs(wl, seed=wl.seed + 1, params="random")
    assert not np.array_equal(a.x, c.x)


def test_random_parameters_differ_per_channel_and_state():
    wl = _small()
    inp = workloads.make_inputs(wl, params="random")
    A = inp.A.reshape(wl.K * wl.D, wl.N)
    assert np.all(A < 0)
    # every (channel, state) entry is its own draw: no two rows and no two columns agree
    assert len({tuple(r) for r in A}) == A.shape[0]
    assert len({tuple(c) for c in A.T}) == A.shape[1]
    assert len(set(inp.Dskip.ravel().tolist())) == inp.Dskip.size
    assert np.all((inp.Dskip >= 0.5) & (inp.Dskip <= 1.5))
    assert np.all((-A >= 0.5) & (-A <= 3.0))


def test_random_parameters_leave_the_shared_draws_unchanged():
    wl = _small()
    paper, rnd = workloads.make_inputs(wl, params="paper"), workloads.make_inputs(wl, params="random")
    for k in ("x", "draw", "Bs", "Cs", "bias"):
        assert np.array_equal(getattr(paper, k), getattr(rnd, k)), k
    # the benchmark recipe: A[c, n] = -(n + 1), Dskip = 1
    A = paper.A.reshape(wl.K * wl.D, wl.N)
    assert np.array_equal(A, np.broadcast_to(-(np.arange(wl.N) + 1.0), A.shape))
    assert np.all(paper.Dskip == 1.0)


def test_channel_identical_shares_everything_over_channels():
    wl = _small()
    inp = workloads.make_inputs(wl, params="random", channel_identical=True)
    x = inp.x.reshape(wl.B, wl.D, -1)
    assert np.array_equal(x, np.broadcast_to(x[:, :1], x.shape))
    draw = inp.draw.reshape(wl.B, wl.K, wl.D, -1)
    assert np.array_equal(draw, np.broadcast_to(draw[:, :, :1], draw.shape))
    A = inp.A.reshape(wl.K, wl.D, wl.N)
    assert np.array_equal(A, np.broadcast_to(A[:, :1], A.shape))
    for v in (inp.Dskip, inp.bias):
        r = v.reshape(wl.K, wl.D)
        assert np.array_equal(r, np.broadcast_to(r[:, :1], r.shape))


def test_bf16_workloads_hold_bf16_values():
    wl = _small(dtype="bf16")
    inp = workloads.make_inputs(wl, params="random")
    for k in ("x", "draw", "Bs", "Cs"):
        v = np.ascontiguousarray(getattr(inp, k), dtype=np.float32)
        low = v.view(np.uint32) & np.uint32(0xFFFF)
        assert not low.any(), f"{k} has bits below the bf16 mantissa"


def test_rejects_unknown_parameter_recipe():
    with pytest.raises(ValueError):
        workloads.make_inputs(_small(), params="nope")


def test_algorithmic_bytes_of_the_benchmark_workload():
    """The per-call byte counts the roofline divides by, against the sizes of
    the scan's operands written out: a scan call reads u, the raw Deltas, B
    and C and writes y (plus the per-channel parameters); a cross-scan or
    cross-merge call moves one map and its four direction rows."""
    wl = workloads.WORKLOADS["batch128_d256_n16_56x56_sigma0.05_f32"]
    B, K, D, N, L, s = 128, 4, 256, 16, 56 * 56, 4
    params = K * D * (N + 2) * 4  # A, Dskip, delta bias in fp32
    assert wl.scan_bytes() == s * (3 * B * K * D * L + 2 * B * K * N * L) + params
    assert abs(wl.scan_bytes() / 1e9 - 5.138) < 1e-3
    assert wl.csm_bytes() == 5 * s * B * D * L
    assert abs(wl.csm_bytes() / 1e9 - 2.055) < 1e-3
    assert wl.scan_elements() == B * K * D * L
