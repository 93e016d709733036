"""The channel-mean approximation itself (Eq. 9 vs the full scan), on the oracle.

The paper prints no value for this error, so it is not a parity target; these
tests only check the properties the method implies: no loss when every channel
of a direction is identical, and an error that grows with the cross-channel
spread of the inputs (Sec. 2.1, Eq. 7 motivates the mean by a small spread)."""
import numpy as np

import oracle
import workloads


def rel_l2(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def mean_vs_full(sigma, seed=31):
    wl = workloads.small_case(B=1, D=24, N=16, H=10, W=10, sigma=sigma, seed=seed)
    inp = workloads.make_inputs(wl)
    _, yf, _ = oracle.ss2d_full(inp)
    _, ym, _, _ = oracle.ss2d_mean(inp)
    return rel_l2(ym, yf)


def test_identical_channels_lose_nothing():
    wl = workloads.small_case(B=1, D=12, N=16, H=6, W=7, seed=32)
    inp = workloads.make_inputs(wl, channel_identical=True)
    _, yf, _ = oracle.ss2d_full(inp)
    _, ym, _, _ = oracle.ss2d_mean(inp)
    assert rel_l2(ym, yf) < 1e-12


def test_error_grows_with_channel_spread():
    errs = [mean_vs_full(s) for s in (0.05, 0.1, 0.5)]
    print("mean-vs-full rel-L2 at sigma 0.05 / 0.1 / 0.5:", ["%.4f" % e for e in errs])
    assert errs[0] > 0
    assert errs[0] < errs[1] < errs[2]
