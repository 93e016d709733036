"""fp64 CPU oracle for the SS2D selective scan (full path) and VMeanba (channel-mean path).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package; the library under
``paper_2412_16602_gb300`` never does, and shares no code with it.

The arithmetic lives in ``oracle.c`` (plain double-precision loops, one
function per step of the paper: cross-scan and cross-merge from App. A
"VMamba", softplus from Eq. 6, discretisation from Eq. 4, the recurrence from
Eq. 3, the channel mean and broadcast from Eq. 9).  This module only converts
numpy arrays to contiguous float64 and calls it.

Every function is pinned by ``tests/test_oracle_pins.py`` against closed
forms, hand-worked cases, invariants and brute-force unrolling, and
``tests/test_oracle_mutants.py`` plants mistakes in a copy of ``oracle.c`` to
show the pins catch them.  The accuracy of the channel-mean approximation
itself (mean path vs full path on noisy inputs) has no printed value in the
paper: that comparison is parity unpinned and only reported as a statistic.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "oracle.c")
LIB_PATH = os.path.join(_HERE, "liboracle.so")

B_EULER, B_ZOH = 0, 1
SKIP_PER_CHANNEL, SKIP_MEAN = 0, 1

CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-pthread", "-fno-fast-math", "-ffp-contract=off"]


def compile_c(src: str, out: str) -> str:
    """Compile one oracle C source into a shared library (gcc, IEEE double)."""
    tmp = out + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", *CFLAGS, src, "-o", tmp, "-lm"])
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so next to it, if missing or stale."""
    if force or not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < os.path.getmtime(SOURCE):
        compile_c(SOURCE, LIB_PATH)
    return LIB_PATH


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


class Oracle:
    """The oracle functions bound to one compiled copy of oracle.c."""

    def __init__(self, lib_path: str):
        lib = ctypes.CDLL(lib_path)
        P = ctypes.POINTER(ctypes.c_double)
        lg, i = ctypes.c_long, ctypes.c_int
        lib.oracle_cross_scan.argtypes = [P, P, lg, lg, lg, lg]
        lib.oracle_cross_scan.restype = None
        lib.oracle_cross_merge.argtypes = [P, P, lg, lg, lg, lg]
        lib.oracle_cross_merge.restype = None
        lib.oracle_selective_scan.argtypes = [P] * 8 + [lg] * 5 + [i, i, i]
        lib.oracle_selective_scan.restype = i
        lib.oracle_mean_scan.argtypes = [P] * 9 + [lg] * 5 + [i, i, i, i]
        lib.oracle_mean_scan.restype = i
        lib.oracle_softplus.argtypes = [P, P, lg]
        lib.oracle_softplus.restype = None
        lib.oracle_discretise.argtypes = [P] * 7 + [lg] * 5 + [i, i]
        lib.oracle_discretise.restype = None
        lib.oracle_discretise_mean.argtypes = [P] * 7 + [lg] * 5 + [i, i]
        lib.oracle_discretise_mean.restype = None
        lib.oracle_scan_only.argtypes = [P] * 4 + [lg] * 5
        lib.oracle_scan_only.restype = None
        lib.oracle_mean_scan_grouped.argtypes = [P] * 9 + [lg] * 6 + [i, i, i]
        lib.oracle_mean_scan_grouped.restype = i
        lib.oracle_selection.argtypes = [P] * 8 + [lg] * 6
        lib.oracle_selection.restype = None
        lib.oracle_mean_scan_bwd.argtypes = [P] * 15 + [lg] * 6 + [i]
        lib.oracle_mean_scan_bwd.restype = None
        self.lib = lib
        self.path = lib_path

    def cross_scan(self, x) -> np.ndarray:
        """x [B, D, H, W] -> xs [B, 4, D, H*W] (App. A, VMamba: unfold along four directions)."""
        x = _f64(x)
        B, D, H, W = x.shape
        xs = np.empty((B, 4, D, H * W), dtype=np.float64)
        self.lib.oracle_cross_scan(_ptr(x), _ptr(xs), B, D, H, W)
        return xs

    def cross_merge(self, ys, H: int, W: int) -> np.ndarray:
        """ys [B, 4, D, H*W] -> out [B, D, H, W] (App. A, VMamba: merge the four directions)."""
        ys = _f64(ys)
        B, K, D, L = ys.shape
        if K != 4 or L != H * W:
            raise ValueError("cross_merge expects ys [B, 4, D, H*W]")
        out = np.empty((B, D, H, W), dtype=np.float64)
        self.lib.oracle_cross_merge(_ptr(ys), _ptr(out), B, D, H, W)
        return out

    def softplus(self, x) -> np.ndarray:
        """Eq. 6 tau_Delta = softplus, in double precision."""
        x = _f64(x)
        out = np.empty_like(x)
        self.lib.oracle_softplus(_ptr(x), _ptr(out), x.size)
        return out

    @staticmethod
    def _scan_args(u, delta, A, Bs, Cs, Dskip, bias):
        u, delta, A, Bs, Cs, Dskip, bias = (_f64(a) for a in (u, delta, A, Bs, Cs, Dskip, bias))
        B, K, D, L = u.shape
        N = Bs.shape[2]
        if delta.shape != u.shape or Bs.shape != (B, K, N, L) or Cs.shape != (B, K, N, L):
            raise ValueError("shape mismatch")
        if A.shape != (K * D, N) or Dskip.shape != (K * D,) or bias.shape != (K * D,):
            raise ValueError("parameter shape mismatch")
        return (u, delta, A, Bs, Cs, Dskip, bias), (B, K, D, N, L)

    def selective_scan(self, u, delta, A, Bs, Cs, Dskip, bias, *, softplus_on=True,
                       b_mode=B_EULER, nthreads: int | None = None) -> np.ndarray:
        """Full-channel selective scan (Eqs. 3, 4, 6): y [B, K, D, L]."""
        arrs, (B, K, D, N, L) = self._scan_args(u, delta, A, Bs, Cs, Dskip, bias)
        y = np.empty((B, K, D, L), dtype=np.float64)
        rc = self.lib.oracle_selective_scan(*(_ptr(a) for a in arrs), _ptr(y), B, K, D, N, L,
                                            int(bool(softplus_on)), int(b_mode),
                                            nthreads or default_threads())
        if rc:
            raise RuntimeError("oracle_selective_scan failed")
        return y

    def mean_scan(self, u, delta, A, Bs, Cs, Dskip, bias, *, softplus_on=True, b_mode=B_EULER,
                  skip_mode=SKIP_PER_CHANNEL, nthreads: int | None = None):
        """VMeanba channel-mean scan (Eq. 9): returns (y [B, K, D, L], ybar [B, K, L])."""
        arrs, (B, K, D, N, L) = self._scan_args(u, delta, A, Bs, Cs, Dskip, bias)
        y = np.empty((B, K, D, L), dtype=np.float64)
        ybar = np.empty((B, K, L), dtype=np.float64)
        rc = self.lib.oracle_mean_scan(*(_ptr(a) for a in arrs), _ptr(y), _ptr(ybar), B, K, D, N,
                                       L, int(bool(softplus_on)), int(b_mode), int(skip_mode),
                                       nthreads or default_threads())
        if rc:
            raise RuntimeError("oracle_mean_scan failed")
        return y, ybar

    def mean_scan_grouped(self, u, delta, A, Bs, Cs, Dskip, bias, groups: int, *, softplus_on=True,
                          b_mode=B_EULER, skip_mode=SKIP_PER_CHANNEL):
        """Grouped basis (reduced channel dimension d = groups): the mean of Eq. 9 over each of
        `groups` consecutive channel groups; returns (y [B, K, D, L], ybar [B, K, groups, L])."""
        arrs, (B, K, D, N, L) = self._scan_args(u, delta, A, Bs, Cs, Dskip, bias)
        y = np.empty((B, K, D, L), dtype=np.float64)
        ybar = np.empty((B, K, groups, L), dtype=np.float64)
        rc = self.lib.oracle_mean_scan_grouped(*(_ptr(a) for a in arrs), _ptr(y), _ptr(ybar), B, K, D, N, L,
                                               int(groups), int(bool(softplus_on)), int(b_mode), int(skip_mode))
        if rc:
            raise ValueError("groups must divide D")
        return y, ybar

    def mean_scan_bwd(self, u, delta, A, Bs, Cs, Dskip, bias, gy, *, groups: int = 1, softplus_on=True):
        """Gradients of the (grouped) channel-mean scan with the Euler Bbar and the per-channel
        skip term (the adjoint of Eq. 9's forward), given gy = dLoss/dy [B, K, D, L]: returns
        dict(u, delta, A, Bs, Cs, Dskip, bias) of gradients with the inputs' shapes (delta is
        the raw Delta before bias and softplus)."""
        arrs, (B, K, D, N, L) = self._scan_args(u, delta, A, Bs, Cs, Dskip, bias)
        gy = _f64(gy)
        if gy.shape != (B, K, D, L):
            raise ValueError("gy must be [B, K, D, L]")
        if groups < 1 or D % groups:
            raise ValueError("groups must divide D")
        out = dict(u=np.empty((B, K, D, L)), delta=np.empty((B, K, D, L)), A=np.empty((K * D, N)),
                   Bs=np.empty((B, K, N, L)), Cs=np.empty((B, K, N, L)), Dskip=np.empty(K * D),
                   bias=np.empty(K * D))
        self.lib.oracle_mean_scan_bwd(*(_ptr(a) for a in arrs), _ptr(gy), _ptr(out["u"]), _ptr(out["delta"]),
                                      _ptr(out["A"]), _ptr(out["Bs"]), _ptr(out["Cs"]), _ptr(out["Dskip"]),
                                      _ptr(out["bias"]), B, K, D, N, L, int(groups), int(bool(softplus_on)))
        return out

    def selection(self, u, WB, WC, Wz, Wup):
        """Eq. 6 selection functions: u [B, K, D, L], WB and WC [K, N, D], Wz [K, R, D],
        Wup [K, D, R] -> (delta_raw [B, K, D, L], Bs [B, K, N, L], Cs [B, K, N, L])."""
        u, WB, WC, Wz, Wup = (_f64(a) for a in (u, WB, WC, Wz, Wup))
        B, K, D, L = u.shape
        N, R = WB.shape[1], Wz.shape[1]
        if WB.shape != (K, N, D) or WC.shape != (K, N, D) or Wz.shape != (K, R, D) or Wup.shape != (K, D, R):
            raise ValueError("weight shape mismatch")
        dr = np.empty((B, K, D, L), dtype=np.float64)
        Bs = np.empty((B, K, N, L), dtype=np.float64)
        Cs = np.empty_like(Bs)
        self.lib.oracle_selection(_ptr(u), _ptr(WB), _ptr(WC), _ptr(Wz), _ptr(Wup), _ptr(Bs), _ptr(Cs), _ptr(dr),
                                  B, K, D, N, R, L)
        return dr, Bs, Cs

    def _disc_args(self, u, delta, A, Bs, bias):
        u, delta, A, Bs, bias = (_f64(a) for a in (u, delta, A, Bs, bias))
        B, K, D, L = u.shape
        N = Bs.shape[2]
        if delta.shape != u.shape or Bs.shape != (B, K, N, L) or A.shape != (K * D, N) or bias.shape != (K * D,):
            raise ValueError("shape mismatch")
        return (u, delta, A, Bs, bias), (B, K, D, N, L)

    def discretise(self, u, delta, A, Bs, bias, *, softplus_on=True, b_mode=B_EULER):
        """Eqs. 4, 6 outside the scan (Sec. 4 kernel setting): (dA, dBu), each [B, K, D, N, L]."""
        arrs, (B, K, D, N, L) = self._disc_args(u, delta, A, Bs, bias)
        dA = np.empty((B, K, D, N, L), dtype=np.float64)
        dBu = np.empty_like(dA)
        self.lib.oracle_discretise(*(_ptr(a) for a in arrs), _ptr(dA), _ptr(dBu), B, K, D, N, L,
                                   int(bool(softplus_on)), int(b_mode))
        return dA, dBu

    def discretise_mean(self, u, delta, A, Bs, bias, *, softplus_on=True, b_mode=B_EULER):
        """Eq. 9's T on the discretised operands: (dAm, dBum), each [B, K, N, L]."""
        arrs, (B, K, D, N, L) = self._disc_args(u, delta, A, Bs, bias)
        dAm = np.empty((B, K, N, L), dtype=np.float64)
        dBum = np.empty_like(dAm)
        self.lib.oracle_discretise_mean(*(_ptr(a) for a in arrs), _ptr(dAm), _ptr(dBum), B, K, D, N, L,
                                        int(bool(softplus_on)), int(b_mode))
        return dAm, dBum

    def scan_only(self, dA, dBu, Cs) -> np.ndarray:
        """The scan alone (Eq. 3 without the skip) on discretised operands.

        dA, dBu [B, K, Dm, N, L] (or [B, K, N, L] for one channel), Cs [B, K, N, L]
        -> y [B, K, Dm, L] (or [B, K, L])."""
        dA, dBu, Cs = _f64(dA), _f64(dBu), _f64(Cs)
        squeeze = dA.ndim == 4
        if squeeze:
            dA, dBu = dA[:, :, None], dBu[:, :, None]
        B, K, Dm, N, L = dA.shape
        if dBu.shape != dA.shape or Cs.shape != (B, K, N, L):
            raise ValueError("shape mismatch")
        dA, dBu = np.ascontiguousarray(dA), np.ascontiguousarray(dBu)
        y = np.empty((B, K, Dm, L), dtype=np.float64)
        self.lib.oracle_scan_only(_ptr(dA), _ptr(dBu), _ptr(Cs), _ptr(y), B, K, Dm, N, L)
        return y[:, :, 0] if squeeze else y

    def ss2d_full(self, inp, **kw):
        """Cross-scan, full scan, cross-merge on one `workloads.Inputs` set."""
        wl = inp.wl
        u = self.cross_scan(inp.x)
        y = self.selective_scan(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias, **kw)
        return u, y, self.cross_merge(y, wl.H, wl.W)

    def ss2d_mean(self, inp, **kw):
        """Cross-scan, channel-mean scan, cross-merge on one `workloads.Inputs` set."""
        wl = inp.wl
        u = self.cross_scan(inp.x)
        y, ybar = self.mean_scan(u, inp.draw, inp.A, inp.Bs, inp.Cs, inp.Dskip, inp.bias, **kw)
        return u, y, ybar, self.cross_merge(y, wl.H, wl.W)


_default = None
_lock = threading.Lock()


def get() -> Oracle:
    """The oracle compiled from oracle.c (built on first use)."""
    global _default
    with _lock:
        if _default is None:
            _default = Oracle(build())
    return _default


def cross_scan(x):
    return get().cross_scan(x)


def cross_merge(ys, H, W):
    return get().cross_merge(ys, H, W)


def softplus(x):
    return get().softplus(x)


def selective_scan(*a, **kw):
    return get().selective_scan(*a, **kw)


def mean_scan(*a, **kw):
    return get().mean_scan(*a, **kw)


def selection(*a, **kw):
    return get().selection(*a, **kw)


def mean_scan_grouped(*a, **kw):
    return get().mean_scan_grouped(*a, **kw)


def discretise(*a, **kw):
    return get().discretise(*a, **kw)


def discretise_mean(*a, **kw):
    return get().discretise_mean(*a, **kw)


def mean_scan_bwd(*a, **kw):
    return get().mean_scan_bwd(*a, **kw)


def scan_only(*a, **kw):
    return get().scan_only(*a, **kw)


def ss2d_full(inp, **kw):
    return get().ss2d_full(inp, **kw)


def ss2d_mean(inp, **kw):
    return get().ss2d_mean(inp, **kw)
