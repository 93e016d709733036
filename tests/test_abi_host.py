"""The C ABI without a GPU: the library loads, exports what include/vmb.h
declares, and rejects invalid arguments before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "vmb.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2412_16602_gb300 import _build
    path = _build.build()
    lib = ctypes.CDLL(path)
    vp, i, u, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint, ctypes.c_size_t
    lib.vmb_cross_scan.argtypes = [vp, vp, i, i, i, i, i, vp]
    lib.vmb_cross_merge.argtypes = [vp, vp, i, i, i, i, i, vp]
    lib.vmb_scan_workspace_bytes.argtypes = [i] * 8
    lib.vmb_scan_workspace_bytes.restype = sz
    lib.vmb_scan_kernel_count.argtypes = [i] * 8
    lib.vmb_scan_kernel_count.restype = i
    lib.vmb_selective_scan_fwd.argtypes = [vp] * 8 + [i] * 6 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_fwd.argtypes = [vp] * 9 + [i] * 6 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_merge_fwd.argtypes = [vp] * 10 + [i] * 5 + [u, i, vp, sz, vp]
    lib.vmb_ss2d_mean_fwd.argtypes = [vp] * 10 + [i] * 5 + [u, i, vp, sz, vp]
    lib.vmb_ss2d_full_fwd.argtypes = [vp] * 10 + [i] * 5 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_grouped_fwd.argtypes = [vp] * 9 + [i] * 7 + [u, i, vp, sz, vp]
    lib.vmb_discretise_fwd.argtypes = [vp] * 7 + [i] * 6 + [u, i, vp]
    lib.vmb_discretise_mean_fwd.argtypes = [vp] * 7 + [i] * 6 + [u, i, vp]
    lib.vmb_scan_only_fwd.argtypes = [vp] * 4 + [i] * 6 + [i, vp]
    lib.vmb_selection_fwd.argtypes = [vp] * 8 + [i] * 7 + [i, vp]
    lib.vmb_selection_lowrank_fwd.argtypes = [vp] * 7 + [i] * 7 + [i, vp]
    lib.vmb_selective_scan_lowrank_fwd.argtypes = [vp] * 9 + [i] * 7 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_lowrank_fwd.argtypes = [vp] * 10 + [i] * 7 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_bwd.argtypes = [vp] * 16 + [i] * 7 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_train_fwd.argtypes = [vp] * 10 + [i] * 7 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_bwd_workspace_bytes.argtypes = [i] * 8
    lib.vmb_mean_scan_bwd_workspace_bytes.restype = sz
    lib.vmb_status_string.argtypes = [i]
    lib.vmb_status_string.restype = ctypes.c_char_p
    lib.vmb_read_status.argtypes = [vp, vp]
    return lib


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(vmb_[a-z_]+)\s*\(", text)))


def test_header_declares_the_four_calls():
    names = declared_functions()
    for n in ["vmb_cross_scan", "vmb_selective_scan_fwd", "vmb_mean_scan_fwd", "vmb_cross_merge"]:
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} declared in vmb.h but not exported"


def test_status_strings(lib):
    for s in range(8):
        assert lib.vmb_status_string(s)
    assert lib.vmb_status_string(99) == b"unknown status"
    assert lib.vmb_version() >= 100


FAKE = 0x10000  # never dereferenced: validation fails before any device access
S = 0  # null stream


def scan_call(lib, fn, *, ptrs=None, B=1, K=4, D=8, N=16, H=4, W=4, flags=1, dtype=0,
              ws=0x100000, ws_bytes=1 << 20, mean=False):
    p = [FAKE] * 8 if ptrs is None else ptrs
    if mean:
        return fn(*p[:8], 0, B, K, D, N, H, W, flags, dtype, ws, ws_bytes, S)
    return fn(*p[:8], B, K, D, N, H, W, flags, dtype, ws, ws_bytes, S)


def test_cross_scan_validation(lib):
    assert lib.vmb_cross_scan(FAKE, FAKE, -1, 4, 4, 4, 0, S) == 1        # negative size
    assert lib.vmb_cross_scan(0, FAKE, 1, 4, 4, 4, 0, S) == 1            # null input
    assert lib.vmb_cross_scan(FAKE, FAKE, 1, 4, 4, 4, 7, S) == 1         # bad dtype
    assert lib.vmb_cross_scan(FAKE + 2, FAKE, 1, 4, 4, 4, 0, S) == 2     # fp32 misaligned
    assert lib.vmb_cross_scan(FAKE + 2, FAKE, 1, 4, 4, 4, 1, S) != 2     # bf16: 2-byte aligned is fine
    assert lib.vmb_cross_scan(0, 0, 0, 4, 4, 4, 0, S) == 0               # empty problem: no launch
    assert lib.vmb_cross_merge(FAKE, 0, 1, 4, 4, 4, 0, S) == 1
    assert lib.vmb_cross_merge(0, 0, 2, 3, 0, 5, 0, S) == 0


@pytest.mark.parametrize("mean", [False, True])
def test_scan_validation(lib, mean):
    fn = lib.vmb_mean_scan_fwd if mean else lib.vmb_selective_scan_fwd
    assert scan_call(lib, fn, B=-1, mean=mean) == 1
    assert scan_call(lib, fn, N=0, mean=mean) == 1
    assert scan_call(lib, fn, N=17, mean=mean) == 3                      # unsupported state size
    assert scan_call(lib, fn, flags=0x100, mean=mean) == 1               # unknown flag
    assert scan_call(lib, fn, dtype=5, mean=mean) == 1
    assert scan_call(lib, fn, ptrs=[FAKE] * 7 + [0], mean=mean) == 1     # null output
    assert scan_call(lib, fn, ptrs=[FAKE + 2] + [FAKE] * 7, mean=mean) == 2  # misaligned fp32
    assert scan_call(lib, fn, ws=0, mean=mean) == 4                      # no workspace
    assert scan_call(lib, fn, ws=FAKE + 16, mean=mean) == 2              # workspace not 256-B aligned
    assert scan_call(lib, fn, ptrs=[0] * 8, B=0, ws=0, mean=mean) == 0   # empty problem
    assert scan_call(lib, fn, ptrs=[0] * 8, H=0, ws=0, mean=mean) == 0


def test_skip_mean_flag_is_mean_only(lib):
    assert scan_call(lib, lib.vmb_selective_scan_fwd, flags=0x5) == 1


def test_workspace_query_invalid_and_empty(lib):
    assert lib.vmb_scan_workspace_bytes(7, 1, 4, 8, 16, 4, 4, 0) == 0
    assert lib.vmb_scan_workspace_bytes(0, 1, 4, 8, 17, 4, 4, 0) == 0
    assert lib.vmb_scan_workspace_bytes(0, -1, 4, 8, 16, 4, 4, 0) == 0
    assert lib.vmb_scan_workspace_bytes(1, 0, 4, 8, 16, 4, 4, 0) == 256


def test_kernel_count_invalid_and_empty(lib):
    assert lib.vmb_scan_kernel_count(7, 1, 4, 8, 16, 4, 4, 0) == 0
    assert lib.vmb_scan_kernel_count(0, 1, 4, 8, 17, 4, 4, 0) == 0
    assert lib.vmb_scan_kernel_count(1, 0, 4, 8, 16, 4, 4, 0) == 0


def test_read_status_rejects_null(lib):
    assert lib.vmb_read_status(0, 0) == 1
    assert lib.vmb_read_status(FAKE + 8, 0) == 2


def merge_call(lib, *, ptrs=None, B=1, D=8, N=16, H=4, W=4, flags=1, dtype=0, ws=0x100000, ws_bytes=1 << 20):
    p = [FAKE] * 7 + [FAKE, FAKE + 0x1000, FAKE + 0x2000] if ptrs is None else ptrs
    return lib.vmb_mean_scan_merge_fwd(*p, B, D, N, H, W, flags, dtype, ws, ws_bytes, S)


def test_mean_scan_merge_validation(lib):
    base = [FAKE] * 7 + [FAKE, FAKE + 0x1000, FAKE + 0x2000]
    assert merge_call(lib, B=-1) == 1
    assert merge_call(lib, ptrs=base[:7] + [0] + base[8:]) == 1                # null x
    assert merge_call(lib, ptrs=base[:8] + [FAKE] + base[9:]) == 1             # out aliases x
    assert merge_call(lib, ptrs=base[:9] + [0]) == 1                           # ybar is required
    assert merge_call(lib, ptrs=base[:7] + [FAKE + 2] + base[8:]) == 2         # misaligned fp32 map
    assert merge_call(lib, N=17) == 3
    assert merge_call(lib, flags=0x100) == 1
    assert merge_call(lib, ws=0) == 4
    assert merge_call(lib, ptrs=[0] * 10, B=0, ws=0) == 0                      # empty problem


def ss2d_call(lib, *, ptrs=None, B=1, D=8, N=16, H=4, W=4, flags=1, dtype=0, ws=0x100000, ws_bytes=1 << 20):
    p = [FAKE, FAKE + 0x3000] + [FAKE] * 6 + [FAKE + 0x1000, FAKE + 0x2000] if ptrs is None else ptrs
    return lib.vmb_ss2d_mean_fwd(*p, B, D, N, H, W, flags, dtype, ws, ws_bytes, S)


def test_ss2d_mean_validation(lib):
    """The scan side of the block from the map: x, xt, out and ybar are checked
    like the fused merge's, the scan inputs like the mean scan's, all before
    any launch."""
    base = [FAKE, FAKE + 0x3000] + [FAKE] * 6 + [FAKE + 0x1000, FAKE + 0x2000]
    assert ss2d_call(lib, B=-1) == 1
    assert ss2d_call(lib, ptrs=[0] + base[1:]) == 1                            # null map
    assert ss2d_call(lib, ptrs=base[:1] + [0] + base[2:]) == 1                 # null transpose scratch
    assert ss2d_call(lib, ptrs=base[:1] + [FAKE] + base[2:]) == 1              # transpose aliases x
    assert ss2d_call(lib, ptrs=base[:8] + [FAKE] + base[9:]) == 1              # out aliases x
    assert ss2d_call(lib, ptrs=base[:9] + [0]) == 1                            # ybar is required
    assert ss2d_call(lib, ptrs=[FAKE + 2] + base[1:]) == 2                     # misaligned fp32 map
    assert ss2d_call(lib, ptrs=base[:1] + [FAKE + 0x3002] + base[2:]) == 2     # misaligned transpose
    assert ss2d_call(lib, N=17) == 3
    assert ss2d_call(lib, flags=0x100) == 1
    assert ss2d_call(lib, ws=0) == 4
    assert ss2d_call(lib, ptrs=[0] * 10, B=0, ws=0) == 0                       # empty problem


def ss2d_full_call(lib, *, ptrs=None, B=1, D=8, N=16, H=4, W=4, flags=1, dtype=0, ws=0x100000, ws_bytes=1 << 20):
    p = [FAKE, FAKE + 0x3000] + [FAKE] * 6 + [FAKE + 0x4000, FAKE + 0x1000] if ptrs is None else ptrs
    return lib.vmb_ss2d_full_fwd(*p, B, D, N, H, W, flags, dtype, ws, ws_bytes, S)


def test_ss2d_full_validation(lib):
    """The full-channel scan side of the block from the map: x, xt, y and out
    must be distinct and aligned, the scan inputs are checked like the full
    scan's, all before any launch."""
    base = [FAKE, FAKE + 0x3000] + [FAKE] * 6 + [FAKE + 0x4000, FAKE + 0x1000]
    assert ss2d_full_call(lib, B=-1) == 1
    assert ss2d_full_call(lib, ptrs=[0] + base[1:]) == 1                       # null map
    assert ss2d_full_call(lib, ptrs=base[:1] + [0] + base[2:]) == 1            # null transpose scratch
    assert ss2d_full_call(lib, ptrs=base[:8] + [0] + base[9:]) == 1            # null y
    assert ss2d_full_call(lib, ptrs=base[:1] + [FAKE] + base[2:]) == 1         # transpose aliases x
    assert ss2d_full_call(lib, ptrs=base[:8] + [FAKE + 0x1000] + base[9:]) == 1  # y aliases out
    assert ss2d_full_call(lib, ptrs=base[:9] + [FAKE]) == 1                    # out aliases x
    assert ss2d_full_call(lib, ptrs=[FAKE + 2] + base[1:]) == 2                # misaligned fp32 map
    assert ss2d_full_call(lib, ptrs=base[:1] + [FAKE + 0x3002] + base[2:]) == 2  # misaligned transpose
    assert ss2d_full_call(lib, N=17) == 3
    assert ss2d_full_call(lib, flags=0x100) == 1
    assert ss2d_full_call(lib, ws=0) == 4
    assert ss2d_full_call(lib, ptrs=[0] * 10, B=0, ws=0) == 0                  # empty problem


def sel_lr_call(lib, *, ptrs=None, B=1, K=4, D=8, N=16, R=6, H=4, W=4, dtype=0):
    p = [FAKE] * 4 + [FAKE + 0x1000, FAKE + 0x2000, FAKE + 0x3000] if ptrs is None else ptrs
    return lib.vmb_selection_lowrank_fwd(*p, B, K, D, N, R, H, W, dtype, S)


def test_selection_lowrank_validation(lib):
    base = [FAKE] * 4 + [FAKE + 0x1000, FAKE + 0x2000, FAKE + 0x3000]
    assert sel_lr_call(lib, B=-1) == 1
    assert sel_lr_call(lib, N=0) == 1
    assert sel_lr_call(lib, R=0) == 1
    assert sel_lr_call(lib, R=17) == 3
    assert sel_lr_call(lib, ptrs=base[:6] + [0]) == 1                          # null z
    assert sel_lr_call(lib, ptrs=base[:6] + [FAKE + 0x3002]) == 2              # misaligned z (fp32)
    assert sel_lr_call(lib, dtype=5) == 1
    assert sel_lr_call(lib, ptrs=[0] * 7, B=0) == 0                            # empty problem


def scan_lr_call(lib, *, ptrs=None, B=1, K=4, D=8, N=16, R=6, H=4, W=4, flags=1, dtype=0, ws=0x100000,
                 ws_bytes=1 << 20):
    p = [FAKE, FAKE + 0x1000] + [FAKE] * 6 + [FAKE + 0x2000] if ptrs is None else ptrs
    return lib.vmb_selective_scan_lowrank_fwd(*p, B, K, D, N, R, H, W, flags, dtype, ws, ws_bytes, S)


def test_selective_scan_lowrank_validation(lib):
    """Rank, the low-rank operands and the usual scan arguments are checked
    before any launch."""
    base = [FAKE, FAKE + 0x1000] + [FAKE] * 6 + [FAKE + 0x2000]
    assert scan_lr_call(lib, B=-1) == 1
    assert scan_lr_call(lib, R=-1) == 1
    assert scan_lr_call(lib, R=0) == 1
    assert scan_lr_call(lib, R=17) == 3
    assert scan_lr_call(lib, N=17) == 3
    assert scan_lr_call(lib, ptrs=base[:2] + [0] + base[3:]) == 1              # null Wup
    assert scan_lr_call(lib, ptrs=base[:1] + [0] + base[2:]) == 1              # null z
    assert scan_lr_call(lib, ptrs=base[:1] + [FAKE + 0x1002] + base[2:]) == 2  # misaligned z
    assert scan_lr_call(lib, ptrs=base[:8] + [FAKE]) == 1                      # y aliases u
    assert scan_lr_call(lib, flags=0x100) == 1
    assert scan_lr_call(lib, ws=0) == 4
    assert scan_lr_call(lib, ptrs=[0] * 9, B=0, ws=0) == 0                     # empty problem


def test_mean_scan_lowrank_validation(lib):
    base = [FAKE, FAKE + 0x1000] + [FAKE] * 6 + [FAKE + 0x2000, 0]

    def call(ptrs=base, R=6, N=16, flags=1, ws=0x100000, B=1):
        return lib.vmb_mean_scan_lowrank_fwd(*ptrs, B, 4, 8, N, R, 4, 4, flags, 0, ws, 1 << 20, S)
    assert call(B=-1) == 1
    assert call(R=0) == 1
    assert call(R=17) == 3
    assert call(N=17) == 3
    assert call(ptrs=base[:2] + [0] + base[3:]) == 1                  # null Wup
    assert call(ptrs=base[:1] + [FAKE + 0x1002] + base[2:]) == 2      # misaligned z
    assert call(ptrs=base[:8] + [FAKE, 0]) == 1                       # y aliases u
    assert call(flags=0x100) == 1
    assert call(ws=0) == 4
    assert call(ptrs=[0] * 10, B=0, ws=0) == 0                        # empty problem


def disc_call(fn, *, ptrs=None, B=1, K=4, D=8, N=16, H=4, W=4, flags=1, dtype=0):
    p = [FAKE] * 7 if ptrs is None else ptrs
    return fn(*p, B, K, D, N, H, W, flags, dtype, S)


@pytest.mark.parametrize("mean", [False, True])
def test_discretise_validation(lib, mean):
    fn = lib.vmb_discretise_mean_fwd if mean else lib.vmb_discretise_fwd
    assert disc_call(fn, B=-1) == 1
    assert disc_call(fn, N=0) == 1
    assert disc_call(fn, N=17) == 3
    assert disc_call(fn, flags=0x4) == 1                                 # skip-mode flag: not a discretisation flag
    assert disc_call(fn, dtype=3) == 1
    assert disc_call(fn, ptrs=[FAKE] * 6 + [0]) == 1                     # null output
    assert disc_call(fn, ptrs=[FAKE] * 5 + [FAKE + 2, FAKE]) == 2        # misaligned fp32 output
    assert disc_call(fn, ptrs=[FAKE + 2] + [FAKE] * 6, dtype=1) != 2     # bf16 input: 2-byte aligned is fine
    assert disc_call(fn, ptrs=[0] * 7, W=0) == 0                         # empty problem


def test_scan_only_validation(lib):
    f = lib.vmb_scan_only_fwd
    assert f(FAKE, FAKE, FAKE, FAKE, -1, 4, 8, 16, 4, 4, 0, S) == 1
    assert f(FAKE, FAKE, FAKE, FAKE, 1, 4, 8, 0, 4, 4, 0, S) == 1
    assert f(FAKE, FAKE, FAKE, FAKE, 1, 4, 8, 17, 4, 4, 0, S) == 3
    assert f(FAKE, FAKE, FAKE, 0, 1, 4, 8, 16, 4, 4, 0, S) == 1          # null y
    assert f(FAKE, FAKE + 2, FAKE, FAKE, 1, 4, 8, 16, 4, 4, 0, S) == 2   # misaligned dBu
    assert f(FAKE, FAKE, FAKE + 1, FAKE, 1, 4, 8, 16, 4, 4, 1, S) == 2   # misaligned bf16 C
    assert f(FAKE, FAKE, FAKE, FAKE, 1, 4, 8, 16, 4, 4, 9, S) == 1       # bad dtype
    assert f(0, 0, 0, 0, 1, 4, 0, 16, 4, 4, 0, S) == 0                   # empty problem


def test_grouped_validation(lib):
    f = lib.vmb_mean_scan_grouped_fwd

    def call(groups, D=8, ptrs=None, ws=0x100000):
        p = [FAKE] * 9 if ptrs is None else ptrs
        return f(*p, 1, 4, D, 16, 4, 4, groups, 1, 0, ws, 1 << 20, S)
    assert call(0) == 1                  # no groups
    assert call(3) == 1                  # does not divide D
    assert call(2, ptrs=[FAKE] * 7 + [0, FAKE]) == 1   # null y
    assert call(2, ws=0) == 4
    assert call(4, D=0, ptrs=[0] * 9, ws=0) == 0        # empty problem


def test_mean_scan_rejects_slabs_beyond_32bit_offsets(lib):
    # D * L >= 2^31: a (b, k) slab no longer fits the mean kernel's 32-bit offsets
    D, H, W = 65536, 182, 182
    assert scan_call(lib, lib.vmb_mean_scan_fwd, D=D, H=H, W=W, mean=True) == 3
    assert lib.vmb_scan_workspace_bytes(1, 1, 4, D, 16, H, W, 0) == 0
    assert scan_call(lib, lib.vmb_mean_scan_fwd, D=D // 2, H=H, W=W, ws=0, mean=True) == 4  # below the limit


def test_selection_validation(lib):
    f = lib.vmb_selection_fwd

    def call(ptrs=None, B=1, K=4, D=8, N=16, R=6, H=4, W=4, dtype=0):
        p = [FAKE] * 8 if ptrs is None else ptrs
        return f(*p, B, K, D, N, R, H, W, dtype, S)
    assert call(B=-1) == 1
    assert call(N=0) == 1
    assert call(R=0) == 1
    assert call(N=17) == 3
    assert call(R=17) == 3
    assert call(dtype=4) == 1
    assert call(ptrs=[FAKE] * 7 + [0]) == 1                 # null delta_raw
    assert call(ptrs=[FAKE + 2] + [FAKE] * 7) == 2          # misaligned fp32 input
    assert call(ptrs=[FAKE, FAKE + 2] + [FAKE] * 6) == 2    # misaligned weights
    assert call(ptrs=[0] * 8, D=0) == 0                     # empty problem


def bwd_call(lib, *, ptrs=None, B=1, K=4, D=8, N=16, H=4, W=4, groups=1, flags=1, dtype=0, ws=0x100000,
             ws_bytes=1 << 30):
    p = [FAKE] * 16 if ptrs is None else ptrs
    return lib.vmb_mean_scan_bwd(*p, B, K, D, N, H, W, groups, flags, dtype, ws, ws_bytes, S)


def test_mean_backward_validation(lib):
    """The backward rejects invalid arguments and the flags it does not
    implement before any launch."""
    assert bwd_call(lib, B=-1) == 1
    assert bwd_call(lib, ptrs=[FAKE] * 15 + [0]) == 1                # a null gradient output
    assert bwd_call(lib, ptrs=[FAKE + 2] + [FAKE] * 15) == 2         # misaligned fp32 input
    assert bwd_call(lib, ptrs=[FAKE] * 8 + [FAKE + 2] + [FAKE] * 7) == 2  # misaligned saved means
    assert bwd_call(lib, groups=3) == 1                              # groups must divide D
    assert bwd_call(lib, groups=0) == 1
    assert bwd_call(lib, N=17) == 3
    assert bwd_call(lib, flags=1 | 2) == 3                           # zero-order hold: not implemented
    assert bwd_call(lib, flags=1 | 4) == 3                           # mean skip term: not implemented
    assert bwd_call(lib, flags=0x100) == 1
    assert bwd_call(lib, ws=0) == 4
    assert bwd_call(lib, ws_bytes=256) == 4
    assert bwd_call(lib, ptrs=[0] * 16, B=0, ws=0) == 0             # empty problem
    assert lib.vmb_mean_scan_bwd_workspace_bytes(1, 4, 8, 16, 4, 4, 3, 0) == 0
    assert lib.vmb_mean_scan_bwd_workspace_bytes(0, 4, 8, 16, 4, 4, 1, 0) == 256
    assert lib.vmb_mean_scan_bwd_workspace_bytes(2, 4, 8, 16, 4, 4, 2, 0) > 256


def test_train_forward_validation(lib):
    """The training forward (mean scan keeping its group means) rejects a
    missing or misaligned buffer and the forms the backward does not cover."""
    def call(ptrs=None, B=1, K=4, D=8, N=16, H=4, W=4, groups=1, flags=1, dtype=0):
        p = [FAKE] * 10 if ptrs is None else ptrs
        return lib.vmb_mean_scan_train_fwd(*p, B, K, D, N, H, W, groups, flags, dtype, 0x100000, 1 << 30, S)
    assert call(ptrs=[FAKE] * 9 + [0]) == 1          # no buffer for the means
    assert call(ptrs=[FAKE] * 9 + [FAKE + 2]) == 2   # misaligned means
    assert call(flags=1 | 2) == 3                    # zero-order hold: the backward does not cover it
    assert call(flags=1 | 4) == 3                    # mean skip term: likewise
    assert call(groups=3) == 1                       # groups must divide D
    assert call(B=0, ptrs=[0] * 10) == 0             # empty problem
