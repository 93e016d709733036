"""Python binding of libvmb (include/vmb.h): argument marshalling only.

Every function has the name of the C entry point it calls and takes torch
CUDA tensors; it checks shapes and dtypes, allocates outputs with torch when
none are given, and passes raw device pointers plus the current CUDA stream
to the library.  All arithmetic runs in the library's kernels: there is no
fallback, and a missing library raises at import.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libvmb.so")

VMB_OK = 0
VMB_ERR_INVALID_ARG = 1
VMB_ERR_MISALIGNED = 2
VMB_ERR_UNSUPPORTED = 3
VMB_ERR_WORKSPACE = 4
VMB_ERR_CUDA = 5
VMB_ERR_TIMEOUT = 6
VMB_ERR_BOUNDS = 7

VMB_F32 = 0
VMB_BF16 = 1

VMB_FLAG_SOFTPLUS = 0x1
VMB_FLAG_B_ZOH = 0x2
VMB_FLAG_SKIP_MEAN = 0x4
VMB_FLAG_TEST_SUPPRESS_PUBLISH = 0x40000000

VMB_PATH_FULL = 0
VMB_PATH_MEAN = 1

EXPORTS = ["vmb_cross_scan", "vmb_cross_merge", "vmb_scan_workspace_bytes", "vmb_scan_kernel_count",
           "vmb_selective_scan_fwd",
           "vmb_mean_scan_fwd", "vmb_mean_scan_merge_fwd", "vmb_mean_scan_grouped_fwd", "vmb_ss2d_mean_fwd",
           "vmb_ss2d_full_fwd", "vmb_discretise_fwd", "vmb_discretise_mean_fwd",
           "vmb_scan_only_fwd", "vmb_selection_fwd", "vmb_selection_lowrank_fwd", "vmb_selective_scan_lowrank_fwd",
           "vmb_mean_scan_lowrank_fwd", "vmb_mean_scan_train_fwd", "vmb_mean_scan_bwd",
           "vmb_mean_scan_bwd_workspace_bytes",
           "vmb_read_status", "vmb_status_string", "vmb_version"]


class VmbError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built: run `python -c \"import __graft_entry__ as g; g.build()\"`")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i, u, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint, ctypes.c_size_t
    lib.vmb_cross_scan.argtypes = [vp, vp, i, i, i, i, i, vp]
    lib.vmb_cross_merge.argtypes = [vp, vp, i, i, i, i, i, vp]
    lib.vmb_scan_workspace_bytes.argtypes = [i, i, i, i, i, i, i, i]
    lib.vmb_scan_workspace_bytes.restype = sz
    lib.vmb_scan_kernel_count.argtypes = [i, i, i, i, i, i, i, i]
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
    lib.vmb_mean_scan_train_fwd.argtypes = [vp] * 10 + [i] * 7 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_bwd.argtypes = [vp] * 16 + [i] * 7 + [u, i, vp, sz, vp]
    lib.vmb_mean_scan_bwd_workspace_bytes.argtypes = [i] * 8
    lib.vmb_mean_scan_bwd_workspace_bytes.restype = sz
    lib.vmb_read_status.argtypes = [vp, vp]
    lib.vmb_status_string.argtypes = [i]
    lib.vmb_status_string.restype = ctypes.c_char_p
    lib.vmb_version.argtypes = []
    for name in ["vmb_cross_scan", "vmb_cross_merge", "vmb_selective_scan_fwd", "vmb_mean_scan_fwd",
                 "vmb_mean_scan_merge_fwd", "vmb_mean_scan_grouped_fwd", "vmb_ss2d_mean_fwd", "vmb_ss2d_full_fwd",
                 "vmb_discretise_fwd",
                 "vmb_discretise_mean_fwd", "vmb_scan_only_fwd", "vmb_selection_fwd", "vmb_mean_scan_bwd",
                 "vmb_selection_lowrank_fwd", "vmb_selective_scan_lowrank_fwd", "vmb_mean_scan_lowrank_fwd",
                 "vmb_read_status", "vmb_version"]:
        getattr(lib, name).restype = i
    return lib


lib = _load()


def status_string(status: int) -> str:
    return lib.vmb_status_string(int(status)).decode()


def vmb_status_string(status: int) -> str:
    return status_string(status)


def vmb_version() -> int:
    return lib.vmb_version()


def _check(status: int, where: str):
    if status != VMB_OK:
        raise VmbError(status, where)


def _dtype_code(t: torch.dtype) -> int:
    if t == torch.float32:
        return VMB_F32
    if t == torch.bfloat16:
        return VMB_BF16
    raise TypeError(f"unsupported dtype {t} (float32 or bfloat16)")


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)


def _dev(t: torch.Tensor, name: str):
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


# ---------------------------------------------------------------- cross-scan / merge


def vmb_cross_scan(x: torch.Tensor, xs: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """x [B, D, H, W] -> xs [B, 4, D, H*W] (bit-exact permutation)."""
    _dev(x, "x")
    B, D, H, W = x.shape
    if xs is None:
        xs = torch.empty((B, 4, D, H * W), dtype=x.dtype, device=x.device)
    _dev(xs, "xs")
    if xs.shape != (B, 4, D, H * W) or xs.dtype != x.dtype:
        raise ValueError("xs must be [B, 4, D, H*W] with the dtype of x")
    _check(lib.vmb_cross_scan(_ptr(x), _ptr(xs), B, D, H, W, _dtype_code(x.dtype), _stream(stream)),
           "vmb_cross_scan")
    return xs


def vmb_cross_merge(ys: torch.Tensor, H: int, W: int, out: torch.Tensor | None = None,
                    stream=None) -> torch.Tensor:
    """ys [B, 4, D, H*W] -> out [B, D, H, W]."""
    _dev(ys, "ys")
    B, K, D, L = ys.shape
    if K != 4 or L != H * W:
        raise ValueError("ys must be [B, 4, D, H*W]")
    if out is None:
        out = torch.empty((B, D, H, W), dtype=ys.dtype, device=ys.device)
    _dev(out, "out")
    if out.shape != (B, D, H, W) or out.dtype != ys.dtype:
        raise ValueError("out must be [B, D, H, W] with the dtype of ys")
    _check(lib.vmb_cross_merge(_ptr(ys), _ptr(out), B, D, H, W, _dtype_code(ys.dtype), _stream(stream)),
           "vmb_cross_merge")
    return out


# ---------------------------------------------------------------- scans


def vmb_scan_workspace_bytes(path: int, B: int, K: int, D: int, N: int, H: int, W: int,
                             dtype: torch.dtype = torch.float32) -> int:
    return int(lib.vmb_scan_workspace_bytes(path, B, K, D, N, H, W, _dtype_code(dtype)))


def vmb_scan_kernel_count(path: int, B: int, K: int, D: int, N: int, H: int, W: int,
                          dtype: torch.dtype = torch.float32) -> int:
    return int(lib.vmb_scan_kernel_count(path, B, K, D, N, H, W, _dtype_code(dtype)))


class Workspace:
    """A zero-initialised device workspace that grows on demand (one per device).

    The library keeps a workspace ready for the next call by itself; only a
    newly allocated buffer needs zero-filling, which torch.zeros does."""

    def __init__(self):
        self._bufs = {}
        self._lock = threading.Lock()

    def get(self, nbytes: int, device: torch.device) -> torch.Tensor:
        key = (device.type, device.index)
        with self._lock:
            buf = self._bufs.get(key)
            if buf is None or buf.numel() < nbytes:
                n = max(nbytes, 256)
                n = (n + 255) // 256 * 256
                buf = torch.zeros(n, dtype=torch.uint8, device=device)
                self._bufs[key] = buf
            return buf


_default_ws = Workspace()


def _scan_shapes(u, delta, A, Bs, Cs, Dskip, delta_bias, H, W):
    for t, n in [(u, "u"), (delta, "delta"), (A, "A"), (Bs, "Bs"), (Cs, "Cs"), (Dskip, "Dskip"),
                 (delta_bias, "delta_bias")]:
        _dev(t, n)
    B, K, D, L = u.shape
    N = Bs.shape[2]
    if L != H * W:
        raise ValueError("u must be [B, K, D, H*W]")
    if delta.shape != u.shape or Bs.shape != (B, K, N, L) or Cs.shape != (B, K, N, L):
        raise ValueError("delta [B,K,D,L], Bs and Cs [B,K,N,L] expected")
    if len({u.dtype, delta.dtype, Bs.dtype, Cs.dtype}) != 1:
        raise ValueError("u, delta, Bs, Cs must share one dtype")
    if A.shape != (K * D, N) or Dskip.shape != (K * D,) or delta_bias.shape != (K * D,):
        raise ValueError("A [K*D, N], Dskip [K*D], delta_bias [K*D] expected")
    if A.dtype != torch.float32 or Dskip.dtype != torch.float32 or delta_bias.dtype != torch.float32:
        raise ValueError("A, Dskip, delta_bias must be float32")
    return B, K, D, N, L


def vmb_selective_scan_fwd(u, delta, A, Bs, Cs, Dskip, delta_bias, H: int, W: int, *,
                           y=None, flags: int = VMB_FLAG_SOFTPLUS, workspace=None,
                           stream=None) -> torch.Tensor:
    """Full-channel selective scan: y [B, K, D, H*W] (dtype of u)."""
    B, K, D, N, L = _scan_shapes(u, delta, A, Bs, Cs, Dskip, delta_bias, H, W)
    if y is None:
        y = torch.empty_like(u)
    _dev(y, "y")
    if y.shape != u.shape or y.dtype != u.dtype:
        raise ValueError("y must match u")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_FULL, B, K, D, N, H, W, u.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, u.device)
    _check(lib.vmb_selective_scan_fwd(_ptr(u), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                      _ptr(delta_bias), _ptr(y), B, K, D, N, H, W, flags,
                                      _dtype_code(u.dtype), _ptr(workspace), workspace.numel(),
                                      _stream(stream)), "vmb_selective_scan_fwd")
    return y


def vmb_mean_scan_fwd(u, delta, A, Bs, Cs, Dskip, delta_bias, H: int, W: int, *,
                      y=None, ybar=None, want_ybar: bool = False, flags: int = VMB_FLAG_SOFTPLUS,
                      workspace=None, stream=None):
    """VMeanba channel-mean scan: returns (y [B, K, D, L], ybar [B, K, L] fp32 or None)."""
    B, K, D, N, L = _scan_shapes(u, delta, A, Bs, Cs, Dskip, delta_bias, H, W)
    if y is None:
        y = torch.empty_like(u)
    _dev(y, "y")
    if y.shape != u.shape or y.dtype != u.dtype:
        raise ValueError("y must match u")
    if ybar is None and want_ybar:
        ybar = torch.empty((B, K, L), dtype=torch.float32, device=u.device)
    if ybar is not None:
        _dev(ybar, "ybar")
        if ybar.shape != (B, K, L) or ybar.dtype != torch.float32:
            raise ValueError("ybar must be float32 [B, K, L]")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_MEAN, B, K, D, N, H, W, u.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, u.device)
    _check(lib.vmb_mean_scan_fwd(_ptr(u), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                 _ptr(delta_bias), _ptr(y), _ptr(ybar), B, K, D, N, H, W, flags,
                                 _dtype_code(u.dtype), _ptr(workspace), workspace.numel(),
                                 _stream(stream)), "vmb_mean_scan_fwd")
    return y, ybar


def vmb_mean_scan_grouped_fwd(u, delta, A, Bs, Cs, Dskip, delta_bias, H: int, W: int, groups: int, *,
                              y=None, ybar=None, want_ybar: bool = False, flags: int = VMB_FLAG_SOFTPLUS,
                              workspace=None, stream=None):
    """Grouped basis (reduced channel dimension d = groups): the channel mean of Eq. 9 over each
    of `groups` channel groups; returns (y [B, K, D, L], ybar [B, K, groups, L] fp32 or None)."""
    B, K, D, N, L = _scan_shapes(u, delta, A, Bs, Cs, Dskip, delta_bias, H, W)
    if groups < 1 or D % groups:
        raise ValueError("groups must be >= 1 and divide D")
    if y is None:
        y = torch.empty_like(u)
    _dev(y, "y")
    if y.shape != u.shape or y.dtype != u.dtype:
        raise ValueError("y must match u")
    if ybar is None and want_ybar:
        ybar = torch.empty((B, K, groups, L), dtype=torch.float32, device=u.device)
    if ybar is not None:
        _dev(ybar, "ybar")
        if ybar.shape != (B, K, groups, L) or ybar.dtype != torch.float32:
            raise ValueError("ybar must be float32 [B, K, groups, L]")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_MEAN, B, K * groups, D // groups, N, H, W, u.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, u.device)
    _check(lib.vmb_mean_scan_grouped_fwd(_ptr(u), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                         _ptr(delta_bias), _ptr(y), _ptr(ybar), B, K, D, N, H, W, groups, flags,
                                         _dtype_code(u.dtype), _ptr(workspace), workspace.numel(),
                                         _stream(stream)), "vmb_mean_scan_grouped_fwd")
    return y, ybar


def vmb_mean_scan_train_fwd(u, delta, A, Bs, Cs, Dskip, delta_bias, H: int, W: int, *, groups: int = 1,
                            y=None, ybar=None, saved=None, flags: int = VMB_FLAG_SOFTPLUS, workspace=None,
                            stream=None):
    """The (grouped) channel-mean scan that also keeps its group means for the backward: returns
    (y [B, K, D, L], saved [B, K, groups, N + 1, L] fp32, ybar or None)."""
    B, K, D, N, L = _scan_shapes(u, delta, A, Bs, Cs, Dskip, delta_bias, H, W)
    if groups < 1 or D % groups:
        raise ValueError("groups must be >= 1 and divide D")
    if y is None:
        y = torch.empty_like(u)
    _dev(y, "y")
    if y.shape != u.shape or y.dtype != u.dtype:
        raise ValueError("y must match u")
    if saved is None:
        saved = torch.empty((B, K, groups, N + 1, L), dtype=torch.float32, device=u.device)
    _dev(saved, "saved")
    if tuple(saved.shape) != (B, K, groups, N + 1, L) or saved.dtype != torch.float32:
        raise ValueError("saved must be float32 [B, K, groups, N + 1, L]")
    if ybar is not None:
        _dev(ybar, "ybar")
        if ybar.shape != (B, K, groups, L) or ybar.dtype != torch.float32:
            raise ValueError("ybar must be float32 [B, K, groups, L]")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_MEAN, B, K * groups, D // groups, N, H, W, u.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, u.device)
    _check(lib.vmb_mean_scan_train_fwd(_ptr(u), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                       _ptr(delta_bias), _ptr(y), _ptr(ybar), _ptr(saved), B, K, D, N, H, W, groups,
                                       flags, _dtype_code(u.dtype), _ptr(workspace), workspace.numel(),
                                       _stream(stream)), "vmb_mean_scan_train_fwd")
    return y, saved, ybar


def vmb_mean_scan_merge_fwd(u, delta, A, Bs, Cs, Dskip, delta_bias, x, H: int, W: int, *,
                            out=None, ybar=None, flags: int = VMB_FLAG_SOFTPLUS, workspace=None, stream=None):
    """Channel-mean path with the broadcast fused into the cross-merge:
    returns (out [B, D, H, W], ybar [B, 4, L] fp32)."""
    B, K, D, N, L = _scan_shapes(u, delta, A, Bs, Cs, Dskip, delta_bias, H, W)
    if K != 4:
        raise ValueError("the fused merge needs the four SS2D directions (K = 4)")
    _dev(x, "x")
    if tuple(x.shape) != (B, D, H, W) or x.dtype != u.dtype:
        raise ValueError("x must be [B, D, H, W] in the storage dtype of u")
    if out is None:
        out = torch.empty_like(x)
    _dev(out, "out")
    if out.shape != x.shape or out.dtype != x.dtype:
        raise ValueError("out must match x")
    if ybar is None:
        ybar = torch.empty((B, 4, L), dtype=torch.float32, device=u.device)
    _dev(ybar, "ybar")
    if ybar.shape != (B, 4, L) or ybar.dtype != torch.float32:
        raise ValueError("ybar must be float32 [B, 4, L]")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_MEAN, B, 4, D, N, H, W, u.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, u.device)
    _check(lib.vmb_mean_scan_merge_fwd(_ptr(u), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                       _ptr(delta_bias), _ptr(x), _ptr(out), _ptr(ybar), B, D, N, H, W, flags,
                                       _dtype_code(u.dtype), _ptr(workspace), workspace.numel(),
                                       _stream(stream)), "vmb_mean_scan_merge_fwd")
    return out, ybar


def vmb_ss2d_mean_fwd(x, delta, A, Bs, Cs, Dskip, delta_bias, *, out=None, ybar=None, xt=None,
                      flags: int = VMB_FLAG_SOFTPLUS, workspace=None, stream=None):
    """The scan side of a VMeanba SS2D block from the map: cross-scan, channel-mean scan and
    cross-merge in one call, xs and y never written.  x [B, D, H, W]; delta [B, 4, D, H*W],
    Bs, Cs [B, 4, N, H*W]; xt [B, D, W, H] scratch for the map's transpose (allocated when not
    given); returns (out [B, D, H, W], ybar [B, 4, H*W] fp32)."""
    _dev(x, "x")
    B, D, H, W = x.shape
    if xt is None:
        xt = torch.empty((B, D, W, H), dtype=x.dtype, device=x.device)
    _dev(xt, "xt")
    if tuple(xt.shape) != (B, D, W, H) or xt.dtype != x.dtype:
        raise ValueError("xt must be [B, D, W, H] in the dtype of x")
    L = H * W
    for t, n in [(delta, "delta"), (A, "A"), (Bs, "Bs"), (Cs, "Cs"), (Dskip, "Dskip"), (delta_bias, "delta_bias")]:
        _dev(t, n)
    N = Bs.shape[2]
    if tuple(delta.shape) != (B, 4, D, L) or tuple(Bs.shape) != (B, 4, N, L) or tuple(Cs.shape) != (B, 4, N, L):
        raise ValueError("delta [B,4,D,H*W], Bs and Cs [B,4,N,H*W] expected")
    if len({x.dtype, delta.dtype, Bs.dtype, Cs.dtype}) != 1:
        raise ValueError("x, delta, Bs, Cs must share one dtype")
    if tuple(A.shape) != (4 * D, N) or tuple(Dskip.shape) != (4 * D,) or tuple(delta_bias.shape) != (4 * D,):
        raise ValueError("A [4*D, N], Dskip [4*D], delta_bias [4*D] expected")
    if A.dtype != torch.float32 or Dskip.dtype != torch.float32 or delta_bias.dtype != torch.float32:
        raise ValueError("A, Dskip, delta_bias must be float32")
    if out is None:
        out = torch.empty_like(x)
    _dev(out, "out")
    if out.shape != x.shape or out.dtype != x.dtype:
        raise ValueError("out must match x")
    if ybar is None:
        ybar = torch.empty((B, 4, L), dtype=torch.float32, device=x.device)
    _dev(ybar, "ybar")
    if tuple(ybar.shape) != (B, 4, L) or ybar.dtype != torch.float32:
        raise ValueError("ybar must be float32 [B, 4, L]")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_MEAN, B, 4, D, N, H, W, x.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, x.device)
    _check(lib.vmb_ss2d_mean_fwd(_ptr(x), _ptr(xt), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                 _ptr(delta_bias),
                                 _ptr(out), _ptr(ybar), B, D, N, H, W, flags, _dtype_code(x.dtype), _ptr(workspace),
                                 workspace.numel(), _stream(stream)), "vmb_ss2d_mean_fwd")
    return out, ybar


def vmb_ss2d_full_fwd(x, delta, A, Bs, Cs, Dskip, delta_bias, *, out=None, y=None, xt=None,
                      flags: int = VMB_FLAG_SOFTPLUS, workspace=None, stream=None):
    """The scan side of a full-channel SS2D block from the map: cross-scan, selective scan and
    cross-merge in one call, xs never written.  x [B, D, H, W]; delta [B, 4, D, H*W], Bs, Cs
    [B, 4, N, H*W]; xt [B, D, W, H] scratch for the map's transpose (allocated when not given);
    returns (out [B, D, H, W], y [B, 4, D, H*W])."""
    _dev(x, "x")
    B, D, H, W = x.shape
    if xt is None:
        xt = torch.empty((B, D, W, H), dtype=x.dtype, device=x.device)
    _dev(xt, "xt")
    if tuple(xt.shape) != (B, D, W, H) or xt.dtype != x.dtype:
        raise ValueError("xt must be [B, D, W, H] in the dtype of x")
    L = H * W
    for t, n in [(delta, "delta"), (A, "A"), (Bs, "Bs"), (Cs, "Cs"), (Dskip, "Dskip"), (delta_bias, "delta_bias")]:
        _dev(t, n)
    N = Bs.shape[2]
    if tuple(delta.shape) != (B, 4, D, L) or tuple(Bs.shape) != (B, 4, N, L) or tuple(Cs.shape) != (B, 4, N, L):
        raise ValueError("delta [B,4,D,H*W], Bs and Cs [B,4,N,H*W] expected")
    if len({x.dtype, delta.dtype, Bs.dtype, Cs.dtype}) != 1:
        raise ValueError("x, delta, Bs, Cs must share one dtype")
    if tuple(A.shape) != (4 * D, N) or tuple(Dskip.shape) != (4 * D,) or tuple(delta_bias.shape) != (4 * D,):
        raise ValueError("A [4*D, N], Dskip [4*D], delta_bias [4*D] expected")
    if A.dtype != torch.float32 or Dskip.dtype != torch.float32 or delta_bias.dtype != torch.float32:
        raise ValueError("A, Dskip, delta_bias must be float32")
    if out is None:
        out = torch.empty_like(x)
    _dev(out, "out")
    if out.shape != x.shape or out.dtype != x.dtype:
        raise ValueError("out must match x")
    if y is None:
        y = torch.empty((B, 4, D, L), dtype=x.dtype, device=x.device)
    _dev(y, "y")
    if tuple(y.shape) != (B, 4, D, L) or y.dtype != x.dtype:
        raise ValueError("y must be [B, 4, D, H*W] in the dtype of x")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_FULL, B, 4, D, N, H, W, x.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, x.device)
    _check(lib.vmb_ss2d_full_fwd(_ptr(x), _ptr(xt), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                 _ptr(delta_bias), _ptr(y), _ptr(out), B, D, N, H, W, flags, _dtype_code(x.dtype),
                                 _ptr(workspace), workspace.numel(), _stream(stream)), "vmb_ss2d_full_fwd")
    return out, y


# ------------------------------------------- the paper's scan-only kernel setting


def _disc_shapes(u, delta, A, Bs, delta_bias, H, W):
    for t, n in [(u, "u"), (delta, "delta"), (A, "A"), (Bs, "Bs"), (delta_bias, "delta_bias")]:
        _dev(t, n)
    B, K, D, L = u.shape
    N = Bs.shape[2]
    if L != H * W or delta.shape != u.shape or Bs.shape != (B, K, N, L):
        raise ValueError("u, delta [B,K,D,H*W] and Bs [B,K,N,H*W] expected")
    if len({u.dtype, delta.dtype, Bs.dtype}) != 1:
        raise ValueError("u, delta, Bs must share one dtype")
    if A.shape != (K * D, N) or delta_bias.shape != (K * D,) or A.dtype != torch.float32 \
            or delta_bias.dtype != torch.float32:
        raise ValueError("A [K*D, N], delta_bias [K*D] float32 expected")
    return B, K, D, N, L


def vmb_discretise_fwd(u, delta, A, Bs, delta_bias, H: int, W: int, *, dA=None, dBu=None,
                       flags: int = VMB_FLAG_SOFTPLUS, stream=None):
    """Eqs. 4, 6 outside the scan: (dA, dBu), each float32 [B, K, D, N, H*W]."""
    B, K, D, N, L = _disc_shapes(u, delta, A, Bs, delta_bias, H, W)
    shape = (B, K, D, N, L)
    dA = torch.empty(shape, dtype=torch.float32, device=u.device) if dA is None else dA
    dBu = torch.empty(shape, dtype=torch.float32, device=u.device) if dBu is None else dBu
    for t, n in [(dA, "dA"), (dBu, "dBu")]:
        _dev(t, n)
        if t.shape != shape or t.dtype != torch.float32:
            raise ValueError(f"{n} must be float32 {shape}")
    _check(lib.vmb_discretise_fwd(_ptr(u), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(delta_bias), _ptr(dA), _ptr(dBu),
                                  B, K, D, N, H, W, flags, _dtype_code(u.dtype), _stream(stream)),
           "vmb_discretise_fwd")
    return dA, dBu


def vmb_discretise_mean_fwd(u, delta, A, Bs, delta_bias, H: int, W: int, *, dAm=None, dBum=None,
                            flags: int = VMB_FLAG_SOFTPLUS, stream=None):
    """Channel means of the discretised operands (Eq. 9's T): (dAm, dBum), float32 [B, K, N, H*W]."""
    B, K, D, N, L = _disc_shapes(u, delta, A, Bs, delta_bias, H, W)
    shape = (B, K, N, L)
    dAm = torch.empty(shape, dtype=torch.float32, device=u.device) if dAm is None else dAm
    dBum = torch.empty(shape, dtype=torch.float32, device=u.device) if dBum is None else dBum
    for t, n in [(dAm, "dAm"), (dBum, "dBum")]:
        _dev(t, n)
        if t.shape != shape or t.dtype != torch.float32:
            raise ValueError(f"{n} must be float32 {shape}")
    _check(lib.vmb_discretise_mean_fwd(_ptr(u), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(delta_bias), _ptr(dAm),
                                       _ptr(dBum), B, K, D, N, H, W, flags, _dtype_code(u.dtype), _stream(stream)),
           "vmb_discretise_mean_fwd")
    return dAm, dBum


def vmb_scan_only_fwd(dA, dBu, Cs, H: int, W: int, *, y=None, stream=None):
    """The scan alone (Eq. 3 without the skip): dA, dBu float32 [B, K, Dm, N, L] (or
    [B, K, N, L] for one channel), Cs [B, K, N, L] -> y float32 [B, K, Dm, L] (or [B, K, L])."""
    for t, n in [(dA, "dA"), (dBu, "dBu"), (Cs, "Cs")]:
        _dev(t, n)
    one = dA.dim() == 4
    B, K = dA.shape[:2]
    Dm = 1 if one else dA.shape[2]
    N, L = dA.shape[-2:]
    if L != H * W or dBu.shape != dA.shape or Cs.shape != (B, K, N, L):
        raise ValueError("dA, dBu [B,K,Dm,N,H*W] and Cs [B,K,N,H*W] expected")
    if dA.dtype != torch.float32 or dBu.dtype != torch.float32:
        raise ValueError("dA, dBu must be float32")
    shape = (B, K, L) if one else (B, K, Dm, L)
    y = torch.empty(shape, dtype=torch.float32, device=dA.device) if y is None else y
    _dev(y, "y")
    if tuple(y.shape) != shape or y.dtype != torch.float32:
        raise ValueError(f"y must be float32 {shape}")
    _check(lib.vmb_scan_only_fwd(_ptr(dA), _ptr(dBu), _ptr(Cs), _ptr(y), B, K, Dm, N, H, W, _dtype_code(Cs.dtype),
                                 _stream(stream)), "vmb_scan_only_fwd")
    return y


def vmb_selection_fwd(u, WB, WC, Wz, Wup, H: int, W: int, *, delta_raw=None, Bs=None, Cs=None, stream=None):
    """Eq. 6 selection functions: u [B, K, D, H*W] -> (delta_raw [B, K, D, L], Bs, Cs [B, K, N, L]),
    all in u's dtype; WB, WC [K, N, D], Wz [K, R, D], Wup [K, D, R] float32."""
    for t, n in [(u, "u"), (WB, "WB"), (WC, "WC"), (Wz, "Wz"), (Wup, "Wup")]:
        _dev(t, n)
    B, K, D, L = u.shape
    N, R = WB.shape[1], Wz.shape[1]
    if L != H * W or tuple(WB.shape) != (K, N, D) or tuple(WC.shape) != (K, N, D) or \
            tuple(Wz.shape) != (K, R, D) or tuple(Wup.shape) != (K, D, R):
        raise ValueError("u [B,K,D,H*W], WB/WC [K,N,D], Wz [K,R,D], Wup [K,D,R] expected")
    if any(w.dtype != torch.float32 for w in (WB, WC, Wz, Wup)):
        raise ValueError("weights must be float32")
    delta_raw = torch.empty_like(u) if delta_raw is None else delta_raw
    Bs = torch.empty((B, K, N, L), dtype=u.dtype, device=u.device) if Bs is None else Bs
    Cs = torch.empty((B, K, N, L), dtype=u.dtype, device=u.device) if Cs is None else Cs
    for t, n, shp in [(delta_raw, "delta_raw", (B, K, D, L)), (Bs, "Bs", (B, K, N, L)), (Cs, "Cs", (B, K, N, L))]:
        _dev(t, n)
        if tuple(t.shape) != shp or t.dtype != u.dtype:
            raise ValueError(f"{n} must be {u.dtype} {shp}")
    _check(lib.vmb_selection_fwd(_ptr(u), _ptr(WB), _ptr(WC), _ptr(Wz), _ptr(Wup), _ptr(Bs), _ptr(Cs),
                                 _ptr(delta_raw), B, K, D, N, R, H, W, _dtype_code(u.dtype), _stream(stream)),
           "vmb_selection_fwd")
    return delta_raw, Bs, Cs


def vmb_selection_lowrank_fwd(u, WB, WC, Wz, H: int, W: int, *, z=None, Bs=None, Cs=None, stream=None):
    """Eq. 6 selection functions with the Delta branch left low-rank: u [B, K, D, H*W] ->
    (z [B, K, R, L] float32, Bs, Cs [B, K, N, L] in u's dtype); WB, WC [K, N, D], Wz [K, R, D]."""
    for t, n in [(u, "u"), (WB, "WB"), (WC, "WC"), (Wz, "Wz")]:
        _dev(t, n)
    B, K, D, L = u.shape
    N, R = WB.shape[1], Wz.shape[1]
    if L != H * W or tuple(WB.shape) != (K, N, D) or tuple(WC.shape) != (K, N, D) or tuple(Wz.shape) != (K, R, D):
        raise ValueError("u [B,K,D,H*W], WB/WC [K,N,D], Wz [K,R,D] expected")
    if any(w.dtype != torch.float32 for w in (WB, WC, Wz)):
        raise ValueError("weights must be float32")
    z = torch.empty((B, K, R, L), dtype=torch.float32, device=u.device) if z is None else z
    Bs = torch.empty((B, K, N, L), dtype=u.dtype, device=u.device) if Bs is None else Bs
    Cs = torch.empty((B, K, N, L), dtype=u.dtype, device=u.device) if Cs is None else Cs
    for t, n, shp, dt in [(z, "z", (B, K, R, L), torch.float32), (Bs, "Bs", (B, K, N, L), u.dtype),
                          (Cs, "Cs", (B, K, N, L), u.dtype)]:
        _dev(t, n)
        if tuple(t.shape) != shp or t.dtype != dt:
            raise ValueError(f"{n} must be {dt} {shp}")
    _check(lib.vmb_selection_lowrank_fwd(_ptr(u), _ptr(WB), _ptr(WC), _ptr(Wz), _ptr(Bs), _ptr(Cs), _ptr(z),
                                         B, K, D, N, R, H, W, _dtype_code(u.dtype), _stream(stream)),
           "vmb_selection_lowrank_fwd")
    return z, Bs, Cs


def vmb_selective_scan_lowrank_fwd(u, z, Wup, A, Bs, Cs, Dskip, delta_bias, H: int, W: int, *, y=None,
                                   flags: int = VMB_FLAG_SOFTPLUS, workspace=None, stream=None) -> torch.Tensor:
    """Full-channel selective scan whose raw Deltas are Wup z, formed inside the scan:
    z [B, K, R, H*W] float32, Wup [K, D, R] float32; returns y [B, K, D, H*W] (dtype of u)."""
    for t, n in [(z, "z"), (Wup, "Wup")]:
        _dev(t, n)
    B, K, D, L = u.shape
    R = z.shape[2]
    if tuple(z.shape) != (B, K, R, L) or z.dtype != torch.float32:
        raise ValueError("z must be float32 [B, K, R, H*W]")
    if tuple(Wup.shape) != (K, D, R) or Wup.dtype != torch.float32:
        raise ValueError("Wup must be float32 [K, D, R]")
    B, K, D, N, L = _scan_shapes(u, u, A, Bs, Cs, Dskip, delta_bias, H, W)
    if y is None:
        y = torch.empty_like(u)
    _dev(y, "y")
    if y.shape != u.shape or y.dtype != u.dtype:
        raise ValueError("y must match u")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_FULL, B, K, D, N, H, W, u.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, u.device)
    _check(lib.vmb_selective_scan_lowrank_fwd(_ptr(u), _ptr(z), _ptr(Wup), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                              _ptr(delta_bias), _ptr(y), B, K, D, N, R, H, W, flags,
                                              _dtype_code(u.dtype), _ptr(workspace), workspace.numel(),
                                              _stream(stream)), "vmb_selective_scan_lowrank_fwd")
    return y


def vmb_mean_scan_lowrank_fwd(u, z, Wup, A, Bs, Cs, Dskip, delta_bias, H: int, W: int, *, y=None, ybar=None,
                              want_ybar: bool = False, flags: int = VMB_FLAG_SOFTPLUS, workspace=None, stream=None):
    """Channel-mean scan whose raw Deltas are Wup z, formed inside the scan: z [B, K, R, H*W]
    float32, Wup [K, D, R] float32; returns (y [B, K, D, L], ybar [B, K, L] fp32 or None)."""
    for t, n in [(z, "z"), (Wup, "Wup")]:
        _dev(t, n)
    B, K, D, L = u.shape
    R = z.shape[2]
    if tuple(z.shape) != (B, K, R, L) or z.dtype != torch.float32:
        raise ValueError("z must be float32 [B, K, R, H*W]")
    if tuple(Wup.shape) != (K, D, R) or Wup.dtype != torch.float32:
        raise ValueError("Wup must be float32 [K, D, R]")
    B, K, D, N, L = _scan_shapes(u, u, A, Bs, Cs, Dskip, delta_bias, H, W)
    if y is None:
        y = torch.empty_like(u)
    _dev(y, "y")
    if y.shape != u.shape or y.dtype != u.dtype:
        raise ValueError("y must match u")
    if ybar is None and want_ybar:
        ybar = torch.empty((B, K, L), dtype=torch.float32, device=u.device)
    if ybar is not None:
        _dev(ybar, "ybar")
        if tuple(ybar.shape) != (B, K, L) or ybar.dtype != torch.float32:
            raise ValueError("ybar must be float32 [B, K, L]")
    ws_bytes = vmb_scan_workspace_bytes(VMB_PATH_MEAN, B, K, D, N, H, W, u.dtype)
    if workspace is None:
        workspace = _default_ws.get(ws_bytes, u.device)
    _check(lib.vmb_mean_scan_lowrank_fwd(_ptr(u), _ptr(z), _ptr(Wup), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip),
                                         _ptr(delta_bias), _ptr(y), _ptr(ybar),
                                         B, K, D, N, R, H, W, flags, _dtype_code(u.dtype), _ptr(workspace),
                                         workspace.numel(), _stream(stream)), "vmb_mean_scan_lowrank_fwd")
    return y, ybar


def vmb_mean_scan_bwd_workspace_bytes(B: int, K: int, D: int, N: int, H: int, W: int, groups: int = 1,
                                      dtype: torch.dtype = torch.float32) -> int:
    return int(lib.vmb_mean_scan_bwd_workspace_bytes(B, K, D, N, H, W, groups, _dtype_code(dtype)))


def vmb_mean_scan_bwd(u, delta, A, Bs, Cs, Dskip, delta_bias, gy, H: int, W: int, *, groups: int = 1,
                      saved=None, flags: int = VMB_FLAG_SOFTPLUS, workspace=None, stream=None) -> dict:
    """Gradients of the (grouped) channel-mean scan given gy = dLoss/dy [B, K, D, H*W]: returns
    dict(u, delta, A, Bs, Cs, Dskip, delta_bias) with the inputs' shapes (delta: the raw Delta).
    saved: the group means vmb_mean_scan_train_fwd kept for these inputs, or None (recomputed)."""
    B, K, D, N, L = _scan_shapes(u, delta, A, Bs, Cs, Dskip, delta_bias, H, W)
    _dev(gy, "gy")
    if gy.shape != u.shape or gy.dtype != u.dtype:
        raise ValueError("gy must match u")
    if groups < 1 or D % groups:
        raise ValueError("groups must be >= 1 and divide D")
    if saved is not None:
        _dev(saved, "saved")
        if tuple(saved.shape) != (B, K, groups, N + 1, L) or saved.dtype != torch.float32:
            raise ValueError("saved must be float32 [B, K, groups, N + 1, L]")
    out = dict(u=torch.empty_like(u), delta=torch.empty_like(u), A=torch.empty_like(A), Bs=torch.empty_like(Bs),
               Cs=torch.empty_like(Cs), Dskip=torch.empty_like(Dskip), delta_bias=torch.empty_like(delta_bias))
    ws_bytes = vmb_mean_scan_bwd_workspace_bytes(B, K, D, N, H, W, groups, u.dtype)
    if workspace is None:
        workspace = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=u.device)
    _check(lib.vmb_mean_scan_bwd(_ptr(u), _ptr(delta), _ptr(A), _ptr(Bs), _ptr(Cs), _ptr(Dskip), _ptr(delta_bias),
                                 _ptr(gy), _ptr(saved), _ptr(out["u"]), _ptr(out["delta"]), _ptr(out["A"]), _ptr(out["Bs"]),
                                 _ptr(out["Cs"]), _ptr(out["Dskip"]), _ptr(out["delta_bias"]), B, K, D, N, H, W,
                                 groups, flags, _dtype_code(u.dtype), _ptr(workspace), workspace.numel(),
                                 _stream(stream)), "vmb_mean_scan_bwd")
    return out


def vmb_read_status(workspace=None, device=None, stream=None) -> int:
    """Synchronise and return (then clear) the device error word of a workspace."""
    if workspace is None:
        dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
        workspace = _default_ws.get(256, dev)
    return int(lib.vmb_read_status(_ptr(workspace), _stream(stream)))


def default_workspace(device=None) -> torch.Tensor:
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    return _default_ws.get(256, dev)
