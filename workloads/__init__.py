"""Seeded synthetic workloads for the SS2D selective scan (full and channel-mean).

This module only draws random numbers and lays them out: it holds none of the
method's arithmetic (no cross-scan, no softplus, no exponentials of the scan,
no recurrence), so that both the fp64 oracle and the CUDA path can take their
inputs from it without sharing any computation.

Shapes (row-major, contiguous):
    x      [B, D, H, W]   the 2-D feature map fed to the cross-scan
    draw   [B, K, D, L]   raw time-step input Delta before the bias and softplus
    Bs, Cs [B, K, N, L]   input-dependent B and C (no channel axis, as in Mamba)
    A      [K*D, N]       continuous-time state matrix diagonal, per channel
    Dskip  [K*D]          skip weight D of y = C h + D u
    bias   [K*D]          Delta bias ("Parameter" of the selection mechanism)

The recipe follows the paper's workloads (VMamba-T stage shapes at 224^2, a
512^2 segmentation map and a batch-128 classification batch; App. D
"Datasets", "Models"): the map x is a shared N(0,1) image plus small
per-channel N(0, sigma^2) noise, which mimics the low cross-channel variance
the paper observes in its activations (Sec. 2.1, Eq. 7).  Trained weights and
the ImageNet/ADE20K images are not available, so these seeded arrays stand in
for them.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import math

import numpy as np

K_DIRECTIONS = 4


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    D: int
    N: int
    H: int
    W: int
    dtype: str = "f32"          # "f32" or "bf16": storage type of x, draw, Bs, Cs, y
    sigma: float = 0.1          # per-channel noise std of the map
    seed: int = 0
    K: int = K_DIRECTIONS

    @property
    def L(self) -> int:
        return self.H * self.W

    @property
    def esize(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def scan_elements(self) -> int:
        """B*K*D*L: the element count the throughput metric is quoted in."""
        return self.B * self.K * self.D * self.L

    def scan_bytes(self) -> int:
        """Algorithmic HBM bytes of one selective-scan call (full or mean path):
        u and delta read once, Bs and Cs read once, y written once, plus the
        per-channel parameters (A, Dskip, bias)."""
        s = self.esize
        bkdl = self.B * self.K * self.D * self.L
        bknl = self.B * self.K * self.N * self.L
        params = self.K * self.D * (self.N + 2) * 4
        return s * (3 * bkdl + 2 * bknl) + params

    def csm_bytes(self) -> int:
        """Algorithmic bytes of one cross-scan or one cross-merge call:
        one map of B*D*L elements on one side, four on the other."""
        return self.esize * 5 * self.B * self.D * self.L

    def fused_mean_bytes(self) -> int:
        """Algorithmic bytes of the channel-mean path with the broadcast fused
        into the cross-merge: u and delta read once, Bs and Cs read once, the
        map x read and the merged map written once, ybar (fp32, [B, K, L])
        written and read back once, plus the per-channel parameters."""
        s = self.esize
        bkdl = self.B * self.K * self.D * self.L
        bknl = self.B * self.K * self.N * self.L
        bdl = self.B * self.D * self.L
        params = self.K * self.D * (self.N + 2) * 4
        return s * (2 * bkdl + 2 * bknl + 2 * bdl) + 2 * 4 * self.B * self.K * self.L + params

    def gathered_mean_bytes(self) -> int:
        """Algorithmic bytes of the scan side of the block from the map (cross-scan,
        channel-mean scan and cross-merge in one call, vmb_ss2d_mean_fwd): delta
        read once, Bs and Cs read once, the map x read once (every direction
        reads the same map) and the merged map written once, ybar (fp32,
        [B, K, L]) written and read back once, plus the per-channel parameters.
        (The implementation also writes and reads a transposed copy of the map
        for the column-major directions; that is not counted.)"""
        s = self.esize
        bkdl = self.B * self.K * self.D * self.L
        bknl = self.B * self.K * self.N * self.L
        bdl = self.B * self.D * self.L
        params = self.K * self.D * (self.N + 2) * 4
        return s * (bkdl + 2 * bknl + 2 * bdl) + 2 * 4 * self.B * self.K * self.L + params

    def gathered_full_bytes(self) -> int:
        """Algorithmic bytes of the full-channel scan side of the block from the
        map (vmb_ss2d_full_fwd: selective scan reading the map, then the
        cross-merge): delta read once, Bs and Cs read once, the map x read once
        (every direction reads the same map), y written once and read back by
        the merge, the merged map written once, plus the per-channel
        parameters.  (The transposed copy of the map the column-major
        directions read is not counted, as in gathered_mean_bytes.)"""
        s = self.esize
        bkdl = self.B * self.K * self.D * self.L
        bknl = self.B * self.K * self.N * self.L
        bdl = self.B * self.D * self.L
        params = self.K * self.D * (self.N + 2) * 4
        return s * (3 * bkdl + 2 * bknl + 2 * bdl) + params

    def replace(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


# The paper's scan shapes (App. D "Models"; Table 1/2 shapes), one GPU each.
WORKLOADS = {
    w.name: w
    for w in [
        Workload("ss2d_b1_d192_n16_14x14_f32", 1, 192, 16, 14, 14, "f32", 0.1, 1000),
        Workload("vmamba_t_stage1_b1_d192_n16_56x56_f32", 1, 192, 16, 56, 56, "f32", 0.1, 1001),
        Workload("vmamba_t_224_b32_stage1_d192_56x56_f32", 32, 192, 16, 56, 56, "f32", 0.1, 1021),
        Workload("vmamba_t_224_b32_stage2_d384_28x28_f32", 32, 384, 16, 28, 28, "f32", 0.1, 1022),
        Workload("vmamba_t_224_b32_stage3_d768_14x14_f32", 32, 768, 16, 14, 14, "f32", 0.1, 1023),
        Workload("vmamba_t_224_b32_stage4_d1536_7x7_f32", 32, 1536, 16, 7, 7, "f32", 0.1, 1024),
        Workload("seg512_stage1_b8_d192_n16_128x128_bf16", 8, 192, 16, 128, 128, "bf16", 0.1, 1003),
        Workload("batch128_d256_n1_56x56_sigma0.05_f32", 128, 256, 1, 56, 56, "f32", 0.05, 1040),
        Workload("batch128_d256_n1_56x56_sigma0.5_f32", 128, 256, 1, 56, 56, "f32", 0.5, 1041),
        Workload("batch128_d256_n16_56x56_sigma0.05_f32", 128, 256, 16, 56, 56, "f32", 0.05, 1042),
        Workload("batch128_d256_n16_56x56_sigma0.5_f32", 128, 256, 16, 56, 56, "f32", 0.5, 1043),
    ]
}

SMALL = "ss2d_b1_d192_n16_14x14_f32"
STAGE1_B1 = "vmamba_t_stage1_b1_d192_n16_56x56_f32"


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even) and return
    them as float32 (exactly representable in bf16).  Storage conversion only."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    bits = a.view(np.uint32).astype(np.uint64)
    rounded = ((bits + 0x7FFF + ((bits >> 16) & 1)) >> 16) << 16
    return rounded.astype(np.uint32).view(np.float32)


@dataclass
class Inputs:
    wl: Workload
    x: np.ndarray
    draw: np.ndarray
    Bs: np.ndarray
    Cs: np.ndarray
    A: np.ndarray
    Dskip: np.ndarray
    bias: np.ndarray
    extra: dict = field(default_factory=dict)

    def arrays(self) -> dict:
        return dict(x=self.x, draw=self.draw, Bs=self.Bs, Cs=self.Cs,
                    A=self.A, Dskip=self.Dskip, bias=self.bias)


PARAMS = ("paper", "random")


def make_inputs(wl: Workload, seed: int | None = None, *, sigma: float | None = None,
                channel_identical: bool = False, params: str = "paper") -> Inputs:
    """Draw one seeded input set for workload `wl`.

    Draw order (fixed): s, e, draw, Bs, Cs, dt.
      x[b,d,h,w] = s[b,h,w] + sigma * e[b,d,h,w],   s, e ~ N(0, 1)
      draw       ~ N(0, 0.5^2)
      Bs, Cs     ~ N(0, 1)
      dt_c       = exp(U[ln 1e-3, ln 1e-1]),  bias_c = the value whose softplus is dt_c
    Per-channel parameters, by `params`:
      "paper"  (the benchmark recipe): A[c, n] = -(n + 1), Dskip_c = 1
      "random" (parity tests): A[c, n] = -U[0.5, 3] drawn independently for
               every (c, n), Dskip_c = U[0.5, 1.5] per channel, from a second
               generator seeded with (seed, 2), so that the draws above are
               the same under both settings.  Every channel then has its own
               A row and skip weight, and a kernel that reads the parameters
               of the wrong channel or state gives a different result.
    bf16 workloads round x, draw, Bs, Cs to bf16 (ties to even) after drawing.

    channel_identical=True makes every channel of a direction identical
    (sigma = 0, draw/bias shared over d, and under "random" the A rows and
    skip weights shared over d): the case in which the channel mean loses
    nothing.
    """
    if params not in PARAMS:
        raise ValueError(f"params must be one of {PARAMS}, not {params!r}")
    seed = wl.seed if seed is None else seed
    sigma = wl.sigma if sigma is None else sigma
    B, K, D, N, H, W, L = wl.B, wl.K, wl.D, wl.N, wl.H, wl.W, wl.L
    rng = np.random.default_rng(seed)
    f32 = np.float32
    s = rng.standard_normal((B, 1, H, W), dtype=f32)
    e = rng.standard_normal((B, D, H, W), dtype=f32)
    if channel_identical:
        x = np.broadcast_to(s, (B, D, H, W)).astype(f32)
    else:
        x = (s + f32(sigma) * e).astype(f32)
    del e
    draw = rng.standard_normal((B, K, D, L), dtype=f32)
    draw *= f32(0.5)
    Bs = rng.standard_normal((B, K, N, L), dtype=f32)
    Cs = rng.standard_normal((B, K, N, L), dtype=f32)
    dt = np.exp(rng.uniform(math.log(1e-3), math.log(1e-1), size=K * D))
    # inverse of softplus: log(exp(dt) - 1) = dt + log(1 - exp(-dt))
    bias = (dt + np.log(-np.expm1(-dt))).astype(f32)
    if channel_identical:
        draw[:] = draw[:, :, :1, :]
        bias = np.repeat(bias.reshape(K, D)[:, :1], D, axis=1).reshape(K * D).astype(f32)
    if params == "random":
        prng = np.random.default_rng([seed, 2])
        A = (-prng.uniform(0.5, 3.0, size=(K * D, N))).astype(f32)
        Dskip = prng.uniform(0.5, 1.5, size=K * D).astype(f32)
        if channel_identical:
            A = np.repeat(A.reshape(K, D, N)[:, :1], D, axis=1).reshape(K * D, N).astype(f32)
            Dskip = np.repeat(Dskip.reshape(K, D)[:, :1], D, axis=1).reshape(K * D).astype(f32)
    else:
        A = np.tile(-(np.arange(N, dtype=f32) + 1.0), (K * D, 1)).astype(f32)
        Dskip = np.ones(K * D, dtype=f32)
    if wl.dtype == "bf16":
        x = round_to_bf16(x)
        draw = round_to_bf16(draw)
        Bs = round_to_bf16(Bs)
        Cs = round_to_bf16(Cs)
    return Inputs(wl, x, draw, Bs, Cs, A, Dskip, bias)


def small_case(B=1, D=5, N=3, H=3, W=4, dtype="f32", sigma=0.1, seed=7) -> Workload:
    """A tiny ad-hoc workload for brute-force and edge-case tests."""
    return Workload(f"tiny_b{B}_d{D}_n{N}_{H}x{W}_{dtype}", B, D, N, H, W, dtype, sigma, seed)


def make_device_inputs(wl: Workload, device, seed: int | None = None, params: str = "paper") -> dict:
    """The recipe of make_inputs drawn on the GPU with torch's generator (same
    distributions and shapes, different values): for timing runs over many and
    large workloads, where only the sizes and the value ranges matter.  Parity
    tests use make_inputs.  Returns torch tensors x, draw, Bs, Cs (storage
    dtype) and A, Dskip, bias (fp32)."""
    import torch

    if params not in PARAMS:
        raise ValueError(f"params must be one of {PARAMS}, not {params!r}")
    seed = wl.seed if seed is None else seed
    B, K, D, N, H, W, L = wl.B, wl.K, wl.D, wl.N, wl.H, wl.W, wl.L
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    f = dict(device=device, dtype=torch.float32, generator=gen)
    x = torch.randn(B, 1, H, W, **f) + wl.sigma * torch.randn(B, D, H, W, **f)
    draw = 0.5 * torch.randn(B, K, D, L, **f)
    Bs = torch.randn(B, K, N, L, **f)
    Cs = torch.randn(B, K, N, L, **f)
    u01 = torch.rand(K * D, device=device, dtype=torch.float64, generator=gen)
    dt = torch.exp(math.log(1e-3) + u01 * (math.log(1e-1) - math.log(1e-3)))
    bias = (dt + torch.log(-torch.expm1(-dt))).float()
    if params == "random":
        A = -(0.5 + 2.5 * torch.rand(K * D, N, **f))
        Dskip = 0.5 + torch.rand(K * D, **f)
    else:
        A = -(torch.arange(N, device=device, dtype=torch.float32) + 1.0).repeat(K * D, 1).contiguous()
        Dskip = torch.ones(K * D, device=device, dtype=torch.float32)
    sdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    return dict(x=x.contiguous().to(sdt), draw=draw.to(sdt), Bs=Bs.to(sdt), Cs=Cs.to(sdt), A=A, Dskip=Dskip,
                bias=bias)
