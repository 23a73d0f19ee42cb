"""Seeded synthetic workloads for one Efficient-Adam round.

This module describes the five workloads (dimension, worker count, quantizers, hyper-parameters,
rounds) and draws their gradients.  It holds none of the method's arithmetic and imports neither
the CUDA binding nor the oracle, so that both sides of every parity check consume identical inputs.

The paper's own experiments (Section 5: a 500-dimensional quadratic toy, ResNet-18 on CIFAR-100, a
bi-GRU on IMDB) need datasets and trained encoders that are not available here; the workloads keep
only their shapes and value distributions:

  c1  d = 65,536, n = 4, 10 rounds, g ~ N(0, 1), 1-bit scaled sign with one scale for the vector.
  c2  the quadratic toy f(x) = 0.5 ||x - x*||^2 at d = 1e6, n = 8, 1,000 rounds:
      g_i = (x - x*) + 0.1 xi_i,  x* ~ N(0, 1), xi ~ N(0, I); whole-vector sign scales.
  c3  a flat vector with the 62 parameter tensors of ResNet-18 (11,689,512 values), n = 16,
      100 rounds, g = Student-t(3) times a per-tensor magnitude 10^(-5 + 4 U) (log-uniform in
      [1e-5, 1e-1]); one sign scale per tensor.
  c4  d = 1.1e8 (BERT-base sized) in 4,096-blocks, n = 8, 50 rounds, g ~ N(0, 1e-3^2) with 1% of
      the coordinates (Bernoulli per worker and round) multiplied by 100; Q_w = 4-bit stochastic
      uniform grid, Q_s = 8-bit deterministic uniform grid (Example 1), per-block l_inf scales.
  c5  d = 1.558e9 (GPT-2-XL sized) in 4,096-blocks, n = 8, 10 rounds, g ~ N(0, 1e-4^2);
      1-bit scaled sign with per-block scales.
"""
from __future__ import annotations

import dataclasses
import hashlib

import numpy as np

# quantizer kinds and placements (the C-ABI's enumerators)
Q_IDENTITY, Q_SIGN_L1, Q_UNIFORM_MAX, Q_POW2 = 0, 1, 2, 3
ADAM_AT_WORKER, ADAM_AT_SERVER = 0, 1

# ResNet-18 (torchvision, 1000-class head) parameter tensors in registration order.
_RESNET18_BLOCK = {  # (conv1, conv2, downsample conv or 0) per stage, channels
    64: (64 * 64 * 9, 64 * 64 * 9, 0),
    128: (128 * 64 * 9, 128 * 128 * 9, 128 * 64),
    256: (256 * 128 * 9, 256 * 256 * 9, 256 * 128),
    512: (512 * 256 * 9, 512 * 512 * 9, 512 * 256),
}


def resnet18_tensor_sizes() -> list[int]:
    sizes = [64 * 3 * 7 * 7, 64, 64]
    for ch in (64, 128, 256, 512):
        c1, c2, ds = _RESNET18_BLOCK[ch]
        # first block of the stage
        sizes += [c1, ch, ch, c2, ch, ch]
        if ds:
            sizes += [ds, ch, ch]
        # second block: both convs are ch -> ch
        sizes += [ch * ch * 9, ch, ch, ch * ch * 9, ch, ch]
    sizes += [512 * 1000, 1000]
    return sizes


@dataclasses.dataclass(frozen=True)
class QuantSpec:
    kind: int
    bits: int
    group: int = 0                 # 0 whole vector, > 0 fixed block length, < 0 segments
    segments: tuple = ()           # segment lengths when group < 0
    stochastic: bool = False
    pow2_k: int = 0
    pow2_K: int = 0


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    d: int
    n: int
    rounds: int
    qw: QuantSpec
    qs: QuantSpec
    alpha: float
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-8
    seed: int = 0
    grad: str = "normal"          # normal | quadratic | student_t | outlier | (scale in grad_std)
    grad_std: float = 1.0

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def sign_q(group: int = 0, segments: tuple = ()) -> QuantSpec:
    return QuantSpec(Q_SIGN_L1, 1, group, segments)


def uniform_q(bits: int, group: int = 4096, stochastic: bool = False) -> QuantSpec:
    return QuantSpec(Q_UNIFORM_MAX, bits, group, (), stochastic)


def pow2_q(k: int = -17, K: int = -11, bits: int = 4) -> QuantSpec:
    return QuantSpec(Q_POW2, bits, 0, (), False, k, K)


def identity_q() -> QuantSpec:
    return QuantSpec(Q_IDENTITY, 32, 0)


_R18 = tuple(resnet18_tensor_sizes())

WORKLOADS = {
    "c1": Workload("c1", 65_536, 4, 10, sign_q(0), sign_q(0), 1e-3, seed=1001, grad="normal"),
    "c2": Workload("c2", 1_000_000, 8, 1000, sign_q(0), sign_q(0), 1e-2, seed=1002, grad="quadratic"),
    "c3": Workload("c3", sum(_R18), 16, 100, sign_q(-1, _R18), sign_q(-1, _R18), 1e-3, seed=1003,
                   grad="student_t"),
    "c4": Workload("c4", 110_000_000, 8, 50, uniform_q(4, 4096, True), uniform_q(8, 4096, False), 1e-4,
                   seed=1004, grad="outlier", grad_std=1e-3),
    "c5": Workload("c5", 1_558_000_000, 8, 10, sign_q(4096), sign_q(4096), 1e-4, seed=1005,
                   grad="normal", grad_std=1e-4),
}


def _mix(*parts) -> int:
    """A 63-bit seed from (workload seed, stream name, worker, round)."""
    h = hashlib.sha256(repr(parts).encode()).digest()
    return int.from_bytes(h[:8], "little") & ((1 << 63) - 1)


# ------------------------------------------------------------------------- host (numpy) draws

def _rng(*parts) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(_mix(*parts)))


def tensor_magnitudes(w: Workload) -> np.ndarray:
    """c3: one log-uniform magnitude in [1e-5, 1e-1] per tensor, drawn once per workload."""
    u = _rng(w.seed, "mag").random(len(w.qw.segments))
    return (10.0 ** (-5.0 + 4.0 * u)).astype(np.float32)


def xstar_host(w: Workload, d: int | None = None) -> np.ndarray:
    d = w.d if d is None else d
    return _rng(w.seed, "xstar").standard_normal(d, dtype=np.float32)


def gradient_host(w: Workload, i: int, t: int, d: int | None = None) -> np.ndarray:
    """Worker i's round-t input for the workloads whose gradient does not depend on x
    (for c2 this is the noise term 0.1 xi; add (x - x*) with quadratic_gradient)."""
    d = w.d if d is None else d
    r = _rng(w.seed, "g", i, t)
    if w.grad == "normal":
        return (r.standard_normal(d, dtype=np.float32) * np.float32(w.grad_std)).astype(np.float32)
    if w.grad == "quadratic":
        return (r.standard_normal(d, dtype=np.float32) * np.float32(0.1)).astype(np.float32)
    if w.grad == "outlier":
        z = r.standard_normal(d, dtype=np.float32) * np.float32(w.grad_std)
        mask = r.random(d) < 0.01
        return np.where(mask, z * np.float32(100.0), z).astype(np.float32)
    if w.grad == "student_t":
        seg = np.asarray(w.qw.segments, dtype=np.int64)
        mags = np.repeat(tensor_magnitudes(w), seg)[:d]
        return (r.standard_t(3, size=d).astype(np.float32) * mags).astype(np.float32)
    raise ValueError(w.grad)


def quadratic_gradient(x, xstar, noise):
    """Gradient of 0.5 ||x - x*||^2 plus the drawn noise (numpy or torch arrays alike)."""
    return (x - xstar) + noise


# ------------------------------------------------------------------------ device (torch) draws

def gradient_device(w: Workload, i: int, t: int, out, d: int | None = None):
    """Fill the float32 torch tensor `out` with worker i's round-t input, drawn on out's device.
    Used where the host draw would be too slow (the 1e8-1e9 coordinate workloads)."""
    import torch

    d = out.numel() if d is None else d
    g = torch.Generator(device=out.device)
    g.manual_seed(_mix(w.seed, "gd", i, t))
    o = out[:d]
    torch.randn(d, generator=g, out=o)
    if w.grad == "normal":
        o.mul_(w.grad_std)
    elif w.grad == "quadratic":
        o.mul_(0.1)
    elif w.grad == "outlier":
        o.mul_(w.grad_std)
        mask = torch.rand(d, generator=g, device=out.device) < 0.01
        o[mask] *= 100.0
    elif w.grad == "student_t":
        z = torch.randn(3, d, generator=g, device=out.device)
        chi = (z * z).sum(0).div_(3.0).sqrt_()
        o.div_(chi)
        seg = torch.tensor(w.qw.segments, device=out.device)
        mags = torch.from_numpy(tensor_magnitudes(w)).to(out.device)
        o.mul_(torch.repeat_interleave(mags, seg)[:d])
    else:
        raise ValueError(w.grad)
    return out


def sample_blocks(w: Workload, count: int, block: int = 4096) -> np.ndarray:
    """A fixed sample of block indices: the first, the last (ragged tail) and count-2 drawn ones."""
    nb = -(-w.d // block)
    rest = _rng(w.seed, "sample").choice(np.arange(1, max(nb - 1, 1)), size=max(0, min(count - 2, nb - 2)),
                                         replace=False)
    return np.unique(np.concatenate([[0, nb - 1], rest]).astype(np.int64))


# ------------------------------------------------------------------- Section 5.1's convex toy
# min_x E || A x - (x* + xi) ||^2 with A in R^{500 x 500}, A_ij ~ N(0, 1), x* ~ N(0, 0.1 I),
# xi ~ N(0, 0.1 I), 10 workers, beta = 0.9, theta = 0.99; quantizers Example 1 with k = 1 ("com1")
# and Example 2 with k = -17, K = -11 ("com2"); "full" is the 32-bit identity.

TOY_D, TOY_N = 500, 10
TOY_QUANTIZERS = {
    "full": QuantSpec(Q_IDENTITY, 32, 0),
    "com1": QuantSpec(Q_UNIFORM_MAX, 2, 0),
    "com2": QuantSpec(Q_POW2, 4, 0, (), False, -17, -11),
}


def toy_case(case: int, d: int = TOY_D):
    """A random case of the toy: (A, x*) in float32 and a generator for the noise draws."""
    r = _rng(2051, "toy", case)
    A = r.standard_normal((d, d), dtype=np.float32)
    xs = (r.standard_normal(d, dtype=np.float32) * np.float32(np.sqrt(0.1))).astype(np.float32)
    return A, xs


def toy_noise(case: int, i: int, t: int, d: int = TOY_D) -> np.ndarray:
    return (_rng(2051, "toy-xi", case, i, t).standard_normal(d, dtype=np.float32) *
            np.float32(np.sqrt(0.1))).astype(np.float32)


def toy_gradient(A: np.ndarray, x: np.ndarray, xs: np.ndarray, xi: np.ndarray) -> np.ndarray:
    """The stochastic gradient 2 A^T (A x - x* - xi) of the toy (formed in binary64, rounded to
    binary32), for any x (numpy)."""
    A64 = A.astype(np.float64)
    r = A64 @ x.astype(np.float64) - xs.astype(np.float64) - xi.astype(np.float64)
    return (2.0 * (A64.T @ r)).astype(np.float32)


def toy_full_gradient_norm(A: np.ndarray, x: np.ndarray, xs: np.ndarray) -> float:
    """|| grad F(x) || = || 2 A^T (A x - x*) ||, the quantity Figure 2 plots."""
    A64 = A.astype(np.float64)
    return float(np.linalg.norm(2.0 * (A64.T @ (A64 @ x.astype(np.float64) - xs.astype(np.float64)))))
