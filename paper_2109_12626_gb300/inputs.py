"""Seeded, counter-based synthetic inputs for the reduction-to-all.

This module holds no arithmetic of the method: it only makes the p input
vectors x_0..x_{p-1}.  Every element is a pure function of
(seed, rank, column), so the same values can be produced for a whole rank on
the GPU or for a few sampled columns on the host, bit for bit: everything is
exact integer arithmetic on int64 tensors, followed by at most one
correctly rounded float64 multiply and one float32 conversion, which torch
computes identically on every device.

Generator: SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom
number generators", OOPSLA 2014).  Stream key k_r = mix(seed*G + rank + 1);
the n-th 64-bit word of rank r is mix(k_r + (n+1)*G) with G the golden gamma
0x9E3779B97F4A7C15 and mix the published 64-bit finaliser.  int64 tensor
multiplication wraps mod 2^64; logical right shifts are an arithmetic shift
followed by a mask.

Distributions (what the workloads of the paper's experiment and the
benchmark configurations ask for):
  uniform_int32(lo, hi)  Lemire's multiply-shift map of a 32-bit word onto
                         [lo, hi] (exact: product < 2^53)
  words_u32              raw uniform 32-bit words (2x2 uint32 matrices)
  near_identity_f32      2x2 float32 matrices I + E, entries of E exact
                         dyadics of magnitude <= 2^-7
  normal_f32(sigma)      Irwin-Hall sum of twelve uniform 16-bit integers,
                         centred and scaled to unit variance (the classic
                         "sum of 12 uniforms" normal approximation, tails
                         truncated at 6 sigma), times sigma in float64,
                         rounded once to float32
"""
from __future__ import annotations

import torch

_G = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB
_MASK32 = 0xFFFFFFFF


def _s64(v: int) -> int:
    """Two's-complement int64 value of a 64-bit unsigned constant."""
    v &= (1 << 64) - 1
    return v - (1 << 64) if v >= (1 << 63) else v


_GS, _M1S, _M2S = _s64(_G), _s64(_M1), _s64(_M2)


def _shr(z: torch.Tensor, k: int) -> torch.Tensor:
    """Logical right shift of int64 bit patterns."""
    return (z >> k) & ((1 << (64 - k)) - 1)


def _mix(z: torch.Tensor) -> torch.Tensor:
    z = (z ^ _shr(z, 30)) * _M1S
    z = (z ^ _shr(z, 27)) * _M2S
    return z ^ _shr(z, 31)


def _key(seed: int, rank: int) -> int:
    z = torch.tensor([_s64(seed * _G + rank + 1)], dtype=torch.int64)
    return int(_mix(z)[0])


def words64(seed: int, rank: int, n: torch.Tensor) -> torch.Tensor:
    """The n-th 64-bit word (as int64 bits) of rank ``rank``'s stream."""
    n = n.to(torch.int64)
    return _mix((n + 1) * _GS + _key(seed, rank))


def _cols(m_or_idx, device) -> torch.Tensor:
    if isinstance(m_or_idx, torch.Tensor):
        return m_or_idx.to(device=device, dtype=torch.int64)
    return torch.arange(int(m_or_idx), device=device, dtype=torch.int64)


def uniform_int32(seed: int, rank: int, cols, lo: int, hi: int,
                  device="cpu") -> torch.Tensor:
    """int32 values uniform on [lo, hi] at the given columns (or 0..m-1)."""
    c = _cols(cols, device)
    r = hi - lo + 1
    assert 0 < r <= (1 << 21) + 1, "range must keep the product exact"
    w = words64(seed, rank, c) & _MASK32
    return (lo + ((w * r) >> 32)).to(torch.int32)


def words_u32(seed: int, rank: int, cols, k: int, device="cpu") -> torch.Tensor:
    """k uniform 32-bit words per column, returned as int32 bit patterns of
    shape [len(cols), k] (k even; two words per 64-bit draw)."""
    assert k % 2 == 0
    c = _cols(cols, device)
    n = c[:, None] * (k // 2) + torch.arange(k // 2, device=c.device)
    z = words64(seed, rank, n.reshape(-1)).reshape(len(c), k // 2)
    lo = z & _MASK32
    hi = _shr(z, 32)
    w = torch.stack([lo, hi], dim=2).reshape(len(c), k)
    w = torch.where(w >= (1 << 31), w - (1 << 32), w)
    return w.to(torch.int32)


def near_identity_f32(seed: int, rank: int, cols, device="cpu") -> torch.Tensor:
    """2x2 float32 matrices I + E, each entry of E an exact dyadic
    k * 2^-22 with k uniform on [-2^15, 2^15) (|E| <= 2^-7), so products of
    thousands of them stay in range; shape [len(cols), 4]."""
    c = _cols(cols, device)
    z = words64(seed, rank, c)
    k = torch.stack([_shr(z, 16 * q) & 0xFFFF for q in range(4)], dim=1) - 32768
    e = k.to(torch.float64) * 2.0**-22
    e[:, 0] += 1.0
    e[:, 3] += 1.0
    return e.to(torch.float32)


def normal_f32(seed: int, rank: int, cols, sigma: float = 1.0,
               device="cpu") -> torch.Tensor:
    """float32 values ~ N(0, sigma^2) (Irwin-Hall of 12 16-bit uniforms)."""
    c = _cols(cols, device)
    s = torch.zeros(len(c), dtype=torch.int64, device=c.device)
    for t in range(3):
        z = words64(seed, rank, c * 3 + t)
        for q in range(4):
            s += _shr(z, 16 * q) & 0xFFFF
    v = (2 * s - 12 * 65535).to(torch.float64) / 131072.0
    if sigma != 1.0:
        v = v * float(sigma)
    return v.to(torch.float32)


# ---------------------------------------------------------------- workloads
# The five workloads: rank count, vector length, element kind, distribution.

def rank_values(kind: str, seed: int, rank: int, cols, device="cpu",
                **kw) -> torch.Tensor:
    """Values of one rank at the given columns, in the element layout the
    library uses: int32 / float32 as [n], 2x2 uint32 matrices as [n, 4]."""
    if kind == "int32":
        return uniform_int32(seed, rank, cols, kw.get("lo", -1000),
                             kw.get("hi", 1000), device)
    if kind == "float32":
        return normal_f32(seed, rank, cols, kw.get("sigma", 1.0), device)
    if kind == "mat2x2u32":
        return words_u32(seed, rank, cols, 4, device)
    if kind == "mat2x2f32":
        return near_identity_f32(seed, rank, cols, device)
    raise ValueError(kind)


WORKLOADS = {
    # p=7 (trees of 3 and 4), int32 in [-1000, 1000], sum, b=4
    "p7_m1000_int32": dict(p=7, m=1000, kind="int32", seed=1, lo=-1000,
                           hi=1000, b=4),
    # p=36, 2x2 uint32 matrices, product mod 2^32, b=16
    "p36_m65536_mat2x2u32": dict(p=36, m=65536, kind="mat2x2u32", seed=2,
                                 b=16),
    # p=1152 = 36x32, int32 in [-2^20, 2^20], sum, m swept 2^0..2^23
    "p1152_int32_sweep": dict(p=1152, m=None, kind="int32", seed=3,
                              lo=-(1 << 20), hi=1 << 20, b=None),
    # p=1152, m=4194304 float32 ~ N(0,1), sum
    "p1152_m4194304_f32": dict(p=1152, m=4194304, kind="float32", seed=4,
                               sigma=1.0, b=None),
    # p=32, m=134217728 float32 ~ N(0, 1e-3^2), sum
    "p32_m134217728_f32": dict(p=32, m=134217728, kind="float32", seed=5,
                               sigma=1e-3, b=1024),
    # non-commutative float32: p=36, 2x2 float32 matrices near identity
    "p36_m65536_mat2x2f32": dict(p=36, m=65536, kind="mat2x2f32", seed=6, b=16),
}


def workload_kwargs(w: dict) -> dict:
    return {k: w[k] for k in ("lo", "hi", "sigma") if k in w}
