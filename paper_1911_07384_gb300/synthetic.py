"""Seeded synthetic inputs shared by the tests, the smoke check and the bench.

This module holds no arithmetic of the training method: it only draws
ImageNet-shaped random tensors (the paper trains ResNet-50 on ImageNet-1k,
Sec. 5.1; that dataset is not used here, these draws stand in for it) and
rounds them to binary16 with numpy's round-to-nearest-even conversion.

Generator: counter-based splitmix64 (Steele, Lea & Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014): output i of stream `seed` is
mix(seed + (i + 1) * 0x9E3779B97F4A7C15).  Uniforms take the top 53 bits,
normals use the Box-Muller transform in binary64.
Seeds are 1911073840 + 16 * config + tensor_id (x=1, w=2, dy=3, v=4, labels=5).
"""
from __future__ import annotations

import numpy as np

BASE_SEED = 1911073840
TENSOR_IDS = {"x": 1, "w": 2, "dy": 3, "v": 4, "labels": 5}

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def seed_for(config: int, tensor: str | int, sub: int = 0) -> int:
    """Seed of tensor `tensor` of workload `config`; `sub` separates layers."""
    tid = TENSOR_IDS[tensor] if isinstance(tensor, str) else int(tensor)
    return BASE_SEED + 16 * int(config) + tid + 1000003 * int(sub)


def splitmix64(seed: int, n: int) -> np.ndarray:
    i = np.arange(1, n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + i * _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        z = z ^ (z >> np.uint64(31))
    return z


def uniform(seed: int, n: int) -> np.ndarray:
    """n uniforms in (0, 1), binary64."""
    z = splitmix64(seed, n)
    return ((z >> np.uint64(11)).astype(np.float64) + 0.5) * (2.0 ** -53)


def normal(seed: int, n: int) -> np.ndarray:
    """n standard normals (Box-Muller on pairs of uniforms), binary64."""
    m = (n + 1) // 2
    u = uniform(seed, 2 * m)
    u1, u2 = u[0::2], u[1::2]
    r = np.sqrt(-2.0 * np.log(u1))
    out = np.empty(2 * m, np.float64)
    out[0::2] = r * np.cos(2.0 * np.pi * u2)
    out[1::2] = r * np.sin(2.0 * np.pi * u2)
    return out[:n]


def to_f16_bits(x: np.ndarray) -> np.ndarray:
    return np.asarray(x, np.float64).astype(np.float16).view(np.uint16)


def normal_f16(seed: int, shape, std: float = 1.0) -> np.ndarray:
    n = int(np.prod(shape))
    return to_f16_bits(normal(seed, n) * std).reshape(shape)


def he_normal_f16(seed: int, K: int, R: int, S: int, C: int) -> np.ndarray:
    """KRSC weights ~ N(0, 2 / (C*R*S))."""
    return normal_f16(seed, (K, R, S, C), std=float(np.sqrt(2.0 / (C * R * S))))


def labels(seed: int, n: int, classes: int = 1000) -> np.ndarray:
    return np.minimum((uniform(seed, n) * classes).astype(np.int32), classes - 1)


def loguniform_pm_f16(seed: int, shape, lo_exp: float = -24.0, hi_exp: float = 4.0) -> np.ndarray:
    """+-2^U(lo_exp, hi_exp) with a random sign, rounded to binary16."""
    n = int(np.prod(shape))
    u = uniform(seed, 2 * n)
    mag = np.exp2(lo_exp + (hi_exp - lo_exp) * u[:n])
    sign = np.where(u[n:] < 0.5, -1.0, 1.0)
    return to_f16_bits(sign * mag).reshape(shape)


def near_one_f16(seed: int, shape, j_max: int = 8) -> np.ndarray:
    """1 + j * 2^-10 with j uniform in [-j_max, j_max] (exact in binary16)."""
    n = int(np.prod(shape))
    j = np.minimum((uniform(seed, n) * (2 * j_max + 1)).astype(np.int64), 2 * j_max) - j_max
    return to_f16_bits(1.0 + j * 2.0 ** -10).reshape(shape)


def images_f16(seed: int, N: int, H: int = 224, W: int = 224, C: int = 3) -> np.ndarray:
    """NHWC images, each channel ~ N(0, 1)."""
    return normal_f16(seed, (N, H, W, C))
