"""Seeded synthetic inputs shared by the oracle side and the CUDA side.

This module holds no arithmetic of the attention method itself: it only draws
random numbers and rounds them to the I/O dtype.  Both the CPU oracle and the
GPU path receive exactly the same (already rounded) values.

Generator: SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom
number generators", OOPSLA 2014).  Every tensor gets its own stream keyed by
(seed, name), so the order in which tensors are drawn does not matter.
Element k of a stream is mix(key + (k + 1) * GOLDEN), turned into a double in
[0, 1) from its top 53 bits; normals come from the Box-Muller transform applied
to consecutive pairs of uniforms.
"""
from __future__ import annotations

import math

import numpy as np

GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def _mix(z: np.ndarray) -> np.ndarray:
    z = z.astype(np.uint64, copy=True)
    with np.errstate(over="ignore"):
        z ^= z >> np.uint64(30)
        z *= _M1
        z ^= z >> np.uint64(27)
        z *= _M2
        z ^= z >> np.uint64(31)
    return z


def _fnv1a64(name: str) -> int:
    h = 0xCBF29CE484222325
    for byte in name.encode("utf-8"):
        h ^= byte
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def stream_key(seed: int, name: str) -> np.uint64:
    """Key of the stream for tensor `name` under integer `seed`."""
    with np.errstate(over="ignore"):
        s = np.array([(int(seed) & 0xFFFFFFFFFFFFFFFF)], dtype=np.uint64)
        k = _mix(s * GOLDEN + GOLDEN)[0] ^ np.uint64(_fnv1a64(name))
    return _mix(np.array([k], dtype=np.uint64))[0]


def raw_u64(seed: int, name: str, count: int) -> np.ndarray:
    key = stream_key(seed, name)
    idx = np.arange(1, count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix(key + idx * GOLDEN)


def uniform01(seed: int, name: str, count: int) -> np.ndarray:
    """Doubles in [0, 1) with 53 random bits."""
    return (raw_u64(seed, name, count) >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def uniform(seed: int, name: str, shape, lo: float, hi: float) -> np.ndarray:
    count = int(np.prod(shape)) if len(shape) else 1
    u = uniform01(seed, name, count)
    return (lo + (hi - lo) * u).reshape(shape)


def normal(seed: int, name: str, shape) -> np.ndarray:
    """Standard normal doubles (Box-Muller on pairs of uniforms)."""
    count = int(np.prod(shape)) if len(shape) else 1
    pairs = (count + 1) // 2
    u = uniform01(seed, name, 2 * pairs)
    u1 = 1.0 - u[0::2]  # in (0, 1]
    u2 = u[1::2]
    r = np.sqrt(-2.0 * np.log(u1))
    z = np.empty(2 * pairs, dtype=np.float64)
    z[0::2] = r * np.cos(2.0 * math.pi * u2)
    z[1::2] = r * np.sin(2.0 * math.pi * u2)
    return z[:count].reshape(shape)


def normal_at(seed: int, name: str, idx) -> np.ndarray:
    """Elements idx (flat indices) of the stream that `normal` draws, without drawing the others: the
    generator is counter-based, so element e takes uniforms 2*(e // 2) and 2*(e // 2) + 1 of its
    stream.  Equal, bit for bit, to normal(seed, name, shape).ravel()[idx]."""
    idx = np.asarray(idx, dtype=np.int64)
    key = stream_key(seed, name)
    pair = (idx // 2).astype(np.uint64)
    with np.errstate(over="ignore"):
        a = _mix(key + (np.uint64(2) * pair + np.uint64(1)) * GOLDEN)
        b = _mix(key + (np.uint64(2) * pair + np.uint64(2)) * GOLDEN)
    u1 = 1.0 - (a >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)
    u2 = (b >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)
    r = np.sqrt(-2.0 * np.log(u1))
    return np.where(idx % 2 == 0, r * np.cos(2.0 * math.pi * u2), r * np.sin(2.0 * math.pi * u2))


def randint(seed: int, name: str, shape, lo: int, hi: int) -> np.ndarray:
    """Integers uniform on [lo, hi] inclusive."""
    count = int(np.prod(shape)) if len(shape) else 1
    span = np.uint64(hi - lo + 1)
    v = raw_u64(seed, name, count) % span
    return (v.astype(np.int64) + lo).reshape(shape)


# ---------------------------------------------------------------------------
# rounding to the I/O dtype (round to nearest even)

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns (uint16), round to nearest even."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))
    with np.errstate(over="ignore"):
        return ((b + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


class IOTensor:
    """A tensor rounded to the I/O dtype.

    `value` holds the exact rounded values as float64 (what the oracle sees);
    `raw` holds the bytes handed to the device (float32 or bf16 bits).
    """

    def __init__(self, x64: np.ndarray, io: str):
        x32 = np.asarray(x64, dtype=np.float32)
        if io == "f32":
            self.raw = np.ascontiguousarray(x32)
            self.value = x32.astype(np.float64)
        elif io == "bf16":
            self.raw = f32_to_bf16_bits(x32)
            self.value = bf16_bits_to_f64(self.raw)
        else:
            raise ValueError(f"unknown io dtype {io!r}")
        self.io = io
        self.shape = tuple(x64.shape)


# ---------------------------------------------------------------------------
# parameter and input recipes

def phi_params(seed: int, d: int, M: int, L: int, hidden: int = 64, shared: bool = False) -> dict:
    """Feature-map parameters, initialised as the paper's listing does.

    W ~ N(0,1)/sqrt(d) and b = 0 for the projections; each channel MLP uses the
    documented default of a linear layer (uniform in +-1/sqrt(fan_in)):
    fc1 (fan_in 1) in U(-1, 1), fc2 (fan_in = hidden) in U(-1/sqrt(hidden), ...).
    With `shared`, one MLP serves all channels (the listing's shared_channels):
    fc1 has `hidden` units (w1, b1 of shape (hidden,)) and fc2 has L outputs.
    All values are rounded to fp32.
    """
    bound2 = 1.0 / math.sqrt(hidden)
    fc1 = (hidden,) if shared else (L, hidden)
    p = {
        "W": normal(seed, "phi.W", (M, d)) / math.sqrt(d),
        "b": np.zeros((M,)),
        "w1": uniform(seed, "phi.w1", fc1, -1.0, 1.0),
        "b1": uniform(seed, "phi.b1", fc1, -1.0, 1.0),
        "w2": uniform(seed, "phi.w2", (L, hidden), -bound2, bound2),
        "b2": uniform(seed, "phi.b2", (L,), -bound2, bound2),
    }
    return {k: np.ascontiguousarray(v, dtype=np.float32) for k, v in p.items()}


def attn_inputs(seed: int, B: int, H: int, n: int, d: int, dv: int, io: str,
                qkv_scale: float = 1.0, len_range=None, with_grad: bool = False) -> dict:
    """Q, K, V (and dO) of shape (B, H, n, d|dv), N(0,1)*qkv_scale, rounded to io.

    len_range=(lo, hi) draws one valid length per batch entry uniformly in
    [lo, hi]; None means every sequence is full length.
    """
    out = {
        "Q": IOTensor(normal(seed, "attn.Q", (B, H, n, d)) * qkv_scale, io),
        "K": IOTensor(normal(seed, "attn.K", (B, H, n, d)) * qkv_scale, io),
        "V": IOTensor(normal(seed, "attn.V", (B, H, n, dv)) * qkv_scale, io),
        "lengths": None,
    }
    if len_range is not None:
        out["lengths"] = randint(seed, "attn.lengths", (B,), len_range[0], len_range[1]).astype(np.int32)
    if with_grad:
        out["dO"] = IOTensor(normal(seed, "attn.dO", (B, H, n, dv)), io)
    return out
