"""Seeded synthetic inputs shared by the CPU oracle and the CUDA path.

This module only draws random numbers and lays out shapes. It holds none of the
method's arithmetic (no distances, means, quantisation or bit accounting), so the
oracle and the CUDA library can both consume its output without sharing code.

Random source: the SplitMix64 generator (Steele, Lea, Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014) evaluated counter-style: the i-th
output of a stream with key ``s`` is ``mix(s + (i + 1) * GOLDEN)``, which is
exactly the i-th output of a SplitMix64 generator seeded with ``s``. Counter
evaluation makes every draw a pure function of (key, position), so the numpy
implementation below vectorises without changing a single bit.

Normals come from the Box-Muller transform in fp64 and are rounded to fp32 once,
at the end. Conv weights are synthesised as a Gaussian mixture standing in for
trained VGG-16 / ResNet-18 3x3 layers (the paper's Section 4 models): ``P``
prototype kernels with iid N(0, sigma^2) entries, sigma = sqrt(2 / (9 p)) (He
fan-in), and every kernel = a uniformly chosen prototype + iid N(0, (0.3 sigma)^2)
noise.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List

import numpy as np

GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)

# Stream tags: independent streams for prototypes, prototype choice, noise and
# the initial-codeword selection of one layer.
TAG_PROTO = 1
TAG_CHOICE = 2
TAG_NOISE = 3
TAG_INIT = 4


def _mix(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function on a uint64 array (wrapping arithmetic)."""
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def stream_key(seed: int, tag: int) -> np.uint64:
    """Key of stream ``tag`` derived from a 64-bit seed."""
    s = np.array([(seed * 0x100000001B3 + tag) & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64)
    return _mix(s)[0]


def u64(key: np.uint64, start: int, count: int) -> np.ndarray:
    """Outputs ``start .. start+count-1`` of the SplitMix64 stream with ``key``."""
    i = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix(key + i * GOLDEN)


def uniform01(key: np.uint64, start: int, count: int) -> np.ndarray:
    """fp64 uniforms in the open interval (0, 1): (top 53 bits + 0.5) / 2^53."""
    return ((u64(key, start, count) >> np.uint64(11)).astype(np.float64) + 0.5) * (2.0 ** -53)


def normal(key: np.uint64, count: int) -> np.ndarray:
    """``count`` fp64 standard normals by Box-Muller (two per uniform pair)."""
    m = (count + 1) // 2
    u = uniform01(key, 0, 2 * m)
    r = np.sqrt(-2.0 * np.log(u[0::2]))
    th = 2.0 * math.pi * u[1::2]
    out = np.empty(2 * m, dtype=np.float64)
    out[0::2] = r * np.cos(th)
    out[1::2] = r * np.sin(th)
    return out[:count]


def below(key: np.uint64, count: int, bound: int) -> np.ndarray:
    """``count`` integers uniform in [0, bound) by 32x32 multiply-high (bound < 2^32)."""
    assert 0 < bound < 2 ** 32
    hi = u64(key, 0, count) >> np.uint64(32)
    return ((hi * np.uint64(bound)) >> np.uint64(32)).astype(np.int64)


@dataclasses.dataclass(frozen=True)
class Layer:
    """One 3x3 conv layer: p input channels, q output channels, K codewords."""

    name: str
    p: int
    q: int
    K: int
    prototypes: int
    seed: int

    @property
    def n(self) -> int:
        return self.p * self.q

    @property
    def sigma(self) -> float:
        return math.sqrt(2.0 / (9.0 * self.p))


@dataclasses.dataclass(frozen=True)
class Workload:
    """A named set of layers fitted with the same iteration count."""

    name: str
    layers: List[Layer]
    iters: int


def conv_weights(layer: Layer) -> np.ndarray:
    """fp32 kernel matrix of shape (n, 9), kernel i = output o, input c with i = o*p + c.

    This is the PyTorch ``[q][p][3][3]`` weight viewed as ``n`` rows of 9 floats.
    """
    n, P, sig = layer.n, layer.prototypes, layer.sigma
    proto = normal(stream_key(layer.seed, TAG_PROTO), P * 9).reshape(P, 9) * sig
    pick = below(stream_key(layer.seed, TAG_CHOICE), n, P)
    noise = normal(stream_key(layer.seed, TAG_NOISE), n * 9).reshape(n, 9) * (0.3 * sig)
    return (proto[pick] + noise).astype(np.float32)


def init_selection(n: int, K: int, seed: int) -> np.ndarray:
    """K distinct row indices in [0, n), by a partial Fisher-Yates shuffle.

    Step j swaps position j with j + r_j, r_j uniform in [0, n - j). The draws are
    positions 0..K-1 of the seed's TAG_INIT stream. Returned as int64.
    """
    assert 1 <= K <= n
    key = stream_key(seed, TAG_INIT)
    draws = u64(key, 0, K)
    span = np.arange(n, n - K, -1, dtype=np.uint64)
    r = (draws % span).astype(np.int64) + np.arange(K, dtype=np.int64)
    perm = {}
    out = np.empty(K, dtype=np.int64)
    for j in range(K):
        rj = int(r[j])
        vj = perm.get(j, j)
        vr = perm.get(rj, rj)
        out[j] = vr
        perm[rj] = vj
        perm[j] = vr
    return out


def _layer(name, p, q, K, cfg, li, proto=None):
    P = min(4 * K, p * q) if proto is None else proto
    return Layer(name, p, q, K, P, 1000 + cfg * 100 + li)


VGG16_3X3 = [(3, 64), (64, 64), (64, 128), (128, 128), (128, 256), (256, 256), (256, 256),
             (256, 512), (512, 512), (512, 512), (512, 512), (512, 512), (512, 512)]
RESNET18_3X3 = ([(64, 64)] * 4 + [(64, 128)] + [(128, 128)] * 3 + [(128, 256)] + [(256, 256)] * 3
                + [(256, 512)] + [(512, 512)] * 3)


def workload(cfg: int) -> Workload:
    """The five seeded workloads, numbered 1..5.

    1: one 64x64 layer, K=16, 64 prototypes, 10 iterations.
    2: one 256x256 layer (VGG-16 conv3_2 shape), K=256, 1024 prototypes, 20 iterations.
    3: the 13 VGG-16 3x3 layers, K_l = min(512, n_l // 4), 20 iterations.
    4: the 16 ResNet-18 3x3 layers, K_l = min(2^14, n_l // 4), 20 iterations.
    5: one 2048x2048 stress layer, K=65536, 262144 prototypes, 10 iterations.
    """
    if cfg == 1:
        return Workload("conv64x64_K16", [_layer("conv", 64, 64, 16, 1, 0, 64)], 10)
    if cfg == 2:
        return Workload("vgg16_conv3_2_256x256_K256", [_layer("conv3_2", 256, 256, 256, 2, 0)], 20)
    if cfg == 3:
        ls = [_layer(f"conv{i + 1}", p, q, min(512, p * q // 4), 3, i) for i, (p, q) in enumerate(VGG16_3X3)]
        return Workload("vgg16_13x3x3_K512", ls, 20)
    if cfg == 4:
        ls = [_layer(f"conv{i + 1}", p, q, min(2 ** 14, p * q // 4), 4, i) for i, (p, q) in enumerate(RESNET18_3X3)]
        return Workload("resnet18_16x3x3_K16384", ls, 20)
    if cfg == 5:
        return Workload("stress_2048x2048_K65536", [_layer("stress", 2048, 2048, 65536, 5, 0, 262144)], 10)
    raise ValueError(f"unknown workload {cfg}")


def layer_inputs(layer: Layer):
    """(W fp32 (n, 9), initial-codeword selection int64 (K,)) for one layer."""
    W = conv_weights(layer)
    sel = init_selection(layer.n, layer.K, layer.seed + 1)
    return W, sel


def random_kernels(n: int, d: int, seed: int, scale: float = 1.0) -> np.ndarray:
    """Plain iid N(0, scale^2) fp32 matrix (n, d) for edge-case tests."""
    return (normal(stream_key(seed, TAG_NOISE), n * d).reshape(n, d) * scale).astype(np.float32)


def random_counts(K: int, seed: int, high: int) -> np.ndarray:
    """int32 counts uniform in [0, high) for codebook-quantisation tests."""
    return below(stream_key(seed, TAG_CHOICE), K, high).astype(np.int32)
