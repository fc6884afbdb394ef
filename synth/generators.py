"""Seeded, counter-based synthetic inputs (host side, numpy).

This module is shared input plumbing: it produces initial parameters and
per-step gradients for the tests and the benchmark.  It holds none of the
optimizer's arithmetic.  ``synth/synth_dev.cu`` implements the same
definition independently for the GPU so that full-size gradients never have
to cross the host link; a GPU test checks the two bit for bit.

Definition (every operation below is exact integer arithmetic or a single
IEEE-754 binary32 operation with round-to-nearest-even, so any conforming
implementation reproduces it bit for bit):

``mix(z)`` is the SplitMix64 output function (Steele, Lea & Flood, "Fast
splittable pseudorandom number generators", OOPSLA 2014), on uint64 with
wrap-around::

    z += 0x9E3779B97F4A7C15
    z  = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9
    z  = (z ^ (z >> 27)) * 0x94D049BB133111EB
    z  =  z ^ (z >> 31)

Keys and words, for seed ``s``, stream ``r`` (1 = gradients, 2 = initial
parameters), worker ``m``, step ``t`` and padded element index ``i``::

    key    = mix(mix(mix(s ^ r) ^ m) ^ t)
    e      = mix(key ^ i)
    word_k = mix(e ^ k)                     k = 0, 1, 2, ...

Standard normal ``Z(k0)`` (Irwin-Hall sum of twelve 16-bit uniforms taken
from words k0, k0+1, k0+2, four 16-bit lanes each, low lane first)::

    S = sum of the 12 lanes                 (integer, 0 .. 786420)
    Z = float32(2*S - 786420) * 2**-17      (both steps exact)

Mean 0, variance 1 - 2**-32, support [-6, 6].

Gradient kinds (``sigma`` rounded to float32 first):

* ``normal``:   g = Z(0) * sigma
* ``student_t3``: a = Z(3)*Z(3); a = a + Z(6)*Z(6); a = a + Z(9)*Z(9);
  a = a / 3; a = max(a, 2**-20); g = (Z(0) / sqrt(a)) * sigma
  (each product, sum, quotient and root rounded separately)
* ``normal_outliers``: g = Z(0) * sigma, then if the low 32 bits of word 12
  are below 42949673 (1 % of 2**32) g = g * 100

bf16 gradients are the float32 value rounded to nearest-even on its upper 16
bits.  Elements outside every tensor (alignment padding) are exactly 0.
"""
from __future__ import annotations

import numpy as np

GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
STREAM_GRAD = 1
STREAM_INIT = 2
KINDS = ("normal", "student_t3", "normal_outliers")
OUTLIER_THRESHOLD = 42949673
OUTLIER_FACTOR = np.float32(100.0)


def mix(z):
    """SplitMix64 output function on uint64 arrays (wrap-around)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = z + GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def key(seed: int, stream: int, m: int, t: int) -> np.uint64:
    k = mix(np.uint64(seed) ^ np.uint64(stream))
    k = mix(k ^ np.uint64(m))
    return mix(k ^ np.uint64(t))


def element_hash(k: np.uint64, idx) -> np.ndarray:
    return mix(np.uint64(k) ^ np.asarray(idx, dtype=np.uint64))


def word(e: np.ndarray, k: int) -> np.ndarray:
    return mix(e ^ np.uint64(k))


def normal(e: np.ndarray, k0: int) -> np.ndarray:
    """Irwin-Hall(12) standard normal from words k0..k0+2 (float32, exact)."""
    s = np.zeros(e.shape, np.int64)
    mask = np.uint64(0xFFFF)
    for k in range(k0, k0 + 3):
        w = word(e, k)
        for lane in range(4):
            s += ((w >> np.uint64(16 * lane)) & mask).astype(np.int64)
    num = (2 * s - 786420).astype(np.float32)          # exact: |num| < 2**24
    return num * np.float32(2.0 ** -17)                 # exact power of two


def _f32(x) -> np.float32:
    return np.float32(x)


def grad_values(kind: str, seed: int, m: int, t: int, idx, sigma: float) -> np.ndarray:
    """Float32 gradient g_t^m at padded element indices ``idx``."""
    e = element_hash(key(seed, STREAM_GRAD, m, t), idx)
    sg = _f32(sigma)
    if kind == "normal":
        return normal(e, 0) * sg
    if kind == "student_t3":
        z0 = normal(e, 0)
        z1, z2, z3 = normal(e, 3), normal(e, 6), normal(e, 9)
        a = z1 * z1
        a = a + z2 * z2
        a = a + z3 * z3
        a = a / np.float32(3.0)
        a = np.maximum(a, np.float32(2.0 ** -20))
        return (z0 / np.sqrt(a)) * sg
    if kind == "normal_outliers":
        g = normal(e, 0) * sg
        low = word(e, 12) & np.uint64(0xFFFFFFFF)
        out = low < np.uint64(OUTLIER_THRESHOLD)
        return np.where(out, g * OUTLIER_FACTOR, g).astype(np.float32)
    raise ValueError("unknown gradient kind %r" % kind)


def init_values(seed: int, idx, sigma: float = 0.02) -> np.ndarray:
    """Initial parameters x_0 ~ N(0, sigma) (float32) at padded indices."""
    e = element_hash(key(seed, STREAM_INIT, 0, 0), idx)
    return normal(e, 0) * _f32(sigma)


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest-even); returns the uint16 bit patterns."""
    b = np.ascontiguousarray(x, np.float32).view(np.uint32).astype(np.uint64)
    b = b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))
    return (b >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_bf16(x: np.ndarray) -> np.ndarray:
    return bf16_bits_to_f32(to_bf16_bits(x))


def in_tensor_mask(idx, offsets, numels) -> np.ndarray:
    """True where a padded index lies inside a tensor (not in padding)."""
    idx = np.asarray(idx, np.int64)
    keep = np.asarray(numels, np.int64) > 0          # zero-size tensors own no index
    offsets = np.asarray(offsets, np.int64)[keep]
    numels = np.asarray(numels, np.int64)[keep]
    pos = np.searchsorted(offsets, idx, side="right") - 1
    pos = np.clip(pos, 0, len(offsets) - 1)
    return (idx >= offsets[pos]) & (idx < offsets[pos] + numels[pos])


def grads(workload: dict, layout: dict, seed: int, m: int, t: int, idx) -> np.ndarray:
    """Gradient values (float32, already rounded to bf16 when the workload's
    gradients are bf16) for worker m, step t at padded indices idx; padding
    positions are 0."""
    g = grad_values(workload["grad_kind"], seed, m, t, idx, workload["grad_sigma"])
    if workload.get("grad_dtype", "f32") == "bf16":
        g = round_bf16(g)
    inside = in_tensor_mask(idx, layout["offsets"], layout["numels"])
    return np.where(inside, g, np.float32(0.0)).astype(np.float32)


def init_params(workload: dict, layout: dict, seed: int, idx) -> np.ndarray:
    x = init_values(seed, idx, workload.get("init_sigma", 0.02))
    inside = in_tensor_mask(idx, layout["offsets"], layout["numels"])
    return np.where(inside, x, np.float32(0.0)).astype(np.float32)


STREAM_TOY_NOISE = 3


def toy_noise(seed: int, m: int, t: int, idx) -> np.ndarray:
    """Standard normal noise of the toy objectives (stream 3), float32."""
    return normal(element_hash(key(seed, STREAM_TOY_NOISE, m, t), idx), 0)


def toy_grad(kind: str, x: np.ndarray, seed: int, t: int, sigma: float, lam=None,
             idx=None) -> np.ndarray:
    """Noisy gradient of a toy objective at the workers' parameters x
    ([M][n], any float type; computed in fp64):
      quadratic   f = sum_i lam_i x_i^2 / 2            g_i = lam_i x_i
      rosenbrock  f = sum_k (1-a_k)^2 + 100 (b_k - a_k^2)^2 over the pairs
                  (a_k, b_k) = (x_2k, x_2k+1)
    plus sigma * Z with Z from stream 3 at padded indices idx (default
    0..n-1; for Rosenbrock idx must hold whole pairs in order)."""
    x = np.asarray(x, np.float64)
    M, n = x.shape
    idx = np.arange(n) if idx is None else np.asarray(idx, np.int64)
    if kind == "quadratic":
        g = np.asarray(lam, np.float64)[None, :] * x
    elif kind == "rosenbrock":
        a, b = x[:, 0::2], x[:, 1::2]
        g = np.empty_like(x)
        g[:, 0::2] = 2.0 * (a - 1.0) - 400.0 * a * (b - a * a)
        g[:, 1::2] = 200.0 * (b - a * a)
    else:
        raise ValueError(kind)
    noise = np.stack([toy_noise(seed, m, t, idx) for m in range(M)]).astype(np.float64)
    return g + float(np.float32(sigma)) * noise
