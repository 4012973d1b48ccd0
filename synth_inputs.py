"""Seeded synthetic inputs for the DeepShift shift operators.

This module is shared by the CPU oracle, the CUDA path's tests and the
benchmark.  It only draws numbers: it holds none of the shift/flip
arithmetic of the method.  Every draw is counter based (splitmix64 of
``key + (i + 1) * GOLDEN``), so the same seed gives the same tensor on any
host (x86-64 or aarch64) and for any sub-range of indices.

Distributions follow the workloads of the DeepShift evaluation:

* activations and biases are int32 Q16.16 fixed point (Sec. 4: 16 integer and
  16 fraction bits), drawn directly as integers;
* shift codes p lie in [-15, 0] and sign codes s in {-1, 0, +1}
  (Sec. 4 shift range; Eq. 2 and Eq. 11 ternary sign);
* "geometric around c" means p = clip(c + G1 - G2, -15, 0) with G1, G2
  independent Geometric(1/2) counts on {0, 1, ...}.
"""
from __future__ import annotations

import numpy as np

MASK64 = (1 << 64) - 1
GOLDEN = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB

# Stream ids: one independent counter stream per tensor role.
STREAM_X = 1
STREAM_P = 2
STREAM_S = 3
STREAM_B = 4
STREAM_G2 = 5
STREAM_F = 6


def _mix(z: np.ndarray) -> np.ndarray:
    """splitmix64 finaliser on a uint64 array (wrapping arithmetic)."""
    z = z.astype(np.uint64, copy=True)
    with np.errstate(over="ignore"):
        z ^= z >> np.uint64(30)
        z *= np.uint64(_M1)
        z ^= z >> np.uint64(27)
        z *= np.uint64(_M2)
        z ^= z >> np.uint64(31)
    return z


def stream_key(seed: int, stream: int) -> int:
    """64-bit key of one stream of one seed."""
    z = np.array([(seed * GOLDEN + stream * 0xD1B54A32D192ED03) & MASK64], dtype=np.uint64)
    return int(_mix(z)[0])


def raw_u64(seed: int, stream: int, n: int, offset: int = 0) -> np.ndarray:
    """n uniform 64-bit words, element i = mix(key + (offset + i + 1) * GOLDEN)."""
    key = np.uint64(stream_key(seed, stream))
    idx = np.arange(offset + 1, offset + n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = key + idx * np.uint64(GOLDEN)
    return _mix(z)


def uniform_int(seed: int, stream: int, shape, lo: int, hi: int) -> np.ndarray:
    """Integers uniform in [lo, hi); hi - lo must be a power of two (exact, no bias)."""
    span = hi - lo
    if span <= 0 or span & (span - 1):
        raise ValueError("span must be a positive power of two")
    bits = span.bit_length() - 1
    n = int(np.prod(shape))
    w = raw_u64(seed, stream, n)
    if bits == 0:
        v = np.zeros(n, dtype=np.int64)
    else:
        v = (w >> np.uint64(64 - bits)).astype(np.int64)
    return (v + lo).reshape(shape)


def sign_codes(seed: int, shape, p_zero_num: int = 1, p_zero_den: int = 10) -> np.ndarray:
    """s in {-1, 0, +1}: P(0) = p_zero, P(-1) = P(+1) = (1 - p_zero) / 2.

    Decided on the top 32 bits t of each word with integer thresholds:
    s = 0 if t < T0, -1 if t < T0 + (2^32 - T0) // 2, else +1.
    """
    n = int(np.prod(shape))
    t = (raw_u64(seed, STREAM_S, n) >> np.uint64(32)).astype(np.int64)
    t0 = ((1 << 32) * p_zero_num) // p_zero_den
    t1 = t0 + ((1 << 32) - t0) // 2
    s = np.where(t < t0, 0, np.where(t < t1, -1, 1)).astype(np.int8)
    return s.reshape(shape)


def shift_codes_uniform(seed: int, shape, p_min: int = -15) -> np.ndarray:
    """p uniform in {p_min, ..., 0}; the count of values must be a power of two."""
    return uniform_int(seed, STREAM_P, shape, p_min, 1).astype(np.int8)


def _ctz64(words: np.ndarray) -> np.ndarray:
    """Trailing-zero count of each uint64 (64 for a zero word)."""
    w = words.astype(np.uint64)
    out = np.full(w.shape, 64, dtype=np.int64)
    nz = w != 0
    low = w & (~w + np.uint64(1))  # isolate lowest set bit (two's complement)
    # log2 of a power of two, exact via float64 for 2^0..2^63
    out[nz] = np.log2(low[nz].astype(np.float64)).astype(np.int64)
    return out


def shift_codes_geometric(seed: int, shape, centre: int = -6) -> np.ndarray:
    """p = clip(centre + G1 - G2, -15, 0), G1, G2 ~ Geometric(1/2) (two-sided geometric)."""
    n = int(np.prod(shape))
    g1 = _ctz64(raw_u64(seed, STREAM_P, n))
    g2 = _ctz64(raw_u64(seed, STREAM_G2, n))
    p = np.clip(centre + g1 - g2, -15, 0)
    return p.astype(np.int8).reshape(shape)


def activations(seed: int, shape, lo: int, hi: int) -> np.ndarray:
    """int32 Q16.16 activations uniform in [lo, hi)."""
    return uniform_int(seed, STREAM_X, shape, lo, hi).astype(np.int32)


def bias(seed: int, n: int, lo: int = -(1 << 16), hi: int = 1 << 16) -> np.ndarray:
    """int32 Q16.16 bias uniform in [lo, hi)."""
    return uniform_int(seed, STREAM_B, (n,), lo, hi).astype(np.int32)


def post_relu_activations(seed: int, shape, hi: int = 1 << 20, zero_frac_num: int = 1,
                          zero_frac_den: int = 2) -> np.ndarray:
    """Post-ReLU-like activations: exact zeros with the given fraction, else uniform in [0, hi)."""
    x = activations(seed, shape, 0, hi)
    n = int(np.prod(shape))
    t = (raw_u64(seed, STREAM_G2 + 10, n) >> np.uint64(32)).astype(np.int64)
    thr = ((1 << 32) * zero_frac_num) // zero_frac_den
    return np.where(t.reshape(shape) < thr, 0, x).astype(np.int32)


def bf16_bits(v: np.ndarray) -> np.ndarray:
    """uint16 bfloat16 bit patterns of float64 values (round to nearest even)."""
    f32 = v.astype(np.float32)
    u = f32.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    u = (u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)
    return u.astype(np.uint16)


def bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """float64 values of uint16 bfloat16 bit patterns (exact)."""
    u32 = bits.astype(np.uint32) << np.uint32(16)
    return u32.view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------
# Workload recipes (shapes and distributions of the evaluated configurations)
# --------------------------------------------------------------------------

def float32_from_fields(sign, exponent, mantissa) -> np.ndarray:
    """float32 values assembled from integer IEEE-754 fields (sign bit, unbiased
    exponent of a normal number, 23-bit mantissa): identical on every platform."""
    sign = np.asarray(sign, dtype=np.uint64)
    biased = (np.asarray(exponent, dtype=np.int64) + 127).astype(np.uint64)
    mant = np.asarray(mantissa, dtype=np.uint64)
    bits = (sign << np.uint64(31)) | (biased << np.uint64(23)) | mant
    return bits.astype(np.uint32).view(np.float32)


def float_weights(seed: int, shape, e_lo: int = -20, e_hi: int = 1) -> np.ndarray:
    """float32 weights with a random sign, a uniform 23-bit mantissa and an
    exponent uniform in [e_lo, e_hi] (a log-uniform magnitude), built from bit
    fields.  One word per element: bit 0 sign, bits 1-23 mantissa, bits 32-63
    the exponent draw."""
    n = int(np.prod(shape))
    w = raw_u64(seed, STREAM_F, n)
    span = e_hi - e_lo + 1
    sign = w & np.uint64(1)
    mant = (w >> np.uint64(1)) & np.uint64(0x7FFFFF)
    expo = e_lo + ((w >> np.uint64(32)) % np.uint64(span)).astype(np.int64)
    return float32_from_fields(sign, expo, mant).reshape(shape)


def float_activations(seed: int, shape, e_lo: int = -20, e_hi: int = 17) -> np.ndarray:
    """float32 activations as float_weights, plus exact Q16.16 rounding ties:
    every 8th element is (2k + 1) / 2^17 for a random |k| < 2^20."""
    x = float_weights(seed, shape, e_lo, e_hi).reshape(-1).copy()
    k = uniform_int(seed, STREAM_X, (x.size,), -(1 << 20), 1 << 20)
    ties = ((2 * k + 1).astype(np.float64) / float(1 << 17)).astype(np.float32)
    x[::8] = ties[::8]
    return x.reshape(shape)


SEED_BASE = 0xD5000000


def fc_layer(seed: int, M: int, K: int, N: int, x_lo: int, x_hi: int, geometric_centre=None):
    """One FC-shift layer: x [M,K] int32, s/p [N,K] int8, b [N] int32."""
    x = activations(seed, (M, K), x_lo, x_hi)
    s = sign_codes(seed, (N, K))
    if geometric_centre is None:
        p = shift_codes_uniform(seed, (N, K))
    else:
        p = shift_codes_geometric(seed, (N, K), geometric_centre)
    b = bias(seed, N)
    return x, s, p, b


def conv_layer(seed: int, N: int, C: int, H: int, W: int, K: int, R: int, S: int,
               x_lo: int = 0, x_hi: int = 1 << 20, centre: int = -6):
    """One conv-shift layer: x [N,C,H,W] int32, s/p [K,C,R,S] int8, b [K] int32."""
    x = activations(seed, (N, C, H, W), x_lo, x_hi)
    s = sign_codes(seed, (K, C, R, S))
    p = shift_codes_geometric(seed, (K, C, R, S), centre)
    b = bias(seed, K)
    return x, s, p, b


def config1(seed: int = SEED_BASE + 1):
    """Single FC-shift layer 64 x 784 -> 512, x uniform in [0, 2^20), uniform codes."""
    return fc_layer(seed, 64, 784, 512, 0, 1 << 20)


def config2(seed: int = SEED_BASE + 2, N: int = 32):
    """ResNet18 conv2_x-shaped 3x3 conv-shift: N x 64 x 56 x 56, stride 1, pad 1."""
    return conv_layer(seed, N, 64, 56, 56, 64, 3, 3, 0, 1 << 20, -6)


def config4_int(seed: int = SEED_BASE + 4, M: int = 8192, K: int = 4096, N: int = 4096):
    """Large FC-shift: M x K x N with signed x uniform in [-2^20, 2^20), uniform codes."""
    return fc_layer(seed, M, K, N, -(1 << 20), 1 << 20)


def layer_centre(c_in: int, r: int, s: int) -> int:
    """Per-layer shift centre -round(log2(C*R*S)/2) - 4 that keeps a chain in range."""
    fan_in = c_in * r * s
    return -int(np.floor(0.5 * np.log2(fan_in) + 0.5)) - 4


def network_params(shapes, seed: int):
    """Codes and biases for every shift layer of a network, in the given order.

    shapes: list of (K, C, R, S) for conv layers or (N, K) for FC layers.
    Layer i uses seed + i; shifts are geometric around the per-layer centre
    -round(log2(fan_in) / 2) - 4 (fan_in = C*R*S or K), which keeps chained
    activations inside the int32 range; signs as in every config.
    """
    params = []
    for i, shp in enumerate(shapes):
        sd = seed + i
        fan_in = int(np.prod(shp[1:]))
        centre = -int(np.floor(0.5 * np.log2(fan_in) + 0.5)) - 4
        s = sign_codes(sd, shp)
        p = shift_codes_geometric(sd, shp, centre)
        b = bias(sd, shp[0])
        params.append((s, p, b))
    return params


def image_batch(seed: int, n: int, c: int = 3, h: int = 224, w: int = 224):
    """Network input stand-in for ImageNet images: int32 uniform in [-2^17, 2^17) (signed, like normalised pixels)."""
    return activations(seed, (n, c, h, w), -(1 << 17), 1 << 17)
