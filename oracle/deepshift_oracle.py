"""CPU oracle for the DeepShift inference operators.  TEST INFRASTRUCTURE ONLY.

Only the tests, the smoke check and the benchmark's CPU-baseline leg may
import this module.  The CUDA library never calls it, and it shares no code
with the CUDA path.  It is plain and slow on purpose: every function spells
out the definition it follows in exact integer (int64 / Python int) or
float64 arithmetic, so a reader can check it against the paper by eye.

Definitions (DeepShift, Elhoushi et al.):

* Eq. 1 -- a shift by p (p <= 0 here, Sec. 4 clips p to [-15, 0]) of a
  fixed-point integer x is the two's-complement arithmetic right shift by -p,
  i.e. floor(x / 2^-p).
* Eq. 2 -- the ternary sign flip: flip(v, s) = -v, 0, v for s = -1, 0, +1.
* Eq. 3 -- LinearShift / ConvShift replace the weight W by flip(2^P, S):
  Y = flip(2^P, S) X + b and Y = flip(2^P, S) (*) X + b.
* Sec. 4 -- activations and bias are 32-bit fixed point with 16 fraction bits.
* Eq. 4-6 (DeepShift-Q) -- a float weight W becomes S = sign(W),
  P = round(log2|W|), W_q = flip(2^P, S); Sec. 4 clips P to the supported
  shift range ([-15, 0], or [-14, 0] for strict 5-bit codes).

Readings taken where the paper is silent:

* R-order: the integer term is s * (x >> -p): shift first, then flip.
* R-acc: the sum is exact (int64), then saturated to int32, then the
  optional ReLU is applied.
* R-conv: convolution is cross-correlation (PyTorch conv2d semantics), OIHW
  weights, zero padding, reduction index order (c, r, s).
* R-pool: max-pool ignores padded taps; average pool is floor(sum / count).
* R-round: round(log2|W|) is the integer n with 2^(n - 1/2) <= |W| < 2^(n + 1/2);
  the bound 2^(1/2) is irrational, so no float weight is a tie.  W = 0 and NaN
  give S = 0 and P = p_min (clip of -inf); W = +-inf gives S = +-1, P = 0.
* R-q16: the Sec. 4 rounding to fixed point is round-half-to-even of x * 2^16,
  saturated to the int32 range; NaN becomes 0.
* Eq. 7 (with its footnote) -- the input gradient of LinearShift is
  dC/dY W_q^T, of ConvShift W_q^rot180 (*) dC/dY.
* R-code5: the strict 5-bit storage of Sec. 4 (shifts in [-14, 0]) numbers the
  31 states 0 (zero weight), 1 + (-p) (s = +1) and 16 + (-p) (s = -1); the
  p of a zero weight is not stored and reads back as 0.
* R-bwd: the backward terms use the forward's fixed-point semantics: the
  Q16.16 gradient dy is shifted (floor) and flipped, s * (dy >> -p), the sum
  is exact, then saturated to int32.

Parity status: every function here is pinned by tests under
``tests/test_oracle_pins.py`` (brute force, float64 library routines on exact
cases, closed forms and invariants), except where a docstring says
"parity unpinned".
"""
from __future__ import annotations

import numpy as np

INT32_MIN = -(1 << 31)
INT32_MAX = (1 << 31) - 1
P_MIN = -15  # Sec. 4: shifts clipped to [-15, 0]
P_MAX = 0


# --------------------------------------------------------------------------
# Eq. 1 and Eq. 2 on one term
# --------------------------------------------------------------------------

def shift(x: int, p: int) -> int:
    """Eq. 1 for p <= 0: 2^p * x on a two's-complement integer = floor(x / 2^-p)."""
    if p > 0:
        raise ValueError("p > 0 is outside the Sec. 4 shift range")
    return x // (1 << (-p))


def flip(v: int, s: int) -> int:
    """Eq. 2: ternary sign flip."""
    if s == -1:
        return -v
    if s == 0:
        return 0
    if s == 1:
        return v
    raise ValueError("s must be -1, 0 or +1")


def term(x: int, s: int, p: int) -> int:
    """One shift-op term s * (x >> -p) (reading R-order: shift, then flip)."""
    return flip(shift(x, p), s)


def sat32(v):
    """Saturate to the int32 range (reading R-acc)."""
    return np.clip(v, INT32_MIN, INT32_MAX)


def _check_codes(s: np.ndarray, p: np.ndarray) -> None:
    """Rejects codes outside s in {-1, 0, +1} (Eq. 2) and p in [-15, 0] (Sec. 4 clipping; reading R-p+)."""
    if s.shape != p.shape:
        raise ValueError("s and p must have the same shape")
    if not np.isin(s, (-1, 0, 1)).all():
        raise ValueError("sign codes must be in {-1, 0, +1} (Eq. 2)")
    if ((p < P_MIN) | (p > P_MAX)).any():
        raise ValueError("shift codes must be in [-15, 0] (Sec. 4)")


# --------------------------------------------------------------------------
# LinearShift (Eq. 3, fully-connected form)
# --------------------------------------------------------------------------

def linear_shift_acc(x: np.ndarray, s: np.ndarray, p: np.ndarray, b=None) -> np.ndarray:
    """Exact int64 accumulator of LinearShift before saturation.

    acc[m, n] = b[n] + sum_k s[n, k] * floor(x[m, k] / 2^-p[n, k]).
    x: [M, K] integer; s, p: [N, K]; b: [N] or None.  Returns int64 [M, N].
    The loop runs over k; each step adds one term to every (m, n).
    Follows Eq. 3 (fully-connected form) with the terms of Eq. 1-2, reading R-order, summed exactly (reading R-acc).
    """
    x = np.asarray(x, dtype=np.int64)
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    _check_codes(s, p)
    M, K = x.shape
    N, K2 = s.shape
    if K != K2:
        raise ValueError("x and codes disagree on K")
    acc = np.zeros((M, N), dtype=np.int64)
    if b is not None:
        acc += np.asarray(b, dtype=np.int64)[None, :]
    for k in range(K):
        divisor = np.left_shift(np.int64(1), -p[:, k])          # 2^-p per output column
        shifted = np.floor_divide(x[:, k][:, None], divisor[None, :])  # Eq. 1
        acc += s[:, k][None, :] * shifted                         # Eq. 2 flip, then sum
    return acc


def linear_shift(x, s, p, b=None, relu: bool = False) -> np.ndarray:
    """LinearShift forward on Q16.16 int32: sat32(acc), then optional ReLU.  Returns int32.

    Follows Eq. 3 (fully-connected form) and reading R-acc (one saturation, after the bias)."""
    y = sat32(linear_shift_acc(x, s, p, b))
    if relu:
        y = np.maximum(y, 0)
    return y.astype(np.int32)


# --------------------------------------------------------------------------
# ConvShift (Eq. 3, convolutional form)
# --------------------------------------------------------------------------

def conv_out_size(h: int, r: int, stride: int, pad: int) -> int:
    """Output extent of the convolutional form of Eq. 3 (reading R-conv: zero padding, stride)."""
    return (h + 2 * pad - r) // stride + 1


def conv2d_shift_acc(x, s, p, b=None, stride=(1, 1), pad=(0, 0)) -> np.ndarray:
    """Exact int64 accumulator of ConvShift before saturation.

    acc[n, k, oh, ow] = b[k] + sum_{c, r, q} s[k, c, r, q] *
        floor(xpad[n, c, oh*sh + r, ow*sw + q] / 2^-p[k, c, r, q])
    with xpad the input zero-padded by pad on each side (reading R-conv).
    x: [N, C, H, W]; s, p: [K, C, R, S]; returns int64 [N, K, OH, OW].
    """
    x = np.asarray(x, dtype=np.int64)
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    _check_codes(s, p)
    N, C, H, W = x.shape
    K, C2, R, S = s.shape
    if C != C2:
        raise ValueError("x and codes disagree on C")
    sh, sw = stride
    ph, pw = pad
    OH = conv_out_size(H, R, sh, ph)
    OW = conv_out_size(W, S, sw, pw)
    xpad = np.zeros((N, C, H + 2 * ph, W + 2 * pw), dtype=np.int64)
    xpad[:, :, ph:ph + H, pw:pw + W] = x
    acc = np.zeros((N, K, OH, OW), dtype=np.int64)
    if b is not None:
        acc += np.asarray(b, dtype=np.int64)[None, :, None, None]
    for c in range(C):
        for r in range(R):
            for q in range(S):
                # input tap seen by every output pixel for this (c, r, q): [N, OH, OW]
                tap = xpad[:, c, r:r + sh * (OH - 1) + 1:sh, q:q + sw * (OW - 1) + 1:sw]
                divisor = np.left_shift(np.int64(1), -p[:, c, r, q])   # [K]
                shifted = np.floor_divide(tap[:, None, :, :], divisor[None, :, None, None])
                acc += s[:, c, r, q][None, :, None, None] * shifted
    return acc


def conv2d_shift(x, s, p, b=None, stride=(1, 1), pad=(0, 0), relu: bool = False) -> np.ndarray:
    """ConvShift forward on Q16.16 int32 NCHW: sat32(acc), then optional ReLU.  Returns int32.

    Follows Eq. 3 (convolutional form), readings R-conv and R-acc."""
    y = sat32(conv2d_shift_acc(x, s, p, b, stride, pad))
    if relu:
        y = np.maximum(y, 0)
    return y.astype(np.int32)


def conv2d_shift_at(x, s, p, b, stride, pad, n: int, k: int, oh: int, ow: int) -> int:
    """One output element of ConvShift (before saturation), as a Python int.

    Used to check sampled outputs of full-size launches one by one.
    Follows Eq. 3 (convolutional form) and reading R-conv, term by term with Eq. 1-2.
    """
    N, C, H, W = x.shape
    _, _, R, S = s.shape
    acc = int(b[k]) if b is not None else 0
    for c in range(C):
        for r in range(R):
            for q in range(S):
                ih = oh * stride[0] + r - pad[0]
                iw = ow * stride[1] + q - pad[1]
                v = int(x[n, c, ih, iw]) if (0 <= ih < H and 0 <= iw < W) else 0
                acc += term(v, int(s[k, c, r, q]), int(p[k, c, r, q]))
    return acc


def linear_shift_at(x, s, p, b, m: int, n: int) -> int:
    """One output element of LinearShift (before saturation), as a Python int.

    Follows Eq. 3 (fully-connected form), term by term with Eq. 1-2."""
    acc = int(b[n]) if b is not None else 0
    for k in range(x.shape[1]):
        acc += term(int(x[m, k]), int(s[n, k]), int(p[n, k]))
    return acc


# --------------------------------------------------------------------------
# Accumulator-width bound (reading R-acc): when int32 accumulation is exact
# --------------------------------------------------------------------------

def absmax(x) -> int:
    """max |x| over an int32 tensor, as a non-negative Python int (|INT32_MIN| = 2^31).

    The input bound of reading R-acc's int32 proof."""
    x = np.asarray(x, dtype=np.int64)
    return int(np.abs(x).max()) if x.size else 0


def column_constants(s, p):
    """Per output column n (rows of the [N, Kred] code matrix):

    A[n]   = sum_k |s[n,k]| * 2^(15 + p[n,k])   (sum of |weights| in units of 2^-15)
    nnz[n] = #{k : s[n,k] != 0}
    Column constants of reading R-acc's int32 proof (|s| 2^p is the magnitude of flip(2^P, S), Eq. 3).
    """
    s = np.asarray(s, dtype=np.int64).reshape(np.shape(s)[0], -1)
    p = np.asarray(p, dtype=np.int64).reshape(np.shape(p)[0], -1)
    A = (np.abs(s) * np.left_shift(np.int64(1), 15 + p)).sum(axis=1)
    nnz = (s != 0).sum(axis=1)
    return A.astype(np.int64), nnz.astype(np.int64)


def int32_accumulation_is_exact(amax: int, A: int, nnz: int, babs: int) -> bool:
    """True when |b| + sum |s * (x >> -p)| <= INT32_MAX for every |x| <= amax.

    |floor(x / 2^k)| <= ceil(|x| / 2^k) <= |x| / 2^k + 1 - 2^-k, so the sum is at
    most ceil(amax * A / 2^15) + nnz + |b|.
    Reading R-acc: when the exact sum provably fits int32, 32-bit accumulation is exact.
    """
    return ((amax * A + (1 << 15) - 1) >> 15) + nnz + babs <= INT32_MAX


# --------------------------------------------------------------------------
# Chain operators (pools, residual) for ResNet / VGG shaped forwards
# --------------------------------------------------------------------------

def maxpool2d(x, k: int, stride: int, pad: int) -> np.ndarray:
    """Integer max-pool; padded taps are ignored (reading R-pool)."""
    x = np.asarray(x, dtype=np.int64)
    N, C, H, W = x.shape
    OH = conv_out_size(H, k, stride, pad)
    OW = conv_out_size(W, k, stride, pad)
    out = np.full((N, C, OH, OW), np.iinfo(np.int64).min, dtype=np.int64)
    for r in range(k):
        for q in range(k):
            for oh in range(OH):
                ih = oh * stride + r - pad
                if not 0 <= ih < H:
                    continue
                for ow in range(OW):
                    iw = ow * stride + q - pad
                    if 0 <= iw < W:
                        out[:, :, oh, ow] = np.maximum(out[:, :, oh, ow], x[:, :, ih, iw])
    return out.astype(np.int32)


def avgpool_floor(x, k: int, stride: int) -> np.ndarray:
    """Integer average pool without padding: floor(sum / (k*k)) (reading R-pool)."""
    x = np.asarray(x, dtype=np.int64)
    N, C, H, W = x.shape
    OH = (H - k) // stride + 1
    OW = (W - k) // stride + 1
    out = np.zeros((N, C, OH, OW), dtype=np.int64)
    for oh in range(OH):
        for ow in range(OW):
            win = x[:, :, oh * stride:oh * stride + k, ow * stride:ow * stride + k]
            out[:, :, oh, ow] = np.floor_divide(win.sum(axis=(2, 3)), k * k)
    return out.astype(np.int32)


def add_relu(a, b) -> np.ndarray:
    """Residual join: ReLU(sat32(a + b)) on int32 tensors.

    Residual join of the ResNet chain (reading R-acc: one saturation, then ReLU; reading R-bn: no BatchNorm)."""
    v = sat32(np.asarray(a, dtype=np.int64) + np.asarray(b, dtype=np.int64))
    return np.maximum(v, 0).astype(np.int32)


# --------------------------------------------------------------------------
# Float variant (bf16 activations, weights s * 2^p, float64 reference)
# --------------------------------------------------------------------------

def linear_shift_float(x_f64, s, p, b=None) -> np.ndarray:
    """y[m, n] = b[n] + sum_k s[n,k] * 2^p[n,k] * x[m,k] in float64 (Eq. 3 with W = flip(2^P, S)).

    x_f64 holds the exact values of the bf16 activations.  Also returns nothing
    else: the tolerance scale sum |terms| comes from :func:`linear_shift_float_absterms`.
    """
    x = np.asarray(x_f64, dtype=np.float64)
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    _check_codes(s, p)
    M, K = x.shape
    N = s.shape[0]
    y = np.zeros((M, N), dtype=np.float64)
    if b is not None:
        y += np.asarray(b, dtype=np.float64)[None, :]
    for k in range(K):
        w = s[:, k].astype(np.float64) * np.ldexp(1.0, p[:, k])   # flip(2^p, s)
        y += x[:, k][:, None] * w[None, :]
    return y


def linear_shift_float_absterms(x_f64, s, p) -> np.ndarray:
    """sum_k |s * 2^p * x| per output, the scale of the float variant's tolerance.

    Scale of reading R-float's tolerance for Eq. 3 with W = flip(2^P, S)."""
    x = np.abs(np.asarray(x_f64, dtype=np.float64))
    w = np.abs(np.asarray(s, dtype=np.float64)) * np.ldexp(1.0, np.asarray(p, dtype=np.int64))
    return x @ w.T


# --------------------------------------------------------------------------
# Packed weight blob (the library's storage format for the codes of Eq. 3;
# layout documented in include/deepshift.h, format "planes6")
# --------------------------------------------------------------------------

BLOB_HEADER = 256
BLOB_MAGIC = 0x31575344
FORMAT_PLANES6 = 1


def blob_layout(n_out: int, k_red: int) -> dict:
    """Byte offsets of the regions of a planes6 blob.

    Storage of the codes of Eq. 3 (reading R-code: 4 shift bits, a sign plane and a non-zero plane)."""
    n_chunks = (k_red + 31) // 32
    nib = BLOB_HEADER
    bits = nib + n_chunks * n_out * 16
    col_a = bits + n_chunks * n_out * 8
    nnz = col_a + n_out * 8
    end = nnz + n_out * 4
    total = (end + 255) // 256 * 256
    return dict(n_chunks=n_chunks, nib=nib, bits=bits, col_a=col_a, nnz=nnz, total=total)


def pack_planes6(s, p) -> np.ndarray:
    """Pack [n_out, k_red] codes into the planes6 blob, one weight at a time.

    Returns the blob as uint8 [total].  The header carries magic, format, dims,
    invalid_count = 0, nnz_max and a_max.
    Storage format of reading R-code (6 bits per weight for the 33 code states of Eq. 2 and Sec. 4).
    """
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    _check_codes(s, p)
    n_out, k_red = s.shape
    L = blob_layout(n_out, k_red)
    nch = L["n_chunks"]
    nib = np.zeros((nch, n_out, 4), dtype=np.uint32)
    bits = np.zeros((nch, n_out, 2), dtype=np.uint32)
    for n in range(n_out):
        for k in range(k_red):
            g, j = divmod(k, 32)
            w, i = divmod(j, 8)
            nib[g, n, w] |= np.uint32((-p[n, k]) << (4 * i))
            if s[n, k] == -1:
                bits[g, n, 0] |= np.uint32(1 << j)
            if s[n, k] != 0:
                bits[g, n, 1] |= np.uint32(1 << j)
    A, nnz = column_constants(s, p)
    blob = np.zeros(L["total"], dtype=np.uint8)
    hdr = np.zeros(BLOB_HEADER, dtype=np.uint8)
    hdr[0:4] = np.frombuffer(np.uint32(BLOB_MAGIC).tobytes(), np.uint8)
    hdr[4:8] = np.frombuffer(np.uint32(FORMAT_PLANES6).tobytes(), np.uint8)
    hdr[8:32] = np.frombuffer(np.array([n_out, k_red, nch], dtype=np.int64).tobytes(), np.uint8)
    hdr[32:36] = 0  # invalid_count
    hdr[36:40] = np.frombuffer(np.uint32(int(nnz.max()) if n_out else 0).tobytes(), np.uint8)
    hdr[40:48] = np.frombuffer(np.uint64(int(A.max()) if n_out else 0).tobytes(), np.uint8)
    blob[:BLOB_HEADER] = hdr
    blob[L["nib"]:L["bits"]] = np.frombuffer(nib.tobytes(), np.uint8)
    blob[L["bits"]:L["col_a"]] = np.frombuffer(bits.tobytes(), np.uint8)
    blob[L["col_a"]:L["nnz"]] = np.frombuffer(A.astype(np.uint64).tobytes(), np.uint8)
    blob[L["nnz"]:L["nnz"] + 4 * n_out] = np.frombuffer(nnz.astype(np.uint32).tobytes(), np.uint8)
    return blob


def unpack_planes6(blob, n_out: int, k_red: int):
    """Inverse of pack_planes6 for the code regions: returns (s, p) int8 [n_out, k_red].

    Reading R-code, read back."""
    blob = np.asarray(blob, dtype=np.uint8)
    L = blob_layout(n_out, k_red)
    nch = L["n_chunks"]
    nib = np.frombuffer(blob[L["nib"]:L["bits"]].tobytes(), np.uint32).reshape(nch, n_out, 4)
    bits = np.frombuffer(blob[L["bits"]:L["col_a"]].tobytes(), np.uint32).reshape(nch, n_out, 2)
    s = np.zeros((n_out, k_red), dtype=np.int8)
    p = np.zeros((n_out, k_red), dtype=np.int8)
    for n in range(n_out):
        for k in range(k_red):
            g, j = divmod(k, 32)
            w, i = divmod(j, 8)
            p[n, k] = -int((int(nib[g, n, w]) >> (4 * i)) & 15)
            neg = (int(bits[g, n, 0]) >> j) & 1
            nz = (int(bits[g, n, 1]) >> j) & 1
            s[n, k] = 0 if not nz else (-1 if neg else 1)
    return s, p


# --------------------------------------------------------------------------
# Strict 5-bit storage (the paper's 5-bit count, Sec. 4, for shifts in
# [-14, 0]); layout documented in include/deepshift.h, format "codes5"
# --------------------------------------------------------------------------

FORMAT_CODES5 = 2
P_MIN_STRICT5 = -14


def code5(s: int, p: int) -> int:
    """The 5-bit code of one weight (reading R-code5): 0 for s = 0, 1 + (-p) for s = +1, 16 + (-p) for s = -1.

    With p in [-14, 0] a ternary sign times 15 shifts plus zero is 31 states, which fit 5 bits (Sec. 4: 4 shift
    bits and a sign bit; the zero weight takes the code a shift of -15 would need)."""
    s, p = int(s), int(p)
    if s == 0 and P_MIN <= p <= P_MAX:
        return 0
    if s not in (-1, 1) or not (P_MIN_STRICT5 <= p <= P_MAX):
        raise ValueError(f"(s, p) = ({s}, {p}) has no 5-bit code")
    return (1 if s == 1 else 16) + (-p)


def decode5(c: int):
    """Inverse of code5: (s, p), with p = 0 for the zero weight; code 31 is never written and decodes as None."""
    c = int(c)
    if c == 0:
        return 0, 0
    if 1 <= c <= 15:
        return 1, -(c - 1)
    if 16 <= c <= 30:
        return -1, -(c - 16)
    return None


def codes5_layout(n_out: int, k_red: int) -> dict:
    """Byte offsets of a codes5 blob: a 256-byte header, then n_out x n_chunks records of 5 u32 bit planes."""
    n_chunks = (k_red + 31) // 32
    planes = BLOB_HEADER
    end = planes + n_out * n_chunks * 20
    return dict(n_chunks=n_chunks, planes=planes, total=(end + 255) // 256 * 256)


def pack_codes5(s, p) -> np.ndarray:
    """Pack [n_out, k_red] codes into the codes5 blob, one weight at a time: record (n, g) holds, in word b, bit b
    of code5 of k = 32 g + j at bit j (zero beyond k_red).  Header: magic, format 2, n_out, k_red, n_chunks,
    invalid_count = 0.  Storage of reading R-code5."""
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    n_out, k_red = s.shape
    L = codes5_layout(n_out, k_red)
    nch = L["n_chunks"]
    rec = np.zeros((n_out, nch, 5), dtype=np.uint32)
    for n in range(n_out):
        for k in range(k_red):
            c = code5(s[n, k], p[n, k])
            g, j = divmod(k, 32)
            for b in range(5):
                if (c >> b) & 1:
                    rec[n, g, b] |= np.uint32(1 << j)
    blob = np.zeros(L["total"], dtype=np.uint8)
    blob[0:4] = np.frombuffer(np.uint32(BLOB_MAGIC).tobytes(), np.uint8)
    blob[4:8] = np.frombuffer(np.uint32(FORMAT_CODES5).tobytes(), np.uint8)
    blob[8:32] = np.frombuffer(np.array([n_out, k_red, nch], dtype=np.int64).tobytes(), np.uint8)
    blob[L["planes"]:L["planes"] + rec.nbytes] = np.frombuffer(rec.tobytes(), np.uint8)
    return blob


def unpack_codes5(blob, n_out: int, k_red: int):
    """Inverse of pack_codes5: (s, p) int8 [n_out, k_red], p = 0 where s = 0.  Reading R-code5, read back."""
    blob = np.asarray(blob, dtype=np.uint8)
    L = codes5_layout(n_out, k_red)
    nch = L["n_chunks"]
    rec = np.frombuffer(blob[L["planes"]:L["planes"] + n_out * nch * 20].tobytes(), np.uint32).reshape(n_out, nch, 5)
    s = np.zeros((n_out, k_red), dtype=np.int8)
    p = np.zeros((n_out, k_red), dtype=np.int8)
    for n in range(n_out):
        for k in range(k_red):
            g, j = divmod(k, 32)
            c = sum(((int(rec[n, g, b]) >> j) & 1) << b for b in range(5))
            d = decode5(c)
            if d is None:
                raise ValueError(f"code 31 at ({n}, {k})")
            s[n, k], p[n, k] = d
    return s, p


def expand_codes(s, p) -> np.ndarray:
    """Expanded execution layout of [n_out, k_red] codes (documented in include/deepshift.h):
    int32 [ceil(n_out/32)][k_red][64], words 0..31 = -p and 32..63 = s of columns 32*cb + c.
    Execution layout of the codes of Eq. 3 (-p and s per weight as 32-bit words)."""
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    _check_codes(s, p)
    n_out, k_red = s.shape
    nb = (n_out + 31) // 32
    out = np.zeros((nb, k_red, 64), dtype=np.int32)
    for n in range(n_out):
        cb, c = divmod(n, 32)
        out[cb, :, c] = -p[n, :]
        out[cb, :, 32 + c] = s[n, :]
    return out


def weights_bf16_bits(s, p) -> np.ndarray:
    """bf16 bit patterns of W = flip(2^P, S) (Eq. 3): sign bit of s, exponent 127 + p, zero mantissa; +0 for s = 0."""
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    _check_codes(s, p)
    bits = ((s < 0).astype(np.int64) << 15) | ((127 + p) << 7)
    return np.where(s == 0, 0, bits).astype(np.uint16)


# ---------------------------------------------------------------------------
# Float -> code and float -> Q16.16 conversion (the step before packing)
# ---------------------------------------------------------------------------
def quantize_weights(W, p_min: int = P_MIN):
    """DeepShift-Q quantizer (Eq. 4-6, clipping of Sec. 4) of float32 weights.

    s = sign(W); p = clip(round(log2|W|), p_min, 0) with the readings R-round.
    Written with frexp: |W| = m 2^e, m in [1/2, 1), so |W| = (2m) 2^(e-1) with
    2m in [1, 2) and log2|W| = (e - 1) + log2(2m); the fractional part rounds
    up exactly when 2m >= 2^(1/2), i.e. m^2 >= 1/2 (exact in float64: m has at
    most 24 significant bits).  Returns int8 arrays s, p of W's shape.
    """
    if not (P_MIN <= p_min <= P_MAX):
        raise ValueError("p_min outside [-15, 0]")
    w = np.asarray(W, dtype=np.float32).astype(np.float64)
    nan = np.isnan(w)
    s = np.where(nan, 0.0, np.sign(w)).astype(np.int8)
    a = np.abs(np.where(nan, 0.0, w))
    finite_nz = np.isfinite(a) & (a > 0)
    m, e = np.frexp(np.where(finite_nz, a, 1.0))
    r = (e.astype(np.int64) - 1) + (m * m >= 0.5)
    p = np.clip(r, p_min, P_MAX)
    p = np.where(np.isinf(a), P_MAX, p)
    p = np.where(a == 0, p_min, p)  # zero and NaN (mapped to 0 above)
    return s, p.astype(np.int8)


def quantize_activations(x) -> np.ndarray:
    """Float32 -> int32 Q16.16 (Sec. 4, reading R-q16): rint(x * 2^16), ties to
    even, saturated to [-2^31, 2^31 - 1], NaN -> 0.  x * 2^16 is exact in
    float64 for every float32 x."""
    y = np.asarray(x, dtype=np.float32).astype(np.float64) * 65536.0
    y = np.where(np.isnan(y), 0.0, np.rint(y))
    return np.clip(y, INT32_MIN, INT32_MAX).astype(np.int64).astype(np.int32)


# ---------------------------------------------------------------------------
# Input gradient (Eq. 7 and its footnote), reading R-bwd
# ---------------------------------------------------------------------------
def linear_shift_backward_x_acc(dy, s, p) -> np.ndarray:
    """Exact int64 dC/dX of LinearShift: dx[m, k] = sum_n s[n, k] * floor(dy[m, n] / 2^-p[n, k]),
    i.e. dC/dY W_q^T with every product a shift and a flip.  dy: [M, N]; s, p: [N, K].
    Follows Eq. 7 (fully-connected form) with reading R-bwd."""
    dy = np.asarray(dy, dtype=np.int64)
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    _check_codes(s, p)
    M, N = dy.shape
    N2, K = s.shape
    if N != N2:
        raise ValueError("dy and codes disagree on N")
    acc = np.zeros((M, K), dtype=np.int64)
    for n in range(N):
        divisor = np.left_shift(np.int64(1), -p[n])  # [K]
        acc += s[n][None, :] * np.floor_divide(dy[:, n][:, None], divisor[None, :])
    return acc


def linear_shift_backward_x(dy, s, p) -> np.ndarray:
    """Eq. 7 (fully-connected form) with reading R-bwd: sat32 of the exact sum."""
    return sat32(linear_shift_backward_x_acc(dy, s, p)).astype(np.int32)


def conv2d_shift_backward_x_acc(dy, s, p, in_hw, stride=(1, 1), pad=(0, 0)) -> np.ndarray:
    """Exact int64 dC/dX of ConvShift, written as the scatter the forward gather
    implies: output (n, k, oh, ow) read input (c, oh*sh + r - ph, ow*sw + q - pw)
    through code (k, c, r, q), so its gradient term s * floor(dy / 2^-p) is added
    there (positions in the padding are dropped).  dy: [N, K, OH, OW];
    s, p: [K, C, R, S]; in_hw = (H, W); returns int64 [N, C, H, W].
    Follows Eq. 7 and its footnote (convolutional form) with reading R-bwd."""
    dy = np.asarray(dy, dtype=np.int64)
    s = np.asarray(s, dtype=np.int64)
    p = np.asarray(p, dtype=np.int64)
    _check_codes(s, p)
    N, K, OH, OW = dy.shape
    K2, C, R, S = s.shape
    H, W = in_hw
    sh, sw = stride
    ph, pw = pad
    if K != K2 or OH != conv_out_size(H, R, sh, ph) or OW != conv_out_size(W, S, sw, pw):
        raise ValueError("dy, codes and geometry disagree")
    gpad = np.zeros((N, C, H + 2 * ph + sh, W + 2 * pw + sw), dtype=np.int64)  # padded input grid
    for k in range(K):
        for r in range(R):
            for q in range(S):
                divisor = np.left_shift(np.int64(1), -p[k, :, r, q])  # [C]
                terms = s[k, :, r, q][None, :, None, None] * np.floor_divide(
                    dy[:, k][:, None, :, :], divisor[None, :, None, None])  # [N, C, OH, OW]
                gpad[:, :, r:r + sh * (OH - 1) + 1:sh, q:q + sw * (OW - 1) + 1:sw] += terms
    return gpad[:, :, ph:ph + H, pw:pw + W]


def conv2d_shift_backward_x(dy, s, p, in_hw, stride=(1, 1), pad=(0, 0)) -> np.ndarray:
    """Eq. 7 and its footnote (convolutional form) with reading R-bwd: sat32 of the exact sum."""
    return sat32(conv2d_shift_backward_x_acc(dy, s, p, in_hw, stride, pad)).astype(np.int32)


def backward_codes(s, p):
    """Code matrix of the input-gradient pass as a forward layer (Eq. 7 footnote):
    column c, reduction index (k, r, q) holds the code of (k, c, R-1-r, S-1-q),
    i.e. W^rot180 with the channel axes swapped.  s, p: [K, C, R, S] (FC:
    [N, K] is taken as [N, K, 1, 1]); returns [C, K, R, S] int8 arrays."""
    s = np.asarray(s)
    p = np.asarray(p)
    if s.ndim == 2:
        s, p = s[:, :, None, None], p[:, :, None, None]
    st = np.ascontiguousarray(np.transpose(s[:, :, ::-1, ::-1], (1, 0, 2, 3)))
    pt = np.ascontiguousarray(np.transpose(p[:, :, ::-1, ::-1], (1, 0, 2, 3)))
    return st.astype(np.int8), pt.astype(np.int8)


def phase_taps(R: int, stride: int, a: int) -> int:
    """Number of taps r = a, a + stride, ... below R.

    Tap count of one phase of a strided input gradient (Eq. 7 footnote, split by stride phase)."""
    return (R - 1 - a) // stride + 1 if a < R else 0


def backward_phase_codes(s, p, stride):
    """Input-gradient codes of a strided layer split by tap phase (a layout,
    following Eq. 7's footnote): input row i = sh i' + rho receives only the
    taps r = a + sh t, a = (rho + pad) mod sh.  For each phase (a, b) returns
    [C, K, Th, Tw] arrays whose index (k, t, u) holds the code of
    (k, c, a + sh (Th-1-t), b + sw (Tw-1-u)) -- rot180 of the phase's taps,
    channels swapped -- or None when no tap has that phase.  Stride 1: the
    single phase equals backward_codes."""
    s = np.asarray(s)
    p = np.asarray(p)
    if s.ndim == 2:
        s, p = s[:, :, None, None], p[:, :, None, None]
    K, C, R, S = s.shape
    sh, sw = stride
    out = {}
    for a in range(sh):
        for b in range(sw):
            th, tw = phase_taps(R, sh, a), phase_taps(S, sw, b)
            if th == 0 or tw == 0:
                out[(a, b)] = None
                continue
            rows = [a + sh * (th - 1 - t) for t in range(th)]
            cols = [b + sw * (tw - 1 - u) for u in range(tw)]
            ss = s[:, :, rows][:, :, :, cols]
            pp = p[:, :, rows][:, :, :, cols]
            out[(a, b)] = (np.ascontiguousarray(np.transpose(ss, (1, 0, 2, 3))).astype(np.int8),
                           np.ascontiguousarray(np.transpose(pp, (1, 0, 2, 3))).astype(np.int8))
    return out
