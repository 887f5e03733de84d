"""Symmetric round-to-nearest quantizers (Sec. 4 setup; Eq. 11-12).

The paper quantizes activations per token, symmetrically, and weights per
output channel with round-to-nearest (RTN) and a clipping ratio.  It does not
fix the arithmetic, so this oracle takes the following readings (each is a
choice the GPU path must reproduce bit for bit):

* symmetric range +-(2^(b-1) - 1): [-127, 127] for 8 bits, [-7, 7] for 4;
* scale  s = fp32( fp32(c * m) / q_max ),  m = max |v| over the row (exact),
  c the clipping ratio (an fp32 number);
* code   = clamp( round_half_even( fp32(v / s) ), -q_max, q_max );
* a row with s == 0 (all zeros, or a scale that underflowed) gets all-zero
  codes;
* int4 latent groups of 128 channels keep an fp16 scale: the fp32 scale is
  rounded to fp16 (nearest even), saturated at 65504, and the codes divide by
  that fp16 value widened to fp32.

Every fp32 operation is emulated by computing the fp64 result and rounding it
to fp32 (``f32``); for a single +, x or / of fp32 operands this equals the
IEEE fp32 result.
"""
from __future__ import annotations

import numpy as np

INT4_GROUP = 128
FP16_MAX = 65504.0


def f32(x):
    """Round fp64 value(s) to the nearest fp32 (ties to even); fp64 result."""
    return np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)


def f16(x):
    """fp32 value(s) -> nearest fp16 (ties to even), saturated at 65504."""
    with np.errstate(over="ignore"):
        h = f32(x).astype(np.float32).astype(np.float16).astype(np.float64)
    return np.where(np.isinf(h), np.sign(h) * FP16_MAX, h)


def qmax(bits: int) -> int:
    if bits not in (4, 8):
        raise ValueError("bits must be 4 or 8")
    return (1 << (bits - 1)) - 1


def _codes(v, s, q):
    """code = clamp(rne(fp32(v / s)), -q, q); zero where s == 0."""
    s = np.asarray(s, dtype=np.float64)
    safe = np.where(s == 0.0, 1.0, s)
    c = np.clip(np.rint(f32(v / safe)), -q, q)
    return np.where(s == 0.0, 0.0, c).astype(np.int64)


def quantize_rows(V, bits: int, clip: float = 1.0):
    """Per-row (per-token) symmetric RTN.  V: [..., n] fp32 values.

    Returns (codes int64 [..., n], scale fp64 [...] holding fp32 values).
    """
    V = np.asarray(V, dtype=np.float64)
    q = qmax(bits)
    m = np.max(np.abs(V), axis=-1) if V.shape[-1] else np.zeros(V.shape[:-1])
    s = f32(f32(np.float64(np.float32(clip)) * m) / q)
    return _codes(V, s[..., None], q), s


def quantize_columns(W, bits: int = 8, clip: float = 1.0):
    """Per-output-channel symmetric RTN of a weight W [d_in, d_out]: one scale
    per column j (the channel of the row-vector product x W)."""
    codes, s = quantize_rows(np.asarray(W, dtype=np.float64).T, bits, clip)
    return codes.T, s


def quantize_int4_groups(V, clip: float = 1.0, group: int = INT4_GROUP):
    """int4 with one fp16 scale per `group` consecutive channels of a row.

    V: [T, n] fp32 values, n % group == 0.  Returns (codes int64 [T, n],
    scales fp64 [T, n/group] holding fp16 values).
    """
    V = np.asarray(V, dtype=np.float64)
    T, n = V.shape
    if n % group:
        raise ValueError("channel count must be a multiple of the group size")
    Vg = V.reshape(T, n // group, group)
    m = np.max(np.abs(Vg), axis=-1)
    s16 = f16(f32(f32(np.float64(np.float32(clip)) * m) / 7))
    codes = _codes(Vg, s16[..., None], 7)
    return codes.reshape(T, n), s16


def dequantize_rows(codes, scale):
    """fp64 code * scale (per row)."""
    return np.asarray(codes, np.float64) * np.asarray(scale, np.float64)[..., None]


def dequantize_int4_groups(codes, s16, group: int = INT4_GROUP):
    c = np.asarray(codes, np.float64)
    T, n = c.shape
    return (c.reshape(T, n // group, group) * np.asarray(s16, np.float64)[..., None]).reshape(T, n)


def pack_int4(codes):
    """Two's-complement nibbles, element 2i in the low nibble of byte i and
    element 2i+1 in the high nibble.  codes [..., n] (n even) -> uint8 [..., n/2]."""
    c = np.asarray(codes, dtype=np.int64)
    lo = c[..., 0::2] & 0xF
    hi = c[..., 1::2] & 0xF
    return (lo | (hi << 4)).astype(np.uint8)


def unpack_int4(packed):
    p = np.asarray(packed, dtype=np.int64)
    lo = p & 0xF
    hi = (p >> 4) & 0xF
    lo = np.where(lo >= 8, lo - 16, lo)
    hi = np.where(hi >= 8, hi - 16, hi)
    out = np.empty(p.shape[:-1] + (2 * p.shape[-1],), dtype=np.int64)
    out[..., 0::2] = lo
    out[..., 1::2] = hi
    return out
