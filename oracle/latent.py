"""The quantized joint down-projection and the latent cache (Sec. 3.1, 3.3).

Eq. 12: C_qkv ~= Q(X H1^T) Q(H1 W^d_qkv H2^T).  H2 folds offline into the
weights (Sec. 2.3 background: X' = XH with the matching H^T applied to W).
H1 is either folded too (H1 = I here: C_qkv ~= Q(X) Q(W_d)) or applied to X
on the fly (``rot``, oracle.rotate) with W_d replaced by H1 W_d:

  1. X [T, d] -> int8 codes Xq (int4 in the W4A4 setting, with int4 codes
     of W_d too) and an fp32 scale s_x per token;
  2. acc[t, j] = sum_k Xq[t, k] * Wq[k, j]      (exact integer arithmetic);
  3. c_hat[t, j] = fp32( fp32( fp32(acc[t,j]) * s_x[t] ) * s_w[j] );
  4. Eq. 11's Q(C_qkv): c_hat is quantized per token again -- int8 with one
     fp32 scale per token, or int4 with one fp16 scale per 128 channels --
     and those codes are what the latent buffer (the KV cache of Fig. 2(f),
     eta_qsvd = rL) stores.
"""
from __future__ import annotations

import numpy as np

from . import quant, rotate


def int_matmul(A, B):
    """Exact integer product of int64 matrices.  Uses fp64 BLAS on the
    integer values; exact because every partial sum of these products is an
    integer of magnitude below 2^53 (checked)."""
    A = np.asarray(A, dtype=np.int64)
    B = np.asarray(B, dtype=np.int64)
    bound = int(np.abs(A).max(initial=0)) * int(np.abs(B).max(initial=0)) * A.shape[-1]
    if bound >= 2 ** 53:
        raise OverflowError("integer GEMM would leave the exact fp64 range")
    return np.rint(A.astype(np.float64) @ B.astype(np.float64)).astype(np.int64)


def quantize_activations(X, act_clip: float = 1.0, x_bits: int = 8):
    """Step 1: per-token codes (int8, or int4 for the W4A4 setting of the
    Sec. 4 setup) and fp32 scales of X (bf16 values)."""
    return quant.quantize_rows(X, x_bits, act_clip)


def down_project(Xq, Wq):
    """Step 2: acc = Xq @ Wq with Wq [d, r] int8 or int4 codes (int64 result)."""
    return int_matmul(Xq, Wq)


def dequantize_acc(acc, s_x, s_w):
    """Step 3: c_hat = (fp32(acc) * s_x[t]) * s_w[j], fp32 at each step."""
    a32 = quant.f32(np.asarray(acc, dtype=np.float64))     # int -> fp32, nearest even
    return quant.f32(quant.f32(a32 * np.asarray(s_x)[:, None]) * np.asarray(s_w)[None, :])


def requantize_latent(c_hat, lat_bits: int, lat_clip: float = 1.0):
    """Step 4: codes and scales the latent cache stores for each token.

    int8: (codes int64 [T, r], scale fp32 [T]);
    int4: (codes int64 [T, r], scale fp16 [T, r/128]).
    """
    if lat_bits == 8:
        return quant.quantize_rows(c_hat, 8, lat_clip)
    if lat_bits == 4:
        return quant.quantize_int4_groups(c_hat, lat_clip)
    raise ValueError("lat_bits must be 8 or 4")


def latent_project(X, Wq, s_w, act_clip=1.0, lat_bits=8, lat_clip=1.0, rot: int = 0, x_bits: int = 8):
    """Steps 1-4 for a block of tokens.  Returns a dict with every
    intermediate the GPU path can expose: xq, s_x, acc, c_hat, codes, scale.
    rot = b > 0: the rows are rotated by H1 (block b, oracle.rotate) before
    step 1, as Eq. 12 quantizes X H1^T; Wq must then be the codes of H1 W^d.
    x_bits = 4 with 4-bit Wq is the W4A4 setting (Sec. 4 setup)."""
    if rot:
        X = rotate.rotate_rows(np.asarray(X, dtype=np.float32), rot)
    xq, s_x = quantize_activations(X, act_clip, x_bits)
    acc = down_project(xq, Wq)
    c_hat = dequantize_acc(acc, s_x, s_w)
    codes, scale = requantize_latent(c_hat, lat_bits, lat_clip)
    return dict(xq=xq, s_x=s_x, acc=acc, c_hat=c_hat, codes=codes, scale=scale)


def dequantize_latent(codes, scale, lat_bits: int):
    """The latent value a cached token stands for, in fp64."""
    if lat_bits == 8:
        return quant.dequantize_rows(codes, scale)
    return quant.dequantize_int4_groups(codes, scale)


class LatentCache:
    """Latent buffer of one layer: per sequence b, positions 0..Tmax-1 hold
    codes and scales of C_qkv rows (never K or V)."""

    def __init__(self, B: int, tmax: int, r: int, lat_bits: int):
        self.B, self.tmax, self.r, self.bits = B, tmax, r, lat_bits
        self.codes = np.zeros((B, tmax, r), dtype=np.int64)
        if lat_bits == 8:
            self.scale = np.zeros((B, tmax), dtype=np.float64)
        else:
            self.scale = np.zeros((B, tmax, r // quant.INT4_GROUP), dtype=np.float64)

    def append(self, seq, pos, codes, scale):
        """Write rows i of (codes, scale) at (seq[i], pos[i])."""
        seq = np.asarray(seq)
        pos = np.asarray(pos)
        if np.any(pos < 0) or np.any(pos >= self.tmax):
            raise IndexError("cache position out of range")
        self.codes[seq, pos] = codes
        self.scale[seq, pos] = scale

    def rows(self, b: int, L: int):
        """Dequantized latent rows 0..L-1 of sequence b (fp64 [L, r])."""
        return dequantize_latent(self.codes[b, :L], self.scale[b, :L], self.bits)

    def packed_codes(self):
        """Storage image of the codes: int8 [B, Tmax, r] or packed uint8
        [B, Tmax, r/2] for int4."""
        if self.bits == 8:
            return self.codes.astype(np.int8)
        return quant.pack_int4(self.codes)
