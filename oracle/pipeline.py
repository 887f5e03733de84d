"""Workload driver for the oracle: weight preparation, prefill, decode steps.

Weight preparation (offline in the paper, Sec. 3.1 and the Sec. 4 setup):
the tiny layer factors a Gaussian W_qkv by the joint SVD (Eq. 2-4, beta = 0.5
since the paper learns beta per layer and prints no value); every layer's
fp32 W_d is quantized per output channel to int8 (RTN, clip ratio 1.0), and
the up-projections are stored in bf16.

Decode order per step (every sequence gets one new token): project the new
tokens (Eq. 12), append their latent codes at position len[b], then attend
over positions 0..len[b] (Eq. 5).  K and V rows are computed once per token
when the token enters the cache: row t of C W^u depends only on row t of C,
so this is the definition evaluated row by row.
"""
from __future__ import annotations

import math
from typing import Dict, Iterable, Optional

import numpy as np

from synthetic import LayerInputs, bf16_bits, bf16_from_bits

from . import attention, latent, quant, rotate, svd

TINY_BETA = 0.5


def prepare_weights(inp: LayerInputs, beta: float = TINY_BETA, w_clip: float = 1.0, rot: int = 0,
                    u_bits: int = 0, w_bits: int = 8):
    """Returns dict(W_d fp32 values [d, r], Wq int64 [d, r], s_w [r],
    U_q/U_k/U_v bf16 bits [r, d], rot).  rot = b > 0: Wq, s_w quantize
    H1 W_d (oracle.rotate, block b) instead of W_d (W_d itself is returned
    unrotated: it is what the caller hands to the GPU's rotating quantizer).
    u_bits = 8 or 4: Eq. 11's Q(H2 W^u) as well (H2 = I): every column of
    U_q, U_k, U_v quantized per output channel (U*_codes, U*_scale), and the
    attention uses the dequantized values (U*_deq).  w_bits = 4: W_d's codes
    are int4 (with x_bits = 4 in OracleLayer, the W4A4 setting of Sec. 4)."""
    s = inp.workload.shape
    if inp.W_qkv is not None:
        d = s.d
        W_d, Uq, Uk, Uv, _ = svd.joint_qkv_factors(
            inp.W_qkv[:, :d], inp.W_qkv[:, d:2 * d], inp.W_qkv[:, 2 * d:], s.r, beta)
        W_d = quant.f32(W_d)
        U_q, U_k, U_v = bf16_bits(Uq), bf16_bits(Uk), bf16_bits(Uv)
    else:
        W_d, U_q, U_k, U_v = inp.W_d, inp.U_q, inp.U_k, inp.U_v
    Wq, s_w = quant.quantize_columns(rotate.rotate_weight(W_d, rot) if rot else W_d, w_bits, w_clip)
    c = np.ascontiguousarray
    out = dict(W_d=c(W_d), Wq=c(Wq), s_w=c(s_w), U_q=c(U_q), U_k=c(U_k), U_v=c(U_v), rot=rot, u_bits=u_bits,
               w_bits=w_bits)
    if u_bits:
        for k in ("U_q", "U_k", "U_v"):
            codes, scale = quantize_up(bf16_from_bits(out[k]), u_bits)
            out[k + "_codes"], out[k + "_scale"] = codes, scale
            out[k + "_deq"] = codes.astype(np.float64) * scale[None, :]
    return out


def quantize_up(U, bits: int = 8):
    """Eq. 11's Q(W^u) for one up-projection U [r, d] (bf16 values): symmetric
    RTN per output channel (column), the weight quantizer of the Sec. 4 setup.
    Returns (codes int64 [r, d], scale fp64 [d] holding fp32 values)."""
    return quant.quantize_columns(np.asarray(U, dtype=np.float64), bits)


class OracleLayer:
    """One layer's latent cache plus explicit K/V rows for tracked sequences."""

    def __init__(self, shape, weights: Dict, B: int, tmax: int, lat_bits: int,
                 act_clip: float = 1.0, lat_clip: float = 1.0,
                 track: Optional[Iterable[int]] = None, x_bits: int = 8):
        self.s = shape
        self.w = weights
        if weights.get("u_bits"):
            self.U_q, self.U_k, self.U_v = (weights[k + "_deq"] for k in ("U_q", "U_k", "U_v"))
        else:
            self.U_q = bf16_from_bits(weights["U_q"])
            self.U_k = bf16_from_bits(weights["U_k"])
            self.U_v = bf16_from_bits(weights["U_v"])
        self.B, self.tmax, self.bits = B, tmax, lat_bits
        self.act_clip, self.lat_clip, self.x_bits = act_clip, lat_clip, x_bits
        self.cache = latent.LatentCache(B, tmax, shape.r, lat_bits)
        self.len = np.zeros(B, dtype=np.int64)
        self.track = set(range(B)) if track is None else set(track)
        self.K = {b: np.zeros((tmax, shape.d)) for b in self.track}
        self.V = {b: np.zeros((tmax, shape.d)) for b in self.track}

    def project(self, X_bits):
        """Eq. 12 for a block of tokens given as bf16 bits [T, d]."""
        X = bf16_from_bits(X_bits)
        return latent.latent_project(X, self.w["Wq"], self.w["s_w"],
                                     self.act_clip, self.bits, self.lat_clip, self.w.get("rot", 0), self.x_bits)

    def _append(self, seq, pos, codes, scale):
        self.cache.append(seq, pos, codes, scale)
        for b in set(int(x) for x in seq) & self.track:
            sel = np.asarray(seq) == b
            rows = latent.dequantize_latent(codes[sel], scale[sel], self.bits)
            p = np.asarray(pos)[sel]
            self.K[b][p] = rows @ self.U_k
            self.V[b][p] = rows @ self.U_v

    def prefill(self, b: int, X_bits):
        """Project and cache the prompt of sequence b (positions len[b]...)."""
        out = self.project(X_bits)
        T = X_bits.shape[0]
        pos = self.len[b] + np.arange(T)
        self._append(np.full(T, b), pos, out["codes"], out["scale"])
        self.len[b] += T
        return out

    def attend(self, b: int):
        L = int(self.len[b])
        C = self.cache.rows(b, L)
        if b in self.track:
            return attention.decode_attention(C, self.U_q, self.U_k, self.U_v,
                                              self.s.H, self.s.dh,
                                              1.0 / math.sqrt(self.s.dh),
                                              K=self.K[b][:L], V=self.V[b][:L])
        return attention.decode_attention(C, self.U_q, self.U_k, self.U_v,
                                          self.s.H, self.s.dh)

    def decode_step(self, x_bits, attend: Optional[Iterable[int]] = None):
        """One decode step: x_bits [B, d] bf16 bits, one token per sequence.
        Returns (projection dict, {b: o_b}) for the sequences in ``attend``
        (default: the tracked ones)."""
        out = self.project(x_bits)
        seq = np.arange(self.B)
        self._append(seq, self.len.copy(), out["codes"], out["scale"])
        self.len += 1
        targets = sorted(self.track) if attend is None else list(attend)
        return out, {b: self.attend(b) for b in targets}
