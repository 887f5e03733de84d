"""Offline preparation of a QSVD layer: importance scores of singular values
(Sec. 3.2, Eq. 8-10), the cross-layer rank budget, and the per-layer choice
of beta (Sec. 3.3, Eq. 13-14).

Eq. 8: removing sigma_i changes W by dW_i = W - W'_i (W'_i: W with sigma_i set
to zero) and the loss by about <dW_i, G>_F, G the gradient of the loss at W.
Eq. 9: the importance score is the mean over calibration samples of that
change squared.  Eq. 10: since dW_i = sigma_i u_i v_i^T, the score equals the
mean of sigma_i^2 [U^T G V]_{ii}^2, which needs no E x E matrix per value.
The rank budget keeps the k highest-scoring singular values over all layers
(a global sort); every other one is truncated.

Eq. 14 picks beta per layer to minimise the squared difference between the
block output with and without quantization over calibration data.  Reading:
the block output is the joint QKV output Y = X W_concat (what the
factorisation approximates; W_o is not compressed), its quantized
counterpart Eq. 11's Y' = Q(C) Q(W^u) with C from Eq. 12 (H1 = H2 = I).

Test infrastructure: only tests/ use this module.
"""
from __future__ import annotations

import numpy as np

from . import latent, quant, svd


def importance_scores_definition(U, s, Vt, grads):
    """Eq. 9 from the definition: for each i, W'_i = U diag(s with s_i = 0) Vt,
    dW_i = W - W'_i, score_i = mean_n <dW_i, G_n>_F^2.  O(k m n) memory per
    value: tiny sizes only."""
    U, s, Vt = (np.asarray(a, dtype=np.float64) for a in (U, s, Vt))
    W = (U * s[None, :]) @ Vt
    scores = np.empty(len(s))
    for i in range(len(s)):
        s_cut = s.copy()
        s_cut[i] = 0.0
        dW = W - (U * s_cut[None, :]) @ Vt
        scores[i] = np.mean([np.sum(dW * np.asarray(G, dtype=np.float64)) ** 2 for G in grads])
    return scores


def importance_scores(U, s, Vt, grads):
    """Eq. 10: score_i = mean_n sigma_i^2 [U^T G_n V]_{ii}^2."""
    U, s, Vt = (np.asarray(a, dtype=np.float64) for a in (U, s, Vt))
    acc = np.zeros(len(s))
    for G in grads:
        diag = np.einsum("ji,jk,ik->i", U, np.asarray(G, dtype=np.float64), Vt)   # [U^T G V]_{ii}
        acc += (s * diag) ** 2
    return acc / len(grads)


def allocate_ranks(scores_per_layer, k: int):
    """Global top-k over every layer's scores.  Returns, per layer, the sorted
    indices of the singular values kept.  Ties go to the lower layer, then the
    lower index (a stable order)."""
    flat = [(-float(sc), layer, i) for layer, scores in enumerate(scores_per_layer) for i, sc in enumerate(scores)]
    if not 0 <= k <= len(flat):
        raise ValueError("rank budget outside [0, number of singular values]")
    kept = sorted(flat)[:k]
    out = [[] for _ in scores_per_layer]
    for _, layer, i in kept:
        out[layer].append(i)
    return [sorted(x) for x in out]


def quantized_qkv_error(W_q, W_k, W_v, r: int, beta: float, X, w_bits: int = 8, u_bits: int = 8,
                        lat_bits: int = 8, quantize: bool = True):
    """Eq. 14's objective for one beta on calibration rows X [N, E]:
    ||Y - Y'||_F^2 with Y = X W_concat and Y' = Q(C) Q(W^u) (Eq. 11-12):
    the factors of Eq. 3 at this beta, W_d quantized per output channel,
    X per token (int8), the latent per token (lat_bits), W^u per output
    channel (u_bits).  quantize=False gives the unquantized rank-r output."""
    W_d, U_q, U_k, U_v, _ = svd.joint_qkv_factors(W_q, W_k, W_v, r, beta)
    return qkv_error_from_factors(np.concatenate([W_q, W_k, W_v], axis=1), W_d,
                                  np.concatenate([U_q, U_k, U_v], axis=1), X, w_bits, u_bits, lat_bits, quantize)


def qkv_error_from_factors(W_concat, W_d, W_u, X, w_bits: int = 8, u_bits: int = 8, lat_bits: int = 8,
                           quantize: bool = True):
    """The objective of quantized_qkv_error for given factors W_d [E, r] and
    W^u [r, n] (Eq. 3 at one beta) of W_concat [E, n]."""
    X = np.asarray(X, dtype=np.float64)
    Y = X @ np.asarray(W_concat, dtype=np.float64)
    if not quantize:
        return float(np.sum((Y - (X @ W_d) @ W_u) ** 2))
    Wq, s_w = quant.quantize_columns(quant.f32(W_d), w_bits)
    out = latent.latent_project(quant.f32(X), Wq, s_w, lat_bits=lat_bits)
    C = latent.dequantize_latent(out["codes"], out["scale"], lat_bits)
    Uc, s_u = quant.quantize_columns(W_u, u_bits)
    Yq = C @ (Uc * s_u[None, :])
    return float(np.sum((Y - Yq) ** 2))


def beta_search(W_q, W_k, W_v, r: int, X, betas=tuple(np.round(np.linspace(0.0, 1.0, 11), 2)), **kw):
    """Eq. 14 by grid search: (best beta, {beta: objective}).  The joint SVD
    is taken once; Eq. 3 then gives the factors of every beta."""
    W_concat = np.concatenate([W_q, W_k, W_v], axis=1)
    Wd_r, sig, Wu_r = svd.truncated_svd(W_concat, r)
    errs = {}
    for b in betas:
        W_d, W_u = svd.factors_at_beta(Wd_r, sig, Wu_r, float(b))
        errs[float(b)] = qkv_error_from_factors(W_concat, W_d, W_u, X, **kw)
    best = min(errs, key=lambda b: (errs[b], b))
    return best, errs
