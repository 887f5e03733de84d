"""Decode attention over the latent cache (Sec. 3.1, Eq. 5).

At a decode step the cache of sequence b holds the latent rows C (L x r) of
its L tokens, the current one last.  Eq. 5 recomputes K = C W^u_k and
V = C W^u_v; the query of the current token is q = c_L W^u_q (Eq. 11 uses the
quantized latent, so C here is the dequantized cache).  Per head h (columns
h*dh .. (h+1)*dh-1 of each up-projection) the output is the textbook

    o_h = softmax( K_h q_h * softmax_scale )^T V_h,

with softmax_scale = 1/sqrt(dh) and every cached token (the current one
included) attended.  ``decode_attention`` materialises K and V -- the plain
definition.  ``decode_attention_absorbed`` regroups the same products
(q~_h = W^u_k,h q_h, scores C q~_h, o_h = (p^T C) W^u_v,h) and exists only so
the tests can check the two agree.

``prefill_attention`` is the prompt's side of the same layer: every prompt
token queries the cache of its own sequence under a decoder's causal mask
(Fig. 2(f): the prompt's latents are cached, then attended).
"""
from __future__ import annotations

import math

import numpy as np


def softmax(s):
    s = np.asarray(s, dtype=np.float64)
    e = np.exp(s - np.max(s, axis=-1, keepdims=True))
    return e / np.sum(e, axis=-1, keepdims=True)


def decode_attention(C, U_q, U_k, U_v, H: int, dh: int, softmax_scale=None,
                     K=None, V=None):
    """One decode step for one sequence.  C: fp64 [L, r] dequantized latent
    rows, the current token last; U_*: fp64 [r, H*dh].  ``K``/``V`` may be
    passed when the caller already holds C @ U_k / C @ U_v (row t of each
    depends only on row t of C).  Returns o fp64 [H*dh]."""
    C = np.asarray(C, dtype=np.float64)
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    q = C[-1] @ U_q
    if K is None:
        K = C @ U_k
    if V is None:
        V = C @ U_v
    o = np.empty(H * dh)
    for h in range(H):
        sl = slice(h * dh, (h + 1) * dh)
        p = softmax((K[:, sl] @ q[sl]) * softmax_scale)
        o[sl] = p @ V[:, sl]
    return o


def decode_attention_absorbed(C, U_q, U_k, U_v, H: int, dh: int, softmax_scale=None):
    """The same step with U_k folded into the query and U_v applied last."""
    C = np.asarray(C, dtype=np.float64)
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    q = C[-1] @ U_q
    o = np.empty(H * dh)
    for h in range(H):
        sl = slice(h * dh, (h + 1) * dh)
        q_t = U_k[:, sl] @ q[sl]                 # q~_h in R^r
        p = softmax((C @ q_t) * softmax_scale)
        o_lat = p @ C                            # sum_t p_t c_t in R^r
        o[sl] = o_lat @ U_v[:, sl]
    return o


def decode_attention_loops(C, U_q, U_k, U_v, H: int, dh: int, softmax_scale=None):
    """Brute force with explicit scalar loops (tiny sizes only)."""
    C = [list(map(float, row)) for row in np.asarray(C, dtype=np.float64)]
    L, r = len(C), len(C[0])
    E = H * dh
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    Uq = np.asarray(U_q, dtype=np.float64).tolist()
    Uk = np.asarray(U_k, dtype=np.float64).tolist()
    Uv = np.asarray(U_v, dtype=np.float64).tolist()
    q = [sum(C[L - 1][j] * Uq[j][e] for j in range(r)) for e in range(E)]
    K = [[sum(C[t][j] * Uk[j][e] for j in range(r)) for e in range(E)] for t in range(L)]
    V = [[sum(C[t][j] * Uv[j][e] for j in range(r)) for e in range(E)] for t in range(L)]
    out = [0.0] * E
    for h in range(H):
        cols = range(h * dh, (h + 1) * dh)
        s = [sum(K[t][e] * q[e] for e in cols) * softmax_scale for t in range(L)]
        mx = max(s)
        w = [math.exp(x - mx) for x in s]
        z = sum(w)
        for e in cols:
            out[e] = sum(w[t] / z * V[t][e] for t in range(L))
    return np.array(out)


def prefill_attention(C, U_q, U_k, U_v, H: int, dh: int, softmax_scale=None, t0: int = 0):
    """Causal attention of the prompt tokens at positions t0 .. L-1 of one
    sequence, L = len(C) (C: fp64 [L, r] dequantized latent rows of
    positions 0 .. L-1).  The decoder's masked self-attention in matrix form:
    Q = C[t0:] U_q, K = C U_k, V = C U_v and per head h

        S_h = Q_h K_h^T * softmax_scale,  S_h[i, t] = -inf for t > t0 + i,
        O_h = softmax_rows(S_h) V_h.

    Returns fp64 [L - t0, H*dh]; row i is the output of position t0 + i."""
    C = np.asarray(C, dtype=np.float64)
    L = C.shape[0]
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    T = L - t0
    Q = C[t0:] @ U_q
    K = C @ U_k
    V = C @ U_v
    masked = np.arange(L)[None, :] > (t0 + np.arange(T))[:, None]    # keys after the query
    O = np.empty((T, H * dh))
    for h in range(H):
        sl = slice(h * dh, (h + 1) * dh)
        S = (Q[:, sl] @ K[:, sl].T) * softmax_scale
        S[masked] = -np.inf
        O[:, sl] = softmax(S) @ V[:, sl]
    return O
