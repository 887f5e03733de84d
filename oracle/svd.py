"""Truncated SVD and the joint-QKV factorisation (Sec. 3.1).

Eq. 1: W ~= U_r Sigma_r V_r^T keeps the r largest singular values.
Eq. 2: W_concat = [W_q, W_k, W_v] (E x 3E) ~= W^d_r Sigma_r W^u_r.
Eq. 3: W^d_qkv = W^d_r Sigma_r^beta,  W^u_qkv = Sigma_r^(1-beta) W^u_r,
       0 <= beta <= 1.
Eq. 4: [W_q, W_k, W_v] ~= W^d_qkv [W^u_q, W^u_k, W^u_v].

The SVD itself is a one-sided (Hestenes) Jacobi iteration written here, so
that it can be checked against numpy's LAPACK SVD as an independent routine.
"""
from __future__ import annotations

import numpy as np


def _round_robin(n: int):
    """n-1 rounds of n/2 disjoint column pairs covering every pair once
    (circle method; n even)."""
    idx = list(range(n))
    for _ in range(n - 1):
        yield [(idx[i], idx[n - 1 - i]) for i in range(n // 2)]
        idx = [idx[0]] + [idx[-1]] + idx[1:-1]


def jacobi_svd(A: np.ndarray, tol: float = 1e-15, max_sweeps: int = 60):
    """Thin SVD of A (m x n) by one-sided Jacobi rotations.

    Returns (U, s, Vt) with U (m x k), s (k,) descending, Vt (k x n),
    k = min(m, n), and A = U diag(s) Vt.
    """
    A = np.asarray(A, dtype=np.float64)
    m, n = A.shape
    if m < n:                       # work on the tall orientation
        U, s, Vt = jacobi_svd(A.T, tol, max_sweeps)
        return Vt.T, s, U.T
    npad = n + (n % 2)
    G = np.zeros((m, npad))
    G[:, :n] = A
    V = np.eye(npad)
    for _ in range(max_sweeps):
        rotated = False
        for pairs in _round_robin(npad):
            p = np.array([a for a, _ in pairs])
            q = np.array([b for _, b in pairs])
            gp, gq = G[:, p], G[:, q]
            alpha = np.einsum("ij,ij->j", gp, gp)
            beta = np.einsum("ij,ij->j", gq, gq)
            gamma = np.einsum("ij,ij->j", gp, gq)
            act = np.abs(gamma) > tol * np.sqrt(alpha * beta)
            act &= gamma != 0.0
            if not np.any(act):
                continue
            rotated = True
            zeta = np.where(act, (beta - alpha) / np.where(act, 2.0 * gamma, 1.0), 0.0)
            t = np.where(act, np.sign(zeta + (zeta == 0)) /
                         (np.abs(zeta) + np.sqrt(1.0 + zeta * zeta)), 0.0)
            c = 1.0 / np.sqrt(1.0 + t * t)
            s = c * t
            G[:, p], G[:, q] = c * gp - s * gq, s * gp + c * gq
            vp, vq = V[:, p], V[:, q]
            V[:, p], V[:, q] = c * vp - s * vq, s * vp + c * vq
        if not rotated:
            break
    sig = np.sqrt(np.einsum("ij,ij->j", G, G))[:n]
    G, V = G[:, :n], V[:n, :n]
    order = np.argsort(-sig, kind="stable")
    sig, G, V = sig[order], G[:, order], V[:, order]
    U = np.zeros_like(G)
    nz = sig > 0
    U[:, nz] = G[:, nz] / sig[nz]
    return U, sig, V.T


def truncated_svd(W: np.ndarray, r: int):
    """Eq. 1: the rank-r factors (U_r, sigma_r, V_r^T) of W."""
    U, s, Vt = jacobi_svd(W)
    return U[:, :r], s[:r], Vt[:r, :]


def joint_qkv_factors(W_q, W_k, W_v, r: int, beta: float):
    """Eq. 2-4: shared down-projection and per-block up-projections.

    Returns (W_d, U_q, U_k, U_v, sigma) with W_d = W^d_r Sigma_r^beta (E x r)
    and U_x = the x block of Sigma_r^(1-beta) W^u_r (r x E each).
    """
    if not 0.0 <= beta <= 1.0:
        raise ValueError("beta must lie in [0, 1] (Eq. 3)")
    W_concat = np.concatenate([W_q, W_k, W_v], axis=1)
    E = W_q.shape[1]
    Wd_r, sig, Wu_r = truncated_svd(W_concat, r)
    W_d, W_u = factors_at_beta(Wd_r, sig, Wu_r, beta)
    return W_d, W_u[:, :E], W_u[:, E:2 * E], W_u[:, 2 * E:], sig


def factors_at_beta(Wd_r, sig, Wu_r, beta: float):
    """Eq. 3 from the rank-r SVD factors: W_d = W^d_r Sigma_r^beta (E x r) and
    W^u = Sigma_r^(1-beta) W^u_r (r x n), in fp64."""
    if not 0.0 <= beta <= 1.0:
        raise ValueError("beta must lie in [0, 1] (Eq. 3)")
    sig = np.asarray(sig, dtype=np.float64)
    W_d = np.asarray(Wd_r, dtype=np.float64) * (sig ** beta)[None, :]
    W_u = (sig ** (1.0 - beta))[:, None] * np.asarray(Wu_r, dtype=np.float64)
    return W_d, W_u
