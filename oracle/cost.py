"""Hardware-cost model of Sec. 3.1 and the ratios of Eq. 15.

Single-head accounting with embedding size E, sequence length L, rank r:

* original  : alpha_fp   = 3 E^2   (weights), eta_fp   = 2 L E (KV cache),
              gamma_fp   = 3 L E^2 (FLOPs of the Q/K/V projections);
* QSVD      : alpha_qsvd = 4 r E,  eta_qsvd = r L,  gamma_qsvd = 4 L r E;
* per-matrix: alpha_ind  = 6 r E,  eta_ind  = 2 r L, gamma_ind  = 6 L r E.

Eq. 15: R1 = alpha_i / alpha_fp (= gamma_i / gamma_fp), R2 = eta_i / eta_fp.

The baselines of Sec. 4 leave W_q undecomposed and factor only W_k and W_v
(experimental setup), so their weight count is E^2 + 4 r E while the cache is
still 2 r L; ``ratios_kv_only`` gives that variant.  With quantization the
ratios count bits: a weight of b_w bits and a cached value of b_a bits weigh
b_w/16 and b_a/16 of their fp16 counterparts.
"""
from __future__ import annotations


def alpha_fp(E):
    return 3 * E * E


def eta_fp(E, L):
    return 2 * L * E


def gamma_fp(E, L):
    return 3 * L * E * E


def alpha_qsvd(E, r):
    return 4 * r * E


def eta_qsvd(r, L):
    return r * L


def gamma_qsvd(E, r, L):
    return 4 * L * r * E


def alpha_ind(E, r):
    return 6 * r * E


def eta_ind(r, L):
    return 2 * r * L


def gamma_ind(E, r, L):
    return 6 * L * r * E


def ratios_qsvd(E, r, w_bits=16, a_bits=16, L=1):
    """(R1, R2) of QSVD at rank r; bit widths scale both against fp16."""
    R1 = alpha_qsvd(E, r) / alpha_fp(E) * (w_bits / 16)
    R2 = eta_qsvd(r, L) / eta_fp(E, L) * (a_bits / 16)
    return R1, R2


def ratios_ind(E, r, L=1):
    """(R1, R2) of per-matrix SVD of all three of W_q, W_k, W_v."""
    return alpha_ind(E, r) / alpha_fp(E), eta_ind(r, L) / eta_fp(E, L)


def ratios_kv_only(E, r, L=1):
    """(R1, R2) of the Sec. 4 baselines: W_q kept, W_k and W_v factored at
    rank r each."""
    return (E * E + 4 * r * E) / alpha_fp(E), eta_ind(r, L) / eta_fp(E, L)
