"""The rotation H1 of Eq. 11-12 (Sec. 3.3, after the orthogonal transforms of
Sec. 2.3): C_qkv ~= Q(X H1^T) Q(H1 W^d), so the per-token quantizer sees the
rotated row x H1^T, whose channel-wise outliers are spread over many
channels, while (x H1^T)(H1 W^d) = x W^d leaves the product unchanged.

Reading (the paper names QuaRot's rotations and fixes no matrix):
H1 = I_{d/b} (x) H_b / sqrt(b), block-diagonal normalized Walsh-Hadamard with
H_b the Sylvester Hadamard matrix of order b, b a power of two dividing d
(by default the largest one, so b = d for d = 4096 and b = 1024 for d = 5120).
H1 is symmetric and orthogonal.  Both sides compute it as the fast
Walsh-Hadamard transform in fp32: stages h = 1, 2, 4, ..., b/2 in that order,
each pair (i, i + h) with (i & h) == 0 becoming (v_i + v_{i+h}, v_i - v_{i+h}),
then every entry times fp32(1 / sqrt(b)).  Rows of X take it on the fly;
columns of W^d take it once, offline.  H2 folds into W^d and W^u offline and
is not applied here.

Test infrastructure: only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline use this module.
"""
from __future__ import annotations

import numpy as np


def default_block(d: int) -> int:
    """Largest power of two dividing d."""
    return d & -d


def fwht_rows(V, b: int):
    """Unnormalized Walsh-Hadamard transform of every length-b block of the
    last axis, fp32 butterflies in stage order (fp32 result)."""
    V = np.array(V, dtype=np.float32, copy=True)
    n = V.shape[-1]
    if b < 1 or b & (b - 1) or n % b:
        raise ValueError("block must be a power of two dividing the row length")
    lead = V.shape[:-1]
    h = 1
    while h < b:
        W = V.reshape(lead + (n // (2 * h), 2, h))
        a = W[..., 0, :].copy()
        c = W[..., 1, :].copy()
        W[..., 0, :] = a + c            # float32 + float32: IEEE single, nearest even
        W[..., 1, :] = a - c
        V = W.reshape(lead + (n,))
        h *= 2
    return V


def rotate_rows(X, b: int):
    """x H1 (= x H1^T) for every row: fp32 values returned as fp64 arrays."""
    scale = np.float32(1.0 / np.sqrt(float(b)))
    return (fwht_rows(X, b) * scale).astype(np.float64)


def rotate_weight(W, b: int):
    """H1 W for W [d, r]: the same transform down every column."""
    return rotate_rows(np.asarray(W, dtype=np.float32).T, b).T.copy()
