"""Pins for oracle.svd (Eq. 1-4, Eq. 13) -- CPU only."""
import numpy as np
import pytest

from oracle import svd


@pytest.mark.parametrize("shape", [(7, 5), (5, 7), (12, 12), (16, 9), (3, 11), (8, 1)])
def test_jacobi_matches_lapack(shape):
    rng = np.random.default_rng(sum(shape))
    A = rng.standard_normal(shape)
    U, s, Vt = svd.jacobi_svd(A)
    s_ref = np.linalg.svd(A, compute_uv=False)
    np.testing.assert_allclose(s, s_ref, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(U @ np.diag(s) @ Vt, A, atol=1e-12)
    k = min(shape)
    np.testing.assert_allclose(U.T @ U, np.eye(k), atol=1e-12)
    np.testing.assert_allclose(Vt @ Vt.T, np.eye(k), atol=1e-12)
    assert np.all(np.diff(s) <= 0)


def test_rank_deficient_and_zero():
    rng = np.random.default_rng(3)
    A = rng.standard_normal((9, 2)) @ rng.standard_normal((2, 6))   # rank 2
    U, s, Vt = svd.jacobi_svd(A)
    np.testing.assert_allclose(s[2:], 0, atol=1e-12)
    np.testing.assert_allclose(U @ np.diag(s) @ Vt, A, atol=1e-12)
    U0, s0, Vt0 = svd.jacobi_svd(np.zeros((4, 3)))
    assert np.all(s0 == 0)


def test_truncation_eckart_young():
    """Eq. 1: the rank-r error is the tail of the spectrum (Eckart-Young)."""
    rng = np.random.default_rng(5)
    W = rng.standard_normal((20, 30))
    s_all = np.linalg.svd(W, compute_uv=False)
    for r in (1, 4, 10, 19, 20):
        Ur, sr, Vtr = svd.truncated_svd(W, r)
        Wr = Ur @ np.diag(sr) @ Vtr
        err = np.linalg.norm(W - Wr, "fro") ** 2
        assert err == pytest.approx(np.sum(s_all[r:] ** 2), rel=1e-10, abs=1e-10)
        # same rank-r matrix as LAPACK's truncation
        u, s, vt = np.linalg.svd(W, full_matrices=False)
        np.testing.assert_allclose(Wr, (u[:, :r] * s[:r]) @ vt[:r], atol=1e-11)


def _qkv(E, seed):
    rng = np.random.default_rng(seed)
    return [rng.standard_normal((E, E)) / np.sqrt(E) for _ in range(3)]


def test_joint_full_rank_reproduces_qkv():
    """Eq. 4 with r = E: X W_d W^u_x equals X W_x for x in q, k, v."""
    E = 12
    Wq, Wk, Wv = _qkv(E, 0)
    X = np.random.default_rng(1).standard_normal((5, E))
    W_d, Uq, Uk, Uv, sig = svd.joint_qkv_factors(Wq, Wk, Wv, E, beta=0.5)
    assert W_d.shape == (E, E) and Uq.shape == (E, E)
    for W, U in ((Wq, Uq), (Wk, Uk), (Wv, Uv)):
        np.testing.assert_allclose(X @ W_d @ U, X @ W, atol=1e-12)


def test_joint_beta_independence_and_column_scaling():
    """Eq. 3: W_d W^u does not depend on beta; Eq. 13: column i of W_d has
    norm sigma_i^beta (W^d_r has orthonormal columns)."""
    E, r = 10, 6
    Wq, Wk, Wv = _qkv(E, 2)
    ref = None
    for beta in (0.0, 0.3, 0.5, 1.0):
        W_d, Uq, Uk, Uv, sig = svd.joint_qkv_factors(Wq, Wk, Wv, r, beta)
        prod = W_d @ np.concatenate([Uq, Uk, Uv], axis=1)
        if ref is None:
            ref = prod
        np.testing.assert_allclose(prod, ref, atol=1e-12)
        np.testing.assert_allclose(np.linalg.norm(W_d, axis=0), sig ** beta, rtol=1e-12)
    # the rank-r product is LAPACK's rank-r approximation of [W_q, W_k, W_v]
    u, s, vt = np.linalg.svd(np.concatenate([Wq, Wk, Wv], axis=1), full_matrices=False)
    np.testing.assert_allclose(ref, (u[:, :r] * s[:r]) @ vt[:r], atol=1e-12)
    with pytest.raises(ValueError):
        svd.joint_qkv_factors(Wq, Wk, Wv, r, 1.5)
