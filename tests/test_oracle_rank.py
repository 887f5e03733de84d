"""Pins for oracle.rank: Eq. 8-10 importance scores, the global rank budget,
and Eq. 14's beta search -- CPU only."""
import numpy as np
import pytest

from oracle import rank, svd


def _factors(m, n, seed):
    rng = np.random.default_rng(seed)
    W = rng.standard_normal((m, n)) * np.linspace(2.0, 0.2, n)[None, :]
    U, s, Vt = np.linalg.svd(W, full_matrices=False)
    grads = [rng.standard_normal((m, n)) for _ in range(5)]
    return W, U, s, Vt, grads


def test_eq10_equals_the_definition():
    """The identity the paper proves: mean (<dW_i, G>)^2 = mean sigma_i^2 [U^T G V]_ii^2."""
    W, U, s, Vt, grads = _factors(12, 9, 0)
    a = rank.importance_scores_definition(U, s, Vt, grads)
    b = rank.importance_scores(U, s, Vt, grads)
    np.testing.assert_allclose(a, b, rtol=1e-10, atol=1e-12 * a.max())


def test_first_order_loss_change_sign_and_size():
    """Eq. 8 on a quadratic loss L(W) = 0.5 ||W - T||^2 (gradient G = W - T):
    L(W) - L(W'_i) = <dW_i, G> - 0.5 ||dW_i||^2 exactly, ||dW_i||_F = sigma_i."""
    rng = np.random.default_rng(1)
    W, U, s, Vt, _ = _factors(8, 6, 1)
    T = rng.standard_normal(W.shape)
    G = W - T
    L = lambda A: 0.5 * np.sum((A - T) ** 2)  # noqa: E731
    for i in range(len(s)):
        s_cut = s.copy()
        s_cut[i] = 0.0
        Wp = (U * s_cut[None, :]) @ Vt
        dW = W - Wp
        assert abs(np.linalg.norm(dW) - s[i]) < 1e-12 * s[0]
        assert abs((L(W) - L(Wp)) - (np.sum(dW * G) - 0.5 * s[i] ** 2)) < 1e-9 * s[0] ** 2


def test_zero_gradient_gives_zero_scores():
    W, U, s, Vt, _ = _factors(6, 5, 2)
    np.testing.assert_array_equal(rank.importance_scores(U, s, Vt, [np.zeros_like(W)]), 0.0)


def test_global_rank_budget():
    scores = [np.array([5.0, 1.0, 0.5]), np.array([4.0, 3.0, 0.1, 2.0]), np.array([0.2])]
    assert rank.allocate_ranks(scores, 0) == [[], [], []]
    assert rank.allocate_ranks(scores, 3) == [[0], [0, 1], []]
    assert rank.allocate_ranks(scores, 5) == [[0, 1], [0, 1, 3], []]
    assert rank.allocate_ranks(scores, 8) == [[0, 1, 2], [0, 1, 2, 3], [0]]
    for k in range(9):                                 # k values kept, nested as k grows
        got = rank.allocate_ranks(scores, k)
        assert sum(len(x) for x in got) == k
        if k:
            prev = rank.allocate_ranks(scores, k - 1)
            assert all(set(p) <= set(g) for p, g in zip(prev, got))
    with pytest.raises(ValueError):
        rank.allocate_ranks(scores, 9)


def test_beta_objective_without_quantization_is_beta_independent():
    """W^d W^u does not depend on beta (Eq. 3), so neither does the unquantized
    objective; with quantization it does, and the search returns its minimum."""
    rng = np.random.default_rng(3)
    E, r = 32, 12
    Wq, Wk, Wv = (rng.standard_normal((E, E)) / np.sqrt(E) for _ in range(3))
    X = rng.standard_normal((40, E))
    X[:, [3, 17]] *= 20.0                               # channel-wise outliers
    base = [rank.quantized_qkv_error(Wq, Wk, Wv, r, b, X, quantize=False) for b in (0.0, 0.5, 1.0)]
    np.testing.assert_allclose(base, base[0], rtol=1e-9)
    best, errs = rank.beta_search(Wq, Wk, Wv, r, X)
    assert errs[best] == min(errs.values())
    assert len(set(round(v, 9) for v in errs.values())) > 1


def test_latent_channel_spread_grows_with_beta():
    """Eq. 13: C = X W_r^d diag(sigma^beta), so the ratio of the largest to the
    smallest latent channel norm grows with beta (sigma decreasing)."""
    rng = np.random.default_rng(4)
    E, r = 24, 10
    Wq, Wk, Wv = (rng.standard_normal((E, E)) * np.linspace(3.0, 0.1, E)[None, :] for _ in range(3))
    X = rng.standard_normal((30, E))
    spread = []
    for b in (0.0, 0.5, 1.0):
        W_d = svd.joint_qkv_factors(Wq, Wk, Wv, r, b)[0]
        cn = np.linalg.norm(X @ W_d, axis=0)
        spread.append(cn.max() / cn.min())
    assert spread[0] < spread[1] < spread[2]


def test_beta_search_matches_the_objective_per_beta():
    """The search (one joint SVD, Eq. 3 per beta) gives, bit for bit, the
    objective quantized_qkv_error computes from its own SVD at each beta; at
    full rank the unquantized objective vanishes (W^d W^u = W_concat)."""
    rng = np.random.default_rng(5)
    E, r = 24, 10
    Wq, Wk, Wv = (rng.standard_normal((E, E)) / np.sqrt(E) for _ in range(3))
    X = rng.standard_normal((30, E))
    X[:, 5] *= 20.0
    _, errs = rank.beta_search(Wq, Wk, Wv, r, X, betas=(0.0, 0.4, 1.0))
    for b, v in errs.items():
        assert v == rank.quantized_qkv_error(Wq, Wk, Wv, r, b, X)
    _, errs4 = rank.beta_search(Wq, Wk, Wv, r, X, betas=(0.3,), u_bits=4)
    assert errs4[0.3] == rank.quantized_qkv_error(Wq, Wk, Wv, r, 0.3, X, u_bits=4)
    full = rank.quantized_qkv_error(Wq, Wk, Wv, E, 0.5, X, quantize=False)
    assert full <= 1e-18 * np.sum((X @ np.concatenate([Wq, Wk, Wv], axis=1)) ** 2)
