"""Pins for oracle.attention (Eq. 5 decode over the latent cache) -- CPU only."""
import math

import numpy as np

from oracle import attention


def _case(L, r, H, dh, seed):
    rng = np.random.default_rng(seed)
    C = rng.standard_normal((L, r))
    U = [rng.standard_normal((r, H * dh)) / math.sqrt(r) * 3 for _ in range(3)]
    return C, U


def test_softmax_normalised_and_shift_invariant():
    rng = np.random.default_rng(0)
    s = rng.standard_normal((4, 9)) * 30
    p = attention.softmax(s)
    np.testing.assert_allclose(p.sum(-1), 1.0, atol=1e-15)
    np.testing.assert_allclose(attention.softmax(s + 1234.5), p, atol=1e-15)
    assert np.all(p > 0)


def test_explicit_equals_brute_force_loops():
    C, (Uq, Uk, Uv) = _case(L=5, r=6, H=2, dh=3, seed=1)
    a = attention.decode_attention(C, Uq, Uk, Uv, 2, 3)
    b = attention.decode_attention_loops(C, Uq, Uk, Uv, 2, 3)
    np.testing.assert_allclose(a, b, atol=1e-12)


def test_absorbed_equals_explicit():
    for seed, (L, r, H, dh) in enumerate([(7, 12, 3, 4), (40, 96, 4, 64), (1, 8, 2, 4)]):
        C, (Uq, Uk, Uv) = _case(L, r, H, dh, seed)
        a = attention.decode_attention(C, Uq, Uk, Uv, H, dh)
        b = attention.decode_attention_absorbed(C, Uq, Uk, Uv, H, dh)
        np.testing.assert_allclose(a, b, atol=1e-12 * max(1.0, np.abs(a).max()))


def test_single_token_returns_its_value_row():
    C, (Uq, Uk, Uv) = _case(L=1, r=10, H=2, dh=5, seed=3)
    np.testing.assert_allclose(attention.decode_attention(C, Uq, Uk, Uv, 2, 5),
                               C[0] @ Uv, atol=1e-13)


def test_zero_query_gives_mean_of_values():
    C, (Uq, Uk, Uv) = _case(L=9, r=10, H=2, dh=5, seed=4)
    o = attention.decode_attention(C, np.zeros_like(Uq), Uk, Uv, 2, 5)
    np.testing.assert_allclose(o, (C @ Uv).mean(0), atol=1e-13)


def test_dominant_token_and_head_blocks():
    """A score gap of ~1e3 selects one token's V row; heads use only their
    own column block of each up-projection."""
    r, H, dh = 4, 2, 2
    C = np.eye(r)[:3] * 1.0
    C = np.vstack([C, np.array([[0.0, 0, 0, 1]])])     # last token = query source
    Uq = np.zeros((r, H * dh)); Uq[3, 0] = 1.0           # q_0 = (1, 0), q_1 = 0
    Uk = np.zeros((r, H * dh)); Uk[1, 0] = 3000.0        # token 1 has key (3000, 0) in head 0
    Uv = np.arange(r * H * dh, dtype=float).reshape(r, H * dh)
    o = attention.decode_attention(C, Uq, Uk, Uv, H, dh, softmax_scale=1.0)
    np.testing.assert_allclose(o[:2], Uv[1, :2], atol=1e-12)
    np.testing.assert_allclose(o[2:], (C @ Uv)[:, 2:].mean(0), atol=1e-12)
