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


# ---------------------------------------------------------------------------
# causal prefill (every prompt token attends to the cached prefix, itself included)
# ---------------------------------------------------------------------------
def test_prefill_rows_equal_decode_on_each_prefix():
    """Row i of the masked matrix form is the decode step of the sequence cut
    after position t0 + i (decode is pinned above by brute force)."""
    for seed, (L, t0, r, H, dh) in enumerate([(9, 0, 12, 3, 4), (33, 20, 40, 2, 8), (5, 4, 6, 2, 3)]):
        C, (Uq, Uk, Uv) = _case(L, r, H, dh, seed + 10)
        O = attention.prefill_attention(C, Uq, Uk, Uv, H, dh, t0=t0)
        assert O.shape == (L - t0, H * dh)
        for i in range(L - t0):
            ref = attention.decode_attention(C[:t0 + i + 1], Uq, Uk, Uv, H, dh)
            np.testing.assert_allclose(O[i], ref, atol=1e-12 * max(1.0, np.abs(ref).max()))


def test_prefill_equals_brute_force_loops():
    C, (Uq, Uk, Uv) = _case(L=6, r=5, H=2, dh=3, seed=31)
    O = attention.prefill_attention(C, Uq, Uk, Uv, 2, 3, t0=1)
    for i in range(5):
        np.testing.assert_allclose(O[i], attention.decode_attention_loops(C[:i + 2], Uq, Uk, Uv, 2, 3),
                                   atol=1e-12)


def test_prefill_is_causal():
    """Changing the latents after position t0 + i leaves row i unchanged and
    changes the later rows."""
    C, (Uq, Uk, Uv) = _case(L=12, r=10, H=2, dh=4, seed=32)
    O = attention.prefill_attention(C, Uq, Uk, Uv, 2, 4)
    C2 = C.copy()
    C2[7:] += 5.0
    O2 = attention.prefill_attention(C2, Uq, Uk, Uv, 2, 4)
    np.testing.assert_array_equal(O[:7], O2[:7])
    assert np.abs(O[7:] - O2[7:]).min(axis=1).max() > 1e-3


def test_prefill_first_token_is_its_value_row():
    """Position 0 sees only itself: o = c_0 U_v whatever the query."""
    C, (Uq, Uk, Uv) = _case(L=4, r=8, H=2, dh=4, seed=33)
    O = attention.prefill_attention(C, Uq, Uk, Uv, 2, 4)
    np.testing.assert_allclose(O[0], C[0] @ Uv, atol=1e-13)
