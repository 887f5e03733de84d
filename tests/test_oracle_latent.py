"""Pins for oracle.latent (Eq. 11-12 on the H = I path) -- CPU only."""
import numpy as np
import pytest

from oracle import latent, quant


def test_int_matmul_brute_force():
    rng = np.random.default_rng(0)
    A = rng.integers(-127, 128, size=(5, 37))
    B = rng.integers(-127, 128, size=(37, 6))
    C = latent.int_matmul(A, B)
    for i in range(5):
        for j in range(6):
            assert C[i, j] == sum(int(A[i, k]) * int(B[k, j]) for k in range(37))
    with pytest.raises(OverflowError):
        latent.int_matmul(np.full((1, 4), 2 ** 40), np.full((4, 1), 2 ** 20))


def test_dequantize_acc_matches_float32_arithmetic():
    """c_hat = (fp32(acc) * s_x) * s_w, done here in numpy float32."""
    rng = np.random.default_rng(1)
    acc = rng.integers(-80_000_000, 80_000_000, size=(4, 9))
    s_x = rng.uniform(1e-3, 1.0, size=4).astype(np.float32)
    s_w = rng.uniform(1e-4, 1e-2, size=9).astype(np.float32)
    got = latent.dequantize_acc(acc, s_x.astype(np.float64), s_w.astype(np.float64))
    ref = (acc.astype(np.float32) * s_x[:, None]) * s_w[None, :]
    np.testing.assert_array_equal(got, ref.astype(np.float64))


@pytest.mark.parametrize("x_bits,w_bits", [(8, 8), (4, 4), (8, 4)])
def test_projection_within_quantization_error(x_bits, w_bits):
    """The dequantized latent differs from the exact X W_d by no more than
    the rounding of X and W_d to their grids allows:
    |X W - s_x s_w Xq Wq| <= sum_k ( s_x/2 |W_kj| + s_x |Xq_k| s_w/2 ),
    for int8 (W8A8) and int4 (W4A4, and int4 weights with int8 X) codes."""
    rng = np.random.default_rng(2)
    T, d, r = 9, 64, 24
    X = rng.standard_normal((T, d)).astype(np.float32).astype(np.float64)
    X[:, 3] *= 20
    W = (rng.standard_normal((d, r)) / 8).astype(np.float32).astype(np.float64)
    Wq, s_w = quant.quantize_columns(W, w_bits)
    out = latent.latent_project(X, Wq, s_w, lat_bits=8, x_bits=x_bits)
    assert np.abs(out["xq"]).max() == (1 << (x_bits - 1)) - 1
    assert np.abs(Wq).max() == (1 << (w_bits - 1)) - 1
    exact = X @ W
    bound = (out["s_x"][:, None] / 2) * np.abs(W).sum(0)[None, :] \
        + (out["s_x"][:, None] * np.abs(out["xq"]).sum(1)[:, None]) * (s_w[None, :] / 2)
    err = np.abs(exact - out["c_hat"])
    assert np.all(err <= bound * (1 + 1e-5) + 1e-6 * np.abs(exact))
    # and the bound is not vacuous: the error is far below |C| (int4 grids are 18x coarser)
    assert np.median(err / (np.abs(exact) + 1e-9)) < (0.05 if x_bits == w_bits == 8 else 0.6)


def test_w4a4_projection_brute_force():
    """W4A4 on a tiny block, every step recomputed by hand in numpy float32:
    4-bit codes from a search over [-7, 7], the integer sums by loops, then
    (fp32(acc) s_x) s_w; and |acc| <= 49 d, the bound that keeps every
    partial sum exact in fp32 for d < 2^24 / 49."""
    rng = np.random.default_rng(21)
    T, d, r = 3, 40, 5
    X = (rng.standard_normal((T, d)) * 2).astype(np.float32)
    W = (rng.standard_normal((d, r)) / 6).astype(np.float32)
    Wq, s_w = quant.quantize_columns(W.astype(np.float64), 4)
    out = latent.latent_project(X.astype(np.float64), Wq, s_w, lat_bits=8, x_bits=4)
    for t in range(T):
        s = np.float32(np.max(np.abs(X[t]))) / np.float32(7)
        assert out["s_x"][t] == float(s)
        for k in range(d):
            x = X[t, k] / s
            c = min(range(-7, 8), key=lambda v: (abs(float(x) - v), v % 2))
            assert out["xq"][t, k] == c
        for j in range(r):
            acc = sum(int(out["xq"][t, k]) * int(Wq[k, j]) for k in range(d))
            assert out["acc"][t, j] == acc and abs(acc) <= 49 * d
            c_hat = (np.float32(acc) * np.float32(out["s_x"][t])) * np.float32(s_w[j])
            assert out["c_hat"][t, j] == float(c_hat)


def test_latent_requant_roundtrip_int8_int4():
    rng = np.random.default_rng(3)
    c = (rng.standard_normal((5, 256)) * np.linspace(3, 0.1, 256)).astype(np.float32).astype(np.float64)
    for bits in (8, 4):
        codes, sc = latent.requantize_latent(c, bits)
        deq = latent.dequantize_latent(codes, sc, bits)
        if bits == 8:
            assert np.all(np.abs(deq - c) <= sc[:, None] * 0.5 * (1 + 1e-6))
        else:
            g = np.repeat(sc, 128, axis=1)
            assert np.all(np.abs(deq - c) <= g * 0.5 * (1 + 1e-3) + 1e-7)


def test_cache_append_and_rows():
    cache = latent.LatentCache(B=2, tmax=4, r=128, lat_bits=4)
    codes = np.arange(-7, 8).repeat(9)[:128][None, :].repeat(3, 0)
    sc = np.array([[0.5], [1.0], [2.0]])
    cache.append([1, 1, 0], [0, 1, 3], codes, sc)
    np.testing.assert_array_equal(cache.rows(1, 2), codes[:2] * np.array([[0.5], [1.0]]))
    assert np.all(cache.rows(0, 3) == 0)
    np.testing.assert_array_equal(cache.packed_codes().shape, (2, 4, 64))
    with pytest.raises(IndexError):
        cache.append([0], [4], codes[:1], sc[:1])
