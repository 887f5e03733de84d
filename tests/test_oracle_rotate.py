"""Pins for oracle.rotate (the rotation H1 of Eq. 11-12) -- CPU only."""
import numpy as np
import pytest

import synthetic
from oracle import latent, quant, rotate

scipy_linalg = pytest.importorskip("scipy.linalg")


def test_default_block():
    assert rotate.default_block(4096) == 4096
    assert rotate.default_block(5120) == 1024
    assert rotate.default_block(256) == 256
    assert rotate.default_block(96) == 32


def test_small_cases_by_hand():
    s2 = np.float32(1 / np.sqrt(2.0))
    got = rotate.rotate_rows(np.array([[3.0, 1.0]], dtype=np.float32), 2)
    np.testing.assert_array_equal(got, [[np.float32(4.0) * s2, np.float32(2.0) * s2]])
    # order 4: rows of the Sylvester matrix [[1,1,1,1],[1,-1,1,-1],[1,1,-1,-1],[1,-1,-1,1]] / 2
    got = rotate.rotate_rows(np.array([[1.0, 2.0, 3.0, 4.0]], dtype=np.float32), 4)
    np.testing.assert_array_equal(got, [[5.0, -1.0, -2.0, 0.0]])


@pytest.mark.parametrize("d,b", [(64, 64), (256, 64), (5120, 1024)])
def test_matches_explicit_block_hadamard(d, b):
    """The butterflies equal multiplication by I (x) H_b / sqrt(b) with the
    Sylvester matrix from scipy, to fp32 rounding."""
    rng = np.random.default_rng(d + b)
    X = rng.standard_normal((5, d)).astype(np.float32)
    H = scipy_linalg.hadamard(b).astype(np.float64) / np.sqrt(b)
    ref = np.concatenate([X[:, k * b:(k + 1) * b].astype(np.float64) @ H for k in range(d // b)], axis=1)
    got = rotate.rotate_rows(X, b)
    assert np.abs(got - ref).max() <= 1e-5 * np.abs(ref).max()


def test_orthogonal_and_invariant():
    """H1 H1 = I, and (x H1)(H1 W) = x W."""
    rng = np.random.default_rng(7)
    X = rng.standard_normal((4, 512)).astype(np.float32)
    W = rng.standard_normal((512, 48)).astype(np.float32)
    back = rotate.rotate_rows(rotate.rotate_rows(X, 512), 512)
    assert np.abs(back - X).max() <= 1e-5 * np.abs(X).max()
    lhs = rotate.rotate_rows(X, 128) @ rotate.rotate_weight(W, 128)
    rhs = X.astype(np.float64) @ W.astype(np.float64)
    assert np.abs(lhs - rhs).max() <= 1e-4 * np.abs(rhs).max()


def test_weight_rotation_is_the_column_transform():
    rng = np.random.default_rng(8)
    W = rng.standard_normal((256, 9)).astype(np.float32)
    got = rotate.rotate_weight(W, 256)
    for j in range(9):
        np.testing.assert_array_equal(got[:, j], rotate.rotate_rows(W[:, j][None, :], 256)[0])


def test_rotation_shrinks_the_quantization_error_of_outlier_rows():
    """Sec. 3.3's point: activations with channel-wise outliers (the
    synthetic recipe: 1 % of channels x 20) lose less to per-token int8
    quantization after H1, and so does the projected latent."""
    wl = synthetic.WORKLOADS["llava7b"]
    inp = synthetic.gen_layer(synthetic.Workload("rot", wl.shape, B=1, n_image=48, n_text=16,
                                                 decode_steps=0, lat_bits=8), seed=11)
    X = synthetic.bf16_from_bits(inp.X_prefill[0]).astype(np.float32)
    W = np.asarray(inp.W_d, dtype=np.float32)
    b = rotate.default_block(X.shape[1])
    exact = X.astype(np.float64) @ W.astype(np.float64)

    def err(rot):
        Wr = rotate.rotate_weight(W, b) if rot else W
        Wq, s_w = quant.quantize_columns(Wr, 8)
        out = latent.latent_project(X, Wq, s_w, rot=b if rot else 0)
        xr = rotate.rotate_rows(X, b) if rot else X.astype(np.float64)
        xerr = np.linalg.norm(xr - out["xq"] * out["s_x"][:, None]) / np.linalg.norm(xr)
        cerr = np.linalg.norm(out["c_hat"] - exact) / np.linalg.norm(exact)
        return xerr, cerr

    (x0, c0), (x1, c1) = err(False), err(True)
    assert x1 < 0.5 * x0
    assert c1 < c0
