"""Pins for oracle.quant (per-token / per-channel symmetric RTN, int4 groups,
nibble packing) -- CPU only.

The checks use numpy float32 arithmetic and exhaustive searches over the code
range, independent of the oracle's fp64-then-round emulation."""
import numpy as np
import pytest

from oracle import quant


def _brute_codes(v32, s32, q):
    """Nearest code to fp32(v/s) by search over [-q, q], ties to the even
    code; computed in numpy float32."""
    out = np.zeros(v32.shape, dtype=np.int64)
    for idx in np.ndindex(v32.shape):
        if s32 == 0:
            continue
        x = np.float32(v32[idx]) / np.float32(s32)       # IEEE fp32 division
        best, bestd = None, None
        for c in range(-q, q + 1):
            dd = abs(float(x) - c)
            if best is None or dd < bestd or (dd == bestd and c % 2 == 0):
                best, bestd = c, dd
        out[idx] = best
    return out


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("clip", [1.0, 0.9, 0.85])
def test_rows_brute_force(bits, clip):
    rng = np.random.default_rng(bits * 7 + int(clip * 100))
    V = (rng.standard_normal((6, 17)) * rng.uniform(0.01, 50, size=(6, 1))).astype(np.float32)
    V[2, 5] *= 40.0                      # an outlier
    codes, s = quant.quantize_rows(V.astype(np.float64), bits, clip)
    q = (1 << (bits - 1)) - 1
    for t in range(V.shape[0]):
        m = np.max(np.abs(V[t]))
        s32 = np.float32(np.float32(clip) * m) / np.float32(q)
        assert s[t] == float(s32)
        np.testing.assert_array_equal(codes[t], _brute_codes(V[t], s32, q))


def test_absmax_maps_to_qmax_and_error_bound():
    rng = np.random.default_rng(11)
    V = rng.standard_normal((20, 64)).astype(np.float32).astype(np.float64)
    for bits, q in ((8, 127), (4, 7)):
        codes, s = quant.quantize_rows(V, bits)
        am = np.argmax(np.abs(V), axis=1)
        np.testing.assert_array_equal(np.abs(codes[np.arange(20), am]), q)
        assert np.all(np.abs(codes) <= q)
        # unclipped: |v - s * code| <= s/2 (plus the fp32 rounding of v/s)
        err = np.abs(V - codes * s[:, None])
        assert np.all(err <= s[:, None] * (0.5 + 1e-6))


def test_ties_to_even_and_exact_scale():
    # m = 127 gives s = 1 exactly, so codes are rint(v) with ties to even
    v = np.array([[127.0, 2.5, -3.5, 0.5, -0.5, 1.5, -126.5, 3.49]])
    codes, s = quant.quantize_rows(v, 8)
    assert s[0] == 1.0
    np.testing.assert_array_equal(codes[0], [127, 2, -4, 0, 0, 2, -126, 3])


def test_zero_row_and_clipping():
    codes, s = quant.quantize_rows(np.zeros((2, 8)), 8)
    assert np.all(s == 0) and np.all(codes == 0)
    v = np.array([[10.0, 9.5, 8.0, -10.0, 1.0]])
    codes, s = quant.quantize_rows(v, 8, clip=0.5)
    # s = 0.5*10/127; |v| > 5 saturates
    np.testing.assert_array_equal(codes[0, [0, 1, 2, 3]], [127, 127, 127, -127])
    assert codes[0, 4] == round(1.0 / float(np.float32(np.float32(5.0) / np.float32(127))))


def test_requantize_idempotent():
    rng = np.random.default_rng(4)
    V = rng.standard_normal((10, 40)).astype(np.float32).astype(np.float64)
    codes, s = quant.quantize_rows(V, 8)
    deq = quant.f32(quant.dequantize_rows(codes, s))
    codes2, _ = quant.quantize_rows(deq, 8)
    np.testing.assert_array_equal(codes2, codes)


def test_columns_are_per_output_channel():
    W = np.array([[1.0, -8.0, 0.0], [-2.0, 4.0, 0.0], [0.5, 1.0, 0.0]])
    codes, s = quant.quantize_columns(W, 8)
    np.testing.assert_array_equal(s, [float(np.float32(2.0) / np.float32(127)),
                                      float(np.float32(8.0) / np.float32(127)), 0.0])
    np.testing.assert_array_equal(codes[:, 0], [64, -127, 32])   # 63.5 -> 64 (even)
    np.testing.assert_array_equal(codes[:, 1], [-127, 64, 16])    # 63.5 -> 64, 15.875 -> 16
    np.testing.assert_array_equal(codes[:, 2], [0, 0, 0])


def test_int4_groups_brute_force_and_fp16_scale():
    rng = np.random.default_rng(8)
    V = (rng.standard_normal((3, 256)) * 3).astype(np.float32)
    V[1, 130] = 900.0
    codes, s16 = quant.quantize_int4_groups(V.astype(np.float64))
    assert codes.shape == (3, 256) and s16.shape == (3, 2)
    for t in range(3):
        for g in range(2):
            blk = V[t, g * 128:(g + 1) * 128]
            s32 = np.float32(np.float32(1.0) * np.max(np.abs(blk))) / np.float32(7)
            h = np.float16(s32)                       # numpy's own fp16 rounding
            assert s16[t, g] == float(h)
            np.testing.assert_array_equal(codes[t, g * 128:(g + 1) * 128],
                                          _brute_codes(blk, np.float32(h), 7))


def test_int4_scale_saturates_and_underflows():
    V = np.zeros((2, 128))
    V[0, 0] = 1.0e6          # 1e6/7 is above the fp16 range -> 65504
    V[0, 1] = -1.0e6
    V[0, 2] = 65504.0 * 3.2
    V[1, 0] = 1e-12          # scale underflows to 0 in fp16 -> all codes 0
    codes, s16 = quant.quantize_int4_groups(V)
    assert s16[0, 0] == 65504.0
    assert codes[0, 0] == 7 and codes[0, 1] == -7 and codes[0, 2] == 3
    assert s16[1, 0] == 0.0 and np.all(codes[1] == 0)


def test_pack_nibble_order_golden():
    # element 2i in the low nibble, 2i+1 in the high nibble, two's complement
    packed = quant.pack_int4(np.array([1, -1, 7, -7, 0, -8 + 1]))
    np.testing.assert_array_equal(packed, np.array([0xF1, 0x97, 0x90], dtype=np.uint8))
    rng = np.random.default_rng(2)
    c = rng.integers(-7, 8, size=(5, 64))
    np.testing.assert_array_equal(quant.unpack_int4(quant.pack_int4(c)), c)
