"""Pins for Eq. 11's quantized up-projection Q(H2 W^u) in the oracle
(pipeline.quantize_up, prepare_weights(u_bits=...)) -- CPU only.  The GPU
path for it is not built yet; these fix the oracle it will be checked against."""
import math

import numpy as np

import synthetic
from oracle import attention, pipeline, quant


def _layer(seed=0):
    wl = synthetic.WORKLOADS["tiny"]
    return wl, synthetic.gen_layer(wl, seed=seed)


def test_per_column_rtn_error_bound_and_exact_scales():
    wl, inp = _layer(1)
    w = pipeline.prepare_weights(inp, u_bits=8)
    for k in ("U_q", "U_k", "U_v"):
        U = synthetic.bf16_from_bits(w[k])
        codes, s = w[k + "_codes"], w[k + "_scale"]
        assert codes.shape == U.shape and s.shape == (U.shape[1],)
        assert np.abs(codes).max() <= 127
        # every column's absmax maps to +-127 and every element is within half a
        # step (plus the fp32 rounding of the quotient v / s before the rounding
        # to an integer: |v/s| <= 127.5, so at most 127.5 * 2^-24 of a step)
        np.testing.assert_array_equal(np.abs(codes).max(axis=0), np.where(np.abs(U).max(axis=0) > 0, 127, 0))
        assert np.all(np.abs(U - codes * s[None, :]) <= s[None, :] * (0.5 + 127.5 * 2.0 ** -24))
        np.testing.assert_array_equal(s, quant.f32(quant.f32(np.abs(U).max(axis=0)) / 127))


def test_int4_up_projection_bound():
    wl, inp = _layer(2)
    w = pipeline.prepare_weights(inp, u_bits=4)
    U = synthetic.bf16_from_bits(w["U_v"])
    assert np.abs(w["U_v_codes"]).max() <= 7
    assert np.all(np.abs(U - w["U_v_deq"]) <= w["U_v_scale"][None, :] * (0.5 + 7.5 * 2.0 ** -24))


def test_attention_with_quantized_up_projections_tracks_bf16():
    """Decode through the dequantized U stays close to the bf16 U (int8: a few
    tenths of a percent of the output norm on the tiny layer), and the oracle
    layer really uses the quantized values."""
    wl, inp = _layer(3)
    s = wl.shape
    w16 = pipeline.prepare_weights(inp)
    w8 = pipeline.prepare_weights(inp, u_bits=8)
    outs = []
    for w in (w16, w8):
        layer = pipeline.OracleLayer(s, w, 1, wl.tmax, 8)
        layer.prefill(0, inp.X_prefill[0])
        _, o = layer.decode_step(inp.X_decode[0])
        outs.append(o[0])
    rel = np.abs(outs[1] - outs[0]).max() / np.linalg.norm(outs[0])
    assert 0 < rel < 2e-2
    layer = pipeline.OracleLayer(s, w8, 1, wl.tmax, 8)
    np.testing.assert_array_equal(layer.U_v, w8["U_v_deq"])
