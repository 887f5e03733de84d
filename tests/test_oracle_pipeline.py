"""Pins for oracle.pipeline: the workload driver composes the pinned steps
and its row-by-row K/V bookkeeping equals recomputing Eq. 5 from the whole
cache -- CPU only."""
import numpy as np

import synthetic
from oracle import attention, latent, pipeline, quant


def test_tiny_workload_end_to_end():
    wl = synthetic.WORKLOADS["tiny"]
    inp = synthetic.gen_layer(wl, seed=0, decode_steps=4)
    w = pipeline.prepare_weights(inp)
    s = wl.shape
    assert w["Wq"].shape == (s.d, s.r) and w["U_q"].shape == (s.r, s.d)
    assert np.abs(w["Wq"]).max() == 127
    lay = pipeline.OracleLayer(s, w, wl.B, wl.tmax, wl.lat_bits)
    pre = lay.prefill(0, inp.X_prefill[0])
    # the prefill is exactly the composition of the pinned steps
    X = synthetic.bf16_from_bits(inp.X_prefill[0])
    xq, s_x = quant.quantize_rows(X, 8)
    np.testing.assert_array_equal(pre["xq"], xq)
    acc = latent.int_matmul(xq, w["Wq"])
    np.testing.assert_array_equal(pre["acc"], acc)
    for step in range(4):
        _, outs = lay.decode_step(inp.X_decode[step])
        L = int(lay.len[0])
        C = lay.cache.rows(0, L)
        ref = attention.decode_attention(C, lay.U_q, lay.U_k, lay.U_v, s.H, s.dh)
        np.testing.assert_allclose(outs[0], ref, atol=1e-12)
    assert lay.len[0] == wl.prefill + 4
    # attention is not degenerate on this workload: the softmax is far from uniform
    q = C[-1] @ lay.U_q
    K = C @ lay.U_k
    p = attention.softmax(K[:, :s.dh] @ q[:s.dh] / np.sqrt(s.dh))
    assert p.max() > 5.0 / L


def test_synthetic_draws_are_seeded_and_prefix_stable():
    wl = synthetic.WORKLOADS["tiny"]
    a = synthetic.gen_layer(wl, seed=0)
    b = synthetic.gen_layer(wl, seed=0, decode_steps=3)
    np.testing.assert_array_equal(a.X_prefill, b.X_prefill)
    np.testing.assert_array_equal(a.X_decode[:3], b.X_decode)
    c = synthetic.gen_layer(wl, seed=1)
    assert not np.array_equal(a.X_prefill, c.X_prefill)
    # bf16 storage: value -> bits -> value is exact and rounds to nearest even
    v = np.array([1.0, 1.00390625, 1.005859375, -3.0e38, 1e-40])
    bits = synthetic.bf16_bits(v)
    assert synthetic.bf16_from_bits(bits)[0] == 1.0
    assert synthetic.bf16_from_bits(bits)[1] == 1.0          # tie -> even
    assert synthetic.bf16_from_bits(bits)[2] == 1.0078125
