"""GPU parity of the 4-bit projection settings of the Sec. 4 setup against the
oracle: W4A4 (int4 codes of W_d and of X; the fp8 tensor-core GEMM on e4m3
images of the codes for prefill-sized T, the integer dot-product kernels for
decode-sized T) and the mixed W8A4 / W4A8 settings (bf16 images of the
codes).  Codes, scales and int32 accumulators must be bit-exact; every int4
value is exact in e4m3 and every partial sum of products |x w| <= 49 is an
exact fp32 integer below 2^24 / 49 terms."""
import numpy as np
import pytest
import torch

import synthetic
from oracle import latent, pipeline, quant

from gpu_util import assert_rows_close, bf16, cache_codes_np, cache_scales_np, dev, i32, q

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def l7b():
    wl = synthetic.WORKLOADS["llava7b"]
    inp = synthetic.gen_layer(wl, seed=3, decode_steps=2)
    return wl, inp


def _weight(W_d, w_bits, x_bits):
    return q().qsvd_quantize_weight(torch.from_numpy(np.asarray(W_d, dtype=np.float32)).to(dev()), w_bits=w_bits,
                                    x_bits=x_bits)


def test_quantize_weight_4bit_bit_exact(l7b):
    wl, inp = l7b
    W = _weight(inp.W_d, 4, 4)
    Wq, s_w = quant.quantize_columns(inp.W_d, 4)
    np.testing.assert_array_equal(W.codes.cpu().numpy().astype(np.int64), Wq.T)
    np.testing.assert_array_equal(W.scale.cpu().numpy().astype(np.float64), s_w)
    np.testing.assert_array_equal(W.codes_bf16.float().cpu().numpy(), Wq.T.astype(np.float32))
    e4 = W.codes_e4m3.view(torch.float8_e4m3fn).float().cpu().numpy()
    np.testing.assert_array_equal(e4, Wq.T.astype(np.float32))


def _project(W, X_bits, r, bits):
    lib = q()
    T, d = X_bits.shape
    xq = torch.empty((T, d), dtype=torch.int8, device=dev())
    xs = torch.empty((T,), dtype=torch.float32, device=dev())
    acc = torch.empty((T, r), dtype=torch.int32, device=dev())
    if bits == 8:
        lc = torch.empty((T, r), dtype=torch.int8, device=dev())
        ls = torch.empty((T,), dtype=torch.float32, device=dev())
    else:
        lc = torch.empty((T, r // 2), dtype=torch.uint8, device=dev())
        ls = torch.empty((T, r // 128), dtype=torch.float16, device=dev())
    lib.qsvd_latent_project(W, bf16(X_bits), 1.0, bits, 1.0, lat_codes=lc, lat_scales=ls, xq_out=xq, xs_out=xs,
                            acc_out=acc)
    lib.qsvd_check()
    return {k: v.cpu().numpy() for k, v in dict(xq=xq, xs=xs, acc=acc, codes=lc, scale=ls).items()}


def _assert_exact(got, ref, bits):
    np.testing.assert_array_equal(got["xq"].astype(np.int64), ref["xq"])
    np.testing.assert_array_equal(got["xs"].astype(np.float64), ref["s_x"])
    np.testing.assert_array_equal(got["acc"].astype(np.int64), ref["acc"])
    if bits == 8:
        np.testing.assert_array_equal(got["codes"].astype(np.int64), ref["codes"])
    else:
        np.testing.assert_array_equal(got["codes"], quant.pack_int4(ref["codes"]))
    np.testing.assert_array_equal(got["scale"].astype(np.float64), ref["scale"])


@pytest.mark.parametrize("bits", [4, 8])
@pytest.mark.parametrize("T", [1, 3, 5, 16, 64, 640, 1000])
def test_project_w4a4_bit_exact(l7b, T, bits):
    """Decode-sized T (fused and split dot-product kernels) and prefill-sized T
    (the fp8 GEMM with the requantize-and-store epilogue, a ragged last tile
    at 1000), int4 and int8 latents."""
    wl, inp = l7b
    W = _weight(inp.W_d, 4, 4)
    Wq, s_w = quant.quantize_columns(inp.W_d, 4)
    X = inp.X_prefill[0][:T] if T <= wl.prefill else np.concatenate([inp.X_prefill[0]] * 2)[:T]
    got = _project(W, X, wl.shape.r, bits)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), Wq, s_w, lat_bits=bits, x_bits=4)
    _assert_exact(got, ref, bits)


@pytest.mark.parametrize("w_bits,x_bits", [(8, 4), (4, 8)])
@pytest.mark.parametrize("T", [3, 640])
def test_project_mixed_settings_bit_exact(l7b, w_bits, x_bits, T):
    """W8A4 and W4A8 run on the bf16 images of the codes."""
    wl, inp = l7b
    W = _weight(inp.W_d, w_bits, x_bits)
    Wq, s_w = quant.quantize_columns(inp.W_d, w_bits)
    X = inp.X_prefill[0][:T]
    got = _project(W, X, wl.shape.r, 8)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), Wq, s_w, lat_bits=8, x_bits=x_bits)
    _assert_exact(got, ref, 8)


def test_project_f8_worst_case_exact():
    """Every code at +-7 over d = 5120 (the 13B width): |acc| = 49 * 5120, the
    largest sum the fp8 path forms, still exact."""
    lib = q()
    T, d, r = 256, 5120, 2048
    rng = np.random.default_rng(8)
    Xv = np.where(rng.random((T, d)) < 0.5, -1.0, 1.0)
    Xv[0] = 1.0                                             # row 0 against column 0: every product +49
    X = synthetic.bf16_bits(Xv)
    W_d = np.where(rng.random((d, r)) < 0.5, -0.25, 0.25)
    W_d[:, 0] = 0.25
    W = _weight(W_d, 4, 4)
    got = _project(W, X, r, 8)
    Wq, s_w = quant.quantize_columns(W_d, 4)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), Wq, s_w, lat_bits=8, x_bits=4)
    assert ref["acc"][0, 0] == 49 * d
    _assert_exact(got, ref, 8)


def test_project_w4a4_13b_batch():
    """The 13B layer's whole prefill batch (8 x 3008 tokens, d = 5120,
    r = 2048) in W4A4 with an int4 latent: every code, scale and accumulator."""
    wl = synthetic.WORKLOADS["llava13b"]
    inp = synthetic.gen_layer(wl, seed=4, decode_steps=0)
    W = _weight(inp.W_d, 4, 4)
    Wq, s_w = quant.quantize_columns(inp.W_d, 4)
    X = inp.X_prefill.reshape(-1, wl.shape.d)
    got = _project(W, X, wl.shape.r, 4)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), Wq, s_w, lat_bits=4, x_bits=4)
    _assert_exact(got, ref, 4)


def test_w4a4_prefill_and_decode_pipeline(l7b):
    """W4A4 with an int4 latent cache (the paper's W4A4 row): a 200-token
    prompt through the fp8 GEMM into the cache, then two decode steps
    (decode-sized projection + decode attention) against OracleLayer."""
    lib = q()
    wl, inp = l7b
    s = wl.shape
    P, steps = 200, 2
    w = pipeline.prepare_weights(inp, w_bits=4)
    ref = pipeline.OracleLayer(s, w, 1, P + steps, 4, x_bits=4)
    ref.prefill(0, inp.X_prefill[0][:P])
    W = _weight(inp.W_d, 4, 4)
    cache = lib.LatentCache.empty(1, P + steps, s.r, 4, dev())
    lib.qsvd_latent_project(W, bf16(inp.X_prefill[0][:P]), 1.0, 4, 1.0, dst=cache, dst_seq=i32(np.zeros(P)),
                            dst_pos=i32(np.arange(P)))
    U = [bf16(w[k]) for k in ("U_q", "U_k", "U_v")]
    for t in range(steps):
        L = P + t + 1
        lib.qsvd_latent_project(W, bf16(inp.X_decode[t]), 1.0, 4, 1.0, dst=cache, dst_seq=i32([0]),
                                dst_pos=i32([L - 1]))
        O = torch.empty((1, s.d), dtype=torch.float32, device=dev())
        lib.qsvd_latent_decode_attn(cache, i32([L]), L, *U, s.H, s.dh, O)
        lib.qsvd_check()
        _, outs = ref.decode_step(inp.X_decode[t])
        assert_rows_close(O.cpu().numpy(), outs[0][None, :], f"W4A4 step {t}")
    np.testing.assert_array_equal(cache_codes_np(cache, 0, P + steps), ref.cache.codes[0])
    np.testing.assert_array_equal(cache_scales_np(cache, 0, P + steps), ref.cache.scale[0])
