"""GPU parity of the quantized up-projections (Eq. 11: Q(H2 W^u) with H2 = I,
per-output-channel symmetric RTN, int8 or int4) against the oracle.

* qsvd_quantize_up: codes and scales bit-exact against
  oracle.pipeline.quantize_up (the oracle's per-column quantizer).
* qsvd_latent_decode_attn_qu: decode outputs within 2e-3 * ||o||_2 per row
  against the oracle's explicit-K/V attention (Eq. 5) over the dequantized
  up-projections (codes x scale), on the 7B shape at B = 1, B = 5 (a pass of
  8 with three empty rows) and B = 16 (the batched passes), int8 and int4
  caches, int8 and int4 weights, and one call mixing the two.
* A whole prefill + decode sequence through qsvd_latent_project and
  qsvd_latent_decode_attn_qu against oracle.pipeline.OracleLayer with
  prepare_weights(u_bits=8).
"""
import math

import numpy as np
import pytest
import torch

import synthetic
from oracle import attention, pipeline, quant

from gpu_util import assert_rows_close, bf16, dev, i32, q

pytestmark = pytest.mark.gpu


def _up(H, dh, r, seed):
    shape = synthetic.LayerShape(H * dh, H, dh, r)
    wl = synthetic.Workload("attn", shape, B=1, n_image=0, n_text=0, decode_steps=0, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=seed, prefill_rows=0, decode_steps=0)
    return inp.U_q, inp.U_k, inp.U_v


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape", [(4096, 1536), (256, 96), (5120, 2048)])
def test_quantize_up_bit_exact(shape, bits):
    d, r = shape
    rng = np.random.default_rng(d + bits)
    U = synthetic.bf16_bits(rng.standard_normal((r, d)) / math.sqrt(r))
    U[:, 7] = 0                                   # an all-zero column: scale 0, codes 0
    uw = q().qsvd_quantize_up(bf16(U), bits)
    codes, scale = pipeline.quantize_up(synthetic.bf16_from_bits(U), bits)
    got = uw.codes.cpu().numpy()
    if bits == 8:
        np.testing.assert_array_equal(got.astype(np.int64), codes)
    else:
        np.testing.assert_array_equal(got, quant.pack_int4(codes))
    np.testing.assert_array_equal(uw.scale.cpu().numpy().astype(np.float64), scale)


def _fill_cache(lib, lens, r, bits, seed, tmax=None):
    rng = np.random.default_rng(seed)
    B = len(lens)
    cache = lib.LatentCache.empty(B, tmax or max(lens), r, bits, dev())
    Cs = []
    for b, L in enumerate(lens):
        x = synthetic.latent_rows(L, r, rng)
        for f in (0.3, 0.8):
            t = int(f * (L - 1))
            if t < L - 1:
                x[t] = x[L - 1]
        if bits == 8:
            codes, s = quant.quantize_rows(x, 8)
            Cs.append(quant.dequantize_rows(codes, s))
            cache.codes[b, :L] = torch.from_numpy(codes.astype(np.int8)).to(dev())
            cache.scales[b, :L] = torch.from_numpy(s.astype(np.float32)).to(dev())
        else:
            codes, s16 = quant.quantize_int4_groups(x)
            Cs.append(quant.dequantize_int4_groups(codes, s16))
            cache.codes[b, :L] = torch.from_numpy(quant.pack_int4(codes)).to(dev())
            cache.scales[b, :L] = torch.from_numpy(s16.astype(np.float16)).to(dev())
    return cache, Cs


@pytest.mark.parametrize("cache_bits,u_bits,lens", [
    (8, (8, 8, 8), [700]),
    (8, (4, 4, 4), [1, 300, 129, 64, 900]),
    (4, (8, 8, 8), [257] * 3 + [1000] * 13),
    (4, (4, 4, 4), [640]),
    (8, (8, 4, 8), [513, 77]),
])
def test_decode_attn_quantized_up(cache_bits, u_bits, lens):
    lib = q()
    H, dh, r = 32, 128, 1536
    U = _up(H, dh, r, seed=len(lens))
    cache, Cs = _fill_cache(lib, lens, r, cache_bits, seed=sum(lens))
    uw, deq = [], []
    for Ub, bits in zip(U, u_bits):
        w = lib.qsvd_quantize_up(bf16(Ub), bits)
        uw.append(w)
        codes, scale = pipeline.quantize_up(synthetic.bf16_from_bits(Ub), bits)
        deq.append(codes.astype(np.float64) * scale[None, :])
    B = len(lens)
    O = torch.full((B, H * dh), float("nan"), dtype=torch.float32, device=dev())
    lib.qsvd_latent_decode_attn_qu(cache, i32(lens), max(lens), *uw, H, dh, O)
    lib.qsvd_check()
    ref = np.stack([attention.decode_attention(C, *deq, H, dh) for C in Cs])
    got = O.cpu().numpy()
    assert np.isfinite(got).all()
    assert_rows_close(got, ref, f"u_bits {u_bits}")


def test_prefill_decode_quantized_up_pipeline():
    """llava7b weights with Q(U_q), Q(U_k), Q(U_v) in int8: a 96-token prompt
    projected into the cache, then 3 decode steps, against OracleLayer."""
    lib = q()
    wl = synthetic.WORKLOADS["llava7b"]
    s = wl.shape
    P, steps = 96, 3
    inp = synthetic.gen_layer(wl, seed=9, prefill_rows=P, decode_steps=steps)
    w = pipeline.prepare_weights(inp, u_bits=8)
    ref = pipeline.OracleLayer(s, w, 1, P + steps, 8)
    ref.prefill(0, inp.X_prefill[0])
    W = lib.qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    U = [lib.qsvd_quantize_up(bf16(w[k]), 8) for k in ("U_q", "U_k", "U_v")]
    for u, k in zip(U, ("U_q", "U_k", "U_v")):
        np.testing.assert_array_equal(u.codes.cpu().numpy().astype(np.int64), w[k + "_codes"])
        np.testing.assert_array_equal(u.scale.cpu().numpy().astype(np.float64), w[k + "_scale"])
    cache = lib.LatentCache.empty(1, P + steps, s.r, 8, dev())
    lib.qsvd_latent_project(W, bf16(inp.X_prefill[0]), dst=cache, dst_seq=i32(np.zeros(P)), dst_pos=i32(np.arange(P)))
    for t in range(steps):
        L = P + t + 1
        lib.qsvd_latent_project(W, bf16(inp.X_decode[t]), dst=cache, dst_seq=i32([0]), dst_pos=i32([L - 1]))
        O = torch.empty((1, s.d), dtype=torch.float32, device=dev())
        lib.qsvd_latent_decode_attn_qu(cache, i32([L]), L, *U, s.H, s.dh, O)
        lib.qsvd_check()
        _, outs = ref.decode_step(inp.X_decode[t])
        assert_rows_close(O.cpu().numpy(), outs[0][None, :], f"step {t}")
    np.testing.assert_array_equal(cache.codes[0].cpu().numpy().astype(np.int64), ref.cache.codes[0])


def test_decode_attn_qu_rejects_bad_weights():
    lib = q()
    H, dh, r = 4, 64, 96
    cache = lib.LatentCache.empty(1, 8, r, 8, dev())
    U = [lib.qsvd_quantize_up(bf16(u), 8) for u in _up(H, dh, r, seed=3)]
    O = torch.empty((1, H * dh), dtype=torch.float32, device=dev())
    bad = lib.UpWeight(U[1].codes, U[1].scale, 5)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_decode_attn_qu(cache, i32([1]), 1, U[0], bad, U[2], H, dh, O)
    assert e.value.status == lib.QSVD_EINVAL
    other_r = lib.qsvd_quantize_up(bf16(_up(H, dh, 128, seed=4)[2]), 4)      # r = 128 against the cache's 96
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_decode_attn_qu(cache, i32([1]), 1, U[0], U[1], other_r, H, dh, O)
    assert e.value.status == lib.QSVD_EINVAL
