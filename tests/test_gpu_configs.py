"""GPU parity at the full sizes of the LLaVA-13B-shaped layer and at the
corners of the 32-layer 7B-shaped sweep, in the launch configuration the
benchmark times (automatic kernel choice, splits and waves).

* 13B layer (d = 5120, H = 40, dh = 128, r = 2048, int8 cache): B = 8
  prompts of 2880 image-like + 128 text-like tokens projected in one call
  (the tensor-core GEMM with the requantize-and-store epilogue), then chained
  decode steps (qsvd_latent_project for the 8 new tokens, then
  qsvd_latent_decode_attn).  Sequences 0, 3 and 7 are checked against the
  oracle with K = C U_k and V = C U_v materialised (Eq. 5): their cache codes
  and scales bit for bit, their outputs within 2e-3 * ||o||_2 per row.
* Sweep corners (7B shape, H = 32, dh = 128): B = 64 sequences of 32768
  cached tokens at r = 3072 (clusters of four CTAs), int8 and int4, and B = 64
  x 16384 at r = 1024.  Sequences 0, 31 and 63 hold oracle-quantized latent
  rows with late high-score tokens and are checked against the oracle; the
  others hold seeded random codes and scales (they share the launch, not the
  check).  At these lengths the oracle takes the absorbed form of the same
  attention (pinned against the explicit form in the oracle tests).
"""
import math

import numpy as np
import pytest
import torch

import synthetic
from oracle import attention, pipeline, quant

from gpu_util import GpuLayer, assert_rows_close, bf16, cache_codes_np, cache_scales_np, dev, i32, q

pytestmark = pytest.mark.gpu


def test_llava13b_full_batch_chained_decode():
    lib = q()
    wl = synthetic.WORKLOADS["llava13b"]
    s = wl.shape
    steps = 2
    inp = synthetic.gen_layer(wl, seed=5, decode_steps=steps)
    w = pipeline.prepare_weights(inp)
    tracked = (0, 3, 7)
    P = wl.prefill
    tmax = P + steps
    ref = pipeline.OracleLayer(s, w, wl.B, tmax, wl.lat_bits, track=tracked)
    for b in tracked:
        ref.prefill(b, inp.X_prefill[b])
    gpu = GpuLayer(s, w, wl.B, tmax, wl.lat_bits)
    # the whole batch's prompts in one projection call, as the benchmark issues them
    X_all = inp.X_prefill.reshape(wl.B * P, s.d)
    seq = np.repeat(np.arange(wl.B), P)
    pos = np.tile(np.arange(P), wl.B)
    lib.qsvd_latent_project(gpu.W, bf16(X_all), 1.0, wl.lat_bits, 1.0, dst=gpu.cache, dst_seq=i32(seq),
                            dst_pos=i32(pos))
    lib.qsvd_check()
    gpu.len[:] = P
    for b in tracked:
        np.testing.assert_array_equal(cache_codes_np(gpu.cache, b, P), ref.cache.codes[b, :P])
        np.testing.assert_array_equal(cache_scales_np(gpu.cache, b, P), ref.cache.scale[b, :P])
    prev = lib.qsvd_set_decode_attn_path(0)
    try:
        for t in range(steps):
            O = gpu.decode_step(inp.X_decode[t])
            lib.qsvd_check()
            _, outs = ref.decode_step(inp.X_decode[t])
            got = O.cpu().numpy()
            assert np.isfinite(got).all()
            assert_rows_close(got[list(tracked)], np.stack([outs[b] for b in tracked]), f"13B step {t}")
    finally:
        lib.qsvd_set_decode_attn_path(prev)
    L = P + steps
    for b in tracked:
        np.testing.assert_array_equal(cache_codes_np(gpu.cache, b, L), ref.cache.codes[b, :L])
        np.testing.assert_array_equal(cache_scales_np(gpu.cache, b, L), ref.cache.scale[b, :L])


def _up_weights(H, dh, r, seed):
    shape = synthetic.LayerShape(H * dh, H, dh, r)
    wl = synthetic.Workload("attn", shape, B=1, n_image=0, n_text=0, decode_steps=0, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=seed, prefill_rows=0, decode_steps=0)
    return inp.U_q, inp.U_k, inp.U_v


def _sweep_corner(B, L, r, bits, seed):
    lib = q()
    H, dh = 32, 128
    checked = (0, B // 2 - 1, B - 1)
    U_q, U_k, U_v = _up_weights(H, dh, r, seed)
    cache = lib.LatentCache.empty(B, L, r, bits, dev())
    g = torch.Generator(device=dev()).manual_seed(seed + 1)
    if bits == 8:
        cache.codes.copy_(torch.randint(-127, 128, cache.codes.shape, generator=g, device=dev(), dtype=torch.int8))
        cache.scales.copy_(torch.rand(cache.scales.shape, generator=g, device=dev()) * 0.01 + 0.005)
    else:
        cache.codes.copy_(torch.randint(0, 256, cache.codes.shape, generator=g, device=dev(), dtype=torch.uint8))
        cache.scales.copy_((torch.rand(cache.scales.shape, generator=g, device=dev()) * 0.2 + 0.05).half())
    rng = np.random.default_rng(seed + 2)
    Uq, Uk, Uv = (synthetic.bf16_from_bits(u) for u in (U_q, U_k, U_v))
    refs = []
    for b in checked:
        x = synthetic.latent_rows(L, r, rng)
        for f in (0.02, 0.5, 0.97):             # late and early repeats of the current token
            x[int(f * (L - 1))] = x[L - 1]
        if bits == 8:
            codes, sc = quant.quantize_rows(x, 8)
            del x
            C = quant.dequantize_rows(codes, sc)
            cache.codes[b] = torch.from_numpy(codes.astype(np.int8)).to(dev())
            cache.scales[b] = torch.from_numpy(sc.astype(np.float32)).to(dev())
        else:
            codes, s16 = quant.quantize_int4_groups(x)
            del x
            C = quant.dequantize_int4_groups(codes, s16)
            cache.codes[b] = torch.from_numpy(quant.pack_int4(codes)).to(dev())
            cache.scales[b] = torch.from_numpy(s16.astype(np.float16)).to(dev())
        del codes
        refs.append(attention.decode_attention_absorbed(C, Uq, Uk, Uv, H, dh))
        del C
    O = torch.full((B, H * dh), float("nan"), dtype=torch.float32, device=dev())
    prev = lib.qsvd_set_decode_attn_path(0)
    try:
        lib.qsvd_latent_decode_attn(cache, i32([L] * B), L, bf16(U_q), bf16(U_k), bf16(U_v), H, dh, O)
        lib.qsvd_check()
    finally:
        lib.qsvd_set_decode_attn_path(prev)
    got = O.cpu().numpy()
    assert np.isfinite(got).all()
    assert_rows_close(got[list(checked)], np.stack(refs), f"B={B} L={L} r={r} int{bits}")


@pytest.mark.parametrize("bits", [8, 4])
def test_sweep_corner_b64_32k_r3072(bits):
    _sweep_corner(64, 32768, 3072, bits, seed=40 + bits)


def test_sweep_corner_b64_16k_r1024():
    _sweep_corner(64, 16384, 1024, 8, seed=50)


def test_sweep_corner_b64_16k_r1024_int4():
    _sweep_corner(64, 16384, 1024, 4, seed=51)
