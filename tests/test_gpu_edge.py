"""Degenerate cases of decode attention (Eq. 5) on every attention kernel.

* q~ = 0 (U_k = 0): every score is 0, the softmax is uniform over the L
  tokens, and the output is the mean of the cached latent rows times U_v.
  The oracle's explicit form gives exactly that; the kernels must reach it
  whatever their query scaling does with an all-zero query block.
* A zero latent cache row next to ordinary ones: scale 0, codes 0, score 0.

Paths: 0 automatic, 1 CUDA cores, 2 tcgen05, 3 warp-level MMA; int8 and int4
caches; per row max |error| <= 2e-3 * ||o_ref||_2.
"""
import numpy as np
import pytest
import torch

import synthetic
from oracle import attention, quant

from gpu_util import assert_rows_close, bf16, dev, i32, q

pytestmark = pytest.mark.gpu


def _fill(cache, b, x, bits):
    """Quantize fp64 rows x with the oracle's quantizer into cache row b;
    returns the dequantized rows."""
    L = x.shape[0]
    if bits == 8:
        codes, s = quant.quantize_rows(x, 8)
        cache.codes[b, :L] = torch.from_numpy(codes.astype(np.int8)).to(dev())
        cache.scales[b, :L] = torch.from_numpy(s.astype(np.float32)).to(dev())
        return quant.dequantize_rows(codes, s)
    codes, s16 = quant.quantize_int4_groups(x)
    cache.codes[b, :L] = torch.from_numpy(quant.pack_int4(codes)).to(dev())
    cache.scales[b, :L] = torch.from_numpy(s16.astype(np.float16)).to(dev())
    return quant.dequantize_int4_groups(codes, s16)


def _up(H, dh, r, seed):
    shape = synthetic.LayerShape(H * dh, H, dh, r)
    wl = synthetic.Workload("edge", shape, B=1, n_image=0, n_text=0, decode_steps=0, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=seed, prefill_rows=0, decode_steps=0)
    return inp.U_q, inp.U_k, inp.U_v


def _decode(lib, cache, lens, Uq, Uk, Uv, H, dh, path):
    prev = lib.qsvd_set_decode_attn_path(path)
    try:
        O = torch.full((len(lens), H * dh), float("nan"), dtype=torch.float32, device=dev())
        lib.qsvd_latent_decode_attn(cache, i32(lens), max(lens), Uq, Uk, Uv, H, dh, O)
        lib.qsvd_check()
    finally:
        lib.qsvd_set_decode_attn_path(prev)
    return O.cpu().numpy()


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("path", [0, 1, 2, 3])
def test_zero_query_gives_the_mean_of_v(bits, path):
    """U_k = 0: uniform softmax, o = mean_t(c_t) U_v (7B head shape, r = 1536,
    lengths 1, 130 and 700)."""
    lib = q()
    H, dh, r = 32, 128, 1536
    lens = [1, 130, 700]
    U_q, _, U_v = _up(H, dh, r, seed=61)
    U_k = np.zeros_like(U_q)                     # bf16 bit patterns of +0
    cache = lib.LatentCache.empty(len(lens), max(lens), r, bits, dev())
    rng = np.random.default_rng(62)
    refs = []
    Uq64, Uk64, Uv64 = (synthetic.bf16_from_bits(u) for u in (U_q, U_k, U_v))
    for b, L in enumerate(lens):
        C = _fill(cache, b, synthetic.latent_rows(L, r, rng), bits)
        ref = attention.decode_attention(C, Uq64, Uk64, Uv64, H, dh)
        np.testing.assert_allclose(ref, C.mean(axis=0) @ Uv64, rtol=1e-12, atol=1e-12)   # the closed form
        refs.append(ref)
    got = _decode(lib, cache, lens, bf16(U_q), bf16(U_k), bf16(U_v), H, dh, path)
    assert_rows_close(got, np.stack(refs), f"q~ = 0, int{bits}, path {path}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("path", [1, 2, 3])
def test_zero_cache_rows(bits, path):
    """Latent rows of zeros (scale 0) among ordinary rows, the current row
    included in one sequence: they score 0 and add nothing to o_lat."""
    lib = q()
    H, dh, r = 32, 128, 1536
    lens = [257, 64]
    U_q, U_k, U_v = _up(H, dh, r, seed=63)
    cache = lib.LatentCache.empty(len(lens), max(lens), r, bits, dev())
    rng = np.random.default_rng(64)
    refs = []
    Uq64, Uk64, Uv64 = (synthetic.bf16_from_bits(u) for u in (U_q, U_k, U_v))
    for b, L in enumerate(lens):
        x = synthetic.latent_rows(L, r, rng)
        x[::7] = 0.0
        if b == 1:
            x[-1] = 0.0                              # the current token's row: q = 0 for this sequence
        C = _fill(cache, b, x, bits)
        refs.append(attention.decode_attention(C, Uq64, Uk64, Uv64, H, dh))
    got = _decode(lib, cache, lens, bf16(U_q), bf16(U_k), bf16(U_v), H, dh, path)
    assert_rows_close(got, np.stack(refs), f"zero rows, int{bits}, path {path}")
