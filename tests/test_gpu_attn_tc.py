"""GPU parity of the tensor-core latent attention (Eq. 5, U_k absorbed into
the query, U_v applied last) against the oracle.

The cache content is an input here: seeded latent rows quantized by the
oracle's own quantizer (per-token int8, or int4 with fp16 scales per 128
channels), written into the device cache as is.  A few tokens repeat the
current token's latent row, so that their scores stand far above the rest and
the running softmax maximum jumps late in the sequence.  Every case runs the
tensor-core kernel (path 2) and, where stated, the CUDA-core kernels (path 1)
on the same cache; both must match the oracle to 2e-3 * ||o_ref||_2 per row.
"""
import math

import numpy as np
import pytest
import torch

import synthetic
from oracle import attention, quant

from gpu_util import assert_rows_close, bf16, dev, i32, q

pytestmark = pytest.mark.gpu


def _up_weights(H, dh, r, seed):
    shape = synthetic.LayerShape(H * dh, H, dh, r)
    wl = synthetic.Workload("attn", shape, B=1, n_image=0, n_text=0, decode_steps=0, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=seed, prefill_rows=0, decode_steps=0)
    return inp.U_q, inp.U_k, inp.U_v


def _cache_rows(lens, r, seed, hot):
    """fp64 latent rows per sequence; rows at the `hot` fractions of the
    length repeat the last (current) row."""
    rng = np.random.default_rng(seed)
    rows = []
    for L in lens:
        x = synthetic.latent_rows(L, r, rng)
        for f in hot:
            t = int(f * (L - 1))
            if 0 <= t < L - 1:
                x[t] = x[L - 1]
        rows.append(x)
    return rows


def _run(H, dh, r, bits, lens, paths=(2, 1), seed=0, hot=(0.3, 0.8), tmax=None):
    lib = q()
    B = len(lens)
    tmax = tmax or max(lens)
    U_q, U_k, U_v = _up_weights(H, dh, r, seed)
    rows = _cache_rows(lens, r, seed + 1, hot)
    cache = lib.LatentCache.empty(B, tmax, r, bits, dev())
    refs = []
    for b, (L, x) in enumerate(zip(lens, rows)):
        if bits == 8:
            codes, s = quant.quantize_rows(x, 8)
            C = quant.dequantize_rows(codes, s)
            cache.codes[b, :L] = torch.from_numpy(codes.astype(np.int8)).to(dev())
            cache.scales[b, :L] = torch.from_numpy(s.astype(np.float32)).to(dev())
        else:
            codes, s16 = quant.quantize_int4_groups(x)
            C = quant.dequantize_int4_groups(codes, s16)
            cache.codes[b, :L] = torch.from_numpy(quant.pack_int4(codes)).to(dev())
            cache.scales[b, :L] = torch.from_numpy(s16.astype(np.float16)).to(dev())
        refs.append(attention.decode_attention_absorbed(
            C, synthetic.bf16_from_bits(U_q), synthetic.bf16_from_bits(U_k), synthetic.bf16_from_bits(U_v), H, dh))
    ref = np.stack(refs)
    Uq, Uk, Uv = bf16(U_q), bf16(U_k), bf16(U_v)
    seq_len = i32(lens)
    outs = {}
    for path in paths:
        prev = lib.qsvd_set_decode_attn_path(path)
        try:
            O = torch.full((B, H * dh), float("nan"), dtype=torch.float32, device=dev())
            lib.qsvd_latent_decode_attn(cache, seq_len, max(lens), Uq, Uk, Uv, H, dh, O)
            lib.qsvd_check()
        finally:
            lib.qsvd_set_decode_attn_path(prev)
        got = O.cpu().numpy()
        assert np.isfinite(got).all(), f"path {path}: non-finite output"
        assert_rows_close(got, ref, f"path {path}")
        outs[path] = got
    return outs, ref


@pytest.mark.parametrize("bits", [8, 4])
def test_attn_tc_7b_ragged(bits):
    """r = 1536, H = 32, dh = 128: lengths 1 (the current token alone), one
    tile minus one, one tile plus one, and several tiles with a ragged tail."""
    _run(32, 128, 1536, bits, [1, 127, 129, 700])


@pytest.mark.parametrize("bits", [8, 4])
def test_attn_tc_long_sequence_multi_tile_splits(bits):
    """One 20000-token sequence: each CTA pair walks several tiles, reusing
    its double buffers, and the late high scores force o_lat rescaling."""
    _run(32, 128, 1536, bits, [20000], paths=(2,), hot=(0.1, 0.55, 0.97))


@pytest.mark.parametrize("H,dh,r,bits", [(8, 128, 512, 8), (20, 64, 768, 8), (20, 64, 768, 4), (16, 64, 256, 4)])
def test_attn_tc_head_and_rank_shapes(H, dh, r, bits):
    """N = 16 (H = 8, 16), padded heads (H = 20 -> 32), 1-3 chunks per CTA."""
    _run(H, dh, r, bits, [300, 64, 1000], seed=2)


@pytest.mark.parametrize("H,dh,r,bits,lens", [(32, 128, 2048, 8, [300, 129, 1000]), (32, 128, 3072, 4, [700, 1]),
                                               (16, 128, 2560, 8, [257, 900]), (32, 128, 2048, 4, [128, 640])])
def test_attn_tc_cluster_of_four(H, dh, r, bits, lens):
    """r > 1536: four CTAs per cluster (r/4 channels each, 4-6 chunks), every
    CTA sends its partial scores to three peers and adds all four in rank
    order; r = 2560 gives five chunks per CTA and N = 16."""
    _run(H, dh, r, bits, lens, paths=(2,), seed=21)


@pytest.mark.parametrize("bits", [8, 4])
def test_attn_tc_cluster_of_four_long_sequence(bits):
    """r = 3072: one 6000-token sequence over several tiles per cluster with
    late high scores (o_lat rescaling in all four CTAs)."""
    _run(32, 128, 3072, bits, [6000], paths=(2,), hot=(0.1, 0.55, 0.97), seed=22)


@pytest.mark.parametrize("bits", [4, 8])
def test_decode7b_full_size_sampled(bits):
    """The decode-heavy 7B shape at full size, in the launch configuration the
    benchmark times (automatic path: the tcgen05 kernel, one wave of CTA pairs
    over 9-tile splits): B = 16 sequences of 4097 cached tokens, r = 1536,
    H = 32.  Sequences 0, 9 and 15 hold oracle-quantized latent rows with late
    high-score tokens and are checked against the oracle; the other 13 hold
    seeded random codes and scales (they share the launch, not the check)."""
    lib = q()
    B, L, r, H, dh = 16, 4097, 1536, 32, 128
    checked = (0, 9, 15)
    U_q, U_k, U_v = _up_weights(H, dh, r, seed=31)
    rng = np.random.default_rng(32)
    cache = lib.LatentCache.empty(B, L, r, bits, dev())
    g = torch.Generator(device=dev()).manual_seed(33)
    if bits == 8:
        cache.codes.copy_(torch.randint(-127, 128, cache.codes.shape, generator=g, device=dev(), dtype=torch.int8))
        cache.scales.copy_(torch.rand(cache.scales.shape, generator=g, device=dev()) * 0.01 + 0.005)
    else:
        cache.codes.copy_(torch.randint(0, 256, cache.codes.shape, generator=g, device=dev(), dtype=torch.uint8))
        cache.scales.copy_((torch.rand(cache.scales.shape, generator=g, device=dev()) * 0.2 + 0.05).half())
    refs = []
    for b in checked:
        x = synthetic.latent_rows(L, r, rng)
        for f in (0.05, 0.5, 0.93):
            x[int(f * (L - 1))] = x[L - 1]
        if bits == 8:
            codes, sc = quant.quantize_rows(x, 8)
            C = quant.dequantize_rows(codes, sc)
            cache.codes[b] = torch.from_numpy(codes.astype(np.int8)).to(dev())
            cache.scales[b] = torch.from_numpy(sc.astype(np.float32)).to(dev())
        else:
            codes, s16 = quant.quantize_int4_groups(x)
            C = quant.dequantize_int4_groups(codes, s16)
            cache.codes[b] = torch.from_numpy(quant.pack_int4(codes)).to(dev())
            cache.scales[b] = torch.from_numpy(s16.astype(np.float16)).to(dev())
        refs.append(attention.decode_attention_absorbed(
            C, synthetic.bf16_from_bits(U_q), synthetic.bf16_from_bits(U_k), synthetic.bf16_from_bits(U_v), H, dh))
    O = torch.full((B, H * dh), float("nan"), dtype=torch.float32, device=dev())
    prev = lib.qsvd_set_decode_attn_path(0)
    try:
        lib.qsvd_latent_decode_attn(cache, i32([L] * B), L, bf16(U_q), bf16(U_k), bf16(U_v), H, dh, O)
        lib.qsvd_check()
    finally:
        lib.qsvd_set_decode_attn_path(prev)
    got = O.cpu().numpy()
    assert np.isfinite(got).all()
    assert_rows_close(got[list(checked)], np.stack(refs), "decode7b full size")


@pytest.mark.parametrize("H,dh,r,bits,lens", [(40, 128, 2048, 8, [3000, 77]), (40, 128, 2048, 4, [1200, 300]),
                                               (48, 64, 1024, 8, [500, 129])])
def test_attn_tc_more_than_32_heads(H, dh, r, bits, lens):
    """H > 32: one launch per group of at most 32 heads over the same splits
    (the 13B shape, H = 40: heads 0-31 then 32-39 with N = 16; H = 48 with
    pairs of CTAs: 32 + 16 heads), each launch's partials at its heads."""
    _run(H, dh, r, bits, lens, paths=(2,), seed=23)


def test_attn_tc_cache_larger_than_lengths():
    """Tmax above every length: the rows after each sequence's end belong to
    no token and must not contribute."""
    _run(32, 128, 1536, 8, [200, 513], tmax=900, seed=4)


@pytest.mark.parametrize("bits", [8, 4])
def test_attn_mma_ragged(bits):
    """The warp-level MMA kernel (path 3): lengths 1, 15, 17, 700 at r = 1536,
    H = 32 (16-token splits), against the oracle and the other kernels."""
    outs, ref = _run(32, 128, 1536, bits, [1, 15, 17, 700], paths=(3, 2, 1), seed=12)


@pytest.mark.parametrize("H,dh,r,bits,lens", [(40, 128, 2048, 8, [3000, 77]), (4, 64, 96, 8, [80, 33]),
                                               (20, 64, 768, 4, [2049, 64]), (32, 128, 3072, 8, [1500, 33]),
                                               (40, 128, 2048, 8, [9000, 300]), (32, 128, 3072, 4, [5000, 17])])
def test_attn_mma_shapes(H, dh, r, bits, lens):
    """H = 40 (five head groups of 8) at the 13B rank with 64-token splits,
    the tiny layer (r = 96, padded heads), a 32-token split with int4,
    r = 3072, where the sub-tile is capped at 32 tokens by shared memory, and
    lengths beyond 64 sub-tiles (each CTA walks several sub-tiles with a
    running softmax) at r = 2048 and r = 3072 (int4)."""
    _run(H, dh, r, bits, lens, paths=(3,), seed=13)


def test_attn_tc_path_selection():
    """The automatic choice uses the tensor cores for a large batch x length
    and the setting is restored; an unsupported shape falls back silently."""
    lib = q()
    assert lib.qsvd_set_decode_attn_path(0) == 0
    assert lib.qsvd_set_decode_attn_path(2) == 0
    assert lib.qsvd_set_decode_attn_path(0) == 2
    with pytest.raises(lib.QsvdError):
        lib.qsvd_set_decode_attn_path(4)
    # r = 2304 does not split into four CTAs of whole 128-channel chunks: path 2 still answers correctly
    _run(8, 128, 2304, 8, [300, 40], paths=(2,), seed=6)
