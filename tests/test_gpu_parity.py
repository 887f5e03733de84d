"""GPU parity: the CUDA path through the C ABI against the CPU oracle on the
same seeded inputs.  Integer results (codes, int32 accumulators, scales) must
be bit-exact; decode outputs must agree to 2e-3 * ||o_ref||_2 max-abs per
row."""
import math

import numpy as np
import pytest
import torch

import synthetic
from oracle import latent, pipeline, quant

from gpu_util import GpuLayer, assert_rows_close, bf16, dev, i32, q

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny():
    wl = synthetic.WORKLOADS["tiny"]
    inp = synthetic.gen_layer(wl, seed=0)
    return wl, inp, pipeline.prepare_weights(inp)


@pytest.fixture(scope="module")
def l7b():
    wl = synthetic.WORKLOADS["llava7b"]
    inp = synthetic.gen_layer(wl, seed=0)
    return wl, inp, pipeline.prepare_weights(inp)


def _project_outputs(W, X_bits, r, bits, act_clip=1.0, lat_clip=1.0):
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
    lib.qsvd_latent_project(W, bf16(X_bits), act_clip, bits, lat_clip, lat_codes=lc, lat_scales=ls,
                            xq_out=xq, xs_out=xs, acc_out=acc)
    lib.qsvd_check()
    return {k: v.cpu().numpy() for k, v in dict(xq=xq, xs=xs, acc=acc, codes=lc, scale=ls).items()}


def _assert_project_exact(got, ref, bits):
    np.testing.assert_array_equal(got["xq"].astype(np.int64), ref["xq"])
    np.testing.assert_array_equal(got["xs"].astype(np.float64), ref["s_x"])
    np.testing.assert_array_equal(got["acc"].astype(np.int64), ref["acc"])
    if bits == 8:
        np.testing.assert_array_equal(got["codes"].astype(np.int64), ref["codes"])
    else:
        np.testing.assert_array_equal(got["codes"], quant.pack_int4(ref["codes"]))
    np.testing.assert_array_equal(got["scale"].astype(np.float64), ref["scale"])


# ---------------------------------------------------------------------------
# weight preparation
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["tiny", "llava7b"])
def test_quantize_weight_bit_exact(name, tiny, l7b):
    wl, inp, w = tiny if name == "tiny" else l7b
    W = q().qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    np.testing.assert_array_equal(W.codes.cpu().numpy().astype(np.int64), w["Wq"].T)
    np.testing.assert_array_equal(W.scale.cpu().numpy().astype(np.float64), w["s_w"])
    np.testing.assert_array_equal(W.codes_bf16.float().cpu().numpy(), w["Wq"].T.astype(np.float32))


# ---------------------------------------------------------------------------
# a1-a4: projection, requantization, append
# ---------------------------------------------------------------------------
def test_project_tiny_bit_exact(tiny):
    wl, inp, w = tiny
    W = q().qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    X = inp.X_prefill[0]
    got = _project_outputs(W, X, wl.shape.r, 8)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), w["Wq"], w["s_w"], lat_bits=8)
    _assert_project_exact(got, ref, 8)


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("T", [1, 3, 4, 9, 16, 37, 64, 65, 640])
def test_project_7b_bit_exact(l7b, bits, T):
    """T <= 3: the decode projection quantizes with the whole CTA; 4 <= T <= 64:
    xquant, the tensor-core dot products in 16-token blocks (a ragged last
    block at 37), requant; larger T: the GEMM."""
    wl, inp, w = l7b
    W = q().qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    X = inp.X_prefill[0][:T]
    got = _project_outputs(W, X, wl.shape.r, bits)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), w["Wq"], w["s_w"], lat_bits=bits)
    _assert_project_exact(got, ref, bits)


def test_project_clip_and_zero_rows(l7b):
    wl, inp, w = l7b
    W = q().qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    X = inp.X_prefill[0][:20].copy()
    X[3] = 0                      # an all-zero token: scale 0, codes 0, latent 0
    X[7, 11] = synthetic.bf16_bits([3.0e4])[0]    # a saturating outlier
    got = _project_outputs(W, X, wl.shape.r, 8, act_clip=0.9, lat_clip=0.85)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), w["Wq"], w["s_w"], 0.9, 8, 0.85)
    _assert_project_exact(got, ref, 8)
    assert got["xs"][3] == 0 and not got["codes"][3].any()


@pytest.mark.parametrize("bits", [8, 4])
def test_cache_append_and_fused_store(l7b, bits):
    """Token-major output + qsvd_cache_append equals the fused store, and both
    equal the oracle's cache image; rows land at the requested (seq, pos)."""
    wl, inp, w = l7b
    lib = q()
    r = wl.shape.r
    W = lib.qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    X = inp.X_prefill[0][:29]
    seq = np.array([i % 3 for i in range(29)])
    pos = np.array([5 + i // 3 for i in range(29)])
    c1 = lib.LatentCache.empty(3, 20, r, bits, dev())
    c2 = lib.LatentCache.empty(3, 20, r, bits, dev())
    lib.qsvd_latent_project(W, bf16(X), lat_bits=bits, dst=c1, dst_seq=i32(seq), dst_pos=i32(pos))
    got = _project_outputs(W, X, r, bits)
    lib.qsvd_cache_append(c2, i32(seq), i32(pos), torch.from_numpy(got["codes"]).to(dev()),
                          torch.from_numpy(got["scale"]).to(dev()))
    lib.qsvd_check()
    ref = latent.latent_project(synthetic.bf16_from_bits(X), w["Wq"], w["s_w"], lat_bits=bits)
    oc = latent.LatentCache(3, 20, r, bits)
    oc.append(seq, pos, ref["codes"], ref["scale"])
    for c in (c1, c2):
        np.testing.assert_array_equal(c.codes.cpu().numpy().view(np.uint8),
                                      oc.packed_codes().view(np.uint8))
        np.testing.assert_array_equal(c.scales.cpu().numpy().astype(np.float64), oc.scale)


# ---------------------------------------------------------------------------
# a5-a8: decode attention, end to end
# ---------------------------------------------------------------------------
def _run_decode(wl, inp, w, steps, check_steps, B=None, track=None):
    B = wl.B if B is None else B
    s = wl.shape
    ref = pipeline.OracleLayer(s, w, B, wl.tmax, wl.lat_bits, track=track)
    gpu = GpuLayer(s, w, B, wl.tmax, wl.lat_bits)
    for b in range(B):
        ref.prefill(b, inp.X_prefill[b])
        gpu.prefill(b, inp.X_prefill[b])
    for step in range(steps):
        _, outs = ref.decode_step(inp.X_decode[step], attend=[] if step not in check_steps else None)
        O = gpu.decode_step(inp.X_decode[step])
        if step in check_steps:
            q().qsvd_check()
            o = O.cpu().numpy()
            bs = sorted(outs)
            assert_rows_close(o[bs], np.stack([outs[b] for b in bs]), f"step {step}")
    q().qsvd_check()
    for b in sorted(ref.track):
        L = int(ref.len[b])
        got = gpu.cache.codes[b, :L].cpu().numpy().view(np.uint8)
        np.testing.assert_array_equal(got, ref.cache.packed_codes()[b, :L].view(np.uint8))
    return ref, gpu


def test_decode_tiny_all_steps(tiny):
    wl, inp, w = tiny
    _run_decode(wl, inp, w, wl.decode_steps, set(range(wl.decode_steps)))


def test_decode_7b_sampled_steps(l7b):
    wl, inp, w = l7b
    _run_decode(wl, inp, w, wl.decode_steps, {0, 1, 63, wl.decode_steps - 1})


@pytest.mark.parametrize("bits", [8, 4])
def test_decode_batch_ragged_lengths(bits):
    """B = 3 sequences of different lengths (one below, one at, one above a
    256-token chunk boundary), int8 and int4 caches, H = 32."""
    base = synthetic.WORKLOADS["llava7b"]
    wl = synthetic.Workload("ragged", base.shape, B=3, n_image=0, n_text=300, decode_steps=3,
                            lat_bits=bits)
    inp = synthetic.gen_layer(wl, seed=5)
    w = pipeline.prepare_weights(inp)
    s = wl.shape
    ref = pipeline.OracleLayer(s, w, 3, wl.tmax, bits)
    gpu = GpuLayer(s, w, 3, wl.tmax, bits)
    for b, n in enumerate((100, 255, 300)):
        ref.prefill(b, inp.X_prefill[b][:n])
        gpu.prefill(b, inp.X_prefill[b][:n])
    for step in range(3):
        _, outs = ref.decode_step(inp.X_decode[step])
        o = gpu.decode_step(inp.X_decode[step]).cpu().numpy()
        assert_rows_close(o, np.stack([outs[b] for b in range(3)]), f"step {step}")


@pytest.mark.parametrize("B,bits", [(5, 8), (6, 4), (9, 8), (17, 4)])
def test_decode_large_batch_tensor_core_products(B, bits):
    """From 5 sequences on, the up-projection products run on the tensor cores
    (16 sequences per pass: B = 5 fills 5 of them, B = 17 takes two passes);
    ragged lengths."""
    base = synthetic.WORKLOADS["llava7b"]
    wl = synthetic.Workload("batch", base.shape, B=B, n_image=0, n_text=160, decode_steps=2, lat_bits=bits)
    inp = synthetic.gen_layer(wl, seed=21)
    w = pipeline.prepare_weights(inp)
    s = wl.shape
    ref = pipeline.OracleLayer(s, w, B, wl.tmax, bits)
    gpu = GpuLayer(s, w, B, wl.tmax, bits)
    lens = [1 + (37 * b) % 160 for b in range(B)]
    for b, n in enumerate(lens):
        ref.prefill(b, inp.X_prefill[b][:n])
        gpu.prefill(b, inp.X_prefill[b][:n])
    for step in range(2):
        _, outs = ref.decode_step(inp.X_decode[step])
        o = gpu.decode_step(inp.X_decode[step]).cpu().numpy()
        assert_rows_close(o, np.stack([outs[b] for b in range(B)]), f"step {step}")


@pytest.mark.parametrize("r,bits", [(512, 8), (1024, 4), (3072, 8)])
def test_decode_batched_weight_rings(r, bits):
    """The batched up-projection kernels stream their weight rows through a
    shared-memory ring: r = 512 takes one slot (one 128-row group of U_q, one
    64-row chunk of U_v per CTA), r = 1024 two slots exactly filled, r = 3072
    six groups / chunks through two slots (the ring wraps three times).
    d = 1024 (8 heads), B = 6, ragged lengths."""
    wl = synthetic.Workload("rings", synthetic.LayerShape(1024, 8, 128, r), B=6, n_image=0, n_text=90,
                            decode_steps=2, lat_bits=bits)
    inp = synthetic.gen_layer(wl, seed=23)
    w = pipeline.prepare_weights(inp)
    s = wl.shape
    ref = pipeline.OracleLayer(s, w, wl.B, wl.tmax, bits)
    gpu = GpuLayer(s, w, wl.B, wl.tmax, bits)
    for b, n in enumerate((1, 17, 40, 64, 77, 90)):
        ref.prefill(b, inp.X_prefill[b][:n])
        gpu.prefill(b, inp.X_prefill[b][:n])
    for step in range(2):
        _, outs = ref.decode_step(inp.X_decode[step])
        o = gpu.decode_step(inp.X_decode[step]).cpu().numpy()
        assert_rows_close(o, np.stack([outs[b] for b in range(wl.B)]), f"r {r} step {step}")


def test_decode_13b_heads_and_rank():
    """H = 40 (five head groups of 8), r = 2048, d = 5120."""
    base = synthetic.WORKLOADS["llava13b"]
    wl = synthetic.Workload("13b_small", base.shape, B=2, n_image=280, n_text=20, decode_steps=2,
                            lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=3)
    w = pipeline.prepare_weights(inp)
    _run_decode(wl, inp, w, 2, {0, 1})


def test_decode_single_token():
    """L = 1: the output is the current token's V row, c_0 U_v."""
    base = synthetic.WORKLOADS["llava7b"]
    wl = synthetic.Workload("one", base.shape, B=2, n_image=0, n_text=0, decode_steps=1, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=9)
    w = pipeline.prepare_weights(inp)
    ref, gpu = _run_decode(wl, inp, w, 1, {0})
    assert list(ref.len) == [1, 1]


# ---------------------------------------------------------------------------
# host-side argument checks and device-side range flags (no GPU fault)
# ---------------------------------------------------------------------------
def test_error_paths(tiny):
    wl, inp, w = tiny
    lib = q()
    r = wl.shape.r
    W = lib.qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    X = bf16(inp.X_prefill[0][:4])
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_project(W, X, lat_bits=8)                  # no destination
    assert e.value.status == lib.QSVD_EINVAL
    lc = torch.empty((4, r), dtype=torch.int8, device=dev())
    ls = torch.empty((4,), dtype=torch.float32, device=dev())
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_project(W, X, lat_bits=4, lat_codes=lc, lat_scales=ls)   # r % 128 != 0
    assert e.value.status == lib.QSVD_EUNSUPPORTED
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_project(W, X, lat_codes=lc, lat_scales=ls,
                                workspace=torch.empty(16, dtype=torch.uint8, device=dev()))
    assert e.value.status == lib.QSVD_ENOSPC
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_project(W, X, act_clip=0.0, lat_codes=lc, lat_scales=ls)
    assert e.value.status == lib.QSVD_EINVAL
    # out-of-range cache position: the row is skipped, qsvd_check reports it
    cache = lib.LatentCache.empty(1, 8, r, 8, dev())
    lib.qsvd_latent_project(W, X, dst=cache, dst_seq=i32([0, 0, 0, 1]), dst_pos=i32([0, 1, 8, 0]))
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_check()
    assert e.value.status == lib.QSVD_ERANGE
    lib.qsvd_check()          # the word was cleared
    assert cache.codes[0, :2].abs().sum() > 0 and cache.codes[0, 2:].abs().sum() == 0
    # decode with a length beyond Tmax
    O = torch.empty((1, wl.shape.d), dtype=torch.float32, device=dev())
    U = bf16(w["U_q"])
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_decode_attn(cache, i32([3]), 9, U, U, U, wl.shape.H, wl.shape.dh, O)
    assert e.value.status == lib.QSVD_EINVAL
    lib.qsvd_latent_decode_attn(cache, i32([0]), 8, U, U, U, wl.shape.H, wl.shape.dh, O)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_check()
    assert e.value.status == lib.QSVD_ERANGE


def test_bounded_wait_expiry_is_reported():
    """Failure detection without a fault: a bounded device wait on a barrier
    nothing completes expires after 5 ms, sets the timeout bit, and qsvd_check
    reports QSVD_ETIMEOUT once; the context keeps running kernels after it."""
    lib = q()
    lib.qsvd_check()
    lib.qsvd_selftest_wait_timeout(5)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_check()
    assert e.value.status == lib.QSVD_ETIMEOUT
    assert lib.qsvd_check() == lib.QSVD_OK          # the word was cleared
    for bad in (0, 1001):
        with pytest.raises(lib.QsvdError) as e:
            lib.qsvd_selftest_wait_timeout(bad)
        assert e.value.status == lib.QSVD_EINVAL
    W = lib.qsvd_quantize_weight(torch.ones((64, 16), dtype=torch.float32, device=dev()))
    assert lib.qsvd_check() == lib.QSVD_OK
    assert int(W.codes.abs().max()) == 127


# ---------------------------------------------------------------------------
# tensor-core projection: exactness at the extremes of the int8 range
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("d,r,T", [(4096, 1536, 200), (5120, 2048, 131)])
def test_project_tc_worst_case_exact(d, r, T):
    """Every code at +-127: |acc| = 127^2 d exceeds 2^24, so the result is
    exact only if the fp32 tensor-core partial sums are drained to int32
    before they leave the exact-integer range of fp32."""
    lib = q()
    rng = np.random.default_rng(d + r)
    W = np.full((d, r), 0.01, dtype=np.float32)
    W[:, 1::3] = -0.02                       # a third of the channels at -127
    X = np.ones((T, d))
    X[1::2, ::2] = -1.0                      # alternate signs along K on odd tokens
    X[5] = rng.standard_normal(d)            # one ordinary row
    Xb = synthetic.bf16_bits(X)
    Wq = lib.qsvd_quantize_weight(torch.from_numpy(W).to(dev()))
    got = _project_outputs(Wq, Xb, r, 8)
    Wc, s_w = quant.quantize_columns(W.astype(np.float64), 8)
    ref = latent.latent_project(synthetic.bf16_from_bits(Xb), Wc, s_w, lat_bits=8)
    assert np.abs(ref["acc"]).max() > 2 ** 24
    _assert_project_exact(got, ref, 8)


@pytest.mark.parametrize("T", [5, 16])
def test_project_small_13b_and_tiny_shapes(T):
    """The decode projection at d = 5120, r = 2048 (K split 640 per warp) and at
    the tiny layer's d = 256 (32 per warp), against the oracle, bit-exact."""
    for name in ("llava13b", "tiny"):
        wl = synthetic.WORKLOADS[name]
        s = wl.shape
        rng = np.random.default_rng(11)
        w = (rng.standard_normal((s.d, s.r)) / np.sqrt(s.d)).astype(np.float32)
        X = synthetic.bf16_bits(rng.standard_normal((T, s.d)) * np.where(rng.random(s.d) < 0.01, 20.0, 1.0))
        wq, s_w = quant.quantize_columns(w.astype(np.float64), 8)
        W = q().qsvd_quantize_weight(torch.from_numpy(w).to(dev()))
        for bits in ((8, 4) if s.r % 128 == 0 else (8,)):      # int4 needs whole 128-channel groups
            got = _project_outputs(W, X, s.r, bits)
            ref = latent.latent_project(synthetic.bf16_from_bits(X), wq, s_w, lat_bits=bits)
            _assert_project_exact(got, ref, bits)


def test_project_13b_shape_tc():
    base = synthetic.WORKLOADS["llava13b"]
    wl = synthetic.Workload("13b_proj", base.shape, B=1, n_image=300, n_text=0, decode_steps=0, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=2)
    w = pipeline.prepare_weights(inp)
    W = q().qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    X = inp.X_prefill[0]
    for bits in (8, 4):
        got = _project_outputs(W, X, wl.shape.r, bits)
        ref = latent.latent_project(synthetic.bf16_from_bits(X), w["Wq"], w["s_w"], lat_bits=bits)
        _assert_project_exact(got, ref, bits)


# ---------------------------------------------------------------------------
# requantization in the GEMM epilogue vs the separate kernel
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("mode", [1, 2])
@pytest.mark.parametrize("shape_name,T", [("llava7b", 300), ("llava13b", 300)])
def test_project_epilogue_modes(mode, shape_name, T):
    """Both requantization placements (separate kernel: mode 1; GEMM
    epilogue, int8 through a cluster of r/256 CTAs: mode 2) give the oracle's
    codes and scales, into the token-major outputs and into the cache."""
    lib = q()
    base = synthetic.WORKLOADS[shape_name]
    wl = synthetic.Workload("epi", base.shape, B=1, n_image=T, n_text=0, decode_steps=0, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=11)
    w = pipeline.prepare_weights(inp)
    W = lib.qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    X = inp.X_prefill[0]
    r = wl.shape.r
    prev = lib.qsvd_set_project_epilogue(mode)
    try:
        for bits in (8, 4):
            got = _project_outputs(W, X, r, bits)
            ref = latent.latent_project(synthetic.bf16_from_bits(X), w["Wq"], w["s_w"], lat_bits=bits)
            _assert_project_exact(got, ref, bits)
            # the cache store of the same call (rows scattered over two sequences)
            cache = lib.LatentCache.empty(2, T, r, bits, dev())
            seq = np.arange(T) % 2
            pos = np.arange(T) // 2
            lib.qsvd_latent_project(W, bf16(X), 1.0, bits, 1.0, dst=cache, dst_seq=i32(seq), dst_pos=i32(pos))
            lib.qsvd_check()
            codes = cache.codes.cpu().numpy()[seq, pos]
            scales = cache.scales.cpu().numpy()[seq, pos]
            if bits == 8:
                np.testing.assert_array_equal(codes.astype(np.int64), ref["codes"])
            else:
                np.testing.assert_array_equal(codes, quant.pack_int4(ref["codes"]))
            np.testing.assert_array_equal(scales.astype(np.float64), ref["scale"])
    finally:
        lib.qsvd_set_project_epilogue(prev)
