"""Causal prefill attention over the latent cache (qsvd_latent_prefill_attn)
against the oracle's masked matrix form (oracle.attention.prefill_attention).

Each test projects prompts into the cache on both sides (codes bit-exact),
then lets every prompt token attend to its own prefix.  Per output row the
bar is the decode tolerance: max |error| <= 2e-3 * ||row||_2."""
import numpy as np
import pytest
import torch

import synthetic
from gpu_util import GpuLayer, assert_rows_close, dev, i32, q
from oracle import attention, pipeline

pytestmark = pytest.mark.gpu


def _layers(name, B, n_text, bits, seed, n_image=0, tmax=None):
    base = synthetic.WORKLOADS[name]
    wl = synthetic.Workload("prefill", base.shape, B=B, n_image=n_image, n_text=n_text, decode_steps=0,
                            lat_bits=bits)
    inp = synthetic.gen_layer(wl, seed=seed)
    w = pipeline.prepare_weights(inp)
    tmax = wl.tmax if tmax is None else tmax
    ref = pipeline.OracleLayer(wl.shape, w, B, tmax, bits, track=[])
    gpu = GpuLayer(wl.shape, w, B, tmax, bits)
    return wl, inp, ref, gpu


def _gpu_prefill(gpu, q_seq, q_len, max_len=None):
    s = gpu.s
    O = torch.full((len(q_seq), s.d), float("nan"), dtype=torch.float32, device=dev())
    max_len = int(max(q_len)) if max_len is None else max_len
    gpu.lib.qsvd_latent_prefill_attn(gpu.cache, i32(q_seq), i32(q_len), max_len, gpu.U_q, gpu.U_k, gpu.U_v,
                                     s.H, s.dh, O)
    return O


def _oracle_rows(ref, b, t0, L):
    """Oracle outputs of positions t0 .. L-1 of sequence b."""
    return attention.prefill_attention(ref.cache.rows(b, L), ref.U_q, ref.U_k, ref.U_v, ref.s.H, ref.s.dh,
                                       t0=t0)


def _assert_cache_equal(ref, gpu, b, L):
    got = gpu.cache.codes[b, :L].cpu().numpy().view(np.uint8)
    np.testing.assert_array_equal(got, ref.cache.packed_codes()[b, :L].view(np.uint8))


@pytest.mark.parametrize("bits", [8, 4])
def test_prefill_one_prompt(bits):
    """A 300-token prompt (two full 128-token tiles and a ragged one): every
    position attends to positions 0 .. itself."""
    wl, inp, ref, gpu = _layers("llava7b", 1, 300, bits, seed=41)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    _assert_cache_equal(ref, gpu, 0, 300)
    O = _gpu_prefill(gpu, np.zeros(300), np.arange(1, 301))
    q().qsvd_check()
    assert_rows_close(O.cpu().numpy(), _oracle_rows(ref, 0, 0, 300), f"prefill int{bits}")


def test_prefill_llava_prompt_all_rows():
    """The 7B-shaped prompt of 576 image-like and 64 text-like tokens, int8:
    640 rows in five groups of 128 that reuse one workspace."""
    wl, inp, ref, gpu = _layers("llava7b", 1, 64, 8, seed=42, n_image=576)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    n = wl.prefill
    prev = q().qsvd_set_prefill_group_rows(128)
    try:
        assert q().qsvd_prefill_workspace_bytes(n, n, wl.shape.r, wl.shape.H, wl.shape.dh) == \
            q().qsvd_decode_workspace_bytes(128, n, wl.shape.r, wl.shape.H, wl.shape.dh)
        O = _gpu_prefill(gpu, np.zeros(n), np.arange(1, n + 1))
        q().qsvd_check()
    finally:
        q().qsvd_set_prefill_group_rows(prev)
    assert_rows_close(O.cpu().numpy(), _oracle_rows(ref, 0, 0, n), "prefill 640")


def test_prefill_continuation_and_mixed_rows():
    """Sequence 0 holds 100 earlier tokens and appends 150 more; sequence 1
    holds a 200-token prompt.  One call takes the 150 + 200 rows in a shuffled
    order (int4 cache)."""
    wl, inp, ref, gpu = _layers("llava7b", 2, 250, 4, seed=43)
    for side in (ref, gpu):
        side.prefill(0, inp.X_prefill[0][:100])
        side.prefill(0, inp.X_prefill[0][100:250])
        side.prefill(1, inp.X_prefill[1][:200])
    rows = [(0, 100 + i + 1) for i in range(150)] + [(1, i + 1) for i in range(200)]
    order = np.random.default_rng(7).permutation(len(rows))
    q_seq = np.array([rows[k][0] for k in order])
    q_len = np.array([rows[k][1] for k in order])
    O = _gpu_prefill(gpu, q_seq, q_len).cpu().numpy()
    q().qsvd_check()
    ref0 = _oracle_rows(ref, 0, 100, 250)
    ref1 = _oracle_rows(ref, 1, 0, 200)
    want = np.stack([ref0[L - 101] if b == 0 else ref1[L - 1] for b, L in zip(q_seq, q_len)])
    assert_rows_close(O, want, "mixed rows")


def test_prefill_13b_more_than_32_heads():
    """d = 5120, H = 40 (two head groups on the tcgen05 path), r = 2048."""
    wl, inp, ref, gpu = _layers("llava13b", 1, 200, 8, seed=44)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    O = _gpu_prefill(gpu, np.zeros(200), np.arange(1, 201))
    q().qsvd_check()
    assert_rows_close(O.cpu().numpy(), _oracle_rows(ref, 0, 0, 200), "prefill 13B")


def test_prefill_13b_long_prompt_sampled():
    """One 13B-shaped prompt of 3008 tokens (5 x 576 image-like + 128 text),
    every row computed on the GPU; sampled rows (tile edges, the middle, the
    last) checked against the oracle's decode over the prefix."""
    wl, inp, ref, gpu = _layers("llava13b", 1, 128, 8, seed=45, n_image=2880)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    n = wl.prefill
    O = _gpu_prefill(gpu, np.zeros(n), np.arange(1, n + 1)).cpu().numpy()
    q().qsvd_check()
    assert np.isfinite(O).all()
    C = ref.cache.rows(0, n)
    s = wl.shape
    for t in (0, 1, 127, 128, 1500, n - 1):
        want = attention.decode_attention(C[:t + 1], ref.U_q, ref.U_k, ref.U_v, s.H, s.dh)
        assert_rows_close(O[t:t + 1], want[None], f"row {t}")


def test_prefill_invalid_rows_are_zero_and_flagged():
    """Rows whose sequence lies outside the cache or whose length is outside
    [1, Tmax] are skipped: zero output, QSVD_ERANGE from qsvd_check; the
    other rows of the call are unaffected."""
    wl, inp, ref, gpu = _layers("llava7b", 2, 40, 8, seed=46)
    for side in (ref, gpu):
        side.prefill(0, inp.X_prefill[0])
        side.prefill(1, inp.X_prefill[1])
    lib = q()
    tmax = gpu.cache.Tmax
    q_seq = np.array([0, -1, 1, 2, 0, 1, 0])
    q_len = np.array([5, 5, 40, 3, 0, tmax + 1, 40])
    O = _gpu_prefill(gpu, q_seq, q_len, max_len=tmax).cpu().numpy()
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_check()
    assert e.value.status == lib.QSVD_ERANGE
    lib.qsvd_check()                       # the flag was cleared
    for i in (1, 3, 4, 5):
        np.testing.assert_array_equal(O[i], 0.0)
    want = np.stack([_oracle_rows(ref, 0, 4, 5)[0], _oracle_rows(ref, 1, 39, 40)[0],
                     _oracle_rows(ref, 0, 39, 40)[0]])
    assert_rows_close(O[[0, 2, 6]], want, "valid rows")


def test_prefill_host_argument_errors():
    wl, inp, ref, gpu = _layers("llava7b", 1, 16, 8, seed=47)
    lib, s = q(), wl.shape
    O = torch.empty((4, s.d), dtype=torch.float32, device=dev())
    with pytest.raises(ValueError):
        lib.qsvd_latent_prefill_attn(gpu.cache, i32([0, 0, 0, 0]), i32([1, 2, 3]), 3, gpu.U_q, gpu.U_k, gpu.U_v,
                                     s.H, s.dh, O)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_prefill_attn(gpu.cache, i32([0] * 4), i32([1, 2, 3, 4]), gpu.cache.Tmax + 1, gpu.U_q,
                                     gpu.U_k, gpu.U_v, s.H, s.dh, O)
    assert e.value.status == lib.QSVD_EINVAL
    small = torch.zeros(256, dtype=torch.uint8, device=dev())
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_prefill_attn(gpu.cache, i32([0] * 4), i32([1, 2, 3, 4]), 4, gpu.U_q, gpu.U_k, gpu.U_v,
                                     s.H, s.dh, O, workspace=small)
    assert e.value.status == lib.QSVD_ENOSPC
    empty = torch.empty((0,), dtype=torch.int32, device=dev())
    lib.qsvd_latent_prefill_attn(gpu.cache, empty, empty, 1, gpu.U_q, gpu.U_k, gpu.U_v, s.H, s.dh, O)
    lib.qsvd_check()


# ---------------------------------------------------------------------------
# whole prompt blocks, K and V materialised (qsvd_latent_prefill)
# ---------------------------------------------------------------------------
def _gpu_blocks(gpu, blocks, Ut=None):
    s = gpu.s
    Ut = gpu.lib.qsvd_prefill_weights(gpu.U_q, gpu.U_k, gpu.U_v) if Ut is None else Ut
    n = sum(T for _, _, T in blocks)
    O = torch.full((n, s.d), float("nan"), dtype=torch.float32, device=dev())
    gpu.lib.qsvd_latent_prefill(gpu.cache, blocks, Ut, s.H, s.dh, O)
    q().qsvd_check()
    return O.cpu().numpy()


def test_prefill_weights_transpose():
    """Ut = [U_q U_k U_v]^T in fp16 (bf16 values are exact in fp16 at these
    magnitudes)."""
    wl, inp, ref, gpu = _layers("llava7b", 1, 4, 8, seed=50)
    Ut = gpu.lib.qsvd_prefill_weights(gpu.U_q, gpu.U_k, gpu.U_v).float().cpu().numpy()
    want = np.concatenate([ref.U_q, ref.U_k, ref.U_v], axis=1).T
    np.testing.assert_array_equal(Ut, want.astype(np.float16).astype(np.float32))


@pytest.mark.parametrize("bits", [8, 4])
def test_latent_prefill_one_prompt(bits):
    wl, inp, ref, gpu = _layers("llava7b", 1, 300, bits, seed=51)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    O = _gpu_blocks(gpu, [(0, 0, 300)])
    assert_rows_close(O, _oracle_rows(ref, 0, 0, 300), f"blocks int{bits}")


def test_latent_prefill_llava_prompt():
    wl, inp, ref, gpu = _layers("llava7b", 1, 64, 8, seed=52, n_image=576)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    n = wl.prefill
    assert_rows_close(_gpu_blocks(gpu, [(0, 0, n)]), _oracle_rows(ref, 0, 0, n), "blocks 640")


def test_latent_prefill_mixed_blocks():
    """Blocks of two sequences in one call: a continued prompt (t0 = 100), a
    short block inside another one's range, a block shorter than a tile, and
    t0 values that are not multiples of 128 (int4 cache)."""
    wl, inp, ref, gpu = _layers("llava7b", 2, 260, 4, seed=53)
    for side in (ref, gpu):
        side.prefill(0, inp.X_prefill[0][:260])
        side.prefill(1, inp.X_prefill[1][:200])
    blocks = [(1, 0, 200), (0, 100, 160), (0, 37, 20), (1, 190, 10), (0, 0, 1)]
    O = _gpu_blocks(gpu, blocks)
    want = np.concatenate([_oracle_rows(ref, b, t0, t0 + T) for b, t0, T in blocks])
    assert_rows_close(O, want, "mixed blocks")


def test_latent_prefill_13b_heads():
    wl, inp, ref, gpu = _layers("llava13b", 1, 300, 8, seed=54)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    assert_rows_close(_gpu_blocks(gpu, [(0, 0, 300)]), _oracle_rows(ref, 0, 0, 300), "blocks 13B")


def test_latent_prefill_13b_batch_sampled():
    """The 13B-shaped batch at full size (8 prompts of 5 x 576 + 128 tokens,
    one call), sampled rows of two prompts checked against the oracle."""
    wl, inp, ref, gpu = _layers("llava13b", 8, 128, 8, seed=55, n_image=2880)
    n = wl.prefill
    for b in range(8):
        gpu.prefill(b, inp.X_prefill[b])
    for b in (0, 7):
        ref.prefill(b, inp.X_prefill[b])
    O = _gpu_blocks(gpu, [(b, 0, n) for b in range(8)])
    assert np.isfinite(O).all()
    s = wl.shape
    for b in (0, 7):
        _assert_cache_equal(ref, gpu, b, n)
        C = ref.cache.rows(b, n)
        K, V = C @ ref.U_k, C @ ref.U_v
        for t in (0, 127, 128, 1500, n - 1):
            want = attention.decode_attention(C[:t + 1], ref.U_q, ref.U_k, ref.U_v, s.H, s.dh,
                                              K=K[:t + 1], V=V[:t + 1])
            assert_rows_close(O[b * n + t:b * n + t + 1], want[None], f"seq {b} row {t}")


def test_latent_prefill_more_than_64_blocks():
    """70 blocks take two launches that reuse one workspace."""
    wl, inp, ref, gpu = _layers("llava7b", 2, 140, 8, seed=56)
    for side in (ref, gpu):
        side.prefill(0, inp.X_prefill[0])
        side.prefill(1, inp.X_prefill[1])
    blocks = [(i % 2, 2 * i, 1 + i % 3) for i in range(70)]
    O = _gpu_blocks(gpu, blocks)
    want = np.concatenate([_oracle_rows(ref, b, t0, t0 + T) for b, t0, T in blocks])
    assert_rows_close(O, want, "70 blocks")


def test_latent_prefill_argument_errors():
    wl, inp, ref, gpu = _layers("llava7b", 1, 16, 8, seed=57)
    lib, s = q(), wl.shape
    Ut = lib.qsvd_prefill_weights(gpu.U_q, gpu.U_k, gpu.U_v)
    O = torch.empty((16, s.d), dtype=torch.float32, device=dev())
    for bad in ([(1, 0, 4)], [(0, -1, 4)], [(0, 0, 0)], [(0, 10, 7)], [(0, 0, 4), (-1, 0, 4)]):
        with pytest.raises(lib.QsvdError) as e:
            lib.qsvd_latent_prefill(gpu.cache, bad, Ut, s.H, s.dh, O)
        assert e.value.status == lib.QSVD_EINVAL
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_prefill(gpu.cache, [(0, 0, 4)], Ut, s.H, s.dh, O,
                                workspace=torch.zeros(256, dtype=torch.uint8, device=dev()))
    assert e.value.status == lib.QSVD_ENOSPC
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_prefill(gpu.cache, [(0, 0, 4)], Ut, 2 * s.H, 64, O)
    assert e.value.status == lib.QSVD_EUNSUPPORTED
    for bad_scale in (0.0, -0.1, float("inf")):
        with pytest.raises(lib.QsvdError) as e:
            lib.qsvd_latent_prefill(gpu.cache, [(0, 0, 4)], Ut, s.H, s.dh, O, softmax_scale=bad_scale)
        assert e.value.status == lib.QSVD_EINVAL
    lib.qsvd_latent_prefill(gpu.cache, [], Ut, s.H, s.dh, O)
    lib.qsvd_check()


def test_prefill_rows_tiny_dh64():
    """The tiny layer (d = 256, H = 4, dh = 64, r = 96, weights from the joint
    SVD): the row path, which also serves dh = 64."""
    wl = synthetic.WORKLOADS["tiny"]
    inp = synthetic.gen_layer(wl, seed=48)
    w = pipeline.prepare_weights(inp)
    ref = pipeline.OracleLayer(wl.shape, w, 1, wl.tmax, 8, track=[])
    gpu = GpuLayer(wl.shape, w, 1, wl.tmax, 8)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    n = wl.prefill
    O = _gpu_prefill(gpu, np.zeros(n), np.arange(1, n + 1))
    q().qsvd_check()
    assert_rows_close(O.cpu().numpy(), _oracle_rows(ref, 0, 0, n), "tiny rows")


def test_latent_prefill_13b_int4_continued():
    """Block path, int4 cache, H = 40: a prompt continued at t0 = 77 (not a
    multiple of 128) and a second sequence's whole prompt."""
    wl, inp, ref, gpu = _layers("llava13b", 2, 260, 4, seed=58)
    for side in (ref, gpu):
        side.prefill(0, inp.X_prefill[0][:260])
        side.prefill(1, inp.X_prefill[1][:150])
    blocks = [(0, 77, 183), (1, 0, 150)]
    O = _gpu_blocks(gpu, blocks)
    want = np.concatenate([_oracle_rows(ref, b, t0, t0 + T) for b, t0, T in blocks])
    assert_rows_close(O, want, "13B int4 blocks")


def test_latent_prefill_fp16_range_guard():
    """Values beyond fp16's range saturate at +-65504 and flag QSVD_ERANGE
    instead of turning into inf silently: an up-projection entry of 1e5 in
    qsvd_prefill_weights (Ut holds 65504), and Q / K / V beyond 65504 in the
    block GEMM (a latent of magnitude ~1e3 against entries ~400)."""
    lib = q()
    H, dh, r, L = 32, 128, 1536, 200
    d = H * dh
    rng = np.random.default_rng(61)
    U = [synthetic.bf16_bits(rng.standard_normal((r, d)) * 400.0) for _ in range(3)]
    Ub = [torch.from_numpy(u.view(np.int16)).view(torch.bfloat16).to(dev()) for u in U]
    big = U[0].copy()
    big[3, 5] = synthetic.bf16_bits(np.array([1e5]))[0]
    Ubig = torch.from_numpy(big.view(np.int16)).view(torch.bfloat16).to(dev())
    Ut = lib.qsvd_prefill_weights(Ubig, Ub[1], Ub[2])
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_check()
    assert e.value.status == lib.QSVD_ERANGE
    assert float(Ut.float().abs().max()) == 65504.0 and torch.isfinite(Ut.float()).all()
    Ut = lib.qsvd_prefill_weights(*Ub)
    lib.qsvd_check()                                        # in range: no flag
    cache = lib.LatentCache.empty(1, L, r, 8, dev())
    cache.codes.copy_(torch.randint(-127, 128, cache.codes.shape, device=dev(), dtype=torch.int8))
    cache.scales.fill_(8.0)                                 # latent entries up to ~1000
    O = torch.empty((L, d), dtype=torch.float32, device=dev())
    lib.qsvd_latent_prefill(cache, [(0, 0, L)], Ut, H, dh, O)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_check()
    assert e.value.status == lib.QSVD_ERANGE           # the saturated operands make this output invalid
