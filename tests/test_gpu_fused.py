"""GPU parity of the one-call decode step (qsvd_decode_step) against the CPU
oracle: cache codes bit-exact, outputs within 2e-3 * ||o_ref||_2.  Up to four
sequences the query kernel requantizes and stores the new latents itself;
from five on a separate requantization launch does (both are covered)."""
import numpy as np
import pytest

import synthetic
from oracle import pipeline

from gpu_util import GpuLayer, assert_rows_close, bf16, dev, i32, q

pytestmark = pytest.mark.gpu


def _run(wl, inp, w, steps, check, lens=None):
    s = wl.shape
    ref = pipeline.OracleLayer(s, w, wl.B, wl.tmax, wl.lat_bits)
    gpu = GpuLayer(s, w, wl.B, wl.tmax, wl.lat_bits)
    for b in range(wl.B):
        n = wl.prefill if lens is None else lens[b]
        ref.prefill(b, inp.X_prefill[b][:n])
        gpu.prefill(b, inp.X_prefill[b][:n])
    for step in range(steps):
        _, outs = ref.decode_step(inp.X_decode[step], attend=None if step in check else [])
        O = gpu.decode_step_fused(inp.X_decode[step])
        if step in check:
            q().qsvd_check()
            assert_rows_close(O.cpu().numpy(), np.stack([outs[b] for b in range(wl.B)]), f"step {step}")
    q().qsvd_check()
    for b in range(wl.B):
        L = int(ref.len[b])
        np.testing.assert_array_equal(gpu.cache.codes[b, :L].cpu().numpy().view(np.uint8),
                                      ref.cache.packed_codes()[b, :L].view(np.uint8))
        np.testing.assert_array_equal(gpu.cache.scales[b, :L].cpu().numpy().astype(np.float64), ref.cache.scale[b, :L])


def test_fused_tiny_all_steps():
    wl = synthetic.WORKLOADS["tiny"]
    inp = synthetic.gen_layer(wl, seed=0)
    _run(wl, inp, pipeline.prepare_weights(inp), wl.decode_steps, set(range(wl.decode_steps)))


def test_fused_7b_sampled():
    wl = synthetic.WORKLOADS["llava7b"]
    inp = synthetic.gen_layer(wl, seed=0)
    _run(wl, inp, pipeline.prepare_weights(inp), wl.decode_steps, {0, 64, wl.decode_steps - 1})


@pytest.mark.parametrize("bits", [8, 4])
def test_fused_batch_ragged(bits):
    base = synthetic.WORKLOADS["llava7b"]
    wl = synthetic.Workload("ragged", base.shape, B=3, n_image=0, n_text=300, decode_steps=2, lat_bits=bits)
    inp = synthetic.gen_layer(wl, seed=7)
    _run(wl, inp, pipeline.prepare_weights(inp), 2, {0, 1}, lens=[1, 63, 300])


@pytest.mark.parametrize("B,bits", [(2, 8), (4, 8), (4, 4), (6, 8), (6, 4), (17, 8)])
def test_fused_batch_sizes(B, bits):
    """Both ways of storing the new latents (in the query kernel up to four
    sequences, in their own launch from five) and the batched query forms."""
    base = synthetic.WORKLOADS["llava7b"]
    wl = synthetic.Workload("batch", base.shape, B=B, n_image=0, n_text=160, decode_steps=3, lat_bits=bits)
    inp = synthetic.gen_layer(wl, seed=11 + B)
    lens = [1 + (37 * b) % 160 for b in range(B)]
    _run(wl, inp, pipeline.prepare_weights(inp), 3, {0, 2}, lens=lens)


def test_fused_matches_two_calls_bit_for_bit():
    """The one-call step and qsvd_latent_project + qsvd_latent_decode_attn give
    the same cache bytes and the same outputs."""
    base = synthetic.WORKLOADS["llava7b"]
    for B in (1, 3):
        wl = synthetic.Workload("pair", base.shape, B=B, n_image=0, n_text=96, decode_steps=2, lat_bits=8)
        inp = synthetic.gen_layer(wl, seed=21 + B)
        w = pipeline.prepare_weights(inp)
        one, two = GpuLayer(wl.shape, w, B, wl.tmax, 8), GpuLayer(wl.shape, w, B, wl.tmax, 8)
        for b in range(B):
            one.prefill(b, inp.X_prefill[b])
            two.prefill(b, inp.X_prefill[b])
        for step in range(2):
            o1 = one.decode_step_fused(inp.X_decode[step]).cpu().numpy()
            o2 = two.decode_step(inp.X_decode[step]).cpu().numpy()
            np.testing.assert_array_equal(o1, o2)
        q().qsvd_check()
        np.testing.assert_array_equal(one.cache.codes.cpu().numpy(), two.cache.codes.cpu().numpy())
        np.testing.assert_array_equal(one.cache.scales.cpu().numpy(), two.cache.scales.cpu().numpy())


def test_fused_13b_shape():
    base = synthetic.WORKLOADS["llava13b"]
    wl = synthetic.Workload("13b_small", base.shape, B=2, n_image=200, n_text=40, decode_steps=2, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=4)
    _run(wl, inp, pipeline.prepare_weights(inp), 2, {0, 1})


def test_fused_rejects_large_batch():
    lib = q()
    base = synthetic.WORKLOADS["llava7b"]
    wl = synthetic.Workload("big", base.shape, B=65, n_image=0, n_text=4, decode_steps=1, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=1)
    gpu = GpuLayer(wl.shape, pipeline.prepare_weights(inp), wl.B, wl.tmax, 8)
    with pytest.raises(lib.QsvdError) as e:
        gpu.decode_step_fused(inp.X_decode[0])
    assert e.value.status == lib.QSVD_EUNSUPPORTED


@pytest.mark.parametrize("B", [2, 6])
def test_fused_invalid_length_flagged(B):
    """A sequence whose length is outside [1, Tmax] gets no cache row and flags
    QSVD_ERANGE; the other sequences of the step are unaffected (both ways of
    storing the new latents: in the query kernel at B = 2, in their own launch
    at B = 6)."""
    import torch
    lib = q()
    base = synthetic.WORKLOADS["llava7b"]
    wl = synthetic.Workload("bad", base.shape, B=B, n_image=0, n_text=40, decode_steps=1, lat_bits=8)
    s = wl.shape
    inp = synthetic.gen_layer(wl, seed=31 + B)
    w = pipeline.prepare_weights(inp)
    ref = pipeline.OracleLayer(s, w, B, wl.tmax, 8)
    gpu = GpuLayer(s, w, B, wl.tmax, 8)
    for b in range(B):
        ref.prefill(b, inp.X_prefill[b])
        gpu.prefill(b, inp.X_prefill[b])
    _, outs = ref.decode_step(inp.X_decode[0])
    codes_before = gpu.cache.codes.clone()
    lens = np.full(B, 41, dtype=np.int32)
    lens[1] = 0
    O = torch.empty((B, s.d), dtype=torch.float32, device=dev())
    lib.qsvd_decode_step(gpu.W, bf16(inp.X_decode[0]), gpu.cache, i32(lens), 41, gpu.U_q, gpu.U_k, gpu.U_v, s.H,
                         s.dh, O)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_check()
    assert e.value.status == lib.QSVD_ERANGE
    lib.qsvd_check()                        # the flag was cleared
    np.testing.assert_array_equal(gpu.cache.codes[1].cpu().numpy(), codes_before[1].cpu().numpy())
    valid = [b for b in range(B) if b != 1]
    got = O.cpu().numpy()
    assert_rows_close(got[valid], np.stack([outs[b] for b in valid]), "valid sequences")
    for b in valid:
        np.testing.assert_array_equal(gpu.cache.codes[b, :41].cpu().numpy().view(np.uint8),
                                      ref.cache.packed_codes()[b, :41].view(np.uint8))
