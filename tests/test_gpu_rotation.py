"""The online rotation H1 of Eq. 11-12 on the GPU against oracle.rotate:
weight codes and scales of H1 W_d, and the rotated projection's X codes,
scales, int32 accumulators and latent codes, all bit-exact; decode through a
rotated layer within the decode tolerance."""
import numpy as np
import pytest
import torch

import synthetic
from gpu_util import GpuLayer, assert_rows_close, dev, q
from oracle import latent, pipeline, rotate
from test_gpu_parity import _assert_project_exact, _project_outputs

pytestmark = pytest.mark.gpu


def _weights(name, rot, seed=0, n_text=300):
    base = synthetic.WORKLOADS[name]
    wl = synthetic.Workload("rot", base.shape, B=1, n_image=0, n_text=n_text, decode_steps=2, lat_bits=8)
    inp = synthetic.gen_layer(wl, seed=seed)
    return wl, inp, pipeline.prepare_weights(inp, rot=rot)


@pytest.mark.parametrize("name,rot", [("llava7b", 4096), ("llava7b", 256), ("llava13b", 1024)])
def test_rotated_weight_bit_exact(name, rot):
    wl, inp, w = _weights(name, rot)
    W = q().qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()), rot=rot)
    q().qsvd_check()
    assert W.rot == rot
    np.testing.assert_array_equal(W.codes.cpu().numpy().astype(np.int64), w["Wq"].T)
    np.testing.assert_array_equal(W.scale.cpu().numpy().astype(np.float64), w["s_w"])
    np.testing.assert_array_equal(W.codes_bf16.float().cpu().numpy(), w["Wq"].T.astype(np.float32))


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("T", [1, 3, 16, 37, 65, 300])
def test_rotated_projection_bit_exact(bits, T):
    """Every T goes through the rotating quantizer: T <= 64 with the
    tensor-core dot products in 16-token blocks, larger T with the GEMM."""
    wl, inp, w = _weights("llava7b", 4096, seed=1)
    W = q().qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()), rot=4096)
    X = inp.X_prefill[0][:T]
    got = _project_outputs(W, X, wl.shape.r, bits)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), w["Wq"], w["s_w"], lat_bits=bits, rot=4096)
    _assert_project_exact(got, ref, bits)


def test_rotated_projection_13b_blocks():
    """d = 5120: blocks of 1024 channels."""
    wl, inp, w = _weights("llava13b", 1024, seed=2, n_text=70)
    W = q().qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()), rot=1024)
    X = inp.X_prefill[0][:70]
    got = _project_outputs(W, X, wl.shape.r, 8)
    ref = latent.latent_project(synthetic.bf16_from_bits(X), w["Wq"], w["s_w"], lat_bits=8, rot=1024)
    _assert_project_exact(got, ref, 8)


def test_rotated_decode_steps():
    """A prompt and two decode steps through the rotated projection."""
    wl, inp, w = _weights("llava7b", 4096, seed=3, n_text=200)
    ref = pipeline.OracleLayer(wl.shape, w, 1, wl.tmax, 8)
    gpu = GpuLayer(wl.shape, w, 1, wl.tmax, 8)
    ref.prefill(0, inp.X_prefill[0])
    gpu.prefill(0, inp.X_prefill[0])
    for step in range(2):
        _, outs = ref.decode_step(inp.X_decode[step])
        o = gpu.decode_step(inp.X_decode[step]).cpu().numpy()
        assert_rows_close(o, outs[0][None], f"step {step}")
    got = gpu.cache.codes[0, :int(ref.len[0])].cpu().numpy().view(np.uint8)
    np.testing.assert_array_equal(got, ref.cache.packed_codes()[0, :int(ref.len[0])].view(np.uint8))


def test_rotation_argument_errors():
    lib = q()
    W_d = torch.zeros((256, 64), dtype=torch.float32, device=dev())
    for bad in (3, 96, 512, 1):
        with pytest.raises(lib.QsvdError) as e:
            lib.qsvd_quantize_weight(W_d, rot=bad)
        assert e.value.status == lib.QSVD_EINVAL
    W = lib.qsvd_quantize_weight(W_d, rot=256)
    X = torch.zeros((2, 256), dtype=torch.bfloat16, device=dev())
    cache = lib.LatentCache.empty(2, 4, 64, 8, dev())
    U = torch.zeros((64, 256), dtype=torch.bfloat16, device=dev())
    O = torch.empty((2, 256), dtype=torch.float32, device=dev())
    seq_len = torch.ones((2,), dtype=torch.int32, device=dev())
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_decode_step(W, X, cache, seq_len, 1, U, U, U, 2, 128, O)
    assert e.value.status == lib.QSVD_EUNSUPPORTED
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_project_static(W, X, dst=cache, dst_seq=torch.zeros((2,), dtype=torch.int32, device=dev()),
                                       dst_pos=torch.zeros((2,), dtype=torch.int32, device=dev()))
    assert e.value.status == lib.QSVD_EUNSUPPORTED
