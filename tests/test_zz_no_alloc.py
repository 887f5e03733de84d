"""The allocation-free decode-size projection (qsvd_latent_project_static).

It serves callers that cannot allocate device memory while they project a
token (a serving process whose device memory was reserved in full at start-up,
or code running under stream capture) and so cannot hand the library a
workspace: its scratch is a fixed array inside the library.  This file runs
last (pytest collects it after the others) and checks, through the C ABI, that
two calls in a row give exactly the codes and scales the workspace-based
qsvd_latent_project gives on the same inputs, both token-major and stored into
a latent cache, for 1-3 tokens (one fused launch whose last CTA requantizes)
and 4-16 tokens (the per-row requantization)."""
import numpy as np
import pytest
import torch

import synthetic
from oracle import pipeline

from gpu_util import bf16, dev, i32, q

pytestmark = pytest.mark.gpu


def _outputs(T, r, bits):
    if bits == 8:
        return (torch.empty((T, r), dtype=torch.int8, device=dev()),
                torch.empty((T,), dtype=torch.float32, device=dev()))
    return (torch.empty((T, r // 2), dtype=torch.uint8, device=dev()),
            torch.empty((T, r // 128), dtype=torch.float16, device=dev()))


@pytest.fixture(scope="module")
def layer():
    lib = q()
    wl = synthetic.WORKLOADS["llava7b"]
    inp = synthetic.gen_layer(wl, seed=11, prefill_rows=40, decode_steps=0)
    w = pipeline.prepare_weights(inp)
    W = lib.qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    return wl, inp.X_prefill[0], W


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("T", [1, 3, 5, 16])
def test_static_projection_matches_workspace_projection_twice(layer, T, bits):
    lib = q()
    wl, X_all, W = layer
    r = wl.shape.r
    for call in range(2):                       # two calls in a row on different rows
        X = bf16(X_all[call * 20: call * 20 + T])
        c_static, s_static = _outputs(T, r, bits)
        c_ref, s_ref = _outputs(T, r, bits)
        lib.qsvd_latent_project_static(W, X, 1.0, bits, 1.0, lat_codes=c_static, lat_scales=s_static)
        lib.qsvd_latent_project(W, X, 1.0, bits, 1.0, lat_codes=c_ref, lat_scales=s_ref)
        lib.qsvd_check()
        np.testing.assert_array_equal(c_static.cpu().numpy(), c_ref.cpu().numpy())
        np.testing.assert_array_equal(s_static.cpu().numpy(), s_ref.cpu().numpy())


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("T", [1, 3, 16])
def test_static_projection_into_cache(layer, T, bits):
    """Rows stored through dst / dst_seq / dst_pos equal the cache rows the
    workspace-based projection stores at the same slots."""
    lib = q()
    wl, X_all, W = layer
    r = wl.shape.r
    got = lib.LatentCache.empty(3, 40, r, bits, dev())
    ref = lib.LatentCache.empty(3, 40, r, bits, dev())
    for call in range(2):
        X = bf16(X_all[call * 20: call * 20 + T])
        seq = i32((np.arange(T) + call) % 3)
        pos = i32(np.arange(T) + 17 * call)
        lib.qsvd_latent_project_static(W, X, 1.0, bits, 1.0, dst=got, dst_seq=seq, dst_pos=pos)
        lib.qsvd_latent_project(W, X, 1.0, bits, 1.0, dst=ref, dst_seq=seq, dst_pos=pos)
        lib.qsvd_check()
    np.testing.assert_array_equal(got.codes.cpu().numpy(), ref.codes.cpu().numpy())
    np.testing.assert_array_equal(got.scales.cpu().numpy(), ref.scales.cpu().numpy())


def test_static_projection_rejects_oversize(layer):
    lib = q()
    wl, X_all, W = layer
    c, s = _outputs(17, wl.shape.r, 8)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_project_static(W, bf16(X_all[:17]), lat_codes=c, lat_scales=s)
    assert e.value.status == lib.QSVD_ENOSPC
    assert "16-token maximum" in str(e.value)


def test_static_projection_rejects_misaligned_cache(layer):
    """A cache whose code rows start 4 bytes off a 16-byte boundary is refused
    before anything is enqueued (the rows are stored as 32-bit words)."""
    lib = q()
    wl, X_all, W = layer
    r = wl.shape.r
    flat = torch.zeros(2 * 8 * r + 16, dtype=torch.int8, device=dev())
    codes = flat[4:4 + 2 * 8 * r].view(2, 8, r)
    cache = lib.LatentCache(codes, torch.zeros((2, 8), dtype=torch.float32, device=dev()), 8, 2, 8, r)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_project_static(W, bf16(X_all[:1]), dst=cache, dst_seq=i32([0]), dst_pos=i32([0]))
    assert e.value.status == lib.QSVD_EINVAL
    lib.qsvd_check()
    assert not flat.any().item()
