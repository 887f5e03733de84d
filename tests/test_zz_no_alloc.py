"""The allocation-free decode-size projection (qsvd_latent_project_static).

It serves callers that cannot allocate device memory while they project a
token (a serving process whose device memory was reserved in full at start-up,
or code running under stream capture) and so cannot hand the library a
workspace: its scratch is a fixed array inside the library.  This file runs
last (pytest collects it after the others) and checks, through the C ABI, that
two calls in a row give exactly the codes and scales the workspace-based
qsvd_latent_project gives on the same inputs."""
import numpy as np
import pytest
import torch

import synthetic
from oracle import pipeline

from gpu_util import bf16, dev, q

pytestmark = pytest.mark.gpu


def _outputs(T, r, bits):
    if bits == 8:
        return (torch.empty((T, r), dtype=torch.int8, device=dev()),
                torch.empty((T,), dtype=torch.float32, device=dev()))
    return (torch.empty((T, r // 2), dtype=torch.uint8, device=dev()),
            torch.empty((T, r // 128), dtype=torch.float16, device=dev()))


def test_static_projection_matches_workspace_projection_twice():
    lib = q()
    wl = synthetic.WORKLOADS["llava7b"]
    inp = synthetic.gen_layer(wl, seed=11, prefill_rows=32, decode_steps=0)
    w = pipeline.prepare_weights(inp)
    W = lib.qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    r = wl.shape.r
    calls = [(inp.X_prefill[0][:5], 8), (inp.X_prefill[0][5:21], 4)]     # two calls in a row
    for X_bits, bits in calls:
        X = bf16(X_bits)
        T = X.shape[0]
        c_static, s_static = _outputs(T, r, bits)
        c_ref, s_ref = _outputs(T, r, bits)
        lib.qsvd_latent_project_static(W, X, 1.0, bits, 1.0, lat_codes=c_static, lat_scales=s_static)
        lib.qsvd_latent_project(W, X, 1.0, bits, 1.0, lat_codes=c_ref, lat_scales=s_ref)
        lib.qsvd_check()
        np.testing.assert_array_equal(c_static.cpu().numpy(), c_ref.cpu().numpy())
        np.testing.assert_array_equal(s_static.cpu().numpy(), s_ref.cpu().numpy())


def test_static_projection_rejects_oversize():
    lib = q()
    wl = synthetic.WORKLOADS["llava7b"]
    inp = synthetic.gen_layer(wl, seed=12, prefill_rows=17, decode_steps=0)
    w = pipeline.prepare_weights(inp)
    W = lib.qsvd_quantize_weight(torch.from_numpy(w["W_d"].astype(np.float32)).to(dev()))
    c, s = _outputs(17, wl.shape.r, 8)
    with pytest.raises(lib.QsvdError) as e:
        lib.qsvd_latent_project_static(W, bf16(inp.X_prefill[0]), lat_codes=c, lat_scales=s)
    assert e.value.status == lib.QSVD_ENOSPC
    assert "16-token maximum" in str(e.value)
