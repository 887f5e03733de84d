"""Helpers for the GPU parity tests: marshal synthetic / oracle arrays to
device tensors and drive the C ABI through the Python binding."""
import math

import numpy as np
import torch

import synthetic
from oracle import pipeline

TOL = 2e-3      # max-abs error per output row, relative to the row's L2 norm


def q():
    import paper_2510_16292_gb300 as lib
    return lib


def dev():
    return torch.device("cuda:0")


def bf16(bits) -> torch.Tensor:
    a = np.ascontiguousarray(np.asarray(bits, dtype=np.uint16))
    return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(dev())


def i32(x) -> torch.Tensor:
    return torch.as_tensor(np.asarray(x, dtype=np.int32), device=dev())


def assert_rows_close(got, ref, what="output"):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape
    for i in range(ref.shape[0]):
        err = np.abs(got[i] - ref[i]).max()
        tol = TOL * np.linalg.norm(ref[i])
        assert err <= tol, f"{what} row {i}: max err {err:.3e} > {tol:.3e}"


def cache_codes_np(cache, b, L):
    """Stored codes of sequence b, positions < L, unpacked to int64."""
    from oracle import quant      # unpacking of the stored image for comparison
    c = cache.codes[b, :L].cpu().numpy()
    if cache.bits == 8:
        return c.astype(np.int64)
    return quant.unpack_int4(c)


def cache_scales_np(cache, b, L):
    return cache.scales[b, :L].cpu().numpy().astype(np.float64)


class GpuLayer:
    """Device-side counterpart of oracle.pipeline.OracleLayer."""

    def __init__(self, shape, weights, B, tmax, bits, act_clip=1.0, lat_clip=1.0):
        lib = q()
        self.lib, self.s, self.B, self.bits = lib, shape, B, bits
        self.act_clip, self.lat_clip = act_clip, lat_clip
        self.W = lib.qsvd_quantize_weight(
            torch.from_numpy(np.asarray(weights["W_d"], dtype=np.float32)).to(dev()), rot=weights.get("rot", 0))
        self.U_q, self.U_k, self.U_v = (bf16(weights[k]) for k in ("U_q", "U_k", "U_v"))
        self.cache = lib.LatentCache.empty(B, tmax, shape.r, bits, dev())
        self.len = np.zeros(B, dtype=np.int64)

    def prefill(self, b, X_bits):
        T = X_bits.shape[0]
        pos = self.len[b] + np.arange(T)
        self.lib.qsvd_latent_project(self.W, bf16(X_bits), self.act_clip, self.bits, self.lat_clip,
                                     dst=self.cache, dst_seq=i32(np.full(T, b)), dst_pos=i32(pos))
        self.len[b] += T

    def decode_step_fused(self, x_bits):
        """One decode step through the single-launch entry point."""
        B = self.B
        self.len += 1
        O = torch.empty((B, self.s.d), dtype=torch.float32, device=dev())
        self.lib.qsvd_decode_step(self.W, bf16(x_bits), self.cache, i32(self.len), int(self.len.max()), self.U_q,
                                  self.U_k, self.U_v, self.s.H, self.s.dh, O, self.act_clip, self.lat_clip)
        return O

    def decode_step(self, x_bits):
        B = self.B
        self.lib.qsvd_latent_project(self.W, bf16(x_bits), self.act_clip, self.bits, self.lat_clip,
                                     dst=self.cache, dst_seq=i32(np.arange(B)), dst_pos=i32(self.len))
        self.len += 1
        O = torch.empty((B, self.s.d), dtype=torch.float32, device=dev())
        self.lib.qsvd_latent_decode_attn(self.cache, i32(self.len), int(self.len.max()), self.U_q, self.U_k,
                                         self.U_v, self.s.H, self.s.dh, O)
        return O
