"""Python binding of the QSVD latent-attention library (include/qsvd.h).

Argument marshalling only: every function below forwards device pointers of
torch tensors and the current CUDA stream to the C ABI of ``libqsvd.so`` and
raises ``QsvdError`` on a non-zero status.  All arithmetic runs in the CUDA
kernels; there is no host fallback.  Importing this package fails loudly if
the library has not been built (``python paper_2510_16292_gb300/build.py``).

Names follow the C ABI: ``qsvd_quantize_weight``, ``qsvd_latent_project``,
``qsvd_cache_append``, ``qsvd_latent_decode_attn``, ``qsvd_latent_prefill_attn``,
``qsvd_check``, plus the
workspace-size queries.  ``DownWeight`` and ``LatentCache`` hold the torch
tensors behind the two C structs.
"""
from __future__ import annotations

import ctypes
import dataclasses
import math
import os
from typing import Optional

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build", "libqsvd.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError(f"QSVD CUDA library not built ({_LIB_PATH} missing); "
                      "run `python paper_2510_16292_gb300/build.py`")
_lib = ctypes.CDLL(_LIB_PATH)

QSVD_OK, QSVD_EINVAL, QSVD_EUNSUPPORTED, QSVD_ECUDA = 0, -1, -2, -3
QSVD_ETIMEOUT, QSVD_ERANGE, QSVD_ENOSPC = -4, -5, -6
EXPORTS = ("qsvd_quantize_weight", "qsvd_quantize_weight_rotated", "qsvd_quantize_weight_ex", "qsvd_importance_scores",
           "qsvd_importance_workspace_bytes", "qsvd_rank_budget", "qsvd_rank_budget_workspace_bytes",
           "qsvd_beta_factors", "qsvd_beta_objective", "qsvd_beta_objective_workspace_bytes",
           "qsvd_latent_project", "qsvd_project_workspace_bytes",
           "qsvd_cache_append", "qsvd_latent_decode_attn", "qsvd_decode_workspace_bytes",
           "qsvd_quantize_up", "qsvd_latent_decode_attn_qu",
           "qsvd_latent_prefill_attn", "qsvd_prefill_workspace_bytes", "qsvd_prefill_weights",
           "qsvd_latent_prefill", "qsvd_latent_prefill_workspace_bytes",
           "qsvd_decode_step", "qsvd_decode_step_workspace_bytes", "qsvd_latent_project_static",
           "qsvd_set_decode_attn_path", "qsvd_set_project_epilogue", "qsvd_set_prefill_group_rows", "qsvd_check", "qsvd_last_error",
           "qsvd_selftest_wait_timeout", "qsvd_version")


class QsvdError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"qsvd status {status}: {msg}")
        self.status = status


class _DownWeight(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("codes_bf16", ctypes.c_void_p), ("scale", ctypes.c_void_p),
                ("d", ctypes.c_int32), ("r", ctypes.c_int32), ("rot", ctypes.c_int32),
                ("w_bits", ctypes.c_int32), ("x_bits", ctypes.c_int32), ("codes_e4m3", ctypes.c_void_p)]


class _Cache(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p), ("bits", ctypes.c_int32),
                ("B", ctypes.c_int32), ("Tmax", ctypes.c_int32), ("r", ctypes.c_int32)]


class _UpWeight(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("scale", ctypes.c_void_p), ("bits", ctypes.c_int32),
                ("r", ctypes.c_int32), ("d", ctypes.c_int32)]


class _PrefillBlock(ctypes.Structure):
    _fields_ = [("seq", ctypes.c_int32), ("t0", ctypes.c_int32), ("T", ctypes.c_int32)]


_vp, _i32, _i64, _f32, _sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
_lib.qsvd_quantize_weight.argtypes = [_vp, _i32, _i32, _f32, _vp, _vp, _vp, _vp]
_lib.qsvd_quantize_weight_rotated.argtypes = [_vp, _i32, _i32, _f32, _i32, _vp, _vp, _vp, _vp]
_lib.qsvd_quantize_weight_ex.argtypes = [_vp, _i32, _i32, _f32, _i32, _i32, _vp, _vp, _vp, _vp, _vp]
_lib.qsvd_importance_scores.argtypes = [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _vp, _vp, _sz, _vp]
_lib.qsvd_importance_workspace_bytes.argtypes = [_i32, _i32, _i32]
_lib.qsvd_rank_budget.argtypes = [_vp, _i32, _i32, _vp, _vp, _sz, _vp]
_lib.qsvd_beta_factors.argtypes = [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _f32, _vp, _vp, _vp, _vp]
_lib.qsvd_beta_objective.argtypes = [_vp, _i64, _i32, _vp, _vp, _i32, _i32, _vp, _vp, _i32, _vp, _vp, _sz, _vp]
_lib.qsvd_beta_objective_workspace_bytes.argtypes = [_i64, _i32]
_lib.qsvd_beta_objective_workspace_bytes.restype = _sz
_lib.qsvd_rank_budget_workspace_bytes.argtypes = []
_lib.qsvd_rank_budget_workspace_bytes.restype = _sz
_lib.qsvd_importance_workspace_bytes.restype = _sz
_lib.qsvd_latent_project.argtypes = [ctypes.POINTER(_DownWeight), _vp, _i64, _f32, _i32, _f32, _vp, _vp,
                                     ctypes.POINTER(_Cache), _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
_lib.qsvd_project_workspace_bytes.argtypes = [_i64, _i32, _i32]
_lib.qsvd_project_workspace_bytes.restype = _sz
_lib.qsvd_cache_append.argtypes = [ctypes.POINTER(_Cache), _vp, _vp, _i64, _vp, _vp, _vp]
_lib.qsvd_latent_decode_attn.argtypes = [ctypes.POINTER(_Cache), _vp, _i32, _vp, _vp, _vp, _i32, _i32, _f32,
                                         _vp, _vp, _sz, _vp]
_lib.qsvd_quantize_up.argtypes = [_vp, _i32, _i32, _i32, _f32, _vp, _vp, _vp]
_lib.qsvd_latent_decode_attn_qu.argtypes = [ctypes.POINTER(_Cache), _vp, _i32, ctypes.POINTER(_UpWeight),
                                            ctypes.POINTER(_UpWeight), ctypes.POINTER(_UpWeight), _i32, _i32, _f32,
                                            _vp, _vp, _sz, _vp]
_lib.qsvd_decode_workspace_bytes.argtypes = [_i32, _i32, _i32, _i32, _i32]
_lib.qsvd_decode_workspace_bytes.restype = _sz
_lib.qsvd_latent_prefill_attn.argtypes = [ctypes.POINTER(_Cache), _vp, _vp, _i64, _i32, _vp, _vp, _vp, _i32, _i32,
                                          _f32, _vp, _vp, _sz, _vp]
_lib.qsvd_prefill_workspace_bytes.argtypes = [_i64, _i32, _i32, _i32, _i32]
_lib.qsvd_prefill_workspace_bytes.restype = _sz
_lib.qsvd_prefill_weights.argtypes = [_vp, _vp, _vp, _i32, _i32, _vp, _vp]
_lib.qsvd_latent_prefill.argtypes = [ctypes.POINTER(_Cache), ctypes.POINTER(_PrefillBlock), _i32, _vp, _i32, _i32,
                                     _f32, _vp, _vp, _sz, _vp]
_lib.qsvd_latent_prefill_workspace_bytes.argtypes = [ctypes.POINTER(_PrefillBlock), _i32, _i32, _i32, _i32]
_lib.qsvd_latent_prefill_workspace_bytes.restype = _sz
_lib.qsvd_decode_step.argtypes = [ctypes.POINTER(_DownWeight), _vp, ctypes.POINTER(_Cache), _vp, _i32, _vp, _vp,
                                  _vp, _i32, _i32, _f32, _f32, _f32, _vp, _vp, _sz, _vp]
_lib.qsvd_decode_step_workspace_bytes.argtypes = [_i32, _i32, _i32, _i32, _i32, _i32]
_lib.qsvd_decode_step_workspace_bytes.restype = _sz
_lib.qsvd_latent_project_static.argtypes = [ctypes.POINTER(_DownWeight), _vp, _i64, _f32, _i32, _f32, _vp, _vp,
                                            ctypes.POINTER(_Cache), _vp, _vp, _vp]
_lib.qsvd_check.argtypes = [_vp]
_lib.qsvd_last_error.restype = ctypes.c_char_p


def library_path() -> str:
    return _LIB_PATH


def _ptr(t: Optional[torch.Tensor], dtype=None, name: str = "tensor"):
    """Device pointer of a contiguous CUDA tensor; `dtype` (one dtype or a
    tuple) is the element type the C ABI reads through that pointer."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name}: device tensor expected")
    if not t.is_contiguous():
        raise ValueError(f"{name}: contiguous tensor expected")
    if dtype is not None:
        ok = t.dtype in dtype if isinstance(dtype, tuple) else t.dtype == dtype
        if not ok:
            raise TypeError(f"{name}: dtype {t.dtype} where {dtype} is expected")
    return t.data_ptr()


_I32, _BF16, _F32 = torch.int32, torch.bfloat16, torch.float32
_CODES, _SCALES = (torch.int8, torch.uint8), (torch.float32, torch.float16)


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def _check(status: int):
    if status != QSVD_OK:
        raise QsvdError(status, _lib.qsvd_last_error().decode(errors="replace"))


@dataclasses.dataclass
class DownWeight:
    """Quantized W_d: codes int8 [r, d], codes_bf16 bf16 [r, d], scale fp32 [r];
    rot > 0: the codes quantize H1 W_d (block Hadamard of rot channels) and
    the projection rotates X by H1 on the fly.  w_bits / x_bits: the setting
    (8/8 W8A8, 8/4 W8A4, 4/4 W4A4); codes_e4m3 uint8 [r, d]: the fp8 image
    of 4-bit codes, the W4A4 tensor-core operand."""
    codes: torch.Tensor
    codes_bf16: torch.Tensor
    scale: torch.Tensor
    rot: int = 0
    w_bits: int = 8
    x_bits: int = 8
    codes_e4m3: Optional[torch.Tensor] = None

    @property
    def d(self):
        return self.codes.shape[1]

    @property
    def r(self):
        return self.codes.shape[0]

    def _c(self):
        return _DownWeight(_ptr(self.codes, torch.int8, "W.codes"), _ptr(self.codes_bf16, _BF16, "W.codes_bf16"),
                           _ptr(self.scale, _F32, "W.scale"), self.d, self.r, self.rot, self.w_bits, self.x_bits,
                           _ptr(self.codes_e4m3, torch.uint8, "W.codes_e4m3"))


@dataclasses.dataclass
class LatentCache:
    """Latent cache tensors: int8 codes [B, Tmax, r] + fp32 scales [B, Tmax],
    or packed uint8 codes [B, Tmax, r/2] + fp16 scales [B, Tmax, r/128]."""
    codes: torch.Tensor
    scales: torch.Tensor
    bits: int
    B: int
    Tmax: int
    r: int

    @staticmethod
    def empty(B: int, Tmax: int, r: int, bits: int, device="cuda") -> "LatentCache":
        if bits == 8:
            codes = torch.zeros((B, Tmax, r), dtype=torch.int8, device=device)
            scales = torch.zeros((B, Tmax), dtype=torch.float32, device=device)
        else:
            codes = torch.zeros((B, Tmax, r // 2), dtype=torch.uint8, device=device)
            scales = torch.zeros((B, Tmax, r // 128), dtype=torch.float16, device=device)
        return LatentCache(codes, scales, bits, B, Tmax, r)

    def _c(self):
        return _Cache(_ptr(self.codes, torch.int8 if self.bits == 8 else torch.uint8, "cache.codes"),
                      _ptr(self.scales, _F32 if self.bits == 8 else torch.float16, "cache.scales"),
                      self.bits, self.B, self.Tmax, self.r)

    def nbytes_per_token(self) -> int:
        return self.r if self.bits == 8 else self.r // 2 + 2 * (self.r // 128)


@dataclasses.dataclass
class UpWeight:
    """Eq. 11's Q(W^u) of one up-projection [r, d]: codes int8 [r, d] (bits 8)
    or packed int4 uint8 [r, d/2] (bits 4), scale fp32 [d] per output channel."""
    codes: torch.Tensor
    scale: torch.Tensor
    bits: int

    @property
    def r(self):
        return self.codes.shape[0]

    @property
    def d(self):
        return self.scale.shape[0]

    def _c(self):
        return _UpWeight(_ptr(self.codes, (torch.int8, torch.uint8), "U.codes"), _ptr(self.scale, _F32, "U.scale"),
                         self.bits, self.r, self.d)


def qsvd_quantize_up(U: torch.Tensor, bits: int = 8, clip: float = 1.0, stream=None) -> UpWeight:
    """U bf16 [r, d] -> UpWeight (per-output-channel RTN to int8 or int4)."""
    r, d = U.shape
    if bits == 8:
        codes = torch.empty((r, d), dtype=torch.int8, device=U.device)
    else:
        codes = torch.empty((r, d // 2), dtype=torch.uint8, device=U.device)
    scale = torch.empty((d,), dtype=torch.float32, device=U.device)
    _check(_lib.qsvd_quantize_up(_ptr(U, _BF16, "U"), r, d, bits, clip, _ptr(codes), _ptr(scale), _stream(stream)))
    return UpWeight(codes, scale, bits)


def qsvd_latent_decode_attn_qu(cache: "LatentCache", seq_len: torch.Tensor, max_seq_len: int, U_q: UpWeight,
                               U_k: UpWeight, U_v: UpWeight, H: int, dh: int, O: torch.Tensor,
                               softmax_scale: Optional[float] = None, workspace=None, stream=None) -> None:
    """Decode attention with quantized up-projections (Eq. 11)."""
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    if workspace is None:
        workspace = torch.zeros(qsvd_decode_workspace_bytes(cache.B, max_seq_len, cache.r, H, dh),
                                dtype=torch.uint8, device=O.device)
    cc, uq, uk, uv = cache._c(), U_q._c(), U_k._c(), U_v._c()
    _check(_lib.qsvd_latent_decode_attn_qu(ctypes.byref(cc), _ptr(seq_len, _I32, "seq_len"), max_seq_len,
                                           ctypes.byref(uq), ctypes.byref(uk), ctypes.byref(uv), H, dh, softmax_scale,
                                           _ptr(O, _F32, "O"), _ptr(workspace), workspace.numel(), _stream(stream)))


def qsvd_quantize_weight(W_d: torch.Tensor, clip: float = 1.0, stream=None, rot: int = 0, w_bits: int = 8,
                         x_bits: int = 8) -> DownWeight:
    """W_d fp32 [d, r] -> DownWeight (per-output-channel RTN, int8 or with
    w_bits = 4 int4 codes plus their e4m3 image); rot > 0: of H1 W_d, and the
    projection then rotates X.  x_bits: how the projection quantizes X."""
    d, r = W_d.shape
    dev = W_d.device
    codes = torch.empty((r, d), dtype=torch.int8, device=dev)
    codes_bf16 = torch.empty((r, d), dtype=torch.bfloat16, device=dev)
    scale = torch.empty((r,), dtype=torch.float32, device=dev)
    if w_bits != 8 or x_bits != 8:
        e4 = torch.empty((r, d), dtype=torch.uint8, device=dev) if w_bits == 4 else None
        _check(_lib.qsvd_quantize_weight_ex(_ptr(W_d, _F32, "W_d"), d, r, clip, w_bits, rot, _ptr(codes),
                                            _ptr(codes_bf16), _ptr(e4), _ptr(scale), _stream(stream)))
        return DownWeight(codes, codes_bf16, scale, rot, w_bits, x_bits, e4)
    if rot:
        _check(_lib.qsvd_quantize_weight_rotated(_ptr(W_d, _F32, "W_d"), d, r, clip, rot, _ptr(codes),
                                                 _ptr(codes_bf16), _ptr(scale), _stream(stream)))
    else:
        _check(_lib.qsvd_quantize_weight(_ptr(W_d, _F32, "W_d"), d, r, clip, _ptr(codes), _ptr(codes_bf16),
                                         _ptr(scale), _stream(stream)))
    return DownWeight(codes, codes_bf16, scale, rot)


def qsvd_importance_scores(U: torch.Tensor, sigma: torch.Tensor, Vt: torch.Tensor, G: torch.Tensor,
                           workspace=None, stream=None) -> torch.Tensor:
    """Eq. 10 scores of the singular values: U [m, k], sigma [k], Vt [k, n],
    G [N, m, n] (one gradient per calibration sample), all fp32 on the device."""
    m, k = U.shape
    N, _, n = G.shape
    scores = torch.empty((k,), dtype=torch.float32, device=U.device)
    if workspace is None:
        workspace = torch.empty(max(1, int(_lib.qsvd_importance_workspace_bytes(N, m, k))), dtype=torch.uint8,
                                device=U.device)
    _check(_lib.qsvd_importance_scores(_ptr(U, _F32, "U"), _ptr(sigma, _F32, "sigma"), _ptr(Vt, _F32, "Vt"),
                                       _ptr(G, _F32, "G"), N, m, n, k, _ptr(scores), _ptr(workspace),
                                       workspace.numel(), _stream(stream)))
    return scores


def qsvd_rank_budget(scores: torch.Tensor, k: int, workspace=None, stream=None) -> torch.Tensor:
    """Cross-layer rank budget: scores fp32 [n] (every layer's scores in layer
    order) -> keep uint8 [n], 1 for the k highest (ties: the lower position)."""
    n = scores.numel()
    keep = torch.empty((n,), dtype=torch.uint8, device=scores.device)
    if workspace is None:
        workspace = torch.empty(int(_lib.qsvd_rank_budget_workspace_bytes()), dtype=torch.uint8, device=scores.device)
    _check(_lib.qsvd_rank_budget(_ptr(scores, _F32, "scores"), n, k, _ptr(keep), _ptr(workspace), workspace.numel(),
                                 _stream(stream)))
    return keep


def qsvd_beta_factors(Wd_r: torch.Tensor, Wu_r: torch.Tensor, fd: torch.Tensor, fu: torch.Tensor, u_bits: int = 8,
                      u_clip: float = 1.0, stream=None):
    """Eq. 3 at one beta (Sec. 3.3): Wd_r fp64 [E, r], Wu_r fp64 [r, n_out] (the
    truncated joint SVD), fd = sigma^beta and fu = sigma^(1-beta) fp64 [r] ->
    (W_d fp32 [E, r], UpWeight Q(W^u) of [r, n_out])."""
    E, r = Wd_r.shape
    n_out = Wu_r.shape[1]
    dev = Wd_r.device
    W_d = torch.empty((E, r), dtype=torch.float32, device=dev)
    codes = torch.empty((r, n_out if u_bits == 8 else n_out // 2), dtype=torch.int8 if u_bits == 8 else torch.uint8,
                        device=dev)
    scale = torch.empty((n_out,), dtype=torch.float32, device=dev)
    f64 = torch.float64
    _check(_lib.qsvd_beta_factors(_ptr(Wd_r, f64, "Wd_r"), _ptr(Wu_r, f64, "Wu_r"), _ptr(fd, f64, "fd"),
                                  _ptr(fu, f64, "fu"), E, r, n_out, u_bits, u_clip, _ptr(W_d), _ptr(codes),
                                  _ptr(scale), _stream(stream)))
    return W_d, UpWeight(codes, scale, u_bits)


def qsvd_beta_objective(Y: torch.Tensor, lat_codes: torch.Tensor, lat_scales: torch.Tensor, lat_bits: int, r: int,
                        U: "UpWeight", workspace=None, stream=None) -> torch.Tensor:
    """Eq. 14's objective sum (Y - Q(C) Q(W^u))^2: Y fp32 [N, n_out] = X W_concat,
    Q(C) token-major as qsvd_latent_project writes it, U from qsvd_beta_factors.
    Returns a one-element fp64 device tensor."""
    N, n_out = Y.shape
    out = torch.empty((1,), dtype=torch.float64, device=Y.device)
    if workspace is None:
        workspace = torch.empty(max(1, int(_lib.qsvd_beta_objective_workspace_bytes(N, n_out))), dtype=torch.uint8,
                                device=Y.device)
    _check(_lib.qsvd_beta_objective(_ptr(Y, _F32, "Y"), N, n_out, _ptr(lat_codes, _CODES, "lat_codes"),
                                    _ptr(lat_scales, _SCALES, "lat_scales"), lat_bits, r,
                                    _ptr(U.codes, _CODES, "U.codes"), _ptr(U.scale, _F32, "U.scale"), U.bits,
                                    _ptr(out), _ptr(workspace), workspace.numel(), _stream(stream)))
    return out


def qsvd_project_workspace_bytes(T: int, d: int, r: int) -> int:
    return int(_lib.qsvd_project_workspace_bytes(T, d, r))


def qsvd_decode_workspace_bytes(B: int, max_seq_len: int, r: int, H: int, dh: int) -> int:
    return int(_lib.qsvd_decode_workspace_bytes(B, max_seq_len, r, H, dh))


def qsvd_latent_project(W: DownWeight, X: torch.Tensor, act_clip: float = 1.0, lat_bits: int = 8,
                        lat_clip: float = 1.0, lat_codes=None, lat_scales=None,
                        dst: Optional[LatentCache] = None, dst_seq=None, dst_pos=None,
                        xq_out=None, xs_out=None, acc_out=None, workspace=None, stream=None) -> None:
    T = X.shape[0]
    if workspace is None:
        workspace = torch.zeros(max(1, qsvd_project_workspace_bytes(T, W.d, W.r)), dtype=torch.uint8,
                                device=X.device)
    cw = W._c()
    cc = dst._c() if dst is not None else None
    _check(_lib.qsvd_latent_project(ctypes.byref(cw), _ptr(X, _BF16, "X"), T, act_clip, lat_bits, lat_clip,
                                    _ptr(lat_codes, _CODES, "lat_codes"), _ptr(lat_scales, _SCALES, "lat_scales"),
                                    ctypes.byref(cc) if cc is not None else None,
                                    _ptr(dst_seq, _I32, "dst_seq"), _ptr(dst_pos, _I32, "dst_pos"),
                                    _ptr(xq_out, torch.int8, "xq_out"), _ptr(xs_out, _F32, "xs_out"),
                                    _ptr(acc_out, _I32, "acc_out"),
                                    _ptr(workspace), workspace.numel(), _stream(stream)))


def qsvd_cache_append(cache: LatentCache, seq: torch.Tensor, pos: torch.Tensor, lat_codes: torch.Tensor,
                      lat_scales: torch.Tensor, stream=None) -> None:
    cc = cache._c()
    _check(_lib.qsvd_cache_append(ctypes.byref(cc), _ptr(seq, _I32, "seq"), _ptr(pos, _I32, "pos"), seq.numel(),
                                  _ptr(lat_codes, _CODES, "lat_codes"), _ptr(lat_scales, _SCALES, "lat_scales"),
                                  _stream(stream)))


def qsvd_latent_decode_attn(cache: LatentCache, seq_len: torch.Tensor, max_seq_len: int, U_q, U_k, U_v,
                            H: int, dh: int, O: torch.Tensor, softmax_scale: Optional[float] = None,
                            workspace=None, stream=None) -> None:
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    if workspace is None:
        workspace = torch.zeros(qsvd_decode_workspace_bytes(cache.B, max_seq_len, cache.r, H, dh),
                                dtype=torch.uint8, device=O.device)
    cc = cache._c()
    _check(_lib.qsvd_latent_decode_attn(ctypes.byref(cc), _ptr(seq_len, _I32, "seq_len"), max_seq_len,
                                        _ptr(U_q, _BF16, "U_q"), _ptr(U_k, _BF16, "U_k"), _ptr(U_v, _BF16, "U_v"),
                                        H, dh, softmax_scale, _ptr(O, _F32, "O"), _ptr(workspace),
                                        workspace.numel(), _stream(stream)))


def qsvd_prefill_workspace_bytes(n: int, max_len: int, r: int, H: int, dh: int) -> int:
    return int(_lib.qsvd_prefill_workspace_bytes(n, max_len, r, H, dh))


def qsvd_latent_prefill_attn(cache: LatentCache, q_seq: torch.Tensor, q_len: torch.Tensor, max_len: int,
                             U_q, U_k, U_v, H: int, dh: int, O: torch.Tensor,
                             softmax_scale: Optional[float] = None, workspace=None, stream=None) -> None:
    """Row i: the token at position q_len[i]-1 of sequence q_seq[i] attends to
    positions 0 .. q_len[i]-1 of that sequence (causal prefill)."""
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    n = q_seq.numel()
    if q_len.numel() != n:
        raise ValueError("q_seq and q_len differ in length")
    if workspace is None:
        workspace = torch.zeros(max(1, qsvd_prefill_workspace_bytes(n, max_len, cache.r, H, dh)),
                                dtype=torch.uint8, device=O.device)
    cc = cache._c()
    _check(_lib.qsvd_latent_prefill_attn(ctypes.byref(cc), _ptr(q_seq, _I32, "q_seq"), _ptr(q_len, _I32, "q_len"),
                                         n, max_len, _ptr(U_q, _BF16, "U_q"), _ptr(U_k, _BF16, "U_k"),
                                         _ptr(U_v, _BF16, "U_v"), H, dh, softmax_scale, _ptr(O, _F32, "O"),
                                         _ptr(workspace), workspace.numel(), _stream(stream)))


def _blocks(blocks):
    arr = (_PrefillBlock * max(1, len(blocks)))()
    for i, (b, t0, T) in enumerate(blocks):
        arr[i] = _PrefillBlock(int(b), int(t0), int(T))
    return arr


def qsvd_prefill_weights(U_q, U_k, U_v, stream=None) -> torch.Tensor:
    """fp16 [3d, r] = [U_q U_k U_v]^T, the weight operand of qsvd_latent_prefill."""
    r, d = U_q.shape
    Ut = torch.empty((3 * d, r), dtype=torch.float16, device=U_q.device)
    _check(_lib.qsvd_prefill_weights(_ptr(U_q, _BF16, "U_q"), _ptr(U_k, _BF16, "U_k"), _ptr(U_v, _BF16, "U_v"),
                                     r, d, _ptr(Ut), _stream(stream)))
    return Ut


def qsvd_latent_prefill_workspace_bytes(blocks, r: int, H: int, dh: int) -> int:
    return int(_lib.qsvd_latent_prefill_workspace_bytes(_blocks(blocks), len(blocks), r, H, dh))


def qsvd_latent_prefill(cache: LatentCache, blocks, Ut: torch.Tensor, H: int, dh: int, O: torch.Tensor,
                        softmax_scale: Optional[float] = None, workspace=None, stream=None) -> None:
    """blocks: (seq, t0, T) triples; block k's T queries (positions t0 ..
    t0+T-1 of sequence seq) attend causally to the cache; their outputs follow
    the earlier blocks' rows in O [sum T, H*dh]."""
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    if workspace is None:
        workspace = torch.zeros(max(1, qsvd_latent_prefill_workspace_bytes(blocks, cache.r, H, dh)),
                                dtype=torch.uint8, device=O.device)
    cc = cache._c()
    _check(_lib.qsvd_latent_prefill(ctypes.byref(cc), _blocks(blocks), len(blocks), _ptr(Ut, torch.float16, "Ut"), H,
                                    dh, softmax_scale, _ptr(O, _F32, "O"), _ptr(workspace), workspace.numel(),
                                    _stream(stream)))


def qsvd_decode_step_workspace_bytes(B: int, max_seq_len: int, d: int, r: int, H: int, dh: int) -> int:
    return int(_lib.qsvd_decode_step_workspace_bytes(B, max_seq_len, d, r, H, dh))


def qsvd_decode_step(W: DownWeight, X: torch.Tensor, cache: LatentCache, seq_len: torch.Tensor, max_seq_len: int,
                     U_q, U_k, U_v, H: int, dh: int, O: torch.Tensor, act_clip: float = 1.0,
                     lat_clip: float = 1.0, softmax_scale: Optional[float] = None, workspace=None,
                     stream=None) -> None:
    """Fused decode step: project the new token of every sequence, store its
    latent at position seq_len[b] - 1, attend over positions < seq_len[b]."""
    if softmax_scale is None:
        softmax_scale = 1.0 / math.sqrt(dh)
    if workspace is None:
        workspace = torch.zeros(qsvd_decode_step_workspace_bytes(cache.B, max_seq_len, W.d, W.r, H, dh),
                                dtype=torch.uint8, device=O.device)
    cw, cc = W._c(), cache._c()
    _check(_lib.qsvd_decode_step(ctypes.byref(cw), _ptr(X, _BF16, "X"), ctypes.byref(cc),
                                 _ptr(seq_len, _I32, "seq_len"), max_seq_len, _ptr(U_q, _BF16, "U_q"),
                                 _ptr(U_k, _BF16, "U_k"), _ptr(U_v, _BF16, "U_v"), H, dh, act_clip, lat_clip,
                                 softmax_scale, _ptr(O, _F32, "O"), _ptr(workspace), workspace.numel(), _stream(stream)))


def qsvd_latent_project_static(W: DownWeight, X: torch.Tensor, act_clip: float = 1.0, lat_bits: int = 8,
                               lat_clip: float = 1.0, lat_codes=None, lat_scales=None,
                               dst: Optional[LatentCache] = None, dst_seq=None, dst_pos=None, stream=None) -> None:
    """Decode-size projection (T <= 16) that uses the library's fixed device
    scratch instead of a workspace; nothing is allocated on the device."""
    cw = W._c()
    cc = dst._c() if dst is not None else None
    _check(_lib.qsvd_latent_project_static(ctypes.byref(cw), _ptr(X, _BF16, "X"), X.shape[0], act_clip, lat_bits,
                                           lat_clip, _ptr(lat_codes, _CODES, "lat_codes"),
                                           _ptr(lat_scales, _SCALES, "lat_scales"),
                                           ctypes.byref(cc) if cc is not None else None,
                                           _ptr(dst_seq, _I32, "dst_seq"), _ptr(dst_pos, _I32, "dst_pos"),
                                           _stream(stream)))


def qsvd_check(stream=None) -> int:
    """Synchronize the stream and return the device status (raises on error)."""
    st = _lib.qsvd_check(_stream(stream))
    _check(st)
    return st


_lib.qsvd_selftest_wait_timeout.argtypes = [_i32, _vp]


def qsvd_selftest_wait_timeout(timeout_ms: int = 5, stream=None) -> None:
    """Enqueue a bounded device wait that expires after `timeout_ms`; the next
    qsvd_check raises QsvdError with status QSVD_ETIMEOUT."""
    _check(_lib.qsvd_selftest_wait_timeout(timeout_ms, _stream(stream)))


def qsvd_version() -> int:
    return int(_lib.qsvd_version())


_lib.qsvd_set_decode_attn_path.argtypes = [_i32]
_lib.qsvd_set_prefill_group_rows.argtypes = [_i32]
_lib.qsvd_set_project_epilogue.argtypes = [_i32]


def qsvd_set_project_epilogue(mode: int) -> int:
    """0 automatic, 1 separate requantization kernel, 2 requantize in the
    tensor-core GEMM epilogue where possible.  Returns the previous setting."""
    st = _lib.qsvd_set_project_epilogue(mode)
    if st < 0:
        _check(st)
    return st


def qsvd_set_prefill_group_rows(rows: int) -> int:
    """Rows per group of qsvd_latent_prefill_attn; 0 automatic.  Returns the
    previous setting."""
    st = _lib.qsvd_set_prefill_group_rows(rows)
    if st < 0:
        _check(st)
    return st


def qsvd_set_decode_attn_path(path: int) -> int:
    """0 automatic, 1 CUDA-core kernels, 2 tcgen05 kernel where the shape
    allows it, 3 warp-level tensor-core kernel (r <= 3072).  Returns the
    previous setting."""
    st = _lib.qsvd_set_decode_attn_path(path)
    if st < 0:
        _check(st)
    return st
