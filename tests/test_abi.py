"""The C-ABI library builds for sm_103a, loads without a GPU, and exports
every entry point include/qsvd.h declares (no compute calls) -- CPU only."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "qsvd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^[A-Za-z_][\w \*]*?\b(qsvd_\w+)\s*\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    path = __graft_entry__._load_builder().build()
    return ctypes.CDLL(path)


def test_header_declares_the_path():
    names = declared_functions()
    for n in ("qsvd_latent_project", "qsvd_cache_append", "qsvd_latent_decode_attn",
              "qsvd_quantize_weight", "qsvd_check", "qsvd_last_error"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, f"not exported: {missing}"


def test_host_only_queries(lib):
    lib.qsvd_project_workspace_bytes.restype = ctypes.c_size_t
    lib.qsvd_project_workspace_bytes.argtypes = [ctypes.c_int64, ctypes.c_int32, ctypes.c_int32]
    lib.qsvd_decode_workspace_bytes.restype = ctypes.c_size_t
    lib.qsvd_decode_workspace_bytes.argtypes = [ctypes.c_int32] * 5
    assert lib.qsvd_project_workspace_bytes(640, 4096, 1536) >= 640 * 1536 * 4
    assert lib.qsvd_project_workspace_bytes(-1, 4096, 1536) == 0
    assert lib.qsvd_decode_workspace_bytes(16, 4352, 1536, 32, 128) > 16 * 32 * 1536 * 4
    assert lib.qsvd_version() >= 100
    lib.qsvd_last_error.restype = ctypes.c_char_p
    assert lib.qsvd_last_error() == b""


class _Block(ctypes.Structure):
    _fields_ = [("seq", ctypes.c_int32), ("t0", ctypes.c_int32), ("T", ctypes.c_int32)]


def _a256(b):
    return (b + 255) // 256 * 256


def test_prefill_workspace_sizes(lib):
    """Host logic of qsvd_latent_prefill: rows padded to 128 per block, launches
    of at most 64 blocks sharing one workspace (the largest launch sizes it):
    latent operand fp16 [R, r] + row scale fp32 [R] + Q, K, V^T fp16 [R, d]."""
    f = lib.qsvd_latent_prefill_workspace_bytes
    f.restype = ctypes.c_size_t
    f.argtypes = [ctypes.POINTER(_Block), ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]

    def expect(blocks, r, d):
        R = 0
        for i0 in range(0, len(blocks), 64):
            R = max(R, sum(-(-(t0 + T) // 128) * 128 for _, t0, T in blocks[i0:i0 + 64]))
        return _a256(R * r * 2) + _a256(R * 4) + 3 * _a256(R * d * 2)

    cases = [[(0, 0, 640)], [(b, 0, 3008) for b in range(8)], [(0, 100, 150), (1, 0, 200), (0, 37, 20)],
             [(i % 2, 2 * i, 1 + i % 3) for i in range(70)], [(0, 0, 1)] * 64 + [(0, 0, 300)] * 3]
    for blocks in cases:
        arr = (_Block * len(blocks))(*[_Block(*b) for b in blocks])
        for r, H in ((1536, 32), (2048, 40)):
            assert f(arr, len(blocks), r, H, 128) == expect(blocks, r, H * 128), blocks[:3]
    assert f(None, 0, 1536, 32, 128) == 0


def test_prefill_row_group_sizes(lib):
    """qsvd_latent_prefill_attn's rows run in groups that share one decode
    workspace: by default the largest power of two up to 1024 whose workspace
    stays within 2 GiB, or the size qsvd_set_prefill_group_rows fixed."""
    pw = lib.qsvd_prefill_workspace_bytes
    pw.restype = ctypes.c_size_t
    pw.argtypes = [ctypes.c_int64, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
    dw = lib.qsvd_decode_workspace_bytes
    dw.restype = ctypes.c_size_t
    dw.argtypes = [ctypes.c_int32] * 5
    setg = lib.qsvd_set_prefill_group_rows
    setg.argtypes = [ctypes.c_int32]
    for n, L, r, H in ((640, 640, 1536, 32), (24064, 3008, 2048, 40), (5, 80, 96, 4)):
        rows = 1024
        while rows > 16 and dw(rows, L, r, H, 128) > (2 << 30):
            rows //= 2
        assert pw(n, L, r, H, 128) == dw(min(rows, n), L, r, H, 128)
    prev = setg(128)
    try:
        assert pw(640, 640, 1536, 32, 128) == dw(128, 640, 1536, 32, 128)
        assert pw(100, 640, 1536, 32, 128) == dw(100, 640, 1536, 32, 128)
    finally:
        setg(prev)
    assert setg(-1) < 0 and setg(65536) < 0


def test_decode_step_workspace(lib):
    """qsvd_decode_step's workspace: the projection's part (a 256-byte
    completion counter, then the X codes, their scales and the fp32 latent rows
    of the B new tokens, each rounded up to 256 bytes) followed by the decode
    attention's workspace for the same B and length."""
    sw = lib.qsvd_decode_step_workspace_bytes
    sw.restype = ctypes.c_size_t
    sw.argtypes = [ctypes.c_int32] * 6
    dw = lib.qsvd_decode_workspace_bytes
    dw.restype = ctypes.c_size_t
    dw.argtypes = [ctypes.c_int32] * 5
    up = lambda x: (x + 255) // 256 * 256  # noqa: E731
    for B, L, d, r, H in ((1, 768, 4096, 1536, 32), (3, 300, 4096, 1536, 32), (16, 4352, 4096, 1536, 32),
                          (8, 3520, 5120, 2048, 40), (64, 1024, 4096, 3072, 32)):
        proj = 256 + up(B * d) + up(4 * B) + up(4 * B * r)
        assert sw(B, L, d, r, H, 128) == proj + dw(B, L, r, H, 128)
    assert sw(0, 768, 4096, 1536, 32, 128) == 0 and sw(1, 768, 4096, 1536, 0, 128) == 0
