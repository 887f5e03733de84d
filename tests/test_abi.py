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
