"""The C-ABI library loads and exports every entry point include/sn.h declares.

CPU only: no call here touches a GPU (only status strings, the launch counter
and argument checks that return before any CUDA call).
"""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sn.h")


def declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sn_[a-z_0-9]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    from paper_2506_01260_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_boundary():
    names = declared()
    for required in ("sn_compress_fwd", "sn_decompress_fwd", "sn_compress_bwd",
                     "sn_decompress_bwd", "sn_project_weight"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_every_declared_symbol():
    from paper_2506_01260_gb300 import sn
    assert sorted(sn.EXPORTS) == declared()
    for name in declared():
        assert callable(getattr(sn, name)), name


def test_status_strings(lib):
    f = lib.sn_status_string
    f.restype = ctypes.c_char_p
    f.argtypes = [ctypes.c_int]
    names = [f(i).decode() for i in range(8)]
    assert names == ["SN_OK", "SN_ERR_INVALID_ARG", "SN_ERR_ALIGNMENT", "SN_ERR_UNSUPPORTED",
                     "SN_ERR_BAD_ID", "SN_ERR_TIMEOUT", "SN_ERR_CUDA", "SN_ERR_NUMERIC"]
    assert f(99).decode() == "SN_ERR_UNKNOWN"


def test_host_side_argument_errors(lib):
    """Argument errors return synchronously, before any CUDA call."""
    P = ctypes.c_void_p
    lib.sn_basis_create.argtypes = [P, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(P), P]
    h = P()
    assert lib.sn_basis_create(None, 256, 8, ctypes.byref(h), None) == 1
    fake = P(0x1000)
    assert lib.sn_basis_create(fake, 8, 8, ctypes.byref(h), None) == 1      # d < 16
    assert lib.sn_basis_create(fake, 260, 8, ctypes.byref(h), None) == 1    # d % 8
    assert lib.sn_basis_create(fake, 256, 0, ctypes.byref(h), None) == 1    # k = 0
    assert lib.sn_basis_create(fake, 256, 129, ctypes.byref(h), None) == 1  # k > 128
    assert lib.sn_basis_create(fake, 16, 17, ctypes.byref(h), None) == 1    # k > d
    assert lib.sn_basis_create(P(0x1004), 256, 8, ctypes.byref(h), None) == 2  # misaligned
    lib.sn_compress_bwd.argtypes = [P, ctypes.c_int, P, ctypes.c_int64, P, P]
    assert lib.sn_compress_bwd(None, 0, fake, 16, fake, None) == 1
    lib.sn_wire_bytes.argtypes = [P, ctypes.c_int, ctypes.c_int64, ctypes.POINTER(ctypes.c_size_t)]
    n = ctypes.c_size_t()
    assert lib.sn_wire_bytes(None, 0, 16, ctypes.byref(n)) == 1
    lib.sn_basis_destroy.argtypes = [P]
    assert lib.sn_basis_destroy(None) == 0


def test_launch_counter_starts_at_zero(lib):
    lib.sn_launch_count.restype = ctypes.c_uint64
    assert lib.sn_launch_count() == 0
