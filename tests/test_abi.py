"""The C ABI library builds, loads without a GPU, and exports every symbol
that include/gmc.h declares; the binding declares the same names."""
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "gmc.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(gmc_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_1905_12948_gb300 import build, gmc
    build.build()
    return gmc.load()


def test_header_declares_the_api():
    names = _declared()
    for must in ("gmc_create", "gmc_step", "gmc_get_params", "gmc_destroy", "gmc_check"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_binding_covers_the_header(lib):
    from paper_1905_12948_gb300 import gmc
    assert sorted(gmc.exported_symbols()) == _declared()


def test_strerror_without_gpu(lib):
    assert lib.gmc_strerror(0) == b"success"
    assert lib.gmc_strerror(1) == b"invalid argument"
    assert lib.gmc_kernel_name(0) == b"accumulate"


def test_invalid_arguments_rejected_without_gpu(lib):
    import ctypes
    h = ctypes.c_void_p()
    # d = 0 (empty), K = 0, beta = 1, eta = 0, ratio = 0 / > 1, bad compressor, RBGS block 0
    bad = [(0, 4, 0.9, 0.1, 0, 0.01, 1), (10, 0, 0.9, 0.1, 0, 0.01, 1),
           (10, 2, 1.0, 0.1, 0, 0.01, 1), (10, 2, 0.9, 0.0, 0, 0.01, 1),
           (10, 2, 0.9, 0.1, 0, 0.0, 1), (10, 2, 0.9, 0.1, 0, 1.5, 1),
           (10, 2, 0.9, 0.1, 7, 0.01, 1), (10, 2, 0.9, 0.1, 1, 0.01, 0),
           (1 << 31, 2, 0.9, 0.1, 0, 0.01, 1), (10, 2, float("nan"), 0.1, 0, 0.01, 1)]
    for args in bad:
        assert lib.gmc_create(ctypes.byref(h), *args) == 1, args
        assert h.value is None
    assert lib.gmc_step(None, None, None) == 1
    assert lib.gmc_set_params(None, None, None) == 1


def test_failure_hooks_without_gpu(lib):
    """The allocation hook round-trips without a device (no handle holds
    memory), the timeout has its own status and message, and the copy hook
    refuses a NULL handle."""
    assert lib.gmc_test_fail_alloc(3) == 0
    assert lib.gmc_test_fail_alloc(-1) == 0
    assert lib.gmc_strerror(8).startswith(b"a bounded wait")
    assert lib.gmc_strerror(9) == b"unknown status"
    assert lib.gmc_test_withhold_copy(None, 0, 0, 1000) == 1
    assert lib.gmc_check(None) == 1
