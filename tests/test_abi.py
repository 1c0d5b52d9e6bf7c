"""The C-ABI library builds, loads without a GPU, and exports every entry
point that include/pss.h declares (no compute calls are made here)."""
import ctypes
import os
import re

import pytest

from paper_2207_10731_gb300 import binding, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "pss.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pss_[a-z_0-9]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.load_library()


def test_header_declares_the_expected_entry_points():
    assert _declared() == sorted(binding.EXPORTS)


def test_every_declared_symbol_is_exported(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    for code in range(8):
        s = binding.status_string(code)
        assert isinstance(s, str) and s
    assert binding.status_string(0) == "ok"


def test_create_rejects_bad_arguments_before_touching_the_device(lib):
    cards = (ctypes.c_int64 * 2)(10, 20)
    h = ctypes.c_void_p()
    # dim 0, Z 0, G 0, M < L, dim > 512, cardinality 0, null out
    bad = [
        (cards, 2, 0, 1024, 4, 4),
        (cards, 2, 16, 1024, 0, 4),
        (cards, 2, 16, 1024, 4, 0),
        (cards, 2, 16, 3, 4, 4),
        (cards, 2, 1024, 1 << 20, 4, 4),
        ((ctypes.c_int64 * 2)(10, 0), 2, 16, 1024, 4, 4),
    ]
    for c, T, d, M, Z, G in bad:
        rc = lib.pss_create(c, T, d, M, Z, G, ctypes.c_uint64(0), 0, ctypes.c_float(1e-10), None,
                            ctypes.byref(h))
        assert rc == binding.PSS_ERR_INVALID_ARG
    rc = lib.pss_create(cards, 2, 16, 1024, 4, 4, ctypes.c_uint64(0), 0, ctypes.c_float(1e-10),
                        None, None)
    assert rc == binding.PSS_ERR_INVALID_ARG
    # keys beyond the hash field: max n_t * T * J > 2^61 - 1
    huge = (ctypes.c_int64 * 1)(1 << 60)
    rc = lib.pss_create(huge, 1, 128, 1 << 20, 32, 4, ctypes.c_uint64(0), 0, ctypes.c_float(1e-10),
                        None, ctypes.byref(h))
    assert rc == binding.PSS_ERR_INVALID_ARG


def test_null_handle_calls_are_rejected(lib):
    assert lib.pss_forward(None, None, 0, None, 0, None, None) == binding.PSS_ERR_INVALID_ARG
    assert lib.pss_backward_update(None, None, ctypes.c_float(0.1), None) == \
        binding.PSS_ERR_INVALID_ARG
    assert lib.pss_set_option(None, 1, 0) == binding.PSS_ERR_INVALID_ARG
    assert lib.pss_destroy(None) == binding.PSS_OK


def test_check_convert_rejects_bad_arguments_before_touching_the_device(lib):
    for direction, n in ((2, 4), (-1, 4), (0, -1)):
        rc = lib.pss_check_convert(direction, None, None, n, None)
        assert rc == binding.PSS_ERR_INVALID_ARG
    assert lib.pss_check_convert(1, None, None, 0, None) == binding.PSS_OK
