"""The C-ABI library builds for sm_103a, loads, and exports every entry point that
include/shallowstream.h declares (no GPU needed: no compute calls)."""
import ctypes
import os
import re
import subprocess

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "shallowstream.h")


def declared_functions() -> list[str]:
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ss_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib_path():
    from paper_2609_02780_gb300 import build
    return build.build()


def test_header_declares_the_api():
    names = declared_functions()
    for required in ("ss_index_create", "ss_index_append", "ss_index_compress",
                     "ss_retrieve", "ss_retrieve_batched", "ss_index_destroy"):
        assert required in names


def test_library_exports_every_declared_symbol(lib_path):
    lib = ctypes.CDLL(lib_path)
    for name in declared_functions():
        assert hasattr(lib, name), name
    nm = subprocess.run(["nm", "-D", "--defined-only", lib_path], capture_output=True,
                        text=True, check=True).stdout
    exported = set(re.findall(r"\bT (ss_\w+)", nm))
    assert set(declared_functions()) <= exported
    # nothing else of ours leaks out of the library's C ABI
    assert {s for s in exported if s.startswith("ss_")} == set(declared_functions())


def test_binding_covers_the_header():
    from paper_2609_02780_gb300 import _abi
    assert set(_abi.SIGNATURES) == set(declared_functions())


def test_status_strings_and_version(lib_path):
    from paper_2609_02780_gb300 import _abi
    lib = _abi.load()
    assert lib.ss_status_string(0) == b"SS_OK"
    assert lib.ss_status_string(3) == b"SS_ERR_CAPACITY"
    assert b"sm_103a" in lib.ss_version()


def test_binding_fails_loudly_without_the_library():
    from paper_2609_02780_gb300 import _abi
    with pytest.raises(RuntimeError, match="not built"):
        _abi.load(os.path.join(ROOT, "does-not-exist.so"))


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-device error path")
def test_create_without_a_device_reports_cuda_error(lib_path):
    from paper_2609_02780_gb300 import _abi
    lib = _abi.load()
    cfg = _abi.IndexConfig(2, 28, 4, 128, 64, 1, 64)
    h = ctypes.c_void_p()
    st = lib.ss_index_create(ctypes.byref(cfg), None, None, ctypes.byref(h))
    assert st == 6 and not h.value
    assert lib.ss_last_error()


def test_invalid_config_rejected_before_any_device_work(lib_path):
    from paper_2609_02780_gb300 import _abi
    lib = _abi.load()
    h = ctypes.c_void_p()
    bad = _abi.IndexConfig(2, 28, 5, 128, 64, 1, 64)        # 28 % 5 != 0
    assert lib.ss_index_create(ctypes.byref(bad), None, None, ctypes.byref(h)) == 1
    bad = _abi.IndexConfig(2, 28, 4, 64, 64, 1, 64)         # head_dim 64
    assert lib.ss_index_create(ctypes.byref(bad), None, None, ctypes.byref(h)) == 2
    assert lib.ss_index_create(None, None, None, ctypes.byref(h)) == 1
