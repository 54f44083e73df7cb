"""The C-ABI library builds for sm_103a, loads without a GPU, and exports
every function include/akashic_mem.h declares (no compute calls here)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "akashic_mem.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(akashic_mem_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib_path():
    from paper_2607_05708_gb300 import _build
    return _build.build()


def test_header_matches_binding():
    import paper_2607_05708_gb300 as pkg
    assert declared_functions() == sorted(pkg.EXPORTS)


def test_library_exports_every_declared_symbol(lib_path):
    out = subprocess.run(["nm", "-D", "--defined-only", lib_path], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (akashic_mem_\w+)", out))
    missing = set(declared_functions()) - exported
    assert not missing, f"not exported: {missing}"
    lib = ctypes.CDLL(lib_path)
    for name in declared_functions():
        assert getattr(lib, name) is not None


def test_binding_loads_and_reports_no_error(lib_path):
    import paper_2607_05708_gb300 as pkg
    lib = pkg.load_library()
    assert lib.akashic_mem_last_error() == b""


def test_invalid_config_is_rejected_without_gpu_work(lib_path):
    """create() validates its arguments before touching any device."""
    import paper_2607_05708_gb300 as pkg
    lib = pkg.load_library()
    h = ctypes.c_void_p()
    for cfg in (pkg._Config(100, 10, 1, 0, 0.0, 0.0),     # dim not a multiple of 64
                pkg._Config(64, 0, 1, 0, 0.0, 0.0),       # capacity 0
                pkg._Config(64, 10, 0, 0, 0.0, 0.0)):     # chunks_per_page 0
        assert lib.akashic_mem_create(ctypes.byref(cfg), ctypes.byref(h)) == 1
        assert b"create" in lib.akashic_mem_last_error()
    assert lib.akashic_mem_create(None, ctypes.byref(h)) == 1


def test_build_targets_sm103a_only(lib_path):
    """Every CUDA source is compiled for sm_103a and nothing else: one
    -gencode pair, arch=compute_103a,code=sm_103a, in the build's flags."""
    from paper_2607_05708_gb300 import _build
    assert _build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]
    flags = " ".join(_build.FLAGS)
    assert "gencode" not in flags and "arch=" not in flags
    assert os.path.exists(lib_path)


def test_sort_pairs_rejects_bad_arguments_without_gpu_work(lib_path):
    """sort_pairs validates n, bits and its buffers before any device call;
    n <= 1 is a no-op."""
    import paper_2607_05708_gb300 as pkg
    lib = pkg.load_library()
    for n, bits in ((-1, 8), (10, 8), (10, 33), (10, -1), (1 << 31, 8)):
        assert lib.akashic_mem_sort_pairs(None, None, n, bits, None) == 1
        assert b"sort_pairs" in lib.akashic_mem_last_error()
    assert lib.akashic_mem_sort_pairs(None, None, 0, 8, None) == 0
    assert lib.akashic_mem_sort_pairs(None, None, 1, 8, None) == 0
