"""The C-ABI library loads, exports every entry point include/as2d.h
declares, and rejects bad arguments on the host before touching the GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_entry_points():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            names += re.findall(r"^(?:as2d_status|void|const char\*)\s+(as2d_\w+)\(", src, re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__._lib_build_module().build()
    import paper_2609_37617_gb300 as p
    return p


def test_every_declared_symbol_exported(lib):
    names = declared_entry_points()
    assert len(names) >= 11
    raw = ctypes.CDLL(lib.LIB_PATH)
    for n in names:
        assert hasattr(raw, n), n
    assert set(lib.EXPORTED) <= set(names)


def test_host_side_argument_errors(lib):
    # NULL config: rejected before any CUDA call
    out = ctypes.c_void_p()
    st = lib._lib.as2d_model_load(None, None, ctypes.byref(out))
    assert st == lib.AS2D_ERR_INVALID_ARG and "config" in lib.as2d_last_error()
    bad = lib.as2d_config(2, 256, 4, 2, 96, 704, 4096, 1e6, 1e-6)   # head_dim 96
    st = lib._lib.as2d_model_load(ctypes.byref(bad), None, ctypes.byref(out))
    assert st == lib.AS2D_ERR_UNSUPPORTED
    bad = lib.as2d_config(2, 256, 4, 3, 64, 704, 4096, 1e6, 1e-6)    # 4 % 3 != 0
    st = lib._lib.as2d_model_load(ctypes.byref(bad), None, ctypes.byref(out))
    assert st == lib.AS2D_ERR_INVALID_ARG
    ok = lib.as2d_config(2, 256, 4, 2, 64, 704, 4096, 1e6, 1e-6)
    st = lib._lib.as2d_model_load(ctypes.byref(ok), None, ctypes.byref(out))
    assert st == lib.AS2D_ERR_INVALID_ARG
    st = lib._lib.as2d_kv_init_prefilled(None, 1, None, 16, None, None, None, ctypes.byref(out))
    assert st == lib.AS2D_ERR_INVALID_ARG
    vo = lib.make_verify_out(0, 0)
    assert lib.as2d_verify_block(0, 0, [0], vo) == lib.AS2D_ERR_INVALID_ARG
    assert lib.as2d_decode_step(0, vo) == lib.AS2D_ERR_INVALID_ARG
    assert lib.as2d_kv_rollback(0, [0], [0]) == lib.AS2D_ERR_INVALID_ARG
    assert lib.as2d_kv_check(0) == lib.AS2D_ERR_INVALID_ARG
    lib.as2d_kv_free(0)
    lib.as2d_model_free(0)


def test_product_path_does_not_import_oracle():
    """The package and its sources never reference the oracle."""
    pkg = os.path.join(ROOT, "paper_2609_37617_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".h", ".cuh")):
                text = open(os.path.join(dirpath, fn)).read()
                assert "import oracle" not in text and "oracle.h" not in text, fn
                assert "from oracle" not in text, fn
