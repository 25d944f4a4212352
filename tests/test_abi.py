"""The C ABI without a GPU: libdas.so loads, exports every function that
include/das.h declares, and rejects bad arguments on the host before any
CUDA call."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "das.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(das_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ["das_workspace_size", "das_mature_v_attention", "das_verify_attention",
              "das_greedy_accept", "das_kv_append", "das_wave_readout", "das_status_string"]:
        assert n in names


def test_library_exports_every_declared_symbol():
    import paper_2609_34538_gb300 as das
    lib = ctypes.CDLL(das.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings():
    import paper_2609_34538_gb300 as das
    assert das.status_string(0) == "ok"
    assert "workspace" in das.status_string(3)
    assert das.status_string(99) == "unknown status"


def test_host_argument_checks():
    import paper_2609_34538_gb300 as das
    L = das.LIB
    null = ctypes.c_void_p(0)
    # null cache
    assert L.das_mature_v_attention(None, 0, 1, 1, null, null, 1, null, null, null, 1, 0.0,
                                    null, null, null, 0, null) == das.DAS_ERR_INVALID_ARG
    c = das.das_kv_cache(16, 16, 4, 1, 1, 64, 1, 128)
    # depth out of range, then a block too large for one pair (G * max_block > 64)
    assert L.das_verify_attention(ctypes.byref(c), 0, 5, null, null, 1, null, null, null, 1, 0.0,
                                  null, null, null, 0, null) == das.DAS_ERR_INVALID_ARG
    c2 = das.das_kv_cache(16, 16, 4, 1, 1, 64, 1, 96)
    assert L.das_verify_attention(ctypes.byref(c2), 0, 1, null, null, 1, null, null, null, 1,
                                  0.0, null, null, null, 0, null) == das.DAS_ERR_UNSUPPORTED
    assert L.das_workspace_size(ctypes.byref(c), 8, 16) == 0        # 8 * 16 rows > 64
    assert L.das_greedy_accept(null, null, 1, 0, 10, null, null, null, null) == das.DAS_ERR_INVALID_ARG
    assert L.das_kv_append(ctypes.byref(c), null, null, null, 1, null, null, null) == das.DAS_ERR_INVALID_ARG
    assert L.das_wave_readout(null, 1, 4, 10, null, 5, null) == das.DAS_ERR_INVALID_ARG
    dummy = ctypes.c_void_p(256)  # never dereferenced: the checks fail first
    assert L.das_wave_readout(dummy, 1, 4, 10, dummy, 4, null) == das.DAS_ERR_INVALID_ARG  # stride < W+1
    assert L.das_wave_readout(dummy, 1, 0, 10, dummy, 4, null) == das.DAS_ERR_INVALID_ARG  # W = 0
