"""The C-ABI library loads and exports every function include/hs.h declares
(no compute calls: this runs without a GPU), and the binding keeps the same
names."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "hs.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hs_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_four_steps():
    names = declared_functions()
    for n in ["hs_fingerprint", "hs_unique_inverse", "hs_retrieve_topk", "hs_scatter_results"]:
        assert n in names


def test_library_builds_and_exports_every_declared_symbol():
    from paper_2607_22578_gb300 import build
    path = build.build()
    lib = ctypes.CDLL(path)
    for name in declared_functions():
        assert hasattr(lib, name), "missing export " + name


def test_host_only_calls_without_gpu():
    """Calls that touch no device: version, workspace sizes of empty inputs,
    and argument validation paths that return before any CUDA call."""
    from paper_2607_22578_gb300 import _lib
    lib = _lib.load()
    assert b"sm_103a" in lib.hs_version()
    assert lib.hs_unique_inverse_workspace(0) > 0
    # n_rows < 0 is rejected before anything is enqueued.
    rc = lib.hs_fingerprint(None, -1, 4, None, 0, None, None)
    assert rc == _lib.HS_ERR_INVALID_ARG
    assert b"n_rows" in lib.hs_last_error()
    rc = lib.hs_scatter_results(None, 1, 0, None, 1, None, None)
    assert rc == _lib.HS_ERR_INVALID_ARG
    rc = lib.hs_retrieve_topk(None, 1, None, 10, 12, 3, None, None, None, 0, None)
    assert rc == _lib.HS_ERR_INVALID_ARG and b"dim" in lib.hs_last_error()
    rc = lib.hs_retrieve_topk(None, 1, None, 10, 64, 11, None, None, None, 0, None)
    assert rc == _lib.HS_ERR_INVALID_ARG and b"k outside" in lib.hs_last_error()
    rc = lib.hs_unique_inverse(None, None, 1 << 30, 4, None, None, None, None, None, 0, None)
    assert rc == _lib.HS_ERR_INVALID_ARG
    rc = lib.hs_merge_queries(None, _lib.HS_MERGE_QUERIES_MAX + 1, 768, 0, None, None, None,
                              None, None, None, None)
    assert rc == _lib.HS_ERR_INVALID_ARG and b"n_queries" in lib.hs_last_error()
    rc = lib.hs_merge_queries(None, 4, 12, 0, None, None, None, None, None, None, None)
    assert rc == _lib.HS_ERR_INVALID_ARG and b"dim" in lib.hs_last_error()
    rc = lib.hs_retrieve_topk_fanout(None, 4, None, None, 4, None, 10, 64, 3, None, None, None,
                                     0, None)
    assert rc == _lib.HS_ERR_INVALID_ARG and b"inverse" in lib.hs_last_error()
    # the wait-limit test hook never allows a wait longer than the default
    assert lib.hs_debug_scan_wait(3_000_000_000, -1) == _lib.HS_ERR_INVALID_ARG
    assert lib.hs_debug_scan_wait(0, -2) == _lib.HS_ERR_INVALID_ARG
    assert lib.hs_debug_scan_wait(0, -1) == _lib.HS_OK
    assert lib.hs_debug_retrieve_wait(3_000_000_000, 0) == _lib.HS_ERR_INVALID_ARG
    assert lib.hs_debug_retrieve_wait(0, 2) == _lib.HS_ERR_INVALID_ARG
    assert lib.hs_debug_retrieve_wait(0, 0) == _lib.HS_OK
    assert lib.hs_memcpy_async(None, None, 0, None) == _lib.HS_OK
    assert lib.hs_memcpy_async(None, None, 16, None) == _lib.HS_ERR_INVALID_ARG


def test_binding_names_match_header():
    import paper_2607_22578_gb300 as hs
    for name in declared_functions():
        if name in ("hs_last_error",):
            continue
        assert hasattr(hs, name), "binding lacks " + name


def test_oracle_is_not_imported_by_the_library():
    pkg = os.path.join(ROOT, "paper_2607_22578_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in src and "from oracle" not in src
                assert "hs_oracle" not in src and "liboracle" not in src


def test_binding_constants_match_header():
    """The status codes and the #define limits the binding restates are the
    header's values."""
    import paper_2607_22578_gb300._lib as lib
    text = open(HEADER).read()
    for name, val in re.findall(r"#define (HS_[A-Z0-9_]+) (0x[0-9a-fA-F]+|\d+)", text):
        assert getattr(lib, name) == int(val, 0), name
    enum = dict(re.findall(r"\b(HS_(?:OK|ERR_[A-Z_]+)) = (\d+)", text))
    assert enum["HS_OK"] == "0"
    for name, val in enum.items():
        if name != "HS_OK":
            assert getattr(lib, name) == int(val), name
