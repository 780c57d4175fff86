"""C ABI checks that need no GPU: the library loads, exports every function that
include/cm.h declares, and rejects invalid arguments before touching CUDA."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", h) for h in sorted(os.listdir(os.path.join(ROOT, "include")))
           if h.endswith(".h")]


def _declared_functions():
    names = set()
    for path in HEADERS:
        text = re.sub(r"/\*.*?\*/", "", open(path).read(), flags=re.S)
        names |= set(re.findall(r"\b(cm_[a-z_]+)\s*\(", text))
    return sorted(names)


@pytest.fixture(scope="module")
def cm():
    import paper_2607_01308_gb300 as cm
    return cm


def test_header_declares_the_documented_calls():
    want = {"cm_abi_version", "cm_context_create", "cm_context_destroy", "cm_set_create",
            "cm_set_destroy", "cm_fragment_id", "cm_ingest", "cm_union", "cm_set_size",
            "cm_set_seq_len", "cm_set_ids", "cm_render", "cm_bagmerge", "cm_status_string",
            "cm_last_error_message", "cm_context_check", "cm_ingest_batch",
            "cm_context_set_timing", "cm_context_kernel_times", "cm_fragment_id_static",
            "cm_render_incremental", "cm_render_paged", "cm_ingest_many", "cm_render_many",
            "cm_set_contains", "cm_set_leq", "cm_measure_int_alu",
            "cm_context_set_render_warps", "cm_context_set_dedup_by_bytes", "cm_ingest_render",
            "cm_context_set_overlap"}
    assert want <= set(_declared_functions())


def test_library_exports_every_declared_symbol(cm):
    lib = ctypes.CDLL(cm.LIB_PATH)
    for name in _declared_functions():
        assert hasattr(lib, name), name
    assert set(_declared_functions()) == set(cm.EXPORTED)


def test_abi_version_and_status_strings(cm):
    assert cm.cm_abi_version() == 5
    for st in cm.Status:
        assert cm.cm_status_string(int(st)) == "CM_" + st.name
    assert cm.cm_status_string(99) == "CM_ERR_UNKNOWN"


def test_null_and_range_arguments_rejected_without_cuda(cm):
    lib = cm.lib
    P = ctypes.c_void_p
    assert lib.cm_context_create(0, 1e6, -1, 0, None) == cm.Status.ERR_INVALID_ARG
    out = P()
    assert lib.cm_context_create(-1, 1e6, -1, 0, ctypes.byref(out)) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_context_create(0, -1.0, -1, 0, ctypes.byref(out)) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_context_create(0, float("nan"), -1, 0, ctypes.byref(out)) == cm.Status.ERR_INVALID_ARG
    assert "rope_theta" in cm.cm_last_error_message()
    assert lib.cm_set_create(None, ctypes.byref(out)) == cm.Status.ERR_INVALID_ARG
    n = ctypes.c_int64()
    assert lib.cm_set_size(None, ctypes.byref(n)) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_set_seq_len(None, ctypes.byref(n)) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_set_ids(None, None, 0) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_union(None, None) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_render(None, None, None, 0, None, None, None) == cm.Status.ERR_INVALID_ARG
    idv = cm.cm_id()
    assert lib.cm_ingest(None, None, None, ctypes.byref(idv), None) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_fragment_id(None, None, None, ctypes.byref(idv), None) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_bagmerge(None, None, 0, None, None, 0, None, None) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_context_check(None, None) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_ingest_batch(None, None, 0, None, None, None) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_context_set_timing(None, 1) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_context_kernel_times(None, None, 0) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_render_paged(None, None, None, None, None) == cm.Status.ERR_INVALID_ARG
    assert lib.cm_render_incremental(None, None, None, 0, None, 0, None, None, None,
                                     None) == cm.Status.ERR_INVALID_ARG
    # destroying NULL handles is a no-op
    assert lib.cm_set_destroy(None) == cm.Status.OK
    assert lib.cm_context_destroy(None) == cm.Status.OK


def test_bounds_checked_build_compiles_and_exports_every_declared_call():
    # the testing build (build.py --bounds) is the same library with checked accesses
    import shutil
    import subprocess
    nm = shutil.which("nm")
    if nm is None:
        pytest.skip("nm is not available")
    from paper_2607_01308_gb300 import build as cm_build
    path = cm_build.build(bounds=True)
    out = subprocess.run([nm, "-D", "--defined-only", path], stdout=subprocess.PIPE, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\b(cm_[a-z_]+)\b", out))
    assert set(_declared_functions()) <= exported
