"""Host-side checks that need no GPU: the library builds and loads, exports
every entry point that include/ace.h declares, and plan validation fails
loudly on a machine without an sm_103 device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "ace.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ace_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_06072_gb300 import _build, ace
    _build.build()
    return ace.load()


@pytest.fixture(scope="module")
def lib_checks():
    from paper_2609_06072_gb300 import _build, ace
    _build.build(checks=True)
    return ace.load(checks=True)


def test_checked_build_exports_the_same_boundary(lib, lib_checks):
    # libace_checks.so: the same sources with ACE_CHECKS; same symbols, and
    # each library reports which build it is
    for s in declared_symbols():
        assert hasattr(lib_checks, s), f"libace_checks.so does not export {s}"
    assert lib.ace_build_checks() == 0
    assert lib_checks.ace_build_checks() == 1
    assert lib_checks.ace_version() == lib.ace_version()


def test_header_declares_the_boundary():
    syms = declared_symbols()
    from paper_2609_06072_gb300 import ace
    assert syms == sorted(ace.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    for s in declared_symbols():
        assert hasattr(lib, s), f"libace.so does not export {s}"


def test_version_and_error_message(lib):
    assert lib.ace_version() == 1
    assert isinstance(lib.ace_last_error_message(), bytes)


def test_plan_rejects_bad_descriptions_without_gpu(lib):
    from paper_2609_06072_gb300 import ace
    e2g = (ctypes.c_int32 * 4)(0, 0, 1, 1)
    ro = (ctypes.c_int32 * 3)(0, 8, 16)
    h = ctypes.c_void_p()
    # k > E
    d = ace.ace_layer_desc(16, 5, 4, 2, e2g, ro, 64, 64, 0)
    assert lib.ace_plan_create(ctypes.byref(h), ctypes.byref(d)) == ace.ACE_ERR_SHAPE
    # map out of range
    bad = (ctypes.c_int32 * 4)(0, 0, 2, 1)
    d = ace.ace_layer_desc(16, 2, 4, 2, bad, ro, 64, 64, 0)
    assert lib.ace_plan_create(ctypes.byref(h), ctypes.byref(d)) == ace.ACE_ERR_INDEX
    # empty group
    d = ace.ace_layer_desc(16, 2, 4, 3, e2g, (ctypes.c_int32 * 4)(0, 8, 16, 24), 64, 64, 0)
    assert lib.ace_plan_create(ctypes.byref(h), ctypes.byref(d)) == ace.ACE_ERR_INDEX
    # rank too large
    d = ace.ace_layer_desc(16, 2, 4, 2, e2g, (ctypes.c_int32 * 3)(0, 200, 208), 64, 64, 0)
    assert lib.ace_plan_create(ctypes.byref(h), ctypes.byref(d)) == ace.ACE_ERR_UNSUPPORTED
    # d not a multiple of 8
    d = ace.ace_layer_desc(16, 2, 4, 2, e2g, ro, 60, 64, 0)
    assert lib.ace_plan_create(ctypes.byref(h), ctypes.byref(d)) == ace.ACE_ERR_SHAPE
    # T_max * k above 2^30 rows
    d = ace.ace_layer_desc((1 << 29) + 1, 2, 4, 2, e2g, ro, 64, 64, 0)
    assert lib.ace_plan_create(ctypes.byref(h), ctypes.byref(d)) == ace.ACE_ERR_SHAPE
    # a valid description on a machine without an sm_103 device: no plan, no fallback
    d = ace.ace_layer_desc(16, 2, 4, 2, e2g, ro, 64, 64, 0)
    st = lib.ace_plan_create(ctypes.byref(h), ctypes.byref(d))
    import torch
    if not torch.cuda.is_available():
        assert st in (ace.ACE_ERR_CUDA, ace.ACE_ERR_UNSUPPORTED)
        assert not h.value


def test_null_arguments_are_rejected(lib):
    from paper_2609_06072_gb300 import ace
    assert lib.ace_plan_create(None, None) == ace.ACE_ERR_ARG
    assert lib.ace_workspace_size(None, 0, None, None, None) == ace.ACE_ERR_ARG
    assert lib.ace_permute(None, None, 0, None, 0, None, None) == ace.ACE_ERR_ARG
    assert lib.ace_get_error(None, None) == ace.ACE_ERR_ARG
    assert lib.ace_plan_rank_cols(None) == 0
    assert lib.ace_fwd_combine(None, None, None, None, None, None, 1.0, None, None, None, None) == ace.ACE_ERR_ARG
    assert lib.ace_bwd_combine(None, None, None, None, None, None, None, None, None, 1.0, None, None, None, None, None,
                               0, None) == ace.ACE_ERR_ARG


def test_cka_shape_checks_without_gpu(lib):
    import ctypes
    from paper_2609_06072_gb300 import ace
    nb = ctypes.c_size_t()
    assert lib.ace_cka_workspace_size(10000, 2048, 1024, 64, 8, ctypes.byref(nb)) == ace.ACE_OK
    # covariance 16 MiB + stacked-rank products, and more for more experts
    assert nb.value >= 4 * 2048 * 2048 + 4 * 512 * 2048 + 4 * 512 * 512
    assert lib.ace_cka_workspace_size(10000, 2000, 1024, 64, 8, ctypes.byref(nb)) == ace.ACE_ERR_SHAPE
    assert lib.ace_cka_workspace_size(10000, 2048, 1024, 64, 33, ctypes.byref(nb)) == ace.ACE_ERR_SHAPE
    assert lib.ace_cka(16, 64, 8, 2, 2, None, None, None, 1, None, None, 0, None) == ace.ACE_ERR_ARG


def test_consolidate_adapters_host_checks_without_gpu(lib):
    import ctypes
    import numpy as np
    from paper_2609_06072_gb300 import ace
    e2g = np.array([0, 1, 0, 1], np.int32)
    ro = np.zeros(3, np.int32)
    dummy = ctypes.c_void_p(16)  # never dereferenced: the checks fail before any launch

    def call(e2g_, anchors_, G):
        return lib.ace_consolidate_adapters(4, 2, 8, 8, e2g_.ctypes.data, anchors_.ctypes.data, G, dummy, dummy,
                                            dummy, dummy, dummy, ro.ctypes.data, None)
    assert call(e2g, np.array([1, 1], np.int32), 2) == ace.ACE_ERR_INDEX  # anchor 1 is not in group 0
    assert call(np.array([0, 2, 0, 1], np.int32), np.array([0, 1], np.int32), 2) == ace.ACE_ERR_INDEX
    assert call(np.array([0, 0, 0, 0], np.int32), np.array([0, 1], np.int32), 2) == ace.ACE_ERR_INDEX  # empty group
    assert call(e2g, np.array([0, 1], np.int32), 0) == ace.ACE_ERR_SHAPE


def test_ffn_null_arguments_without_gpu(lib):
    from paper_2609_06072_gb300 import ace
    assert lib.ace_ffn_workspace_size(None, 0, None) == ace.ACE_ERR_ARG
    assert lib.ace_ffn_fwd(None, None, None, None, None, None, None, None, 1.0, None, None, None, None, None, None,
                           None, 0, None) == ace.ACE_ERR_ARG
    assert lib.ace_ffn_bwd(None, None, None, None, None, None, None, None, None, 1.0, None, None, None, None, None,
                           None, None, None, None, 0, None, 0, None) == ace.ACE_ERR_ARG
