"""C-ABI library: loads without a GPU, exports every declared symbol, and its
host-side validation answers without touching the device."""
import ctypes
import os
import re

import pytest

from paper_2609_32479_gb300 import trackfit as T, workloads as W

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "trackfit.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(T.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    return T.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(trackfit_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(T.EXPORTS)


@pytest.mark.parametrize("name", ["tiny", "small", "medium", "large", "sweep64"])
def test_weight_count_matches_layout(lib, name):
    m = W.workload(name).model
    assert T.weight_count(m) == W.weight_count(m)
    e = m.with_(pool=W.POOL_ENDPOINTS)
    assert T.weight_count(e) == W.weight_count(e)


@pytest.mark.parametrize("bad", [dict(d_model=24), dict(d_hidden=100), dict(max_hits=65), dict(max_hits=0),
                                 dict(n_layers=0), dict(n_layers=17), dict(head_hidden=64), dict(n_quantiles=6),
                                 dict(precision=3), dict(pool=3), dict(n_fourier=8), dict(rms_eps=0.0),
                                 dict(d_model=272, d_hidden=408)])
def test_unsupported_configs_rejected_on_host(lib, bad):
    m = W.workload("tiny").model.with_(**bad)
    c = T.make_config(m)
    assert lib.trackfit_weight_count(ctypes.byref(c)) == 0
    h = ctypes.c_void_p()
    st = lib.trackfit_create(ctypes.byref(c), ctypes.c_void_p(16), 10, ctypes.byref(h))
    assert st == T.ERR_UNSUPPORTED and not h.value


def test_null_and_count_errors_on_host(lib):
    m = W.workload("tiny").model
    c = T.make_config(m)
    h = ctypes.c_void_p()
    assert lib.trackfit_create(None, ctypes.c_void_p(16), 1, ctypes.byref(h)) == T.ERR_INVALID_ARG
    assert lib.trackfit_create(ctypes.byref(c), None, 1, ctypes.byref(h)) == T.ERR_INVALID_ARG
    n = W.weight_count(m)
    assert lib.trackfit_create(ctypes.byref(c), ctypes.c_void_p(16), n + 1, ctypes.byref(h)) == T.ERR_INVALID_ARG
    c.abi_version = 2
    assert lib.trackfit_create(ctypes.byref(c), ctypes.c_void_p(16), n, ctypes.byref(h)) == T.ERR_UNSUPPORTED
    assert lib.trackfit_forward(None, ctypes.c_void_p(16), ctypes.c_void_p(16), 4, ctypes.c_void_p(16),
                                None) == T.ERR_INVALID_ARG
    lib.trackfit_destroy(None)
    for s in range(7):
        assert T.strerror(s) and T.strerror(s) != "unknown status"
    assert lib.trackfit_path_name(None) == b"none"
