"""The C-ABI library loads and exports every function include/jarq.h declares.

No compute call is made here: only argument checks that return before any
CUDA work, the default options and the status strings.
"""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "jarq.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(jarq_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def jarq():
    from paper_2609_38599_gb300 import build as b
    if not os.path.exists(b.LIB):
        b.build()
    from paper_2609_38599_gb300 import jarq as mod
    return mod


def test_header_declares_the_boundary():
    names = declared_functions()
    for fn in ("jarq_prepare_hessian", "jarq_refine_layer", "jarq_objective",
               "jarq_hessian_destroy", "jarq_status_string", "jarq_default_options"):
        assert fn in names


def test_library_exports_every_declared_symbol(jarq):
    lib = jarq.library()
    for fn in declared_functions():
        assert hasattr(lib, fn), fn
    assert set(jarq.EXPORTS) <= set(declared_functions())


def test_default_options_follow_the_paper(jarq):
    o = jarq.default_options()
    assert o.max_iters == 3 and o.early_stop == 1
    assert o.tau_rel == pytest.approx(1e-5) and o.tau_abs == pytest.approx(1e-5)
    assert o.ridge == pytest.approx(1e-4) and o.rcond == pytest.approx(1e-10)
    assert o.eps == pytest.approx(2.0 ** -23)


def test_status_strings(jarq):
    for s in range(7):
        assert isinstance(jarq.status_string(s), str) and jarq.status_string(s)


def test_argument_errors_return_before_cuda_work(jarq):
    lib = jarq.library()
    h = ctypes.c_void_p()
    buf = (ctypes.c_float * 16)()
    # din not a multiple of the group size, group size 0, > 128, NULL H, NULL out
    assert lib.jarq_prepare_hessian(ctypes.addressof(buf), 6, 4, 0.0, ctypes.byref(h), None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_prepare_hessian(ctypes.addressof(buf), 4, 0, 0.0, ctypes.byref(h), None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_prepare_hessian(ctypes.addressof(buf), 256, 256, 0.0, ctypes.byref(h), None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_prepare_hessian(ctypes.addressof(buf), 256, 32, 0.0, ctypes.byref(h), None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_prepare_hessian(ctypes.addressof(buf), 192, 128, 0.0, ctypes.byref(h), None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_prepare_hessian(None, 4, 4, 0.0, ctypes.byref(h), None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_prepare_hessian(ctypes.addressof(buf), 4, 4, 0.0, None, None) == jarq.JARQ_ERR_ARG
    # NULL handle, bad bits, negative dout
    o = jarq.default_options()
    assert lib.jarq_refine_layer(None, None, None, None, None, 1, 3, ctypes.byref(o), None, None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_objective(None, None, None, None, None, 1, 3, None, None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_hessian_din(None) == 0 and lib.jarq_hessian_group_size(None) == 0
    lib.jarq_hessian_destroy(None)


def test_writeback_of_an_empty_layer_returns_ok_without_cuda_work(jarq):
    """dout = 0: the write-back calls validate their sizes and return JARQ_OK
    before touching any pointer (which may then be NULL)."""
    lib = jarq.library()
    assert lib.jarq_canonicalize(None, None, None, 0, 256, 64, 3, None) == 0
    assert lib.jarq_dequantize(None, None, None, 0, 256, 64, 3, 1, None, None) == 0
    assert lib.jarq_pack_codes(None, 0, 256, 3, None, None) == 0
    # the sizes are still checked
    assert lib.jarq_canonicalize(None, None, None, 0, 250, 64, 3, None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_dequantize(None, None, None, 0, 256, 64, 9, 1, None, None) == jarq.JARQ_ERR_ARG
    assert lib.jarq_pack_codes(None, -1, 256, 3, None, None) == jarq.JARQ_ERR_ARG
