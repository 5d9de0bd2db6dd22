"""C-ABI checks that need no GPU: the library loads, exports every entry
point declared in include/prunepath.h, and rejects bad arguments on the host
(before any CUDA call) with the documented status codes."""
import ctypes
import os
import re

import pytest

from paper_2605_28283_gb300 import binding as pp
from paper_2605_28283_gb300 import build as ppbuild

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "prunepath.h")


@pytest.fixture(scope="module")
def lib():
    ppbuild.build()
    return pp.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(pp_[a-z_]+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(pp.EXPORTS), "binding and header disagree"


def test_status_strings(lib):
    assert pp.pp_status_string(0) == "PP_OK"
    assert pp.pp_status_string(7) == "PP_ERR_TIMEOUT"
    assert pp.pp_status_string(99) == "PP_ERR_UNKNOWN"
    assert re.match(r"\d+\.\d+\.\d+", pp.pp_version())


def test_workspace_size(lib):
    d = pp.make_desc(4096, 172, "bf16", "swiglu")
    s1, s64 = pp.pp_workspace_size(d, 1), pp.pp_workspace_size(d, 64)
    assert 0 < s1 < s64
    assert s1 % 256 == 0
    bad = pp.make_desc(4096, 172, "bf16", "swiglu", d_expert=32)
    assert pp.pp_workspace_size(bad, 1) == 0


class FakeT:
    """Stands in for a tensor: only an address and a byte size (never dereferenced)."""

    def __init__(self, addr, nbytes=1 << 30):
        self.addr, self.n = addr, nbytes

    def data_ptr(self):
        return self.addr

    def numel(self):
        return self.n

    def element_size(self):
        return 1


A = 0x10000  # aligned fake device addresses (validation never dereferences them)


def call_layer(desc, T=1, x=A, Wr=A, Wg=A, Wu=A, Wd=A, p=0.5, y=A, ws=A, ws_bytes=1 << 30, sel=True):
    s = pp.pp_selection(A, A, A, None) if sel else None
    return pp.load().pp_layer(ctypes.byref(desc), ctypes.c_void_p(x), T, ctypes.c_void_p(Wr),
                              ctypes.c_void_p(Wg) if Wg else None, ctypes.c_void_p(Wu),
                              ctypes.c_void_p(Wd), p, ctypes.byref(s) if s else None,
                              ctypes.c_void_p(y), ctypes.c_void_p(ws), ws_bytes, None)


def test_argument_validation(lib):
    good = pp.make_desc(4096, 172, "bf16", "swiglu")
    assert call_layer(good, p=float("nan")) == pp.PP_ERR_INVALID_ARG
    assert call_layer(good, x=0) == pp.PP_ERR_INVALID_ARG
    assert call_layer(good, Wg=0) == pp.PP_ERR_INVALID_ARG          # SwiGLU needs W_gate
    assert call_layer(good, x=A + 8) == pp.PP_ERR_ALIGN
    assert call_layer(good, Wd=A + 2) == pp.PP_ERR_ALIGN
    assert call_layer(good, ws=A + 16) == pp.PP_ERR_WORKSPACE       # 256-byte alignment
    assert call_layer(good, ws_bytes=1024) == pp.PP_ERR_WORKSPACE
    assert call_layer(good, T=-1) == pp.PP_ERR_SHAPE
    for kw in ({"d_expert": 32}, {"n_experts": 300}, {"d_model": 4100}, {"d_model": 8200}):
        args = dict(d_model=4096, n_experts=172, dtype="bf16", act="swiglu")
        args.update(kw)
        assert call_layer(pp.make_desc(**args)) == pp.PP_ERR_SHAPE, kw
    bad = pp.make_desc(4096, 172, "bf16", "swiglu")
    bad.dtype = 7
    assert call_layer(bad) == pp.PP_ERR_DTYPE
    bad = pp.make_desc(4096, 172, "bf16", "swiglu")
    bad.rule = 5
    assert call_layer(bad) == pp.PP_ERR_INVALID_ARG
    relu = pp.make_desc(256, 16, "f32", "relu")
    # valid arguments reach the device check, which fails without a GPU
    import torch
    if not torch.cuda.is_available():
        assert call_layer(relu, Wg=0) in (pp.PP_ERR_CUDA, pp.PP_ERR_UNSUPPORTED)


def test_select_and_stats_validation(lib):
    d = pp.make_desc(64, 16, "bf16", "swiglu")
    sel = pp.pp_selection(A, A, A, None)
    L = pp.load()
    assert L.pp_select(ctypes.byref(d), None, 4, 0.5, ctypes.byref(sel), ctypes.c_void_p(A), 1 << 30,
                       None) == pp.PP_ERR_INVALID_ARG
    bad_sel = pp.pp_selection(A, 0, A, None)
    assert L.pp_select(ctypes.byref(d), ctypes.c_void_p(A), 4, 0.5, ctypes.byref(bad_sel),
                       ctypes.c_void_p(A), 1 << 30, None) == pp.PP_ERR_INVALID_ARG
    assert L.pp_sparsity_stats(None, 4, 16, ctypes.c_void_p(A), None) == pp.PP_ERR_INVALID_ARG
    assert L.pp_sparsity_stats(ctypes.c_void_p(A), 4, 300, ctypes.c_void_p(A), None) == pp.PP_ERR_INVALID_ARG
    assert L.pp_debug_wait_timeout(ctypes.c_void_p(A), 1 << 20, 0, None) == pp.PP_ERR_INVALID_ARG
    assert L.pp_workspace_init(ctypes.c_void_p(A + 8), 1 << 20, None) == pp.PP_ERR_WORKSPACE
    ws = ctypes.c_void_p(A)
    assert L.pp_router_stats(ctypes.byref(d), ctypes.c_void_p(A), 0, 1e-9, ctypes.c_void_p(A), ws, 1 << 30,
                             None) == pp.PP_ERR_SHAPE
    assert L.pp_router_stats(ctypes.byref(d), None, 4, 1e-9, ctypes.c_void_p(A), ws, 1 << 30,
                             None) == pp.PP_ERR_INVALID_ARG
    assert L.pp_router_stats(ctypes.byref(d), ctypes.c_void_p(A), 4, float("nan"), ctypes.c_void_p(A), ws,
                             1 << 30, None) == pp.PP_ERR_INVALID_ARG
    assert L.pp_router_stats(ctypes.byref(d), ctypes.c_void_p(A), 4, 1e-9, ctypes.c_void_p(A + 4), ws,
                             1 << 30, None) == pp.PP_ERR_ALIGN
    bad_rule = pp.make_desc(64, 16, "bf16", "swiglu")
    bad_rule.rule = 4
    assert L.pp_select(ctypes.byref(bad_rule), ctypes.c_void_p(A), 4, 0.5, ctypes.byref(sel),
                       ctypes.c_void_p(A), 1 << 30, None) == pp.PP_ERR_INVALID_ARG
    for rule in (pp.PP_SEL_TOPK, pp.PP_SEL_LTE):
        d2 = pp.make_desc(64, 16, "bf16", "swiglu", rule=rule)
        assert L.pp_select(ctypes.byref(d2), ctypes.c_void_p(A), 4, float("nan"), ctypes.byref(sel),
                           ctypes.c_void_p(A), 1 << 30, None) == pp.PP_ERR_INVALID_ARG
