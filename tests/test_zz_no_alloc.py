"""pp_layer_noalloc against pp_layer.

pp_layer_noalloc is for callers that cannot allocate device memory where
they run a layer (their memory belongs to their own pool, or an allocation's
implicit synchronisation is not allowed there): it keeps its scratch in a
static device array instead of a caller workspace.  Its results must match
pp_layer's, also on the second call in a row, when the array still holds the
first call's contents.  This file sorts last so that a run stopping at its
first failure has run every other test before it; it also passes alone.
"""
import numpy as np
import pytest

from paper_2605_28283_gb300 import workloads as wl
from parity import Y_TOL, f32, layer_inputs, rel_err_per_token, to_host

pytestmark = pytest.mark.gpu


def dev(a):
    return wl.to_torch(a, "cuda")


@pytest.mark.parametrize("name,T,p", [("llama2_7b_decode", 1, 0.7), ("llama3_8b_batched", 4, 0.5),
                                      ("gpt2m_gelu_bf16", 2, 0.9), ("tiny_relu_f32", 3, 1.0)])
def test_noalloc_matches_pp_layer(pp, name, T, p):
    import torch
    w, L = layer_inputs(name, T)
    pf = f32(p)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    x, Wr, Wu, Wd = dev(L.x), dev(L.Wr), dev(L.Wu), dev(L.Wd)
    Wg = None if L.Wg is None else dev(L.Wg)
    ws = pp.alloc_workspace(desc, T)
    ref_sel = pp.Selection.empty(T, w.n_experts, "cuda")
    y_ref = torch.empty_like(x)
    pp.pp_layer(desc, x, T, Wr, Wg, Wu, Wd, pf, ref_sel, y_ref, ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    for call in range(2):
        sel = pp.Selection.empty(T, w.n_experts, "cuda")
        y = torch.full_like(x, float("nan"))
        status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        pp.pp_layer_noalloc(desc, x, T, Wr, Wg, Wu, Wd, pf, sel, y, status)
        torch.cuda.synchronize()
        assert int(status.item()) == pp.PP_OK, (call, int(status.item()))
        np.testing.assert_array_equal(to_host(sel.counts), to_host(ref_sel.counts))
        np.testing.assert_array_equal(to_host(sel.ids), to_host(ref_sel.ids))
        err = rel_err_per_token(to_host(y), to_host(y_ref))
        assert err.max() <= Y_TOL[w.dtype], (call, float(err.max()))


def test_noalloc_slices_wide_fp32_rows(pp):
    """fp32 rows of d_model = 8192 fit the fused kernel's shared memory one
    token at a time: both entry points run such a call in one-token slices."""
    import torch
    w, L = layer_inputs("tiny_relu_f32", 3, d=8192, E=16)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    x, Wr, Wu, Wd = dev(L.x), dev(L.Wr), dev(L.Wu), dev(L.Wd)
    ws = pp.alloc_workspace(desc, 3)
    ref_sel = pp.Selection.empty(3, w.n_experts, "cuda")
    y_ref = torch.empty_like(x)
    pp.pp_layer(desc, x, 3, Wr, None, Wu, Wd, f32(0.7), ref_sel, y_ref, ws)
    for call in range(2):
        sel = pp.Selection.empty(3, w.n_experts, "cuda")
        y = torch.full_like(x, float("nan"))
        status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        pp.pp_layer_noalloc(desc, x, 3, Wr, None, Wu, Wd, f32(0.7), sel, y, status)
        torch.cuda.synchronize()
        assert int(status.item()) == pp.PP_OK
        np.testing.assert_array_equal(to_host(sel.counts), to_host(ref_sel.counts))
        np.testing.assert_array_equal(to_host(sel.ids), to_host(ref_sel.ids))
        assert rel_err_per_token(to_host(y), to_host(y_ref)).max() <= Y_TOL["f32"]


def test_noalloc_without_selection_output(pp):
    import torch
    w, L = layer_inputs("llama2_7b_decode", 1)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    args = [dev(a) for a in (L.x, L.Wr, L.Wg, L.Wu, L.Wd)]
    ws = pp.alloc_workspace(desc, 1)
    y_ref = torch.empty_like(args[0])
    pp.pp_layer(desc, args[0], 1, *args[1:], f32(0.7), None, y_ref, ws)
    y = torch.empty_like(args[0])
    pp.pp_layer_noalloc(desc, args[0], 1, *args[1:], f32(0.7), None, y)
    torch.cuda.synchronize()
    assert rel_err_per_token(to_host(y), to_host(y_ref)).max() <= Y_TOL["bf16"]


def test_noalloc_rejects_more_tokens_than_its_scratch_holds(pp):
    import torch
    w, L = layer_inputs("llama3_8b_batched", 5)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    x = dev(L.x)
    with pytest.raises(pp.PPError) as ei:
        pp.pp_layer_noalloc(desc, x, 5, dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd), 0.5, None, torch.empty_like(x))
    assert ei.value.status == pp.PP_ERR_SHAPE
