"""GPU parity of the chained decode step (pp_layer_chained):
x = RMSNorm(x_prev + y_prev) * gamma against the oracle's fp64 form, then the
layer on exactly that x against the oracle like any other layer call.  The
fused decode kernel forms x in its prologue (up to 4 bf16 / 8 fp32 tokens);
larger calls run a separate normalisation kernel first."""
import dataclasses

import numpy as np
import pytest

import oracle
from paper_2605_28283_gb300 import workloads as wl
from parity import (Y_TOL, check_route_selection, check_y, f32, layer_inputs, logit_tolerance, to_host, widen)
from test_gpu_parity import dev

pytestmark = pytest.mark.gpu

# |x_gpu - x_ref| per element: the rounding to the storage type (half an ulp:
# 2^-9 relative for bf16) plus fp32 sums
X_RTOL = {"bf16": 2.0 ** -8, "f32": 1e-5}


def host_bits(t):
    """A device tensor back to the host storage form the oracle takes."""
    import torch
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


def chained(pp, name, T, p, with_y=True, with_gamma=True, d=None, E=None, eps=1e-6, rule="min_prefix"):
    import torch
    w, L = layer_inputs(name, T, 0, 0, d, E)
    x_prev = L.x
    y_prev = wl.host_tokens(w, T, 5, 1) if with_y else None
    rng = np.random.default_rng(T)
    gamma = None
    if with_gamma:
        g32 = rng.uniform(0.5, 1.5, w.d_model).astype(np.float32)
        gamma = wl.f32_to_bf16_bits(g32) if w.dtype == "bf16" else g32
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act, "sigmoid", rule)
    ws = pp.alloc_workspace(desc, T)
    xp = dev(x_prev)
    x = torch.empty_like(xp)
    y = torch.empty_like(xp)
    sel = pp.Selection.empty(T, w.n_experts, "cuda")
    pf = f32(p)
    pp.pp_layer_chained(desc, xp, None if y_prev is None else dev(y_prev), None if gamma is None else dev(gamma),
                        eps, T, dev(L.Wr), None if L.Wg is None else dev(L.Wg), dev(L.Wu), dev(L.Wd), pf, sel, x, y,
                        ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    # the normalised input
    x_ref = oracle.rmsnorm_residual(x_prev, y_prev, gamma, float(np.float32(eps)))
    xg = to_host(x).astype(np.float64)
    scale = np.abs(x_ref).max(axis=1, keepdims=True)
    assert np.all(np.abs(xg - x_ref) <= X_RTOL[w.dtype] * np.abs(x_ref) + 1e-6 * scale), "x"
    # the layer on that x
    xb = host_bits(x)
    g_ref = oracle.logits(xb, L.Wr)
    lg = to_host(sel.logits)
    assert np.all(np.abs(lg - g_ref) <= logit_tolerance(xb, L.Wr)), "router logits"
    eps_g = np.abs(lg - g_ref).max(axis=1)
    counts, ids = to_host(sel.counts), to_host(sel.ids)
    unique, _ = check_route_selection(counts, ids, g_ref, eps_g, pf, rule)
    rc, ri, _, _ = oracle.select(g_ref, pf, rule)
    Lx = dataclasses.replace(L, x=xb)
    return check_y(Lx, to_host(y), rc, ri, g_ref, w.n_experts, w.act, "sigmoid", Y_TOL[w.dtype], unique, counts, ids)


@pytest.mark.parametrize("with_y,with_gamma", [(True, True), (True, False), (False, True), (False, False)])
def test_chained_decode_fused(pp, with_y, with_gamma):
    chained(pp, "llama2_7b_decode", 1, 0.7, with_y, with_gamma)


@pytest.mark.parametrize("name,T,d,E", [("llama2_7b_decode", 3, 512, 40), ("llama3_8b_batched", 4, None, None),
                                        ("tiny_relu_f32", 8, None, None), ("gpt2m_gelu_bf16", 2, None, None)])
def test_chained_fused_shapes(pp, name, T, d, E):
    chained(pp, name, T, 0.7, d=d, E=E)


@pytest.mark.parametrize("name,T", [("tiny_relu_f32", 64), ("gpt2m_gelu_bf16", 16), ("llama3_8b_batched", 64),
                                    ("llama2_13b_prefill", 300)])
def test_chained_separate_norm(pp, name, T):
    chained(pp, name, T, 0.7)


@pytest.mark.parametrize("rule,p", [("topk", 5.0), ("lte", 0.99)])
def test_chained_rules(pp, rule, p):
    chained(pp, "llama2_7b_decode", 2, p, rule=rule, d=1024, E=64)


def test_chained_eps_and_large_values(pp):
    """Large eps dominates the mean square; a scaled residual stream normalises to the same x."""
    chained(pp, "llama2_7b_decode", 1, 0.7, eps=4.0, d=512, E=40)


def test_chained_sequence_matches_step_by_step(pp):
    """Three chained layers through the fused kernel equal the same three
    layers with the normalisation done by the oracle's formula on the host."""
    import torch
    w = wl.scaled(wl.WORKLOADS["llama2_7b_decode"], 1024, 48)
    T = 1
    layers = [wl.host_layer(w, T, seed=3, layer=l) for l in range(3)]
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    ws = pp.alloc_workspace(desc, T)
    x_prev = dev(layers[0].x)
    y_prev = None
    for l, L in enumerate(layers):
        x = torch.empty_like(x_prev)
        y = torch.empty_like(x_prev)
        pp.pp_layer_chained(desc, x_prev, y_prev, None, 1e-6, T, dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd),
                            0.7, None, x, y, ws)
        torch.cuda.synchronize()
        ref = oracle.rmsnorm_residual(host_bits(x_prev), None if y_prev is None else host_bits(y_prev), None, 1e-6)
        xg = to_host(x).astype(np.float64)
        assert np.all(np.abs(xg - ref) <= X_RTOL["bf16"] * np.abs(ref) + 1e-6), ("x", l)
        x_prev, y_prev = x, y
    assert pp.pp_get_device_status(ws) == pp.PP_OK


def test_chained_rejects_aliasing(pp):
    import torch
    w, L = layer_inputs("llama2_7b_decode", 1, 0, 0, 512, 40)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    ws = pp.alloc_workspace(desc, 1)
    xp = dev(L.x)
    y = torch.empty_like(xp)
    with pytest.raises(pp.PPError):
        pp.pp_layer_chained(desc, xp, None, None, 1e-6, 1, dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd), 0.7, None,
                            xp, y, ws)
