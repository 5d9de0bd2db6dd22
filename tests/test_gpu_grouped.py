"""GPU parity of the tensor-core grouped path (bf16, T >= 5): router GEMM,
selection from K-split partials, dispatch, grouped gate/up and down GEMMs.

The full-size Llama-2-13B prefill case (4 x 2048 tokens) is checked on a
sample of tokens the oracle evaluates one by one."""
import numpy as np
import pytest

import oracle
from paper_2605_28283_gb300 import workloads as wl
from parity import (Y_TOL, check_route_selection, check_y, f32, layer_inputs, logit_tolerance, to_host)
from test_gpu_parity import dev, layer_parity

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("T,p", [(5, 0.7), (8, 0.3), (32, 0.5), (64, 0.7), (64, 0.95), (127, 0.9),
                                 (128, 0.7), (129, 0.7), (256, 0.7), (257, 0.5)])
def test_grouped_llama3_batched(pp, T, p):
    layer_parity(pp, "llama3_8b_batched", T, p)


@pytest.mark.parametrize("T,p", [(16, 0.5), (16, 0.9), (40, 1.0)])
def test_grouped_gelu(pp, T, p):
    layer_parity(pp, "gpt2m_gelu_bf16", T, p)


@pytest.mark.parametrize("d,E,T", [(200, 9, 20), (1000, 40, 160)])
def test_grouped_gelu_odd_shapes(pp, d, E, T):
    """Non-gated FFN with d not a multiple of the 64-wide K chunk."""
    layer_parity(pp, "gpt2m_gelu_bf16", T, 0.8, d=d, E=E)


@pytest.mark.parametrize("rule,gate", [("paper", "sigmoid"), ("min_prefix", "none"), ("paper", "none")])
def test_grouped_rules_gates(pp, rule, gate):
    layer_parity(pp, "llama2_7b_decode", 24, 0.6, rule, gate, d=1024, E=48)


@pytest.mark.parametrize("d,E,T", [(128, 3, 5), (200, 33, 9), (512, 256, 33), (8192, 20, 6), (1024, 1, 7),
                                   (200, 33, 150), (328, 7, 300)])
def test_grouped_odd_shapes(pp, d, E, T):
    layer_parity(pp, "llama3_8b_batched", T, 0.8, d=d, E=E)


def test_grouped_all_experts(pp):
    """p >= 1 sends every token to every expert (the largest dispatch)."""
    layer_parity(pp, "llama3_8b_batched", 200, 1.0, d=512, E=64)


@pytest.mark.parametrize("T", [300, 2048])
def test_grouped_prefill_13b_shape(pp, T):
    layer_parity(pp, "llama2_13b_prefill", T, 0.7) if T <= 300 else _sampled_prefill(pp, T, 48)


def test_grouped_prefill_13b_full(pp):
    """The full 4 x 2048-token Llama-2-13B-shaped prefill, sampled."""
    _sampled_prefill(pp, 8192, 64)


def _sampled_prefill(pp, T, n_sample):
    import torch
    w = wl.WORKLOADS["llama2_13b_prefill"]
    L = wl.host_layer(w, T, seed=7, layer=3)
    p = f32(0.7)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    ws = pp.alloc_workspace(desc, T)
    x = dev(L.x)
    y = torch.empty_like(x)
    sel = pp.Selection.empty(T, w.n_experts, "cuda")
    pp.pp_layer(desc, x, T, dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd), p, sel, y, ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    rng = np.random.default_rng(11)
    rows = np.sort(np.concatenate([[0, T - 1], rng.choice(np.arange(1, T - 1), n_sample - 2, replace=False)]))
    xs = L.x[rows]
    g_ref = oracle.logits(xs, L.Wr)
    lg = to_host(sel.logits)[rows]
    assert np.all(np.abs(lg - g_ref) <= logit_tolerance(xs, L.Wr))
    eps = np.abs(lg - g_ref).max(axis=1)
    counts, ids = to_host(sel.counts)[rows], to_host(sel.ids)[rows]
    unique, _ = check_route_selection(counts, ids, g_ref, eps, p, "min_prefix")
    rc, ri, _, _ = oracle.select(g_ref, p, "min_prefix")

    class Sub:
        pass
    S = Sub()
    S.x, S.Wg, S.Wu, S.Wd = xs, L.Wg, L.Wu, L.Wd
    check_y(S, to_host(y)[rows], rc, ri, g_ref, w.n_experts, w.act, "sigmoid", Y_TOL["bf16"], unique, counts, ids)
    # every token got a non-empty selection and finite output
    assert np.all(to_host(sel.counts) >= 1)
    assert torch.isfinite(y.float()).all()
