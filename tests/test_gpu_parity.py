"""GPU parity: the CUDA library (through its C ABI) against the CPU oracle.

Cases cover all five workload shapes (tiny ReLU fp32, GPT-2-medium GELU,
Llama-2-7B / Llama-3-8B SwiGLU decode, Llama-2-13B SwiGLU), the two
cumulative-mass cut rules plus top-k and LTE's threshold, both gate modes, p from <= 0 to >= 1, token counts that exercise the fused
decode kernel (T <= 4 bf16 / 8 fp32), its token slices and the stand-alone
router + selection kernels, plus the degenerate inputs (ties, signed zeros,
huge and non-finite logits, T = 0).
"""
import numpy as np
import pytest

import oracle
from paper_2605_28283_gb300 import workloads as wl
from parity import (BOUNDARY, Y_TOL, check_route_selection, check_select_exact, check_y, f32,
                    layer_inputs, logit_tolerance, to_host, widen)

pytestmark = pytest.mark.gpu


def dev(a):
    return wl.to_torch(a, "cuda")


def run_layer(pp, w, L, p, rule="min_prefix", gate="sigmoid", T=None):
    import torch
    T = L.x.shape[0] if T is None else T
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act, gate, rule)
    ws = pp.alloc_workspace(desc, T)
    x, Wr, Wu, Wd = dev(L.x), dev(L.Wr), dev(L.Wu), dev(L.Wd)
    Wg = None if L.Wg is None else dev(L.Wg)
    sel = pp.Selection.empty(T, w.n_experts, "cuda")
    y = torch.empty_like(x)
    pp.pp_layer(desc, x, T, Wr, Wg, Wu, Wd, p, sel, y, ws)
    torch.cuda.synchronize()
    status = pp.pp_get_device_status(ws)
    return (to_host(sel.counts), to_host(sel.ids), to_host(sel.logits), to_host(y), status)


def layer_parity(pp, name, T, p, rule="min_prefix", gate="sigmoid", d=None, E=None, seed=0, layer=0):
    w, L = layer_inputs(name, T, seed, layer, d, E)
    pf = f32(p)
    counts, ids, logits, y, status = run_layer(pp, w, L, pf, rule, gate)
    assert status == pp.PP_OK, pp.status_name(status)
    g_ref = oracle.logits(L.x, L.Wr)
    tol_g = logit_tolerance(L.x, L.Wr)
    assert np.all(np.abs(logits - g_ref) <= tol_g), "router logits"
    eps = np.abs(logits - g_ref).max(axis=1)
    unique, n_nonunique = check_route_selection(counts, ids, g_ref, eps, pf, rule)
    ro_counts, ro_ids, _, _ = oracle.select(g_ref, pf, rule)
    err = check_y(L, y, ro_counts, ro_ids, g_ref, w.n_experts, w.act, gate, Y_TOL[w.dtype], unique, counts, ids)
    return err, n_nonunique


# ------------------------------------------------------------------ pp_layer
@pytest.mark.parametrize("p", [0.5, 0.9, 1.0])
@pytest.mark.parametrize("T", [1, 3, 8, 64])
def test_layer_tiny_relu_f32(pp, T, p):
    layer_parity(pp, "tiny_relu_f32", T, p)


@pytest.mark.parametrize("p", [0.5, 0.7, 0.9])
@pytest.mark.parametrize("T", [1, 4, 16])
def test_layer_gpt2m_gelu(pp, T, p):
    layer_parity(pp, "gpt2m_gelu_bf16", T, p)


@pytest.mark.parametrize("p", [0.3, 0.5, 0.7, 0.9, 1.0])
def test_layer_llama2_7b_decode(pp, p):
    layer_parity(pp, "llama2_7b_decode", 1, p)


@pytest.mark.parametrize("T,p", [(1, 0.3), (1, 0.95), (2, 0.7), (8, 0.5), (8, 0.9)])
def test_layer_llama3_8b(pp, T, p):
    layer_parity(pp, "llama3_8b_batched", T, p)


@pytest.mark.parametrize("T", [1, 4, 37])
def test_layer_llama2_13b(pp, T):
    layer_parity(pp, "llama2_13b_prefill", T, 0.7)


@pytest.mark.parametrize("rule", ["min_prefix", "paper"])
@pytest.mark.parametrize("gate", ["sigmoid", "none"])
@pytest.mark.parametrize("p", [-0.5, 0.0, 0.4, 0.99, 1.0, 1.5])
def test_layer_rules_gates(pp, rule, gate, p):
    layer_parity(pp, "llama2_7b_decode", 3, p, rule, gate, d=512, E=40)


# Top-k (Sec. 4.3) and LTE's threshold (Eq. lte_hard_set) on the same
# kernels: the fused decode kernel (T <= 4 bf16, fp32 slices), the router +
# selection kernels and the grouped tensor-core path (bf16, T >= 5).  LTE at
# delta = 0.999 leaves some tokens without any expert (y = 0).
RULE_CASES = [("topk", 1.0), ("topk", 2.5), ("topk", 7.0), ("topk", 500.0), ("lte", -1.0), ("lte", 0.5),
              ("lte", 0.9), ("lte", 0.999), ("lte", 1.0)]


@pytest.mark.parametrize("rule,p", RULE_CASES)
@pytest.mark.parametrize("gate", ["sigmoid", "none"])
def test_layer_topk_lte_decode(pp, rule, p, gate):
    layer_parity(pp, "llama2_7b_decode", 3, p, rule, gate, d=512, E=40)


@pytest.mark.parametrize("rule,p", [("topk", 3.0), ("lte", 0.95), ("lte", 0.999)])
@pytest.mark.parametrize("name,T", [("tiny_relu_f32", 64), ("gpt2m_gelu_bf16", 16), ("llama3_8b_batched", 8),
                                    ("llama3_8b_batched", 64), ("llama2_13b_prefill", 300)])
def test_layer_topk_lte_batched(pp, name, T, rule, p):
    layer_parity(pp, name, T, p, rule, "none" if rule == "lte" else "sigmoid")


def test_layer_lte_empty_tokens(pp):
    """Tokens whose every score stays at or below delta get no expert and y = 0."""
    for T in (2, 37):
        w, L = layer_inputs("llama2_7b_decode", T, d=512, E=40)
        counts, ids, logits, y, status = run_layer(pp, w, L, 1.0, "lte", "none")
        assert status == pp.PP_OK
        assert np.all(counts == 0) and np.all(ids == -1) and np.all(y == 0.0)
        counts, ids, logits, y, status = run_layer(pp, w, L, -2.0, "lte", "none")
        assert status == pp.PP_OK and np.all(counts == w.n_experts)


@pytest.mark.parametrize("d,E,T", [(64, 1, 2), (128, 3, 5), (200, 33, 4), (2048, 256, 3), (8192, 100, 1)])
def test_layer_odd_shapes(pp, d, E, T):
    layer_parity(pp, "llama3_8b_batched", T, 0.8, d=d, E=E)


def test_layer_dense_identity(pp):
    """p >= 1 with unit gates is the dense FFN (Eq. moefication_decomp)."""
    w, L = layer_inputs("gpt2m_gelu_bf16", 4)
    counts, ids, logits, y, status = run_layer(pp, w, L, 1.0, gate="none")
    assert np.all(counts == w.n_experts)
    ref = oracle.dense_ffn(L.x, L.Wg, L.Wu, L.Wd, w.act)
    err = np.abs(y - ref).max(axis=1) / np.abs(ref).max(axis=1)
    assert err.max() <= Y_TOL["bf16"]


# ---------------------------------------------------------- pp_sparse_ffn
@pytest.mark.parametrize("name,T", [("tiny_relu_f32", 64), ("gpt2m_gelu_bf16", 16),
                                    ("llama2_7b_decode", 1), ("llama3_8b_batched", 8),
                                    ("llama2_13b_prefill", 5)])
def test_sparse_ffn_given_selection(pp, name, T):
    """Selection made by the oracle, FFN on the GPU."""
    import torch
    w, L = layer_inputs(name, T)
    g = oracle.logits(L.x, L.Wr)
    counts, ids, _, _ = oracle.select(g, 0.7, "min_prefix")
    gates = np.zeros(ids.shape, np.float32)
    for t in range(T):
        for r in range(counts[t]):
            gates[t, r] = 1.0 / (1.0 + np.exp(-g[t, ids[t, r]]))
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    ws = pp.alloc_workspace(desc, T)
    sel = pp.Selection(dev(ids), dev(counts), dev(gates))
    x = dev(L.x)
    y = torch.empty_like(x)
    pp.pp_sparse_ffn(desc, x, T, None if L.Wg is None else dev(L.Wg), dev(L.Wu), dev(L.Wd), sel, y, ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    ref = oracle.sparse_ffn(L.x, L.Wg, L.Wu, L.Wd, counts, ids, g, w.n_experts, w.act, "sigmoid")
    err = np.abs(to_host(y) - ref).max(axis=1) / np.abs(ref).max(axis=1)
    assert err.max() <= Y_TOL[w.dtype]


# ---------------------------------------------------------------- pp_route
@pytest.mark.parametrize("name,T", [("tiny_relu_f32", 64), ("gpt2m_gelu_bf16", 4),
                                    ("llama2_7b_decode", 1), ("llama3_8b_batched", 64),
                                    ("llama2_13b_prefill", 300)])
@pytest.mark.parametrize("rule", ["min_prefix", "paper"])
def test_route(pp, name, T, rule):
    import torch
    w, L = layer_inputs(name, T)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act, "sigmoid", rule)
    ws = pp.alloc_workspace(desc, T)
    sel = pp.Selection.empty(T, w.n_experts, "cuda")
    p = f32(0.7)
    pp.pp_route(desc, dev(L.x), T, dev(L.Wr), p, sel, ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    g_ref = oracle.logits(L.x, L.Wr)
    lg = to_host(sel.logits)
    assert np.all(np.abs(lg - g_ref) <= logit_tolerance(L.x, L.Wr))
    eps = np.abs(lg - g_ref).max(axis=1)
    counts, ids = to_host(sel.counts), to_host(sel.ids)
    check_route_selection(counts, ids, g_ref, eps, p, rule)
    gates = to_host(sel.gates)
    for t in range(T):
        k = counts[t]
        np.testing.assert_allclose(gates[t, :k], 1.0 / (1.0 + np.exp(-g_ref[t, ids[t, :k]])), rtol=1e-5, atol=1e-7)
        assert np.all(gates[t, k:] == 0)


@pytest.mark.parametrize("name,T", [("llama2_7b_decode", 1), ("gpt2m_gelu_bf16", 4), ("tiny_relu_f32", 64),
                                    ("llama3_8b_batched", 64), ("llama2_13b_prefill", 300)])
@pytest.mark.parametrize("rule,p", [("topk", 4.0), ("lte", 0.9)])
def test_route_topk_lte(pp, name, T, rule, p):
    import torch
    w, L = layer_inputs(name, T)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act, "sigmoid", rule)
    ws = pp.alloc_workspace(desc, T)
    sel = pp.Selection.empty(T, w.n_experts, "cuda")
    pp.pp_route(desc, dev(L.x), T, dev(L.Wr), p, sel, ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    g_ref = oracle.logits(L.x, L.Wr)
    lg = to_host(sel.logits)
    assert np.all(np.abs(lg - g_ref) <= logit_tolerance(L.x, L.Wr))
    eps = np.abs(lg - g_ref).max(axis=1)
    check_route_selection(to_host(sel.counts), to_host(sel.ids), g_ref, eps, p, rule)


# --------------------------------------------------------------- pp_select
def select_gpu(pp, logits, p, rule, gate="sigmoid"):
    import torch
    T, E = logits.shape
    desc = pp.make_desc(64, E, "bf16", "swiglu", gate, rule)
    ws = pp.alloc_workspace(desc, T)
    sel = pp.Selection.empty(T, E, "cuda", with_logits=False)
    pp.pp_select(desc, dev(logits.astype(np.float32)), T, p, sel, ws)
    torch.cuda.synchronize()
    return to_host(sel.counts), to_host(sel.ids), to_host(sel.gates), pp.pp_get_device_status(ws)


# T <= 64 runs the one-CTA-per-token counting selection, larger T the
# warp-per-token sorting selection: both are checked.
@pytest.mark.parametrize("T", [40, 2000])
@pytest.mark.parametrize("E", [1, 5, 16, 33, 64, 100, 172, 216, 224, 256])
@pytest.mark.parametrize("rule", ["min_prefix", "paper"])
def test_select_bit_exact(pp, E, rule, T):
    logits = wl.host_logits(T, E, std=3.0, seed=E)
    total_boundary = 0
    for p in (0.0, 0.3, 0.5, 0.7, 0.9, 0.95, 1.0):
        pf = f32(p)
        counts, ids, gates, status = select_gpu(pp, logits, pf, rule)
        assert status == pp.PP_OK
        g = logits.astype(np.float64)
        total_boundary += check_select_exact(counts, ids, g, pf, rule)
        for t in range(0, T, 97):
            k = counts[t]
            ref = 1.0 / (1.0 + np.exp(-g[t, ids[t, :k]]))
            np.testing.assert_allclose(gates[t, :k], ref, rtol=2e-6, atol=1e-30)
            assert np.all(gates[t, k:] == 0)
    assert total_boundary <= max(2, T * 7 * 0.01)


@pytest.mark.parametrize("T", [40, 2000])
@pytest.mark.parametrize("E", [1, 5, 33, 64, 172, 224, 256])
@pytest.mark.parametrize("rule", ["topk", "lte"])
def test_select_topk_lte_bit_exact(pp, E, rule, T):
    """Top-k is exact (no boundary); LTE is exact except scores within 1e-6 of delta."""
    logits = wl.host_logits(T, E, std=3.0, seed=E + 1)
    params = (0.0, 0.5, 1.0, 2.0, 5.5, E - 1.0, float(E), 1e9) if rule == "topk" else \
        (-1.0, 0.0, 0.05, 0.3, 0.5, 0.8, 0.97, 0.9999, 1.0, 3.0)
    nb = 0
    for p in params:
        pf = f32(p)
        counts, ids, gates, status = select_gpu(pp, logits, pf, rule)
        assert status == pp.PP_OK
        g = logits.astype(np.float64)
        nb += check_select_exact(counts, ids, g, pf, rule)
        for t in range(0, T, 97):
            k = counts[t]
            ref = 1.0 / (1.0 + np.exp(-g[t, ids[t, :k]]))
            np.testing.assert_allclose(gates[t, :k], ref, rtol=2e-6, atol=1e-30)
            assert np.all(gates[t, k:] == 0)
    assert nb <= max(2, T * len(params) * 0.01)


def test_select_lte_exact_threshold(pp):
    """A logit exactly at ln(delta / (1 - delta)) is not activated (strict >),
    the next float above it is: sigmoid(0) = 0.5 exactly."""
    E = 8
    logits = np.zeros((3, E), np.float32)
    logits[1, 3] = np.nextafter(np.float32(0.0), np.float32(1.0))
    logits[2, :] = np.float32(-0.0)
    logits[2, 5] = np.float32(1e-3)
    counts, ids, gates, status = select_gpu(pp, logits, 0.5, "lte")
    assert status == pp.PP_OK
    assert counts.tolist() == [0, 1, 1]
    assert ids[1, 0] == 3 and ids[2, 0] == 5


@pytest.mark.parametrize("T", [16, 500])
def test_select_ties_and_zeros(pp, T):
    rng = np.random.default_rng(5)
    E = 172
    logits = (np.round(rng.standard_normal((T, E)) * 4) / 2).astype(np.float32)  # many exact ties
    logits[0, :] = 0.0
    logits[1, ::2] = -0.0
    logits[2, :] = np.float32(-1e4)
    logits[2, 7] = np.float32(1e4)
    logits[3, :] = np.linspace(30, -30, E).astype(np.float32)
    for rule, ps in (("min_prefix", (0.1, 0.5, 0.75, 0.999, 1.0)), ("paper", (0.1, 0.5, 0.75, 0.999, 1.0)),
                     ("topk", (1.0, 3.0, 50.0)), ("lte", (0.5, 0.9))):
        for gate in ("sigmoid", "none"):
            for p in ps:
                pf = f32(p)
                counts, ids, gates, status = select_gpu(pp, logits, pf, rule, gate)
                assert status == pp.PP_OK
                check_select_exact(counts, ids, logits.astype(np.float64), pf, rule)
                if gate == "none":
                    for t in range(T):
                        assert np.all(gates[t, :counts[t]] == 1.0)


@pytest.mark.parametrize("T", [6, 100])
def test_select_nonfinite(pp, T):
    logits = wl.host_logits(T, 40)
    logits[1, 3] = np.nan
    logits[4, 0] = np.inf
    logits[5, 9] = -np.inf
    counts, ids, gates, status = select_gpu(pp, logits, 0.5, "min_prefix")
    assert status == pp.PP_ERR_NONFINITE
    assert counts[1] == 0 and counts[4] == 0 and counts[5] == 0
    assert np.all(ids[1] == -1) and np.all(gates[4] == 0)
    ok = [t for t in range(T) if t not in (1, 4, 5)]
    check_select_exact(counts[ok], ids[ok], logits[ok].astype(np.float64), 0.5, "min_prefix")


def test_empty_inputs(pp):
    import torch
    desc = pp.make_desc(256, 16, "f32", "relu")
    ws = pp.alloc_workspace(desc, 0)
    x = torch.empty((0, 256), device="cuda")
    w = torch.empty((16, 256), device="cuda")
    wu = torch.empty((1024, 256), device="cuda")
    wd = torch.empty((256, 1024), device="cuda")
    sel = pp.Selection.empty(1, 16, "cuda")
    y = torch.empty((1, 256), device="cuda")
    pp.pp_layer(desc, y, 0, w, None, wu, wd, 0.5, sel, y, ws)
    pp.pp_route(desc, y, 0, w, 0.5, sel, ws)
    pp.pp_select(desc, sel.logits, 0, 0.5, sel, ws)
    pp.pp_sparse_ffn(desc, y, 0, None, wu, wd, sel, y, ws)
    assert pp.pp_get_device_status(ws) == pp.PP_OK


# -------------------------------------------------------------- auxiliaries
@pytest.mark.parametrize("name,T,p,rule", [("llama2_7b_decode", 1, 0.7, "min_prefix"),
                                            ("llama3_8b_batched", 64, 0.5, "min_prefix"),
                                            ("gpt2m_gelu_bf16", 16, 0.9, "paper"),
                                            ("llama3_8b_batched", 300, 0.999, "lte")])
def test_sparsity_stats(pp, name, T, p, rule):
    """Sec. 4.1 s_FFN: pp_sparsity_stats accumulated over several layers of
    counts that the GPU's own pp_route produced, against the oracle's
    ppo_ffn_sparsity on the same counts (exact integers), and the GPU's
    counts against the oracle's selection for the tokens whose cut is unique."""
    import torch
    w = wl.WORKLOADS[name]
    n_layers = 4
    gate = "none" if rule == "lte" else "sigmoid"
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act, gate, rule)
    ws = pp.alloc_workspace(desc, T)
    acc = torch.zeros(w.n_experts + 2, dtype=torch.int64, device="cuda")
    pf = f32(p)
    all_counts = []
    for l in range(n_layers):
        L = wl.host_layer(w, T, seed=5, layer=l)
        sel = pp.Selection.empty(T, w.n_experts, "cuda")
        pp.pp_route(desc, dev(L.x), T, dev(L.Wr), pf, sel, ws)
        pp.pp_sparsity_stats(sel.counts, T, w.n_experts, acc)
        torch.cuda.synchronize()
        counts, ids, logits = to_host(sel.counts), to_host(sel.ids), to_host(sel.logits)
        g_ref = oracle.logits(L.x, L.Wr)
        assert np.all(np.abs(logits - g_ref) <= logit_tolerance(L.x, L.Wr)), "router logits"
        check_route_selection(counts, ids, g_ref, np.abs(logits - g_ref).max(axis=1), pf, rule)
        all_counts.append(counts)
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    s_ref, k_ref, hist_ref = oracle.ffn_sparsity(np.stack(all_counts), w.n_experts)
    a = to_host(acc)
    assert int(a[0]) == k_ref
    np.testing.assert_array_equal(a[1:], hist_ref)
    assert 1.0 - int(a[0]) / (T * n_layers * w.n_experts) == s_ref


@pytest.mark.parametrize("T,E,std", [(1, 16, 3.0), (37, 172, 3.0), (256, 64, 1.0), (257, 224, 4.0),
                                     (8192, 216, 3.0)])
def test_router_stats(pp, T, E, std):
    """L_ent, L_bal, L_gate against the oracle (fp32 softmax on the GPU)."""
    import torch
    logits = wl.host_logits(T, E, std=std, seed=T + E)
    desc = pp.make_desc(64, E, "bf16", "swiglu")
    ws = pp.alloc_workspace(desc, T)
    out = torch.zeros(3, dtype=torch.float64, device="cuda")
    for eps in (1e-9, 1e-2):
        pp.pp_router_stats(desc, dev(logits), T, eps, out, ws)
        torch.cuda.synchronize()
        assert pp.pp_get_device_status(ws) == pp.PP_OK
        ref = oracle.router_stats(logits.astype(np.float64), float(np.float32(eps)))
        np.testing.assert_allclose(to_host(out), ref, rtol=2e-5, atol=1e-9)
        again = torch.zeros_like(out)
        pp.pp_router_stats(desc, dev(logits), T, eps, again, ws)
        assert torch.equal(out, again)  # fixed reduction order


def test_router_stats_closed_forms(pp):
    import torch
    E = 64
    desc = pp.make_desc(64, E, "bf16", "swiglu")
    ws = pp.alloc_workspace(desc, E)
    out = torch.zeros(3, dtype=torch.float64, device="cuda")
    g = np.full((E, E), -1e4, np.float32)
    g[np.arange(E), np.arange(E)] = 1e4  # one expert per token, each expert once
    pp.pp_router_stats(desc, dev(g), E, 1e-9, out, ws)
    o = to_host(out)
    assert abs(o[1] - 1.0) < 1e-6 and abs(o[0]) < 1e-6 and abs(o[2] - 1.0 / E) < 1e-7
    g = np.zeros((E, E), np.float32)  # uniform routing
    pp.pp_router_stats(desc, dev(g), E, 1e-9, out, ws)
    o = to_host(out)
    assert abs(o[0] - np.log(E)) < 1e-5 and abs(o[1] - 1.0) < 1e-6 and abs(o[2] - 0.5) < 1e-7
    g[5, 7] = np.inf
    pp.pp_router_stats(desc, dev(g), E, 1e-9, out, ws)
    assert np.isnan(to_host(out)[0])
    assert pp.pp_get_device_status(ws) == pp.PP_ERR_NONFINITE


def test_bounded_wait_times_out(pp):
    """Failure detection: a wait on a flag nothing sets gives up and reports."""
    import torch
    desc = pp.make_desc(256, 16, "f32", "relu")
    ws = pp.alloc_workspace(desc, 1)
    pp.pp_debug_wait_timeout(ws, 2_000_000)
    assert pp.pp_get_device_status(ws) == pp.PP_ERR_TIMEOUT
    pp.pp_workspace_init(ws)
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    # the context is still usable
    layer_parity(pp, "tiny_relu_f32", 3, 0.5)


def test_graph_capture_matches_eager(pp):
    import torch
    w, L = layer_inputs("llama2_7b_decode", 1, d=1024, E=64)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    ws = pp.alloc_workspace(desc, 1)
    x, Wr, Wg, Wu, Wd = (dev(a) for a in (L.x, L.Wr, L.Wg, L.Wu, L.Wd))
    y0 = torch.empty_like(x)
    y1 = torch.empty_like(x)
    pp.pp_layer(desc, x, 1, Wr, Wg, Wu, Wd, 0.7, None, y0, ws)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            pp.pp_layer(desc, x, 1, Wr, Wg, Wu, Wd, 0.7, None, y1, ws, stream=s)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert torch.equal(y0, y1)
    assert pp.pp_get_device_status(ws) == pp.PP_OK


@pytest.mark.parametrize("T", [4, 64, 300])
def test_deterministic(pp, T):
    """Selection, logits and y are bitwise reproducible.  On the fused decode
    path (T <= 4) every reduction has a fixed order; on the grouped path each
    token's expert rows are summed in ascending expert order by the combine
    (its fp32 overflow reduction is used only past T * min(E, 64) assignment
    rows, which a top-p selection of these shapes never reaches)."""
    w, L = layer_inputs("llama3_8b_batched", T)
    a = run_layer(pp, w, L, 0.7)
    b = run_layer(pp, w, L, 0.7)
    assert int(a[0].sum()) < T * min(w.n_experts, 64)
    for u, v in zip(a[:4], b[:4]):
        assert np.array_equal(np.asarray(u), np.asarray(v))


@pytest.mark.parametrize("d,T", [(5120, 8), (8192, 5)])
def test_layer_f32_large_d(pp, d, T):
    """fp32 shapes whose x no longer fits 8 tokens per launch are sliced."""
    layer_parity(pp, "tiny_relu_f32", T, 0.7, d=d, E=16)


def test_workspace_reuse_across_calls(pp):
    """CTAs of the fused decode kernel hand logits and activations to each
    other through tagged words that stay in the workspace between calls.  A
    sequence of calls with changing token counts, p, entry points and a
    re-initialisation on ONE workspace must give exactly what each call gives
    on a fresh workspace (a stale word taken for current would change it)."""
    import torch
    w, L = layer_inputs("llama2_7b_decode", 4, d=1024, E=64)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    x, Wr, Wg, Wu, Wd = (dev(a) for a in (L.x, L.Wr, L.Wg, L.Wu, L.Wd))
    shared = pp.alloc_workspace(desc, 4)

    def call(kind, T, p, ws):
        sel = pp.Selection.empty(T, w.n_experts, "cuda")
        y = torch.zeros((T, w.d_model), dtype=x.dtype, device="cuda")
        if kind == "layer":
            pp.pp_layer(desc, x[:T], T, Wr, Wg, Wu, Wd, p, sel, y, ws)
        elif kind == "route":
            pp.pp_route(desc, x[:T], T, Wr, p, sel, ws)
        else:  # sparse FFN over the selection of the same tokens
            pp.pp_route(desc, x[:T], T, Wr, p, sel, ws)
            pp.pp_sparse_ffn(desc, x[:T], T, Wg, Wu, Wd, sel, y, ws)
        torch.cuda.synchronize()
        return to_host(sel.counts), to_host(sel.ids), to_host(y)

    seq = [("layer", 4, 0.9), ("layer", 1, 0.3), ("route", 2, 0.7), ("layer", 3, 1.0), ("ffn", 2, 0.5),
           ("layer", 1, 0.0), ("layer", 4, 0.7), ("init", 0, 0), ("layer", 2, 0.9), ("layer", 2, 0.9)]
    for kind, T, p in seq:
        if kind == "init":
            pp.pp_workspace_init(shared)
            continue
        pf = f32(p)
        got = call(kind, T, pf, shared)
        want = call(kind, T, pf, pp.alloc_workspace(desc, 4))
        for a, b in zip(got, want):
            assert np.array_equal(a, b), (kind, T, p)
        assert pp.pp_get_device_status(shared) == pp.PP_OK


def test_decode_timeline_entry_point(pp):
    """pp_debug_decode_timeline runs the timeline instantiation of the fused
    decode kernel: the same y as pp_layer, bitwise (the stamps only add
    stores), and for every CTA the recorded phase boundaries are ordered in
    time (entry, release, x loaded, router published, selection made)."""
    import torch
    w, L = layer_inputs("llama2_7b_decode", 1)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    ws = pp.alloc_workspace(desc, 1)
    args = [dev(a) for a in (L.x, L.Wr, L.Wg, L.Wu, L.Wd)]
    y_ref = torch.empty_like(args[0])
    pp.pp_layer(desc, args[0], 1, *args[1:], f32(0.7), None, y_ref, ws)
    stamps = torch.zeros(256 * 16, dtype=torch.int64, device="cuda")
    y = torch.empty_like(args[0])
    pp.pp_debug_decode_timeline(desc, args[0], *args[1:], f32(0.7), y, ws, stamps)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    assert torch.equal(y.view(torch.int16), y_ref.view(torch.int16))
    sm = torch.cuda.get_device_properties(0).multi_processor_count
    st = stamps.view(256, 16)[:sm].cpu().numpy()
    assert np.all(st[:, 0] > 0)  # every CTA stamped its entry
    for i in range(1, 5):  # entry <= released <= x <= router <= selected
        assert np.all(st[:, i] >= st[:, i - 1]), i
    # the timeline exists for one bf16 token only
    d32 = pp.make_desc(256, 16, "f32", "relu")
    with pytest.raises(pp.PPError) as ei:
        pp.pp_debug_decode_timeline(d32, args[0], *args[1:], 0.7, y, ws, stamps)
    assert ei.value.status == pp.PP_ERR_DTYPE
