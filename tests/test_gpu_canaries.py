"""Guard bands around every output (a stand-in for a memory sanitizer, which
this GPU pool does not offer): each output tensor is the middle of a larger
allocation whose 512-byte bands before and after it hold a sentinel byte.
A call must leave the bands untouched, and the interior must equal what the
same call writes into a plain allocation (the library is deterministic).
Covered: the fused decode path (T <= 4), the grouped tensor-core path
(T >= 5, including ragged token counts), the fp32 path in 8-token slices,
the chained step, pp_route, and the MoEfication repacking."""
import dataclasses

import numpy as np
import pytest

from paper_2605_28283_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

GUARD = 512       # bytes on each side; keeps the interior 16-byte aligned
SENTINEL = 0xA5


class Guarded:
    """A device tensor of `shape` inside sentinel bands."""

    def __init__(self, shape, dtype, device="cuda"):
        import torch
        self.esz = torch.empty((), dtype=dtype).element_size()
        self.n = int(np.prod(shape))
        self.g = GUARD // self.esz
        self.buf = torch.empty(self.n + 2 * self.g, dtype=dtype, device=device)
        self.buf.view(torch.uint8).fill_(SENTINEL)
        self.t = self.buf[self.g:self.g + self.n].view(shape)

    def bands_intact(self):
        b = self.buf.view(dtype=__import__("torch").uint8)
        lo, hi = b[:GUARD], b[(self.g + self.n) * self.esz:]
        return bool((lo == SENTINEL).all()) and bool((hi == SENTINEL).all()) and hi.numel() == GUARD


def bitwise_equal(a, b):
    import torch
    if a.dtype == torch.bfloat16:
        return torch.equal(a.view(torch.int16), b.view(torch.int16))
    if a.dtype == torch.float32:
        return torch.equal(a.view(torch.int32), b.view(torch.int32))
    return torch.equal(a, b)


def test_guard_helper_on_host():
    """The helper itself: bands start intact and a write next to the
    interior is seen (host tensors)."""
    import torch
    g = Guarded((3, 5), torch.bfloat16, device="cpu")
    assert g.bands_intact() and g.t.data_ptr() - g.buf.data_ptr() == GUARD
    g.t.zero_()
    assert g.bands_intact()
    g.buf[g.g + g.n] = 1.0
    assert not g.bands_intact()


def layer_case(name, T, d=None, E=None):
    w = wl.WORKLOADS[name]
    if d is not None:
        w = wl.scaled(w, d, E)
    return w, wl.host_layer(w, T, seed=T, layer=1)


def run_guarded_layer(pp, w, L, T, p, rule="min_prefix"):
    import torch
    dev = lambda a: None if a is None else wl.to_torch(a, "cuda")
    x, Wr, Wg, Wu, Wd = dev(L.x), dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act, "sigmoid", rule)
    E = w.n_experts
    outs = {}
    for guarded in (False, True):
        ws = pp.alloc_workspace(desc, T)
        if guarded:
            gy = Guarded((T, w.d_model), x.dtype)
            gids, gcnt = Guarded((T, E), torch.int32), Guarded((T,), torch.int32)
            ggat, glog = Guarded((T, E), torch.float32), Guarded((T, E), torch.float32)
            y = gy.t
            sel = pp.Selection(gids.t, gcnt.t, ggat.t, glog.t)
        else:
            y = torch.empty((T, w.d_model), dtype=x.dtype, device="cuda")
            sel = pp.Selection.empty(T, E, "cuda")
        pp.pp_layer(desc, x, T, Wr, Wg, Wu, Wd, p, sel, y, ws)
        torch.cuda.synchronize()
        assert pp.pp_get_device_status(ws) == pp.PP_OK
        outs[guarded] = (y, sel)
        if guarded:
            for g, what in ((gy, "y"), (gids, "ids"), (gcnt, "counts"), (ggat, "gates"), (glog, "logits")):
                assert g.bands_intact(), "a write outside %s" % what
    (y0, s0), (y1, s1) = outs[False], outs[True]
    assert bitwise_equal(y0, y1)
    for a, b in ((s0.ids, s1.ids), (s0.counts, s1.counts), (s0.gates, s1.gates), (s0.logits, s1.logits)):
        assert bitwise_equal(a, b)


@pytest.mark.parametrize("T", [1, 3, 4, 5, 8, 37, 64, 130])
def test_layer_bf16_outputs_stay_in_bounds(pp, T):
    w, L = layer_case("llama2_7b_decode", T, 1024, 48)
    run_guarded_layer(pp, w, L, T, float(np.float32(0.7)))


@pytest.mark.parametrize("rule,p", [("topk", 3.0), ("lte", 0.9), ("paper", 0.5)])
def test_layer_rules_outputs_stay_in_bounds(pp, rule, p):
    for T in (2, 9):
        w, L = layer_case("gpt2m_gelu_bf16", T, 512, 24)
        run_guarded_layer(pp, w, L, T, float(np.float32(p)), rule)


@pytest.mark.parametrize("T", [1, 7, 13])
def test_layer_f32_outputs_stay_in_bounds(pp, T):
    w, L = layer_case("tiny_relu_f32", T)
    run_guarded_layer(pp, w, L, T, float(np.float32(0.9)))


def test_route_outputs_stay_in_bounds(pp):
    import torch
    T = 3
    w, L = layer_case("llama2_7b_decode", T, 1024, 48)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    E = w.n_experts
    gids, gcnt = Guarded((T, E), torch.int32), Guarded((T,), torch.int32)
    ggat, glog = Guarded((T, E), torch.float32), Guarded((T, E), torch.float32)
    ws = pp.alloc_workspace(desc, T)
    pp.pp_route(desc, wl.to_torch(L.x, "cuda"), T, wl.to_torch(L.Wr, "cuda"), float(np.float32(0.7)),
                pp.Selection(gids.t, gcnt.t, ggat.t, glog.t), ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    assert all(g.bands_intact() for g in (gids, gcnt, ggat, glog))


@pytest.mark.parametrize("T", [2, 6])
def test_chained_outputs_stay_in_bounds(pp, T):
    import torch
    w, L = layer_case("llama2_7b_decode", T, 1024, 48)
    dev = lambda a: None if a is None else wl.to_torch(a, "cuda")
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    xp = dev(L.x)
    yp = dev(wl.host_tokens(w, T, 9, 1))
    gx, gy = Guarded((T, w.d_model), xp.dtype), Guarded((T, w.d_model), xp.dtype)
    ws = pp.alloc_workspace(desc, T)
    pp.pp_layer_chained(desc, xp, yp, None, 1e-6, T, dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd),
                        float(np.float32(0.7)), None, gx.t, gy.t, ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    assert gx.bands_intact() and gy.bands_intact()


@pytest.mark.parametrize("dtype,act,d,E", [("bf16", "swiglu", 1024, 48), ("f32", "relu", 68, 5)])
def test_moefy_permute_outputs_stay_in_bounds(pp, dtype, act, d, E):
    import torch
    w = dataclasses.replace(wl.scaled(wl.WORKLOADS["tiny_relu_f32"], d, E), dtype=dtype, act=act)
    L = wl.host_layer(w, 1, seed=2)
    dev = lambda a: None if a is None else wl.to_torch(a, "cuda")
    tg, tu, td = dev(L.Wg), dev(L.Wu), dev(L.Wd)
    perm = dev(np.random.default_rng(5).permutation(w.d_ff).astype(np.int32))
    gg = None if tg is None else Guarded(tuple(tg.shape), tg.dtype)
    gu, gd = Guarded(tuple(tu.shape), tu.dtype), Guarded(tuple(td.shape), td.dtype)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    ws = pp.alloc_workspace(desc, 0)
    pp.pp_moefy_permute(desc, perm, tg, tu, td, None if gg is None else gg.t, gu.t, gd.t, ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    assert gu.bands_intact() and gd.bands_intact() and (gg is None or gg.bands_intact())
    pl = perm.long()
    assert bitwise_equal(gu.t, tu[pl]) and bitwise_equal(gd.t, td[:, pl])
