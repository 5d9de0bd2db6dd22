"""GPU parity of the MoEfication repacking (Sec. 2.2, Eq. permuted_weights)
through the C ABI: pp_moefy_permute against the oracle's indexing
(W_gate[perm], W_up[perm], W_down[:, perm]), bit for bit, on random bit
patterns (the repacking is a copy, so every pattern -- NaN and Inf included --
must come through unchanged), at the workloads' shapes up to a full
Llama-2-7B-shaped layer and at ragged ones.  Then the whole preprocessing:
clustering (library, host) + repacking (library, GPU) + the sparse layer at
p >= 1 with unit gates reproduces the dense FFN of the original weights
(Eq. moefication_decomp)."""
import dataclasses

import numpy as np
import pytest

import oracle
from oracle import moefy
from paper_2605_28283_gb300 import workloads as wl
from parity import Y_TOL, rel_err_per_token, to_host

pytestmark = pytest.mark.gpu


def random_bits(rng, shape, dtype):
    if dtype == "bf16":
        return rng.integers(0, 1 << 16, size=shape, dtype=np.uint16)
    return rng.integers(0, 1 << 32, size=shape, dtype=np.uint32).view(np.float32)


def host_bits(t):
    import torch
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy().view(np.uint32)


def as_bits(a):
    return a.view(np.uint16) if a.dtype == np.uint16 else a.view(np.uint32)


def permute_gpu(pp, desc, perm, Wg, Wu, Wd):
    import torch
    dev = lambda a: None if a is None else wl.to_torch(a, "cuda")
    tg, tu, td = dev(Wg), dev(Wu), dev(Wd)
    outs = [None if tg is None else torch.empty_like(tg), torch.empty_like(tu), torch.empty_like(td)]
    ws = pp.alloc_workspace(desc, 0)
    pp.pp_moefy_permute(desc, dev(perm), tg, tu, td, *outs, ws)
    torch.cuda.synchronize()
    return outs, pp.pp_get_device_status(ws)


@pytest.mark.parametrize("dtype,act,d,E", [
    ("f32", "relu", 256, 16),        # tiny ReLU shape
    ("bf16", "gelu_tanh", 1024, 64),  # GPT-2-medium shape
    ("bf16", "swiglu", 4096, 172),   # Llama-2-7B shape, one full layer
    ("bf16", "swiglu", 72, 3),       # ragged: 9 16-byte chunks per row
    ("f32", "swiglu", 68, 5),        # ragged fp32
    ("bf16", "swiglu", 64, 1),       # one expert
])
def test_permute_bit_exact(pp, dtype, act, d, E):
    rng = np.random.default_rng(d * 7 + E)
    dff = 64 * E
    Wg = random_bits(rng, (dff, d), dtype) if act == "swiglu" else None
    Wu = random_bits(rng, (dff, d), dtype)
    Wd = random_bits(rng, (d, dff), dtype)
    perm = rng.permutation(dff).astype(np.int32)
    desc = pp.make_desc(d, E, dtype, act)
    (og, ou, od), status = permute_gpu(pp, desc, perm, Wg, Wu, Wd)
    assert status == pp.PP_OK
    rg, ru, rd = moefy.permuted_weights(Wg, Wu, Wd, perm)
    assert np.array_equal(host_bits(ou), as_bits(ru))
    assert np.array_equal(host_bits(od), as_bits(rd))
    if Wg is not None:
        assert np.array_equal(host_bits(og), as_bits(rg))


def test_permute_identity_and_reversal(pp):
    rng = np.random.default_rng(3)
    d, E = 128, 8
    Wg, Wu = random_bits(rng, (512, d), "bf16"), random_bits(rng, (512, d), "bf16")
    Wd = random_bits(rng, (d, 512), "bf16")
    desc = pp.make_desc(d, E, "bf16", "swiglu")
    (og, ou, od), status = permute_gpu(pp, desc, np.arange(512, dtype=np.int32), Wg, Wu, Wd)
    assert status == pp.PP_OK
    assert np.array_equal(host_bits(og), Wg) and np.array_equal(host_bits(ou), Wu)
    assert np.array_equal(host_bits(od), Wd)
    (og, ou, od), status = permute_gpu(pp, desc, np.arange(511, -1, -1, dtype=np.int32), Wg, Wu, Wd)
    assert status == pp.PP_OK
    assert np.array_equal(host_bits(ou), Wu[::-1]) and np.array_equal(host_bits(od), Wd[:, ::-1])


def test_permute_rejects_non_permutations(pp):
    """A repeated entry, or one outside [0, d_ff), is reported in the workspace
    status; out-of-range positions are written as zeros, the rest still
    follows perm."""
    rng = np.random.default_rng(4)
    d, E = 64, 2
    Wg, Wu = random_bits(rng, (128, d), "bf16"), random_bits(rng, (128, d), "bf16")
    Wd = random_bits(rng, (d, 128), "bf16")
    desc = pp.make_desc(d, E, "bf16", "swiglu")
    perm = np.arange(128, dtype=np.int32)
    perm[7] = 3  # 3 twice, 7 missing
    (og, ou, od), status = permute_gpu(pp, desc, perm, Wg, Wu, Wd)
    assert status == pp.PP_ERR_INVALID_ARG
    assert np.array_equal(host_bits(ou), Wu[perm])
    perm = np.arange(128, dtype=np.int32)
    perm[5], perm[9] = 128 + 7, -3
    (og, ou, od), status = permute_gpu(pp, desc, perm, Wg, Wu, Wd)
    assert status == pp.PP_ERR_INVALID_ARG
    hu, hd = host_bits(ou), host_bits(od)
    assert not hu[[5, 9]].any() and not hd[:, [5, 9]].any()
    keep = [j for j in range(128) if j not in (5, 9)]
    assert np.array_equal(hu[keep], Wu[keep]) and np.array_equal(hd[:, keep], Wd[:, keep])


@pytest.mark.parametrize("T", [3, 8])
def test_moefied_layer_reproduces_dense_ffn(pp, T):
    """Cluster (library, host), repack (library, GPU), then the layer with
    every expert active and unit gates equals the dense FFN of the original
    weights (oracle, fp64); the repacked weights equal the oracle's indexing."""
    import torch
    w = dataclasses.replace(wl.scaled(wl.WORKLOADS["llama2_7b_decode"], 1024, 24))
    L = wl.host_layer(w, T, seed=6)
    init = np.random.default_rng(6).choice(w.d_ff, size=w.n_experts, replace=False).astype(np.int32)
    desc = pp.make_desc(w.d_model, w.n_experts, "bf16", "swiglu", "none")
    perm, labels, iters, obj = pp.pp_moefy_cluster(desc, L.Wg, L.Wu, init, 30)
    assert sorted(perm.tolist()) == list(range(w.d_ff)) and iters >= 2
    (og, ou, od), status = permute_gpu(pp, desc, perm, L.Wg, L.Wu, L.Wd)
    assert status == pp.PP_OK
    rg, ru, rd = moefy.permuted_weights(L.Wg, L.Wu, L.Wd, perm)
    assert np.array_equal(host_bits(og), rg) and np.array_equal(host_bits(ou), ru)
    assert np.array_equal(host_bits(od), rd)
    x = wl.to_torch(L.x, "cuda")
    y = torch.empty_like(x)
    ws = pp.alloc_workspace(desc, T)
    pp.pp_layer(desc, x, T, wl.to_torch(L.Wr, "cuda"), og, ou, od, 1.0, None, y, ws)
    torch.cuda.synchronize()
    assert pp.pp_get_device_status(ws) == pp.PP_OK
    ref = oracle.dense_ffn(L.x, L.Wg, L.Wu, L.Wd, "swiglu")
    assert rel_err_per_token(to_host(y), ref).max() <= Y_TOL["bf16"]
