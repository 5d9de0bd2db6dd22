"""MoEfication clustering (Sec. 2.2) through the C ABI against the oracle.

pp_moefy_cluster is the library's offline host routine (balanced k-means
over the neurons' input weights, exact equal-size assignment by successive
shortest paths); it touches no GPU, so these tests run on the CPU.  The
oracle solves each assignment with scipy's linear assignment over d_ff slots
instead: the two share nothing but the seeded inputs.  On random weights the
least-cost assignment is unique, so labels, permutation and iteration count
must be equal, and the objective equal to rounding (fp64 sums in different
orders).
"""
import ctypes
import dataclasses

import numpy as np
import pytest

from oracle import moefy
from paper_2605_28283_gb300 import binding as pp
from paper_2605_28283_gb300 import build as ppbuild
from paper_2605_28283_gb300 import workloads as wl


@pytest.fixture(scope="module")
def lib():
    ppbuild.build()
    return pp.load()


def case(dtype, act, d, E, seed=0):
    w = dataclasses.replace(wl.scaled(wl.WORKLOADS["tiny_relu_f32"], d, E), dtype=dtype, act=act)
    L = wl.host_layer(w, 1, seed=seed)
    init = np.random.default_rng(seed + 100).choice(w.d_ff, size=E, replace=False).astype(np.int32)
    return w, L, init


@pytest.mark.parametrize("dtype,act,d,E,max_iter", [
    ("f32", "swiglu", 64, 4, 100),
    ("bf16", "swiglu", 64, 8, 100),
    ("f32", "relu", 64, 4, 100),
    ("bf16", "gelu_tanh", 128, 6, 100),
    ("bf16", "swiglu", 64, 16, 100),
    ("f32", "swiglu", 64, 8, 1),
    ("f32", "swiglu", 64, 8, 3),
    ("bf16", "swiglu", 64, 1, 10),
])
def test_cluster_matches_oracle(lib, dtype, act, d, E, max_iter):
    w, L, init = case(dtype, act, d, E, seed=d + E + max_iter)
    desc = pp.make_desc(w.d_model, E, dtype, act)
    perm, labels, iters, obj = pp.pp_moefy_cluster(desc, L.Wg, L.Wu, init, max_iter)
    F = moefy.features(L.Wu, L.Wg)
    a_ref, it_ref, obj_ref, _ = moefy.balanced_kmeans(F, E, init, max_iter)
    assert iters == it_ref
    assert np.array_equal(labels, a_ref)
    assert np.array_equal(perm, moefy.permutation(a_ref, E))
    assert abs(obj - obj_ref) <= 1e-9 * obj_ref
    assert np.array_equal(np.bincount(labels, minlength=E), np.full(E, 64))


def test_planted_clusters_recovered(lib):
    """E groups of 64 neurons around far-apart centres, shuffled: the library
    finds exactly the groups (cluster h = the group of neuron init[h])."""
    rng = np.random.default_rng(8)
    E, d = 12, 64
    centres = rng.normal(size=(E, 2 * d)) * 0.5
    group = np.repeat(np.arange(E), 64)
    feats = (centres[group] + 0.01 * rng.normal(size=(E * 64, 2 * d))).astype(np.float32)
    shuffle = rng.permutation(E * 64)
    feats, group = feats[shuffle], group[shuffle]
    Wg, Wu = np.ascontiguousarray(feats[:, :d]), np.ascontiguousarray(feats[:, d:])
    init = np.array([np.flatnonzero(group == h)[5] for h in range(E)], np.int32)
    desc = pp.make_desc(d, E, "f32", "swiglu")
    perm, labels, iters, obj = pp.pp_moefy_cluster(desc, Wg, Wu, init, 50)
    assert np.array_equal(labels, group)
    for e in range(E):
        assert sorted(perm[e * 64:(e + 1) * 64].tolist()) == np.flatnonzero(group == e).tolist()
    assert iters == 2


def test_one_neuron_cluster_start_is_stable(lib):
    """Identical neurons within each planted block and inits on distinct
    blocks: zero objective after the first update."""
    E, d = 4, 64
    rng = np.random.default_rng(1)
    base = rng.normal(size=(E, d)).astype(np.float32)
    Wu = np.ascontiguousarray(np.repeat(base, 64, axis=0))
    init = np.array([0, 64, 128, 192], np.int32)
    desc = pp.make_desc(d, E, "f32", "relu")
    perm, labels, iters, obj = pp.pp_moefy_cluster(desc, None, Wu, init, 10)
    assert np.array_equal(labels, np.repeat(np.arange(E), 64)) and obj == 0.0
    assert np.array_equal(perm, np.arange(E * 64))


def test_argument_errors(lib):
    w, L, init = case("f32", "swiglu", 64, 4)
    desc = pp.make_desc(64, 4, "f32", "swiglu")
    call = lambda **kw: _raw_cluster(lib, kw.pop("desc", desc), kw.pop("Wg", L.Wg), kw.pop("Wu", L.Wu),
                                     kw.pop("init", init), kw.pop("max_iter", 10))
    assert call() == pp.PP_OK
    assert call(init=np.array([0, 1, 2, 2], np.int32)) == pp.PP_ERR_INVALID_ARG   # repeated
    assert call(init=np.array([0, 1, 2, 256], np.int32)) == pp.PP_ERR_INVALID_ARG  # out of range
    assert call(init=np.array([-1, 1, 2, 3], np.int32)) == pp.PP_ERR_INVALID_ARG
    assert call(max_iter=0) == pp.PP_ERR_INVALID_ARG
    assert call(Wg=None) == pp.PP_ERR_INVALID_ARG                                  # SwiGLU needs W_gate
    assert call(desc=pp.make_desc(64, 4, "f32", "swiglu", d_expert=32)) == pp.PP_ERR_SHAPE
    assert call(desc=pp.make_desc(60, 4, "f32", "swiglu")) == pp.PP_ERR_SHAPE


def _raw_cluster(lib, desc, Wg, Wu, init, max_iter):
    perm = np.empty(desc.d_ff, np.int32)
    h = lambda a: None if a is None else a.ctypes.data_as(ctypes.c_void_p)
    return lib.pp_moefy_cluster(ctypes.byref(desc), h(Wg), h(Wu), h(np.ascontiguousarray(init, np.int32)),
                                int(max_iter), h(perm), None, None, None)


def test_permute_argument_errors_on_the_host(lib):
    """pp_moefy_permute rejects bad arguments before any CUDA call (fake,
    never dereferenced device addresses)."""
    desc = pp.make_desc(256, 4, "bf16", "swiglu")
    mat = 256 * 256 * 2
    A = 1 << 32
    base = dict(perm=A, Wg=A + 1 * mat, Wu=A + 2 * mat, Wd=A + 3 * mat, og=A + 4 * mat, ou=A + 5 * mat,
                od=A + 6 * mat, ws=A + 8 * mat, ws_bytes=1 << 20)

    def call(d=desc, **kw):
        a = dict(base, **kw)
        v = lambda x: None if x is None else ctypes.c_void_p(x)
        return lib.pp_moefy_permute(ctypes.byref(d), v(a["perm"]), v(a["Wg"]), v(a["Wu"]), v(a["Wd"]), v(a["og"]),
                                    v(a["ou"]), v(a["od"]), v(a["ws"]), a["ws_bytes"], None)

    assert call() in (pp.PP_ERR_CUDA, pp.PP_ERR_UNSUPPORTED)       # valid: stops at the device check
    assert call(perm=None) == pp.PP_ERR_INVALID_ARG
    assert call(og=None) == pp.PP_ERR_INVALID_ARG                 # SwiGLU needs W_gate_out
    assert call(Wg=None) == pp.PP_ERR_INVALID_ARG
    assert call(ou=A + 2 * mat + 512) == pp.PP_ERR_INVALID_ARG    # output overlaps W_up
    assert call(od=A + 5 * mat + 4096) == pp.PP_ERR_INVALID_ARG   # outputs overlap each other
    assert call(ou=A) == pp.PP_ERR_INVALID_ARG                    # output overlaps perm
    assert call(od=A + 6 * mat + 8) == pp.PP_ERR_ALIGN
    assert call(ws_bytes=64) == pp.PP_ERR_WORKSPACE
    assert call(d=pp.make_desc(256, 4, "bf16", "swiglu", d_expert=16)) == pp.PP_ERR_SHAPE
    relu = pp.make_desc(256, 4, "bf16", "relu")
    assert call(d=relu, Wg=None, og=None) in (pp.PP_ERR_CUDA, pp.PP_ERR_UNSUPPORTED)


# ------------------------------------------------ full-size optimality check
def no_improving_exchange(D, labels, k, tol=1e-9):
    """An equal-size assignment is optimal iff no cyclic exchange of neurons
    between clusters lowers the cost, i.e. the graph on the clusters with
    edge h -> h' = min over members j of h of D[j, h'] - D[j, h] has no
    negative cycle (min-plus closure, Floyd-Warshall)."""
    W = np.full((k, k), np.inf)
    for h in range(k):
        m = np.flatnonzero(labels == h)
        W[h] = (D[m] - D[m, h][:, None]).min(axis=0)
    np.fill_diagonal(W, 0.0)
    for m in range(k):
        W = np.minimum(W, W[:, m:m + 1] + W[m:m + 1, :])
    return float(np.diag(W).min()) >= -tol


def sq_dist(F32, C):
    """||f - c||^2 for all pairs, fp64, in row blocks."""
    out = np.empty((F32.shape[0], C.shape[0]))
    cn = (C * C).sum(axis=1)
    for i in range(0, F32.shape[0], 2048):
        f = F32[i:i + 2048].astype(np.float64)
        out[i:i + 2048] = (f * f).sum(axis=1)[:, None] - 2.0 * f @ C.T + cn[None, :]
    return out


@pytest.mark.parametrize("name", ["gpt2m_gelu_bf16", "llama2_7b_decode"])
def test_full_size_assignments_are_optimal(lib, name):
    """At the full layer shapes: the first assignment is optimal for the
    initial centroids, and the converged labels are optimal for their own
    cluster means (the fixed point of the iteration)."""
    w = wl.WORKLOADS[name]
    rng = np.random.default_rng(17)
    mk = lambda: wl.f32_to_bf16_bits(rng.standard_normal((w.d_ff, w.d_model), dtype=np.float32) * np.float32(0.02))
    Wg = mk() if w.gated else None
    Wu = mk()
    init = rng.choice(w.d_ff, size=w.n_experts, replace=False).astype(np.int32)
    desc = pp.make_desc(w.d_model, w.n_experts, "bf16", w.act)
    F32 = wl.bf16_bits_to_f32(Wu) if Wg is None else np.concatenate(
        [wl.bf16_bits_to_f32(Wg), wl.bf16_bits_to_f32(Wu)], axis=1)
    k = w.n_experts
    # one assignment from the initial centroids
    perm1, lab1, it1, obj1 = pp.pp_moefy_cluster(desc, Wg, Wu, init, 1)
    assert it1 == 1 and np.array_equal(np.bincount(lab1, minlength=k), np.full(k, 64))
    D1 = sq_dist(F32, F32[init].astype(np.float64))
    assert no_improving_exchange(D1, lab1, k)
    assert abs(D1[np.arange(w.d_ff), lab1].sum() - obj1) <= 1e-9 * obj1
    # the check has teeth: swapping two neurons of different clusters leaves
    # an improving exchange (the swap back)
    i, j = 0, int(np.flatnonzero(lab1 != lab1[0])[0])
    bad = lab1.copy()
    bad[i], bad[j] = lab1[j], lab1[i]
    assert not no_improving_exchange(D1, bad, k)
    # the fixed point
    perm, lab, it, obj = pp.pp_moefy_cluster(desc, Wg, Wu, init, 20)
    assert 2 <= it < 20
    C = np.stack([F32[lab == h].astype(np.float64).mean(axis=0) for h in range(k)])
    D = sq_dist(F32, C)
    assert no_improving_exchange(D, lab, k)
    assert abs(D[np.arange(w.d_ff), lab].sum() - obj) <= 1e-9 * obj
