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
