"""Pins for the MoEfication oracle (Sec. 2.2: balanced k-means over the
intermediate neurons, the permutation Pi and Eq. permuted_weights).

Each check ties the oracle to something other than itself:
* brute force: every labelling of a few neurons with exactly d_ff / E per
  cluster is enumerated, for the assignment step and for the fixed point the
  iteration stops at (its labels are optimal for their own cluster means);
* planted clusters: E well-separated groups are recovered exactly;
* properties of the method: in one dimension the converged clusters are
  intervals of the sorted values (an optimal equal-size assignment to sorted
  centroids is monotone), the objective never increases, k = 1 and
  one-neuron clusters reduce to the identity;
* Eq. (moefication_decomp): the dense FFN of the permuted weights equals the
  dense FFN of the original ones (Pi Pi^T = I), checked with the C oracle's
  dense FFN;
* hand cases of the feature layout and of the block order of Pi.

``PINS`` also runs against broken copies of the oracle
(test_planted_mistakes_are_caught): each plausible mistake fails a pin.
"""
import dataclasses

import numpy as np
import pytest

import oracle
from oracle import moefy
from paper_2605_28283_gb300 import workloads as wl


# ------------------------------------------------------------- references
def brute_balanced(D, cap):
    """Least sum_n D[n, a[n]] over all labellings with exactly cap neurons per
    cluster, by enumeration."""
    n, k = D.shape
    best = [np.inf]
    counts = [0] * k

    def rec(i, cost):
        if cost >= best[0]:
            return
        if i == n:
            best[0] = cost
            return
        for h in range(k):
            if counts[h] < cap:
                counts[h] += 1
                rec(i + 1, cost + D[i, h])
                counts[h] -= 1

    rec(0, 0.0)
    return best[0]


def cost_of(F, C, a):
    """sum_n ||F[n] - C[a[n]]||^2 written directly."""
    return float(sum(((F[n] - C[a[n]]) ** 2).sum() for n in range(len(a))))


def member_means(F, a, k):
    return np.stack([F[np.asarray(a) == h].mean(axis=0) for h in range(k)])


# ------------------------------------------------------------------- pins
def pin_assign_bruteforce(m):
    """Step 2a against enumeration of every balanced labelling."""
    rng = np.random.default_rng(11)
    for n, k in [(4, 2), (6, 2), (6, 3), (8, 4), (9, 3), (8, 2)]:
        cap = n // k
        for _ in range(3):
            D = rng.uniform(0.0, 10.0, (n, k))
            a = np.asarray(m.balanced_assign(D, cap))
            assert a.shape == (n,)
            assert np.array_equal(np.bincount(a, minlength=k), np.full(k, cap)), "not balanced"
            got = float(D[np.arange(n), a].sum())
            assert abs(got - brute_balanced(D, cap)) <= 1e-9, (n, k, got)


def pin_fixed_point(m):
    """Where the iteration stops, its labels are a least-cost balanced
    labelling for their own cluster means, and the reported objective is that
    cost."""
    rng = np.random.default_rng(5)
    for n, k, f in [(8, 2, 3), (9, 3, 2), (8, 4, 3), (6, 2, 5)]:
        for s in range(3):
            F = rng.normal(size=(n, f))
            init = rng.choice(n, size=k, replace=False)
            a, it, obj, hist = m.balanced_kmeans(F, k, init, 100)
            a = np.asarray(a)
            assert 2 <= it < 100 and len(hist) == it, (it, len(hist))
            C = member_means(F, a, k)
            D = np.array([[((F[i] - C[h]) ** 2).sum() for h in range(k)] for i in range(n)])
            best = brute_balanced(D, n // k)
            assert abs(cost_of(F, C, a) - best) <= 1e-9
            assert abs(obj - best) <= 1e-9 * max(1.0, best)


def pin_planted_clusters(m):
    """E groups of 64 neurons around far-apart centres are recovered exactly."""
    rng = np.random.default_rng(7)
    k, cap, f = 4, 64, 16
    centres = rng.normal(size=(k, f)) * 10.0
    group = np.repeat(np.arange(k), cap)
    F = centres[group] + 0.1 * rng.normal(size=(k * cap, f))
    shuffle = rng.permutation(k * cap)
    F, group = F[shuffle], group[shuffle]
    init = np.array([np.flatnonzero(group == h)[0] for h in range(k)])
    a, it, obj, _ = m.balanced_kmeans(F, k, init, 50)
    assert np.array_equal(np.asarray(a), group)
    # a different starting member of each group gives the same partition
    init2 = np.array([np.flatnonzero(group == h)[-1] for h in range(k)])
    assert np.array_equal(np.asarray(m.balanced_kmeans(F, k, init2, 50)[0]), group)


def pin_one_dimension_intervals(m):
    """In one dimension the converged clusters are intervals of the sorted
    values (exchange argument for equal sizes and squared distances)."""
    rng = np.random.default_rng(3)
    for n, k in [(40, 4), (60, 6), (24, 3)]:
        F = rng.normal(size=(n, 1))
        init = rng.choice(n, size=k, replace=False)
        a = np.asarray(m.balanced_kmeans(F, k, init, 200)[0])
        seq = a[np.argsort(F[:, 0], kind="stable")]
        changes = int((seq[1:] != seq[:-1]).sum())
        assert changes == k - 1, seq
        assert np.array_equal(np.bincount(a, minlength=k), np.full(k, n // k))


def pin_objective_non_increasing(m):
    """Neither step can raise sum ||f - c||^2."""
    rng = np.random.default_rng(9)
    F = rng.normal(size=(128, 8))
    init = rng.choice(128, size=4, replace=False)
    a, it, obj, hist = m.balanced_kmeans(F, 4, init, 100)
    assert all(hist[i + 1] <= hist[i] + 1e-9 for i in range(len(hist) - 1)), hist
    assert it >= 2


def pin_special_cases(m):
    rng = np.random.default_rng(2)
    F = rng.normal(size=(12, 3))
    # one cluster: everything in it, identity permutation
    a, it, obj, _ = m.balanced_kmeans(F, 1, [5], 10)
    assert np.array_equal(np.asarray(a), np.zeros(12, np.int32)) and it == 2
    assert np.array_equal(np.asarray(m.permutation(a, 1)), np.arange(12))
    # one neuron per cluster, started on the neurons themselves: neuron
    # init[h] stays in cluster h with zero cost
    init = rng.permutation(12)
    a, it, obj, _ = m.balanced_kmeans(F, 12, init, 10)
    a = np.asarray(a)
    assert np.array_equal(a[init], np.arange(12)) and obj == 0.0 and it == 2
    assert np.array_equal(np.asarray(m.permutation(a, 12)), init)


def pin_permutation_hand(m):
    """Hand case: labels (1, 0, 1, 0, 2, 2) -> expert 0 = neurons 1, 3;
    expert 1 = neurons 0, 2; expert 2 = neurons 4, 5."""
    assert np.asarray(m.permutation(np.array([1, 0, 1, 0, 2, 2]), 3)).tolist() == [1, 3, 0, 2, 4, 5]
    assert np.asarray(m.permutation(np.array([2, 2, 1, 1, 0, 0]), 3)).tolist() == [4, 5, 2, 3, 0, 1]


def pin_features_hand(m):
    """Hand case: a gated neuron's feature is (gate row, up row), widened exactly."""
    Wg = np.array([[1.0, 2.0], [3.0, 4.0]], np.float32)
    Wu = np.array([[5.0, 6.0], [7.0, 8.0]], np.float32)
    assert np.asarray(m.features(Wu, Wg)).tolist() == [[1, 2, 5, 6], [3, 4, 7, 8]]
    assert np.asarray(m.features(Wu)).tolist() == [[5, 6], [7, 8]]
    # bf16 bit patterns: 0x3FC0 = 1.5, 0xC020 = -2.5, 0x3F81 = 1 + 2^-7
    bits = np.array([[0x3FC0, 0xC020, 0x3F81]], np.uint16)
    assert np.asarray(m.features(bits)).tolist() == [[1.5, -2.5, 1.0 + 2.0 ** -7]]


def pin_moefication_identity(m):
    """Eq. (moefication_decomp): the permuted weights give the same dense FFN
    (C oracle, fp64); at p >= 1 with unit gates the MoEfied layer is that FFN."""
    for dtype, kind in [("f32", "swiglu"), ("bf16", "swiglu"), ("f32", "relu")]:
        w = dataclasses.replace(wl.scaled(wl.WORKLOADS["tiny_relu_f32"], 32, 4), dtype=dtype, act=kind)
        L = wl.host_layer(w, 3, seed=21)
        init = np.random.default_rng(4).choice(w.n_experts * 64, size=w.n_experts, replace=False)
        perm, a, it, obj, Wg2, Wu2, Wd2 = m.moefy(L.Wg, L.Wu, L.Wd, w.n_experts, init, 50)
        perm = np.asarray(perm)
        assert sorted(perm.tolist()) == list(range(w.n_experts * 64))
        for e in range(w.n_experts):
            assert set(perm[e * 64:(e + 1) * 64].tolist()) == set(np.flatnonzero(np.asarray(a) == e).tolist())
        ref = oracle.dense_ffn(L.x, L.Wg, L.Wu, L.Wd, kind)
        np.testing.assert_allclose(oracle.dense_ffn(L.x, Wg2, Wu2, Wd2, kind), ref, rtol=1e-11, atol=1e-13)
        g, counts, ids, y = oracle.layer(L.x, L.Wr, Wg2, Wu2, Wd2, 1.0, kind, "none")
        np.testing.assert_allclose(y, ref, rtol=1e-11, atol=1e-13)
        # neuron j of the new layout is neuron perm[j] of the old one
        j = 77
        assert np.array_equal(Wu2[j], L.Wu[perm[j]]) and np.array_equal(Wd2[:, j], L.Wd[:, perm[j]])


PINS = [pin_assign_bruteforce, pin_fixed_point, pin_planted_clusters, pin_one_dimension_intervals,
        pin_objective_non_increasing, pin_special_cases, pin_permutation_hand, pin_features_hand,
        pin_moefication_identity]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(ppo, pin):
    pin(moefy)


# ----------------------------------------------------- planted mistakes (CPU)
_orig = {name: getattr(moefy, name) for name in
         ("balanced_assign", "update_centroids", "sq_distances", "permutation", "permuted_weights", "features",
          "balanced_kmeans")}


def _assign_slot_mod(D, cap):
    from scipy.optimize import linear_sum_assignment
    n, k = D.shape
    rows, cols = linear_sum_assignment(np.repeat(D, cap, axis=1))
    a = np.empty(n, np.int32)
    a[rows] = cols % k
    return a


def _update_first_member(F, a, k):
    return np.stack([F[np.asarray(a) == h][0] for h in range(k)])


def _update_sum(F, a, k):
    return np.stack([F[np.asarray(a) == h].sum(axis=0) for h in range(k)])


def _l1_distances(F, C):
    return np.stack([np.abs(F - C[h]).sum(axis=1) for h in range(C.shape[0])], axis=1)


def _perm_descending(a, k):
    a = np.asarray(a)
    return np.concatenate([np.flatnonzero(a == h)[::-1] for h in range(k)]).astype(np.int32)


def _perm_clusters_reversed(a, k):
    a = np.asarray(a)
    return np.concatenate([np.flatnonzero(a == h) for h in range(k - 1, -1, -1)]).astype(np.int32)


def _down_rows(Wg, Wu, Wd, perm):
    return (None if Wg is None else Wg[perm], Wu[perm], np.ascontiguousarray(Wd[perm % Wd.shape[0]]))


def _down_unpermuted(Wg, Wu, Wd, perm):
    return (None if Wg is None else Wg[perm], Wu[perm], Wd)


def _features_up_first(Wu, Wg=None):
    up = moefy.widen(Wu)
    return up if Wg is None else np.concatenate([up, moefy.widen(Wg)], axis=1)


def _stop_after_first(F, k, init, max_iter=100):
    return _orig["balanced_kmeans"](F, k, init, 1)


MUTANTS = {
    "assign_unbalanced_argmin": ("balanced_assign", lambda D, cap: D.argmin(axis=1).astype(np.int32)),
    "assign_maximises": ("balanced_assign", lambda D, cap: _orig["balanced_assign"](-D, cap)),
    "assign_slot_to_cluster_mod": ("balanced_assign", _assign_slot_mod),
    "update_first_member": ("update_centroids", _update_first_member),
    "update_sum_not_mean": ("update_centroids", _update_sum),
    "distance_l1": ("sq_distances", _l1_distances),
    "perm_descending_within_expert": ("permutation", _perm_descending),
    "perm_experts_reversed": ("permutation", _perm_clusters_reversed),
    "down_rows_not_columns": ("permuted_weights", _down_rows),
    "down_not_permuted": ("permuted_weights", _down_unpermuted),
    "features_up_before_gate": ("features", _features_up_first),
    "stops_after_first_assignment": ("balanced_kmeans", _stop_after_first),
}


def test_planted_mistakes_are_caught(ppo):
    escaped = []
    try:
        for name, (attr, bad) in MUTANTS.items():
            setattr(moefy, attr, bad)
            caught = False
            for pin in PINS:
                try:
                    pin(moefy)
                except Exception:
                    caught = True
                    break
            setattr(moefy, attr, _orig[attr])
            if not caught:
                escaped.append(name)
    finally:
        for attr, fn in _orig.items():
            setattr(moefy, attr, fn)
    assert not escaped, "planted mistakes not caught by any pin: %s" % escaped
