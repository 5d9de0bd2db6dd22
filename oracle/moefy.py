"""MoEfication preprocessing (Sec. 2.2) -- CPU oracle, TEST INFRASTRUCTURE.

Not product code: only ``tests/`` may import this module.  It shares no code
with the CUDA library and never imports it.  Plain numpy in fp64; the exact
balanced assignment of each iteration is one library call
(``scipy.optimize.linear_sum_assignment``), the only step that is not
written out here.

What it computes, in the order of Sec. 2.2:
  1. the feature vector of each intermediate neuron n: its input weights,
     row n of W_up, preceded by row n of W_gate for a gated FFN (the weights
     that make h_n), widened exactly to fp64;                    features()
  2. balanced k-means (constrained k-means of Bradley, Bennett and Demiriz,
     2000, with every one of the E clusters holding exactly d_ff / E
     neurons, so that each becomes one expert of d_e neurons).  Starting from
     the features of E given neurons as centroids, repeat
       a. cluster assignment: among the assignments that put exactly d_ff / E
          neurons in every cluster, one with the least
          sum_n ||f_n - c_{a(n)}||^2                         balanced_assign()
       b. cluster update: c_h = mean of the features assigned to h
                                                            update_centroids()
     until an assignment equals the previous one (the centroids are then
     fixed) or max_iter assignments have been made;        balanced_kmeans()
  3. the permutation Pi that makes each cluster a contiguous block: new
     position j holds old neuron perm[j], neurons ordered by (cluster, old
     index);                                                   permutation()
  4. Eq. (permuted_weights): W~_gate = W_gate Pi, W~_up = W_up Pi,
     W~_down = Pi^T W_down.  With neurons stored as rows of W_gate / W_up
     ([d_ff][d]) and as columns of W_down ([d][d_ff]), that is
     W_gate[perm], W_up[perm], W_down[:, perm].           permuted_weights()

Readings (the paper names the method, not these details):
  - the clustered vectors are the neurons' raw input weights (no
    normalisation); for a gated FFN the gate and up rows are concatenated;
  - the initial centroids are the features of E distinct neurons chosen by
    the caller (the random draw is an input, not part of the method);
  - cluster h becomes expert h; within an expert the neurons keep their
    original relative order.
"""
import numpy as np
from scipy.optimize import linear_sum_assignment


def widen(a):
    """Stored weights (float32, float64 or uint16 bf16 bit patterns) to fp64, exactly."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    if a.dtype in (np.float32, np.float64):
        return a.astype(np.float64)
    raise TypeError("weights must be float32, float64 or uint16 (bf16 bits), got %s" % a.dtype)


def features(W_up, W_gate=None):
    """Step 1: [d_ff][f] fp64, row n = (W_gate[n], W_up[n]) or W_up[n]."""
    up = widen(W_up)
    if W_gate is None:
        return up
    return np.concatenate([widen(W_gate), up], axis=1)


def sq_distances(F, C):
    """D[n, h] = sum_i (F[n, i] - C[h, i])^2, one cluster at a time."""
    D = np.empty((F.shape[0], C.shape[0]), np.float64)
    for h in range(C.shape[0]):
        diff = F - C[h]
        D[:, h] = (diff * diff).sum(axis=1)
    return D


def balanced_assign(D, cap):
    """Step 2a: labels a[n] with exactly `cap` neurons per cluster minimising
    sum_n D[n, a[n]].  Exact: a linear assignment of the n neurons to n slots,
    cluster h owning slots [h * cap, (h + 1) * cap)."""
    n, k = D.shape
    assert n == k * cap, "every cluster holds exactly cap neurons"
    slots = np.repeat(D, cap, axis=1)  # column h * cap + r is cluster h
    rows, cols = linear_sum_assignment(slots)
    a = np.empty(n, np.int64)
    a[rows] = cols // cap
    return a.astype(np.int32)


def update_centroids(F, a, k):
    """Step 2b: c_h = mean of the features of the neurons labelled h."""
    C = np.zeros((k, F.shape[1]), np.float64)
    for h in range(k):
        C[h] = F[a == h].mean(axis=0)
    return C


def balanced_kmeans(F, k, init, max_iter=100):
    """Step 2.  Returns (labels [n] int32, assignments made, objective of the
    last assignment, objective after every assignment)."""
    F = np.asarray(F, np.float64)
    n = F.shape[0]
    init = np.asarray(init, np.int64)
    assert n % k == 0 and init.shape == (k,) and len(set(init.tolist())) == k
    assert init.min() >= 0 and init.max() < n and max_iter >= 1
    cap = n // k
    C = F[init].copy()
    prev = None
    history = []
    it = 0
    a = None
    while it < max_iter:
        it += 1
        D = sq_distances(F, C)
        a = balanced_assign(D, cap)
        history.append(float(D[np.arange(n), a].sum()))
        if prev is not None and np.array_equal(a, prev):
            break
        C = update_centroids(F, a, k)
        prev = a
    return a, it, history[-1], history


def permutation(a, k):
    """Step 3: perm[j] = the old neuron at new position j, ordered by
    (cluster, old index)."""
    a = np.asarray(a)
    return np.concatenate([np.flatnonzero(a == h) for h in range(k)]).astype(np.int32)


def permuted_weights(W_gate, W_up, W_down, perm):
    """Step 4, Eq. (permuted_weights), in the neuron-row storage."""
    perm = np.asarray(perm)
    return (None if W_gate is None else np.ascontiguousarray(np.asarray(W_gate)[perm]),
            np.ascontiguousarray(np.asarray(W_up)[perm]),
            np.ascontiguousarray(np.asarray(W_down)[:, perm]))


def moefy(W_gate, W_up, W_down, n_experts, init, max_iter=100):
    """Steps 1-4.  Returns (perm, labels, assignments made, objective, permuted
    W_gate, W_up, W_down)."""
    F = features(W_up, W_gate)
    a, it, obj, _ = balanced_kmeans(F, n_experts, init, max_iter)
    perm = permutation(a, n_experts)
    Wg, Wu, Wd = permuted_weights(W_gate, W_up, W_down, perm)
    return perm, a, it, obj, Wg, Wu, Wd
