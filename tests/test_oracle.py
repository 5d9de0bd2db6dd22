"""Pins for the CPU oracle: each check ties it to something other than itself.

* hand-worked cases of the paper's definitions (tests/golden/hand_cases.json),
  including the top-k rule of Sec. 4.3 and LTE's threshold (Eq. lte_hard_set);
* brute force over all 2^E expert subsets for the cumulative-mass cut
  (Eq. tau_thresh_activate), and an O(E^2) rank-by-comparison restatement;
* library routines: numpy matmul for Eq. (routing_logits) and the dense FFN,
  scipy's softmax / expit and torch's GELU / SiLU for the closed forms,
  numpy's lexsort for the top-k order, expit for LTE's set;
* invariants: the MoEfication identity (Eq. moefication_decomp: all experts
  with unit gates = dense FFN), neuron-permutation invariance (Eq.
  permuted_weights), softmax shift invariance, p >= 1 -> all experts,
  p <= 0 -> top-1, overflow-free huge logits.

The ``PINS`` list is also run against deliberately broken copies of the
oracle (test_planted_mistakes_are_caught) to show that each plausible
mistake fails at least one pin.
"""
import json
import math
import os
import shutil
import subprocess
import tempfile

import numpy as np
import pytest
import scipy.special

import oracle
from oracle import build as obuild
from paper_2605_28283_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_cases.json")


# ---------------------------------------------------------------- references
def np_act(kind, a, b=None):
    """Library closed forms: scipy expit for SiLU, torch for tanh-GELU."""
    import torch
    if kind == "swiglu":
        return b * scipy.special.expit(b) * a
    if kind == "relu":
        return np.maximum(a, 0.0)
    return torch.nn.functional.gelu(torch.from_numpy(a), approximate="tanh").numpy()


def widen(a):
    if a is None:
        return None
    if a.dtype == np.uint16:
        return wl.bf16_bits_to_f32(a).astype(np.float64)
    return a.astype(np.float64)


def np_dense(x, Wg, Wu, Wd, kind, block_scale=None, de=64):
    """Eq. (ffn) by numpy matmul; block_scale[t, e] scales expert block e of h."""
    x, Wg, Wu, Wd = widen(x), widen(Wg), widen(Wu), widen(Wd)
    a = x @ Wu.T
    b = None if Wg is None else x @ Wg.T
    h = np_act(kind, a, b)
    if block_scale is not None:
        h = h * np.repeat(block_scale, de, axis=1)
    return h @ Wd.T


def brute_min_prefix(probs, p):
    """Minimum-cardinality subset with mass >= p (max mass among those)."""
    E = probs.shape[0]
    if p >= 1.0:
        return set(range(E)), False
    masks = ((np.arange(1 << E)[:, None] >> np.arange(E)[None, :]) & 1).astype(np.float64)
    mass = masks @ probs
    card = masks.sum(1)
    ok = mass >= p
    if not ok.any():
        return set(range(E)), True
    kmin = card[ok].min()
    cand = np.where(ok & (card == kmin))[0]
    best = cand[np.argmax(mass[cand])]
    masses = np.sort(mass[cand])
    ambiguous = (len(cand) > 1 and masses[-1] - masses[-2] < 1e-12) or np.any(np.abs(mass - p) < 1e-9)
    return set(np.nonzero(masks[best])[0].tolist()), ambiguous


def rank_prefix(probs):
    """Inclusive prefix mass of each expert by pairwise comparison (no sort).

    Expert i precedes j when p_i > p_j, or p_i == p_j and i < j.
    """
    P = probs
    E = P.shape[0]
    idx = np.arange(E)
    ahead = (P[None, :] > P[:, None]) | ((P[None, :] == P[:, None]) & (idx[None, :] <= idx[:, None]))
    return (ahead * P[None, :]).sum(1)


# ---------------------------------------------------------------------- pins
def pin_hand_selection(o):
    cases = json.load(open(GOLDEN))["selection"]
    for group in cases:
        g = np.array([group["logits"]], np.float64)
        for c in group["cases"]:
            for rule in ("paper", "min_prefix"):
                counts, ids, _, _ = o.select(g, c["p"], rule)
                got = ids[0, :counts[0]].tolist()
                assert got == c[rule], (group["logits"], c["p"], rule, got)


def pin_hand_topk_lte(o):
    """Hand-worked top-k (Sec. 4.3) and LTE (Eq. lte_hard_set) selections."""
    for group in json.load(open(GOLDEN))["selection_topk_lte"]:
        g = np.array([group["logits"]], np.float64)
        for c in group["cases"]:
            counts, ids, _, _ = o.select(g, c["param"], c["rule"])
            assert ids[0, :counts[0]].tolist() == c["ids"], (c, ids[0, :counts[0]])
            assert np.all(ids[0, counts[0]:] == -1)


def pin_hand_ffn(o):
    f = json.load(open(GOLDEN))["ffn"]
    x = np.array(f["x"], np.float64)
    Wr, Wg, Wu, Wd = (np.array(f[k], np.float64) for k in ("W_r", "W_gate", "W_up", "W_down"))
    for c in f["cases"]:
        g, counts, ids, y = o.layer(x, Wr, Wg, Wu, Wd, c["p"], "swiglu", c["gate"], c["rule"])
        assert ids[0, :counts[0]].tolist() == c["ids"]
        np.testing.assert_allclose(y[0], c["y"], rtol=1e-13, atol=0)


def pin_logits_vs_matmul(o):
    rng = np.random.default_rng(11)
    for dt in ("f32", "bf16"):
        x32 = rng.standard_normal((5, 48), dtype=np.float32)
        W32 = rng.standard_normal((7, 48), dtype=np.float32)
        x = wl.f32_to_bf16_bits(x32) if dt == "bf16" else x32
        W = wl.f32_to_bf16_bits(W32) if dt == "bf16" else W32
        g = o.logits(x, W)
        ref = widen(x) @ widen(W).T
        np.testing.assert_allclose(g, ref, rtol=1e-13, atol=1e-13)


def pin_cum_vs_scipy_softmax(o):
    rng = np.random.default_rng(12)
    g = rng.standard_normal((20, 37)) * 3.0
    counts, ids, cum, probs = o.select(g, 0.6)
    P = scipy.special.softmax(g, axis=1)
    np.testing.assert_allclose(probs, P, rtol=1e-12, atol=1e-15)
    for t in range(g.shape[0]):
        ref_order = sorted(range(g.shape[1]), key=lambda j: (-g[t, j], j))
        np.testing.assert_allclose(cum[t], np.cumsum(P[t, ref_order]), rtol=1e-12, atol=1e-15)


def pin_bruteforce_min_prefix(o):
    rng = np.random.default_rng(13)
    checked = 0
    for E in (2, 3, 5, 8, 11):
        for _ in range(40):
            g = rng.standard_normal((1, E)) * rng.uniform(0.5, 4.0)
            p = float(rng.uniform(0.05, 0.99))
            P = scipy.special.softmax(g[0])
            want, ambiguous = brute_min_prefix(P, p)
            if ambiguous:
                continue
            counts, ids, _, _ = o.select(g, p, "min_prefix")
            assert set(ids[0, :counts[0]].tolist()) == want, (E, p)
            checked += 1
    assert checked > 150


def pin_rank_restatement(o):
    """Both rules against an O(E^2) comparison-based restatement of Eq. tau_thresh_activate."""
    rng = np.random.default_rng(14)
    for E in (4, 16, 64, 172, 256):
        g = rng.standard_normal((8, E)) * 3.0
        g[0, 3] = g[0, 1]  # exact tie
        for p in (0.0, 0.3, 0.7, 0.95, 1.0, 1.05):
            for rule in ("paper", "min_prefix"):
                counts, ids, _, _ = o.select(g, p, rule)
                for t in range(g.shape[0]):
                    P = scipy.special.softmax(g[t])
                    S = rank_prefix(P)
                    if np.any(np.abs(S - p) < 1e-9):
                        continue
                    top = int(np.argmin(S))  # the rank-1 expert has the smallest prefix
                    if p >= 1.0:
                        want = set(range(E))
                    elif rule == "paper":
                        want = set(np.nonzero(S < p)[0].tolist()) | {top}
                    else:
                        want = set(np.nonzero(S - P < p)[0].tolist()) | {top}
                    got = ids[t, :counts[t]].tolist()
                    assert set(got) == want, (E, p, rule, t)
                    # rank order: the prefixes of the listed experts increase
                    assert np.all(np.diff(S[got]) > 0)


def pin_rule_relation(o):
    """k_paper = max(1, k_min - 1) whenever the full mass reaches p."""
    rng = np.random.default_rng(15)
    g = rng.standard_normal((200, 64)) * 3.0
    for p in (0.2, 0.5, 0.8, 0.95):
        kp, idp, _, _ = o.select(g, p, "paper")
        km, idm, cum, _ = o.select(g, p, "min_prefix")
        assert np.all(kp == np.maximum(1, km - 1))
        for t in range(g.shape[0]):
            assert idp[t, :kp[t]].tolist() == idm[t, :kp[t]].tolist()


def rank_order(gt):
    """Descending logit, ties by lower index, by numpy's lexsort."""
    return np.lexsort((np.arange(gt.shape[0]), -gt))


def pin_topk_vs_lexsort(o):
    """Top-k against a library sort; every kept logit beats every dropped one."""
    rng = np.random.default_rng(19)
    E = 48
    g = np.round(rng.standard_normal((12, E)) * 3.0, 1)  # rounding makes exact ties
    for k in (0.0, 0.5, 1.0, 2.0, 3.7, 7.0, E - 1.0, float(E), E + 5.0, 1e9):
        counts, ids, _, _ = o.select(g, k, "topk")
        want_k = min(E, max(1, int(math.floor(k))))
        assert np.all(counts == want_k), (k, counts)
        for t in range(g.shape[0]):
            ref = rank_order(g[t])
            assert ids[t, :want_k].tolist() == ref[:want_k].tolist()
            kept, dropped = g[t, ids[t, :want_k]], np.delete(g[t], ids[t, :want_k])
            assert dropped.size == 0 or kept.min() >= dropped.max()


def pin_lte_vs_expit(o):
    """LTE's set (Eq. lte_hard_set) against scipy's expit, each expert on its own."""
    rng = np.random.default_rng(20)
    E = 40
    g = rng.standard_normal((16, E)) * 3.0
    g[0, :4] = 0.0  # sigmoid(0) = 0.5 exactly: excluded at delta = 0.5 (strict >)
    g[1, :] = -1000.0  # sigmoid underflows to 0 in fp64
    for delta in (-1.0, 0.0, 1e-30, 0.1, 0.5, 0.73, 0.9, 0.999, 1.0, 2.0):
        counts, ids, _, _ = o.select(g, delta, "lte")
        s = scipy.special.expit(g)
        for t in range(g.shape[0]):
            if delta <= 0.0:
                want = set(range(E))  # a sigmoid is positive everywhere
            else:
                if np.any(np.abs(s[t] - delta) < 1e-12) and delta != 0.5:
                    continue
                want = set(np.nonzero(s[t] > delta)[0].tolist())
            got = ids[t, :counts[t]].tolist()
            assert set(got) == want and len(got) == len(want), (delta, t)
            # listed in the order pi
            ref = [j for j in rank_order(g[t]).tolist() if j in want]
            assert got == ref
            assert np.all(ids[t, counts[t]:] == -1)
    with pytest.raises(oracle.OracleError):
        o.select(g, float("nan"), "lte")
    with pytest.raises(oracle.OracleError):
        o.select(g, float("nan"), "topk")


def pin_router_stats(o):
    """Eq. entropy_loss, Eq. load_balance_loss and L_gate: closed forms and a
    scipy restatement."""
    E, B, eps = 16, 5, 1e-9
    # equal logits: p = 1/E everywhere
    ent, bal, gate = o.router_stats(np.full((B, E), 0.7), eps)
    assert abs(ent - (-math.log(1.0 / E + eps))) <= 1e-14 * math.log(E)
    assert abs(bal - 1.0) <= 1e-14
    assert abs(gate - scipy.special.expit(0.7)) <= 1e-15
    # one-hot tokens (exp underflows to exactly 0): all on expert 3, then one per expert
    g = np.full((B, E), -1e4)
    g[:, 3] = 1e4
    ent, bal, gate = o.router_stats(g, eps)
    assert abs(ent - (-math.log(1.0 + eps))) <= 1e-20 and abs(bal - E) <= 1e-12
    assert abs(gate - 1.0 / E) <= 1e-15
    g = np.full((E, E), -1e4)
    g[np.arange(E), np.arange(E)] = 1e4
    assert abs(o.router_stats(g, eps)[1] - 1.0) <= 1e-14
    # random batch against scipy's softmax and expit
    rng = np.random.default_rng(21)
    for E, B in ((7, 3), (172, 40), (224, 64)):
        g = rng.standard_normal((B, E)) * 3.0
        P = scipy.special.softmax(g, axis=1)
        ent_ref = -np.sum(P * np.log(P + eps)) / B
        bal_ref = E * np.sum(P.mean(axis=0) ** 2)
        gate_ref = scipy.special.expit(g).mean()
        ent, bal, gate = o.router_stats(g, eps)
        assert abs(ent - ent_ref) <= 1e-12 * abs(ent_ref)
        assert abs(bal - bal_ref) <= 1e-12 * bal_ref
        assert abs(gate - gate_ref) <= 1e-13 * gate_ref
    with pytest.raises(oracle.OracleError):
        o.router_stats(np.array([[0.0, np.inf]]))


def pin_rmsnorm_residual(o):
    """x_{l+1} = RMSNorm(x_l + y_l): closed forms, invariants and a numpy restatement."""
    rng = np.random.default_rng(22)
    # constant rows: c / sqrt(c^2 + eps)
    x = np.full((2, 8), 3.0)
    out = o.rmsnorm_residual(x, None, None, 0.25)
    np.testing.assert_allclose(out, 3.0 / math.sqrt(9.25), rtol=1e-15)
    # unit mean square at eps = 0; scale invariance; the residual is a plain sum
    x = rng.standard_normal((5, 64))
    y = rng.standard_normal((5, 64))
    out = o.rmsnorm_residual(x, y, None, 0.0)
    np.testing.assert_allclose((out ** 2).mean(axis=1), 1.0, rtol=1e-13)
    np.testing.assert_allclose(o.rmsnorm_residual(7.5 * x, 7.5 * y, None, 0.0), out, rtol=1e-13)
    np.testing.assert_allclose(o.rmsnorm_residual(x + y, None, None, 0.0), out, rtol=1e-13)
    gamma = rng.uniform(0.5, 2.0, 64)
    v = x + y
    ref = v / np.sqrt((v ** 2).mean(axis=1, keepdims=True) + 1e-5) * gamma
    np.testing.assert_allclose(o.rmsnorm_residual(x, y, gamma, 1e-5), ref, rtol=1e-13)
    # bf16 inputs are widened exactly
    xb, yb, gb = (wl.f32_to_bf16_bits(a.astype(np.float32)) for a in (x, y, gamma))
    vb = widen(xb) + widen(yb)
    refb = vb / np.sqrt((vb ** 2).mean(axis=1, keepdims=True) + 1e-6) * widen(gb)
    np.testing.assert_allclose(o.rmsnorm_residual(xb, yb, gb, 1e-6), refb, rtol=1e-13)


def pin_special_p(o):
    rng = np.random.default_rng(16)
    E = 40
    g = rng.standard_normal((10, E)) * 5.0
    g[3, :] = np.linspace(0, -60, E)  # spread makes the tail vanish in fp64
    for rule in ("paper", "min_prefix"):
        for p in (0.0, -0.5, 1e-12):
            counts, ids, _, _ = o.select(g, p, rule)
            assert np.all(counts == 1)
            assert np.all(ids[:, 0] == np.argmax(g, axis=1))
        for p in (1.0, 1.05, 3.0):
            counts, ids, _, _ = o.select(g, p, rule)
            assert np.all(counts == E)
            for t in range(g.shape[0]):
                assert ids[t].tolist() == sorted(range(E), key=lambda j: (-g[t, j], j))
    with pytest.raises(oracle.OracleError):
        o.select(g, float("nan"))


def pin_shift_invariance_and_huge_logits(o):
    rng = np.random.default_rng(17)
    g = (rng.standard_normal((30, 50)) * 3.0).astype(np.float32).astype(np.float64)
    for p in (0.3, 0.8):
        a = o.select(g, p)[:2]
        b = o.select(g + 3.0, p)[:2]
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    big = np.array([[1e4, -1e4, 9990.0, 0.0], [-1e4, -1e4 + 1.0, -1e4 + 2.0, -1e4]], np.float64)
    counts, ids, cum, probs = o.select(big, 0.9)
    assert np.all(np.isfinite(cum)) and np.all(np.isfinite(probs))
    assert ids[0, :counts[0]].tolist() == [0]
    # second row: probabilities e^2, e^1, 1, 1 over Z
    assert ids[1, :counts[1]].tolist() == [2, 1, 0]


def pin_nonfinite(o):
    g = np.array([[0.0, float("nan"), 1.0], [0.0, 1.0, 2.0]])
    counts, ids, _, _ = o.select(g, 0.5, allow_nonfinite=True)
    assert counts[0] == 0 and counts[1] >= 1
    with pytest.raises(oracle.OracleError):
        o.select(g, 0.5)


def pin_activations(o):
    import torch
    vs = np.array([-6.0, -2.5, -1.0, -0.1, 0.0, 0.3, 1.0, 2.0, 7.5])
    ref_gelu = torch.nn.functional.gelu(torch.from_numpy(vs), approximate="tanh").numpy()
    ref_silu = torch.nn.functional.silu(torch.from_numpy(vs)).numpy()
    for v, rg, rs in zip(vs, ref_gelu, ref_silu):
        assert abs(o.act("gelu_tanh", v) - rg) <= 1e-14 * max(1.0, abs(rg))
        assert abs(o.act("swiglu", 1.0, v) - rs) <= 1e-14 * max(1.0, abs(rs))
        assert abs(o.act("swiglu", 2.5, v) - 2.5 * rs) <= 1e-13 * max(1.0, abs(rs))
        assert o.act("relu", v) == max(v, 0.0)


def _small_layer(kind, dtype="bf16", d=32, E=6, T=5, seed=3):
    w = wl.Workload("pin", d, E * 64, E, 1, dtype, kind, (T,), (0.5,), (3.0, 3.0), False)
    return wl.host_layer(w, T, seed=seed)


def pin_dense_identity(o):
    """Eq. (moefication_decomp): all experts with unit gates equal the dense FFN."""
    for kind in ("swiglu", "relu", "gelu_tanh"):
        L = _small_layer(kind)
        E = L.Wr.shape[0]
        g, counts, ids, y = o.layer(L.x, L.Wr, L.Wg, L.Wu, L.Wd, 1.0, kind, "none")
        assert np.all(counts == E)
        ref = np_dense(L.x, L.Wg, L.Wu, L.Wd, kind)
        np.testing.assert_allclose(y, ref, rtol=1e-11, atol=1e-13)
        np.testing.assert_allclose(o.dense_ffn(L.x, L.Wg, L.Wu, L.Wd, kind), ref,
                                   rtol=1e-11, atol=1e-13)
        # Eq. (moe_output) at p >= 1: every block scaled by its sigmoid gate
        g, counts, ids, y = o.layer(L.x, L.Wr, L.Wg, L.Wu, L.Wd, 1.05, kind, "sigmoid")
        ref = np_dense(L.x, L.Wg, L.Wu, L.Wd, kind, block_scale=scipy.special.expit(g))
        np.testing.assert_allclose(y, ref, rtol=1e-11, atol=1e-13)


def pin_masked_dense(o):
    """A partial selection equals the dense FFN with unselected blocks masked out."""
    for kind in ("swiglu", "gelu_tanh"):
        L = _small_layer(kind, T=9, E=8)
        E = 8
        for p in (0.3, 0.7):
            for rule in ("min_prefix", "paper"):
                g, counts, ids, y = o.layer(L.x, L.Wr, L.Wg, L.Wu, L.Wd, p, kind, "sigmoid", rule)
                scale = np.zeros((L.x.shape[0], E))
                for t in range(L.x.shape[0]):
                    for e in ids[t, :counts[t]]:
                        scale[t, e] = scipy.special.expit(g[t, e])
                ref = np_dense(L.x, L.Wg, L.Wu, L.Wd, kind, block_scale=scale)
                np.testing.assert_allclose(y, ref, rtol=1e-11, atol=1e-13)


def pin_permutation_invariance(o):
    """Eq. (permuted_weights): permuting neurons leaves the dense FFN unchanged."""
    L = _small_layer("swiglu", dtype="f32", E=4, T=3)
    perm = np.random.default_rng(18).permutation(L.Wu.shape[0])
    Wg2, Wu2, Wd2 = L.Wg[perm], L.Wu[perm], L.Wd[:, perm]
    ref = np_dense(L.x, L.Wg, L.Wu, L.Wd, "swiglu")
    np.testing.assert_allclose(o.dense_ffn(L.x, Wg2, Wu2, Wd2, "swiglu"), ref, rtol=1e-11, atol=1e-13)
    g, counts, ids, y = o.layer(L.x, L.Wr, Wg2, Wu2, Wd2, 1.0, "swiglu", "none")
    np.testing.assert_allclose(y, ref, rtol=1e-11, atol=1e-13)


def pin_ffn_sparsity(o):
    """Sec. 4.1 s_FFN: a hand-worked case, closed forms through the oracle's
    own selection (p >= 1 activates all E, top-k exactly k, LTE at delta >= 1
    none) and the histogram's two sums."""
    case = json.load(open(GOLDEN))["ffn_sparsity"]
    s, k_sum, hist = o.ffn_sparsity(np.array(case["counts"]), case["E"])
    assert k_sum == case["k_sum"] and list(hist) == case["hist"]
    assert abs(s - case["s_ffn_num"] / case["s_ffn_den"]) <= 1e-15
    rng = np.random.default_rng(23)
    E, N, L = 24, 7, 3
    g = rng.standard_normal((L * N, E)) * 3.0
    for p, rule, s_ref in ((1.0, "min_prefix", 0.0), (5.0, "topk", 1.0 - 5.0 / E), (1.0, "lte", 1.0),
                           (0.0, "paper", 1.0 - 1.0 / E)):
        counts = o.select(g, p, rule)[0].reshape(L, N)
        s, k_sum, hist = o.ffn_sparsity(counts, E)
        assert abs(s - s_ref) <= 1e-15, (p, rule, s)
    # a mixed selection: the histogram counts every (token, layer) once and
    # its first moment is the sum of the set sizes
    counts = o.select(g, 0.7, "min_prefix")[0].reshape(L, N)
    s, k_sum, hist = o.ffn_sparsity(counts, E)
    assert hist.sum() == N * L and int((np.arange(E + 1) * hist).sum()) == k_sum
    assert abs(s - (1.0 - k_sum / (N * L * E))) <= 1e-15
    assert np.all(hist[np.bincount(counts.ravel(), minlength=E + 1) == 0] == 0)
    with pytest.raises(oracle.OracleError):
        o.ffn_sparsity(np.array([[E + 1]]), E)


PINS = [pin_hand_selection, pin_hand_topk_lte, pin_hand_ffn, pin_logits_vs_matmul, pin_cum_vs_scipy_softmax,
        pin_bruteforce_min_prefix, pin_rank_restatement, pin_rule_relation, pin_special_p,
        pin_shift_invariance_and_huge_logits, pin_nonfinite, pin_activations, pin_dense_identity,
        pin_masked_dense, pin_permutation_invariance, pin_topk_vs_lexsort, pin_lte_vs_expit,
        pin_router_stats, pin_rmsnorm_residual, pin_ffn_sparsity]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(ppo, pin):
    pin(ppo)


def test_bf16_rounding_helper():
    # round-to-nearest-even on ties, exact on representable values
    vals = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 3.0e-3], np.float32)
    back = wl.bf16_bits_to_f32(wl.f32_to_bf16_bits(vals))
    assert back[0] == 1.0 and back[1] == 1.0 and back[2] == np.float32(1.0 + 2 ** -6)
    assert back[3] == -2.5
    assert abs(back[4] - 3.0e-3) <= 3.0e-3 * 2 ** -8


# ----------------------------------------------------- planted mistakes (CPU)
MUTANTS = {
    "paper_rule_drops_top1": ("k = below > 1 ? below : 1;", "k = below;"),
    "cut_not_strict": ("if (S < p)", "if (S <= p)"),
    "ascending_order": ("if (a->g > b->g)\n        return -1;", "if (a->g < b->g)\n        return -1;"),
    "tie_break_reversed": ("return (a->j > b->j) - (a->j < b->j);", "return (a->j < b->j) - (a->j > b->j);"),
    "min_prefix_off_by_one": ("k = below + 1 < E ? below + 1 : E;", "k = below < E ? below : E;"),
    "no_max_shift": ("prob[j] = exp(gt[j] - m);", "prob[j] = exp(gt[j]);"),
    "p_ge_1_not_special": ("if (p >= 1.0) {", "if (p > 1.0) {"),
    "router_transposed": ("acc += ld(Wr, wr_dt, (size_t)j * d + i)", "acc += ld(Wr, wr_dt, (size_t)i * E + j)"),
    "gate_from_rank": ("ppo_sigmoid(g[(size_t)t * E + e])", "ppo_sigmoid(g[(size_t)t * E + r])"),
    "gate_sign": ("return 1.0 / (1.0 + exp(-v));", "return 1.0 / (1.0 + exp(v));"),
    "swiglu_swapped": ("return ppo_silu(b) * a;", "return ppo_silu(a) * b;"),
    "down_neighbour_column": ("yt[j] += w * h * ld(Wd, w_dt, (size_t)j * dff + n);",
                              "yt[j] += w * h * ld(Wd, w_dt, (size_t)j * dff + (n ^ 1));"),
    "gelu_constant": ("0.044715", "0.0447"),
    "topk_rounds_up": ("(p >= 1.0 ? (int)floor(p) : 1)", "(p >= 1.0 ? (int)ceil(p) : 1)"),
    "topk_allows_zero": ("(p >= 1.0 ? (int)floor(p) : 1)", "(p >= 1.0 ? (int)floor(p) : 0)"),
    "lte_not_strict": ("ppo_sigmoid(order[r].g) > p)", "ppo_sigmoid(order[r].g) >= p)"),
    "lte_delta_le0_not_special": ("if (p <= 0.0 || ppo_sigmoid(order[r].g) > p)", "if (ppo_sigmoid(order[r].g) > p)"),
    "stats_no_eps": ("ent -= pj * log(pj + eps);", "ent -= pj * log(pj);"),
    "stats_ent_not_averaged": ("out[0] = ent / (double)T;", "out[0] = ent;"),
    "stats_bal_not_squared": ("bal += f * f;", "bal += f;"),
    "stats_bal_no_E": ("out[1] = (double)E * bal;", "out[1] = bal;"),
    "stats_gate_raw_logit": ("gate += ppo_sigmoid(gt[j]);", "gate += gt[j];"),
    "norm_no_eps": ("const double r = 1.0 / sqrt(ss / (double)d + eps);", "const double r = 1.0 / sqrt(ss / (double)d);"),
    "norm_sum_not_mean": ("const double r = 1.0 / sqrt(ss / (double)d + eps);", "const double r = 1.0 / sqrt(ss + eps);"),
    "norm_no_residual": ("                v += ld(y_prev, dt, (size_t)t * d + i);", "                v += 0.0;"),
    "norm_gamma_index": ("ld(gamma, dt, (size_t)i)", "ld(gamma, dt, (size_t)(d - 1 - i))"),
    "lte_expert_order": ("idt[k++] = order[r].j;", "idt[k++] = order[E - 1 - r].j;"),
    "sparsity_hist_off_by_one": ("hist[c] += 1ull;", "hist[c > 0 ? c - 1 : 0] += 1ull;"),
    "sparsity_without_layers": ("((double)N * (double)L * (double)E)", "((double)N * (double)E)"),
    "sparsity_not_complement": ("*s_ffn = 1.0 - (double)total", "*s_ffn = (double)total"),
    "expert_block_offset": ("for (int n = e * de; n < (e + 1) * de; n++) {",
                            "for (int n = e * de + (de > 1); n < (e + 1) * de; n++) {"),
}


def test_planted_mistakes_are_caught(tmp_path):
    src = open(obuild.SRC).read()
    good = oracle.load()
    escaped = []
    try:
        for name, (old, new) in MUTANTS.items():
            assert src.count(old) >= 1, name
            mutated = src.replace(old, new)
            msrc = tmp_path / ("ppo_%s.c" % name)
            msrc.write_text(mutated)
            lib = str(tmp_path / ("libppo_%s.so" % name))
            subprocess.run(["gcc", "-O2", "-std=c11", "-D_DEFAULT_SOURCE", "-fPIC", "-shared",
                            "-fopenmp", str(msrc), "-o", lib, "-lm"], check=True)
            oracle.load(lib)
            caught = False
            for pin in PINS:
                try:
                    pin(oracle)
                except Exception:
                    caught = True
                    break
            if not caught:
                escaped.append(name)
    finally:
        oracle.load(obuild.LIB)
    assert good is not None
    assert not escaped, "planted mistakes not caught by any pin: %s" % escaped
