"""Helpers for the GPU-vs-oracle parity tests.

Inputs come from the seeded host recipe in ``paper_2605_28283_gb300.workloads``;
expected values come only from the CPU oracle, and every GPU value is taken
through the library's C ABI.  The bars:

* selection, identical logits (pp_select): counts and ids bit-exact, except
  "boundary" tokens whose oracle prefix mass S_i (LTE: a sigmoid score) lies
  within 1e-6 of p; those must take a count that some p' within 1e-6 of p
  gives, with the same ids (top-k has no boundary tokens);
* selection from x (pp_route / pp_layer): the GPU's fp32 logits differ from
  the oracle's fp64 ones by at most eps (checked).  Tokens whose cut is
  unique under that perturbation (no prefix mass within 1e-6 + eps of p, no
  two logits of the activated prefix or across the cut within 2 eps) must
  match exactly; for the others the GPU's selection must be a valid one (a
  count some p' within the margin gives, a set whose logits all exceed the
  unselected ones by -2 eps at worst, rank order non-increasing up to 2 eps);
* y: per-token max|y - y_ref| / max|y_ref| <= 2e-2 (bf16) or 1e-4 (fp32),
  y_ref being the oracle's FFN on the oracle's selection, or on the GPU's
  validated selection for the non-unique tokens above.
"""
import functools

import numpy as np

import oracle
from paper_2605_28283_gb300 import workloads as wl

Y_TOL = {"bf16": 2e-2, "f32": 1e-4}
BOUNDARY = 1e-6


def f32(p):
    """The fp32 value the C ABI receives for p; the oracle is given the same."""
    return float(np.float32(p))


@functools.lru_cache(maxsize=6)
def layer_inputs(name, T, seed=0, layer=0, d=None, E=None):
    w = wl.WORKLOADS[name]
    if d is not None:
        w = wl.scaled(w, d, E)
    return w, wl.host_layer(w, T, seed=seed, layer=layer)


def widen(a):
    if a is None:
        return None
    if a.dtype == np.uint16:
        return wl.bf16_bits_to_f32(a).astype(np.float64)
    return a.astype(np.float64)


def rel_err_per_token(y, ref):
    y = np.asarray(y, np.float64)
    ref = np.asarray(ref, np.float64)
    num = np.abs(y - ref).max(axis=1)
    den = np.maximum(np.abs(ref).max(axis=1), 1e-30)
    return num / den


def to_host(t):
    import torch
    if t.dtype == torch.bfloat16:
        t = t.float()
    return t.detach().cpu().numpy()


def logit_tolerance(x, Wr):
    """Bound on |g_gpu - g_ref| for an fp32-accumulated dot product of length
    d: 1e-5 * sum_i |W_r[j,i] x_i| (each fp32 partial sum is a chain of at most
    ~160 additions, gamma_160 < 1e-5)."""
    return 1e-5 * (np.abs(widen(x)) @ np.abs(widen(Wr)).T) + 1e-30


MASS_RULES = ("min_prefix", "paper")


def _count_range(g_row, p, rule, margin):
    """Counts the oracle gives for parameters within `margin` of p (a mass
    margin for the cumulative-mass rules, a score margin for LTE)."""
    if rule == "topk":
        k = oracle.select(g_row[None], p, rule)[0][0]
        return k, k
    if rule == "lte":
        klo = oracle.select(g_row[None], p + margin, rule)[0][0]
        khi = oracle.select(g_row[None], p - margin, rule)[0][0]
        return min(klo, khi), max(klo, khi)
    if p >= 1.0:
        k = g_row.shape[-1]
        return k, k
    klo = oracle.select(g_row[None], max(p - margin, -1.0), rule)[0][0]
    khi = oracle.select(g_row[None], min(p + margin, 1.0 - 1e-15), rule)[0][0]
    return min(klo, khi), max(klo, khi)


def near_cut(g_row, cum_row, p, rule, margin):
    """Whether the token's cut lies within `margin` of a decision: a prefix
    mass within margin of p (cumulative-mass rules) or a sigmoid score within
    margin of delta (LTE).  The top-k cut depends on the order only."""
    if rule in MASS_RULES:
        return p < 1.0 and bool(np.any(np.abs(cum_row - p) <= margin))
    if rule == "lte":
        with np.errstate(over="ignore"):
            score = 1.0 / (1.0 + np.exp(-g_row))
        return 0.0 < p < 1.0 and bool(np.any(np.abs(score - p) <= margin))
    return False


def check_select_exact(gpu_counts, gpu_ids, g, p, rule):
    """pp_select parity (identical logits).  Returns #boundary tokens."""
    counts, ids, cum, _ = oracle.select(g, p, rule)
    nb = 0
    for t in range(len(counts)):
        k = int(gpu_counts[t])
        boundary = near_cut(g[t], cum[t], p, rule, BOUNDARY)
        if boundary:
            nb += 1
            lo, hi = _count_range(g[t], p, rule, BOUNDARY)
            assert lo <= k <= hi, ("boundary count", t, k, lo, hi)
            kk = min(k, int(counts[t]))
            assert gpu_ids[t, :kk].tolist() == ids[t, :kk].tolist(), ("ids", t)
        else:
            assert k == counts[t], ("count", t, k, int(counts[t]))
            assert gpu_ids[t, :k].tolist() == ids[t, :k].tolist(), ("ids", t)
        assert np.all(gpu_ids[t, k:] == -1), ("padding", t)
    return nb


def check_route_selection(gpu_counts, gpu_ids, g_ref, eps, p, rule):
    """pp_route/pp_layer selection parity.  eps[t] bounds the logit error of
    token t.  Returns (unique mask, number of non-unique tokens)."""
    counts, ids, cum, _ = oracle.select(g_ref, p, rule)
    T, E = g_ref.shape
    unique = np.ones(T, bool)
    for t in range(T):
        e2 = 2.0 * float(eps[t])
        # a logit error eps moves a prefix mass by at most eps and a sigmoid
        # score by at most eps / 4
        margin = BOUNDARY + float(eps[t]) * (0.25 if rule == "lte" else 1.0)
        ko = int(counts[t])
        k = int(gpu_counts[t])
        full = np.argsort(-g_ref[t], kind="stable")
        gs = g_ref[t, full]
        top = min(ko + 1, E)
        ties = np.any(np.diff(gs[:top]) > -e2) if top > 1 else False
        boundary = near_cut(g_ref[t], cum[t], p, rule, margin)
        if not boundary and not ties:
            assert k == ko, ("count", t, k, ko)
            assert gpu_ids[t, :k].tolist() == ids[t, :k].tolist(), ("ids", t)
        else:
            unique[t] = False
            lo, hi = _count_range(g_ref[t], p, rule, margin)
            assert lo <= k <= hi, ("count range", t, k, lo, hi)
            sel = gpu_ids[t, :k]
            assert len(set(sel.tolist())) == k and np.all((sel >= 0) & (sel < E)), ("ids valid", t)
            gsel = g_ref[t, sel]
            assert np.all(np.diff(gsel) <= e2), ("rank order", t)
            rest = np.setdiff1d(np.arange(E), sel)
            if len(rest) and k > 0:
                assert gsel.min() >= g_ref[t, rest].max() - e2, ("top set", t)
        assert np.all(gpu_ids[t, k:] == -1), ("padding", t)
    return unique, int((~unique).sum())


def check_y(L, y_gpu, counts_ref, ids_ref, g_ref, E, act, gate, tol, unique=None, gpu_counts=None,
            gpu_ids=None):
    """y parity against the oracle FFN.  Tokens not in `unique` are compared
    on the GPU's validated selection.  Returns the max relative error."""
    counts = np.array(counts_ref, np.int32)
    ids = np.array(ids_ref, np.int32)
    if unique is not None:
        for t in np.nonzero(~unique)[0]:
            counts[t] = gpu_counts[t]
            ids[t] = gpu_ids[t]
    y_ref = oracle.sparse_ffn(L.x, L.Wg, L.Wu, L.Wd, counts, ids, g_ref, E, act, gate)
    err = rel_err_per_token(y_gpu, y_ref)
    worst = int(np.argmax(err))
    assert err[worst] <= tol, ("y", worst, float(err[worst]), tol)
    return float(err.max())
