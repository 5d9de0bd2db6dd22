"""CPU oracle for the PrunePath sparse-FFN path (test infrastructure).

This package is NOT part of the product.  Only ``tests/``,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference leg of
``bench.py`` may import it.  It shares no code with the CUDA library and
never imports it.  The arithmetic lives in ``ppo.c`` (plain C, fp64); this
module only marshals numpy arrays into it.

Array conventions: fp32 inputs are ``numpy.float32`` arrays, bf16 inputs are
``numpy.uint16`` arrays holding the bf16 bit patterns, fp64 inputs are
``numpy.float64``.  Outputs are fp64 / int32 numpy arrays.
"""
import ctypes
import os

import numpy as np

from . import build as _build

F32, BF16, F64 = 0, 1, 2
RELU, GELU_TANH, SWIGLU = 0, 1, 2
GATE_SIGMOID, GATE_NONE = 0, 1
RULE_MIN_PREFIX, RULE_PAPER, RULE_TOPK, RULE_LTE = 0, 1, 2, 3
OK, ERR_ARG, ERR_NONFINITE = 0, 1, 9

_ACTS = {"relu": RELU, "gelu_tanh": GELU_TANH, "gelu": GELU_TANH, "swiglu": SWIGLU}
_GATES = {"sigmoid": GATE_SIGMOID, "none": GATE_NONE}
_RULES = {"min_prefix": RULE_MIN_PREFIX, "paper": RULE_PAPER, "topk": RULE_TOPK, "lte": RULE_LTE}

_lib = None
_lib_path = None

_P = ctypes.c_void_p
_I = ctypes.c_int
_D = ctypes.c_double


def load(path: str = None):
    """Load (building first if needed) the oracle library; returns the CDLL."""
    global _lib, _lib_path
    if path is None and _lib is not None:
        return _lib
    path = path or _build.build()
    if _lib is not None and _lib_path == path:
        return _lib
    lib = ctypes.CDLL(path)
    for name in ("ppo_sigmoid", "ppo_silu", "ppo_gelu_tanh", "ppo_relu"):
        getattr(lib, name).restype = _D
        getattr(lib, name).argtypes = [_D]
    lib.ppo_act.restype = _D
    lib.ppo_act.argtypes = [_I, _D, _D]
    lib.ppo_logits.restype = _I
    lib.ppo_logits.argtypes = [_P, _I, _I, _I, _P, _I, _I, _P]
    lib.ppo_select.restype = _I
    lib.ppo_select.argtypes = [_P, _I, _I, _D, _I, _P, _P, _P, _P]
    lib.ppo_sparse_ffn.restype = _I
    lib.ppo_sparse_ffn.argtypes = [_P, _I, _I, _I, _I, _I, _I, _I, _P, _P, _P, _I, _P, _P, _P, _P]
    lib.ppo_dense_ffn.restype = _I
    lib.ppo_dense_ffn.argtypes = [_P, _I, _I, _I, _I, _I, _P, _P, _P, _I, _P]
    lib.ppo_router_stats.restype = _I
    lib.ppo_router_stats.argtypes = [_P, _I, _I, _D, _P]
    lib.ppo_rmsnorm_residual.restype = _I
    lib.ppo_rmsnorm_residual.argtypes = [_P, _P, _P, _I, _I, _I, _D, _P]
    lib.ppo_ffn_sparsity.restype = _I
    lib.ppo_ffn_sparsity.argtypes = [_P, _I, _I, _I, _P, _P, _P]
    lib.ppo_layer.restype = _I
    lib.ppo_layer.argtypes = [_P, _I, _I, _I, _I, _I, _I, _I, _I, _D, _P, _P, _P, _P, _I, _P,
                              _P, _P, _P]
    _lib, _lib_path = lib, path
    return lib


class OracleError(RuntimeError):
    def __init__(self, code, what):
        super().__init__("%s returned status %d" % (what, code))
        self.code = code


def _dt(a):
    if a.dtype == np.float32:
        return F32
    if a.dtype == np.uint16:
        return BF16
    if a.dtype == np.float64:
        return F64
    raise TypeError("oracle inputs must be float32, float64 or uint16 (bf16 bits), got %s" % a.dtype)


def _c(a):
    return np.ascontiguousarray(a)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _code(x, table):
    return table[x] if isinstance(x, str) else int(x)


def act(kind, a, b=0.0):
    """h for one neuron: kind in {'relu','gelu_tanh','swiglu'}; a = up, b = gate."""
    return load().ppo_act(_code(kind, _ACTS), float(a), float(b))


def logits(x, Wr):
    """Eq. (routing_logits): g[t, j] = sum_i Wr[j, i] x[t, i], in fp64."""
    lib = load()
    x, Wr = _c(x), _c(Wr)
    T, d = x.shape
    E = Wr.shape[0]
    assert Wr.shape[1] == d
    g = np.empty((T, E), np.float64)
    s = lib.ppo_logits(_ptr(x), _dt(x), T, d, _ptr(Wr), _dt(Wr), E, _ptr(g))
    if s:
        raise OracleError(s, "ppo_logits")
    return g


def select(g, p, rule="min_prefix", allow_nonfinite=False):
    """Softmax, descending order and cumulative-mass cut for each row of g
    (rule 'topk': p is k; rule 'lte': p is the sigmoid threshold delta).

    Returns (counts[T] int32, ids[T,E] int32 (rank order, -1 padded),
    cum[T,E] fp64 inclusive prefix masses S_i, probs[T,E] fp64).
    """
    lib = load()
    g = np.ascontiguousarray(g, dtype=np.float64)
    T, E = g.shape
    counts = np.empty(T, np.int32)
    ids = np.empty((T, E), np.int32)
    cum = np.empty((T, E), np.float64)
    probs = np.empty((T, E), np.float64)
    s = lib.ppo_select(_ptr(g), T, E, float(p), _code(rule, _RULES), _ptr(counts), _ptr(ids),
                       _ptr(cum), _ptr(probs))
    if s and not (s == ERR_NONFINITE and allow_nonfinite):
        raise OracleError(s, "ppo_select")
    return counts, ids, cum, probs


def sparse_ffn(x, Wg, Wu, Wd, counts, ids, g, n_experts, act_kind="swiglu", gate="sigmoid"):
    """Eq. (moe_output) over the given selection.  Returns y [T, d] fp64."""
    lib = load()
    x, Wu, Wd = _c(x), _c(Wu), _c(Wd)
    Wg = None if Wg is None else _c(Wg)
    counts = np.ascontiguousarray(counts, dtype=np.int32)
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    g = np.ascontiguousarray(g, dtype=np.float64)
    T, d = x.shape
    dff = Wu.shape[0]
    E = int(n_experts)
    assert dff % E == 0 and Wu.shape[1] == d and Wd.shape == (d, dff)
    assert ids.shape == (T, E) and g.shape == (T, E)
    w_dt = _dt(Wu)
    assert _dt(Wd) == w_dt and (Wg is None or _dt(Wg) == w_dt)
    y = np.empty((T, d), np.float64)
    s = lib.ppo_sparse_ffn(_ptr(x), _dt(x), T, d, E, dff // E, _code(act_kind, _ACTS),
                           _code(gate, _GATES), _ptr(Wg), _ptr(Wu), _ptr(Wd), w_dt,
                           _ptr(counts), _ptr(ids), _ptr(g), _ptr(y))
    if s:
        raise OracleError(s, "ppo_sparse_ffn")
    return y


def dense_ffn(x, Wg, Wu, Wd, act_kind="swiglu"):
    """Eq. (ffn) with no routing.  Returns y [T, d] fp64."""
    lib = load()
    x, Wu, Wd = _c(x), _c(Wu), _c(Wd)
    Wg = None if Wg is None else _c(Wg)
    T, d = x.shape
    dff = Wu.shape[0]
    y = np.empty((T, d), np.float64)
    s = lib.ppo_dense_ffn(_ptr(x), _dt(x), T, d, dff, _code(act_kind, _ACTS), _ptr(Wg), _ptr(Wu),
                          _ptr(Wd), _dt(Wu), _ptr(y))
    if s:
        raise OracleError(s, "ppo_dense_ffn")
    return y


def router_stats(g, eps=1e-9):
    """Eq. (entropy_loss), Eq. (load_balance_loss) and the gate-magnitude
    term L_gate over the batch of logits g [B, E].  Returns (L_ent, L_bal,
    L_gate) as floats."""
    lib = load()
    g = np.ascontiguousarray(g, dtype=np.float64)
    T, E = g.shape
    out = np.empty(3, np.float64)
    s = lib.ppo_router_stats(_ptr(g), T, E, float(eps), _ptr(out))
    if s:
        raise OracleError(s, "ppo_router_stats")
    return float(out[0]), float(out[1]), float(out[2])


def rmsnorm_residual(x_prev, y_prev=None, gamma=None, eps=1e-6):
    """x = RMSNorm(x_prev + y_prev) * gamma per row, fp64.  Inputs share one
    storage type; y_prev and gamma may be None."""
    lib = load()
    x_prev = _c(x_prev)
    y_prev = None if y_prev is None else _c(y_prev)
    gamma = None if gamma is None else _c(gamma)
    T, d = x_prev.shape
    dt = _dt(x_prev)
    assert y_prev is None or (y_prev.shape == x_prev.shape and _dt(y_prev) == dt)
    assert gamma is None or (gamma.shape == (d,) and _dt(gamma) == dt)
    out = np.empty((T, d), np.float64)
    s = lib.ppo_rmsnorm_residual(_ptr(x_prev), _ptr(y_prev), _ptr(gamma), dt, T, d, float(eps), _ptr(out))
    if s:
        raise OracleError(s, "ppo_rmsnorm_residual")
    return out


def ffn_sparsity(counts, n_experts):
    """Sec. 4.1: s_FFN of the activated-set sizes counts[L, N] (layer-major).
    Returns (s_FFN, k_sum, hist) with hist[c] = #{(token, layer) : |A| = c},
    c = 0..E."""
    lib = load()
    counts = np.ascontiguousarray(counts, dtype=np.int32)
    if counts.ndim == 1:
        counts = counts[None, :]
    L, N = counts.shape
    E = int(n_experts)
    k_sum = np.zeros(1, np.uint64)
    hist = np.zeros(E + 1, np.uint64)
    s_ffn = np.zeros(1, np.float64)
    s = lib.ppo_ffn_sparsity(_ptr(counts), N, L, E, _ptr(k_sum), _ptr(hist), _ptr(s_ffn))
    if s:
        raise OracleError(s, "ppo_ffn_sparsity")
    return float(s_ffn[0]), int(k_sum[0]), hist.astype(np.int64)


def layer(x, Wr, Wg, Wu, Wd, p, act_kind="swiglu", gate="sigmoid", rule="min_prefix"):
    """Logits, selection and sparse FFN.  Returns (g, counts, ids, y)."""
    lib = load()
    x, Wr, Wu, Wd = _c(x), _c(Wr), _c(Wu), _c(Wd)
    Wg = None if Wg is None else _c(Wg)
    T, d = x.shape
    E = Wr.shape[0]
    dff = Wu.shape[0]
    g = np.empty((T, E), np.float64)
    counts = np.empty(T, np.int32)
    ids = np.empty((T, E), np.int32)
    y = np.empty((T, d), np.float64)
    s = lib.ppo_layer(_ptr(x), _dt(x), T, d, E, dff // E, _code(act_kind, _ACTS),
                      _code(gate, _GATES), _code(rule, _RULES), float(p), _ptr(Wr), _ptr(Wg),
                      _ptr(Wu), _ptr(Wd), _dt(Wu), _ptr(g), _ptr(counts), _ptr(ids), _ptr(y))
    if s:
        raise OracleError(s, "ppo_layer")
    return g, counts, ids, y
