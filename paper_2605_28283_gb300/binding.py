"""ctypes binding over ``libprunepath.so`` -- argument marshalling only.

Each function has the name and argument order of its C entry point in
``include/prunepath.h``; torch tensors are passed as raw device pointers and
streams as ``cudaStream_t`` handles (default: torch's current stream).  Every
step of the computation runs in the CUDA library; there is no Python or CPU
fallback: if the library is not built, ``load()`` raises.
"""
import ctypes
import os

from . import build as _build

PP_OK, PP_ERR_INVALID_ARG, PP_ERR_SHAPE, PP_ERR_DTYPE, PP_ERR_ALIGN = 0, 1, 2, 3, 4
PP_ERR_WORKSPACE, PP_ERR_CUDA, PP_ERR_TIMEOUT, PP_ERR_CAPACITY, PP_ERR_NONFINITE = 5, 6, 7, 8, 9
PP_ERR_UNSUPPORTED, PP_ERR_HOST = 10, 11
PP_F32, PP_BF16 = 0, 1
PP_ACT_RELU, PP_ACT_GELU_TANH, PP_ACT_SWIGLU = 0, 1, 2
PP_GATE_SIGMOID, PP_GATE_NONE = 0, 1
PP_SEL_MIN_PREFIX, PP_SEL_PAPER, PP_SEL_TOPK, PP_SEL_LTE = 0, 1, 2, 3

ACTS = {"relu": PP_ACT_RELU, "gelu_tanh": PP_ACT_GELU_TANH, "gelu": PP_ACT_GELU_TANH,
        "swiglu": PP_ACT_SWIGLU}
GATES = {"sigmoid": PP_GATE_SIGMOID, "none": PP_GATE_NONE}
RULES = {"min_prefix": PP_SEL_MIN_PREFIX, "paper": PP_SEL_PAPER, "topk": PP_SEL_TOPK, "lte": PP_SEL_LTE}
DTYPES = {"f32": PP_F32, "bf16": PP_BF16}


class pp_desc(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int), ("d_ff", ctypes.c_int), ("n_experts", ctypes.c_int),
                ("d_expert", ctypes.c_int), ("dtype", ctypes.c_int), ("act", ctypes.c_int),
                ("gate", ctypes.c_int), ("rule", ctypes.c_int)]


class pp_selection(ctypes.Structure):
    _fields_ = [("ids", ctypes.c_void_p), ("counts", ctypes.c_void_p), ("gates", ctypes.c_void_p),
                ("logits", ctypes.c_void_p)]


class PPError(RuntimeError):
    def __init__(self, status, what):
        super().__init__("%s failed: %s" % (what, status_name(status)))
        self.status = status


_lib = None
_P, _I, _F, _Z, _LL = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t, ctypes.c_longlong
_PD = ctypes.POINTER(pp_desc)
_PS = ctypes.POINTER(pp_selection)

EXPORTS = {
    "pp_workspace_size": (_Z, [_PD, _I]),
    "pp_workspace_init": (_I, [_P, _Z, _P]),
    "pp_route": (_I, [_PD, _P, _I, _P, _F, _PS, _P, _Z, _P]),
    "pp_select": (_I, [_PD, _P, _I, _F, _PS, _P, _Z, _P]),
    "pp_sparse_ffn": (_I, [_PD, _P, _I, _P, _P, _P, _PS, _P, _P, _Z, _P]),
    "pp_layer": (_I, [_PD, _P, _I, _P, _P, _P, _P, _F, _PS, _P, _P, _Z, _P]),
    "pp_layer_chained": (_I, [_PD, _P, _P, _P, _F, _I, _P, _P, _P, _P, _F, _PS, _P, _P, _P, _Z, _P]),
    "pp_layer_noalloc": (_I, [_PD, _P, _I, _P, _P, _P, _P, _F, _PS, _P, _P, _P]),
    "pp_sparsity_stats": (_I, [_P, _I, _I, _P, _P]),
    "pp_router_stats": (_I, [_PD, _P, _I, _F, _P, _P, _Z, _P]),
    "pp_moefy_cluster": (_I, [_PD, _P, _P, _P, _I, _P, _P, _P, _P]),
    "pp_moefy_permute": (_I, [_PD, _P, _P, _P, _P, _P, _P, _P, _P, _Z, _P]),
    "pp_get_device_status": (_I, [_P, _P]),
    "pp_debug_wait_timeout": (_I, [_P, _Z, _LL, _P]),
    "pp_debug_decode_timeline": (_I, [_PD, _P, _P, _P, _P, _P, _F, _P, _P, _Z, _P, _Z, _P]),
    "pp_status_string": (ctypes.c_char_p, [_I]),
    "pp_version": (ctypes.c_char_p, []),
}


def library_path() -> str:
    return _build.LIB


def load(path: str = None):
    """Load libprunepath.so (raises if it has not been built)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    path = path or library_path()
    if not os.path.exists(path):
        raise RuntimeError("libprunepath.so is not built (%s); run __graft_entry__.build()" % path)
    lib = ctypes.CDLL(path)
    for name, (res, args) in EXPORTS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def status_name(s: int) -> str:
    try:
        return load().pp_status_string(int(s)).decode()
    except RuntimeError:
        return "status %d" % s


def _check(s, what):
    if s != PP_OK:
        raise PPError(s, what)


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def make_desc(d_model, n_experts, dtype="bf16", act="swiglu", gate="sigmoid", rule="min_prefix",
              d_expert=64) -> pp_desc:
    return pp_desc(int(d_model), int(n_experts) * int(d_expert), int(n_experts), int(d_expert),
                   DTYPES.get(dtype, dtype), ACTS.get(act, act), GATES.get(gate, gate),
                   RULES.get(rule, rule))


class Selection:
    """Device tensors of a selection: ids/gates [T, E], counts [T], logits [T, E] or None."""

    def __init__(self, ids, counts, gates, logits=None):
        self.ids, self.counts, self.gates, self.logits = ids, counts, gates, logits

    @classmethod
    def empty(cls, T, E, device, with_logits=True):
        import torch
        return cls(torch.empty((T, E), dtype=torch.int32, device=device),
                   torch.empty((T,), dtype=torch.int32, device=device),
                   torch.empty((T, E), dtype=torch.float32, device=device),
                   torch.empty((T, E), dtype=torch.float32, device=device) if with_logits else None)

    def c(self) -> pp_selection:
        return pp_selection(self.ids.data_ptr(), self.counts.data_ptr(), self.gates.data_ptr(),
                            None if self.logits is None else self.logits.data_ptr())


def pp_workspace_size(desc, T) -> int:
    return int(load().pp_workspace_size(ctypes.byref(desc), int(T)))


def pp_workspace_init(ws, stream=None):
    _check(load().pp_workspace_init(_ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
           "pp_workspace_init")


def alloc_workspace(desc, T, device="cuda", stream=None):
    """A zero-initialised workspace tensor for calls with up to T tokens."""
    import torch
    ws = torch.empty(max(256, pp_workspace_size(desc, T)), dtype=torch.uint8, device=device)
    pp_workspace_init(ws, stream)
    return ws


def _wsargs(ws):
    return _ptr(ws), ws.numel() * ws.element_size()


def pp_route(desc, x, T, W_r, p, out, ws, stream=None):
    sel = out.c()
    _check(load().pp_route(ctypes.byref(desc), _ptr(x), int(T), _ptr(W_r), float(p), ctypes.byref(sel),
                           *_wsargs(ws), _stream(stream)), "pp_route")


def pp_select(desc, logits, T, p, out, ws, stream=None):
    sel = out.c()
    _check(load().pp_select(ctypes.byref(desc), _ptr(logits), int(T), float(p), ctypes.byref(sel),
                            *_wsargs(ws), _stream(stream)), "pp_select")


def pp_sparse_ffn(desc, x, T, W_gate, W_up, W_down, sel, y, ws, stream=None):
    s = sel.c()
    _check(load().pp_sparse_ffn(ctypes.byref(desc), _ptr(x), int(T), _ptr(W_gate), _ptr(W_up),
                                _ptr(W_down), ctypes.byref(s), _ptr(y), *_wsargs(ws), _stream(stream)),
           "pp_sparse_ffn")


def pp_layer(desc, x, T, W_r, W_gate, W_up, W_down, p, sel_out, y, ws, stream=None):
    s = None if sel_out is None else sel_out.c()
    _check(load().pp_layer(ctypes.byref(desc), _ptr(x), int(T), _ptr(W_r), _ptr(W_gate), _ptr(W_up),
                           _ptr(W_down), float(p), None if s is None else ctypes.byref(s), _ptr(y),
                           *_wsargs(ws), _stream(stream)), "pp_layer")


def pp_layer_chained(desc, x_prev, y_prev, gamma, eps, T, W_r, W_gate, W_up, W_down, p, sel_out, x, y, ws,
                     stream=None):
    """x = RMSNorm(x_prev + y_prev) * gamma, then y = pp_layer(x) (y_prev, gamma may be None)."""
    s = None if sel_out is None else sel_out.c()
    _check(load().pp_layer_chained(ctypes.byref(desc), _ptr(x_prev), _ptr(y_prev), _ptr(gamma), float(eps), int(T),
                                   _ptr(W_r), _ptr(W_gate), _ptr(W_up), _ptr(W_down), float(p),
                                   None if s is None else ctypes.byref(s), _ptr(x), _ptr(y), *_wsargs(ws),
                                   _stream(stream)), "pp_layer_chained")


def pp_layer_noalloc(desc, x, T, W_r, W_gate, W_up, W_down, p, sel_out, y, status_out=None, stream=None):
    """pp_layer without a workspace (library-owned static scratch, T <= 4)."""
    s = None if sel_out is None else sel_out.c()
    _check(load().pp_layer_noalloc(ctypes.byref(desc), _ptr(x), int(T), _ptr(W_r), _ptr(W_gate), _ptr(W_up),
                                   _ptr(W_down), float(p), None if s is None else ctypes.byref(s), _ptr(y),
                                   _ptr(status_out), _stream(stream)), "pp_layer_noalloc")


def pp_sparsity_stats(counts, T, n_experts, acc, stream=None):
    _check(load().pp_sparsity_stats(_ptr(counts), int(T), int(n_experts), _ptr(acc), _stream(stream)),
           "pp_sparsity_stats")


def pp_router_stats(desc, logits, T, eps, out, ws, stream=None):
    """L_ent, L_bal, L_gate of the logits [T][E] into out (3 float64, device)."""
    _check(load().pp_router_stats(ctypes.byref(desc), _ptr(logits), int(T), float(eps), _ptr(out),
                                  *_wsargs(ws), _stream(stream)), "pp_router_stats")


def _host(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def pp_moefy_cluster(desc, W_gate, W_up, init, max_iter=100):
    """Balanced k-means of the neurons (host numpy arrays: float32, or uint16
    bf16 bit patterns; init int32 [E]).  Returns (perm, labels, iters,
    objective)."""
    import numpy as np
    W_up = np.ascontiguousarray(W_up)
    W_gate = None if W_gate is None else np.ascontiguousarray(W_gate)
    init = np.ascontiguousarray(init, dtype=np.int32)
    perm = np.empty(desc.d_ff, np.int32)
    labels = np.empty(desc.d_ff, np.int32)
    iters = ctypes.c_int(0)
    obj = ctypes.c_double(0.0)
    _check(load().pp_moefy_cluster(ctypes.byref(desc), _host(W_gate), _host(W_up), _host(init), int(max_iter),
                                   _host(perm), _host(labels), ctypes.byref(iters), ctypes.byref(obj)),
           "pp_moefy_cluster")
    return perm, labels, iters.value, obj.value


def pp_moefy_permute(desc, perm, W_gate, W_up, W_down, W_gate_out, W_up_out, W_down_out, ws, stream=None):
    """Eq. (permuted_weights) on the device: *_out = the weights with neuron j = old neuron perm[j]."""
    _check(load().pp_moefy_permute(ctypes.byref(desc), _ptr(perm), _ptr(W_gate), _ptr(W_up), _ptr(W_down),
                                   _ptr(W_gate_out), _ptr(W_up_out), _ptr(W_down_out), *_wsargs(ws),
                                   _stream(stream)), "pp_moefy_permute")


def pp_get_device_status(ws, stream=None) -> int:
    return int(load().pp_get_device_status(_ptr(ws), _stream(stream)))


def pp_debug_decode_timeline(desc, x, W_r, W_gate, W_up, W_down, p, y, ws, stamps, stream=None):
    """stamps: a device uint64 tensor of at least 256 * 16 entries."""
    _check(load().pp_debug_decode_timeline(ctypes.byref(desc), _ptr(x), _ptr(W_r), _ptr(W_gate), _ptr(W_up),
                                           _ptr(W_down), float(p), _ptr(y), *_wsargs(ws), _ptr(stamps),
                                           stamps.numel() * stamps.element_size(), _stream(stream)),
           "pp_debug_decode_timeline")


def pp_debug_wait_timeout(ws, timeout_ns, stream=None):
    _check(load().pp_debug_wait_timeout(*_wsargs(ws), int(timeout_ns), _stream(stream)),
           "pp_debug_wait_timeout")


def pp_status_string(s) -> str:
    return load().pp_status_string(int(s)).decode()


def pp_version() -> str:
    return load().pp_version().decode()
