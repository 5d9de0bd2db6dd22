"""Seeded synthetic inputs shaped like the paper's models.

This module holds only shapes and random-number recipes; none of the
method's arithmetic lives here.  Both the CUDA path's tests/benchmark and the
CPU oracle draw their inputs from it.

Recipe (per layer ``l`` of a workload, base seed ``s``):
  * a numpy ``PCG64`` stream per tensor, seeded ``SeedSequence([s, l, k])``
    with k = 0 (W_r), 1 (W_gate), 2 (W_up), 3 (W_down), 4 (x).  numpy's
    generators are bit-reproducible across platforms, so the same seed gives
    the same inputs on any host;
  * x ~ N(0, 1) per element; for the Llama-shaped workloads each token row is
    then rescaled to unit root-mean-square ("RMS-normalised");
  * W_gate, W_up, W_down ~ N(0, 0.02);
  * W_r ~ N(0, s_l / sqrt(d)), so a router logit has standard deviation
    about s_l: s_l = 3 for the tiny, GPT-2-medium and Llama-2-13B shapes, and
    s_l ~ U[2, 4] drawn per layer for the Llama-2-7B / Llama-3-8B shapes;
  * bf16 tensors are the round-to-nearest-even bf16 of the fp32 draws, held
    on the host as ``uint16`` bit patterns.
For speed, ``device_layer`` draws the same distributions with torch's CUDA
generator instead (different values, same recipe): the benchmark uses it for
its many full-size layers, the parity tests use the host recipe above.
"""
from dataclasses import dataclass, field
from typing import Optional, Tuple

import numpy as np

D_EXPERT = 64


@dataclass(frozen=True)
class Workload:
    name: str
    d_model: int
    d_ff: int
    n_experts: int
    n_layers: int
    dtype: str            # "f32" or "bf16"
    act: str              # "relu", "gelu_tanh", "swiglu"
    tokens: Tuple[int, ...]
    ps: Tuple[float, ...]
    router_std: Tuple[float, float]   # (lo, hi): s_l ~ U[lo, hi]; lo == hi means fixed
    rms_norm_x: bool
    description: str = ""
    d_expert: int = D_EXPERT

    @property
    def gated(self) -> bool:
        return self.act == "swiglu"


WORKLOADS = {
    "tiny_relu_f32": Workload(
        "tiny_relu_f32", 256, 1024, 16, 1, "f32", "relu", (64,), (0.5, 0.9, 1.0),
        (3.0, 3.0), False,
        "Tiny ReLU FFN, fp32, d=256, d_ff=1024, E=16, 1 layer, 64 tokens"),
    "gpt2m_gelu_bf16": Workload(
        "gpt2m_gelu_bf16", 1024, 4096, 64, 24, "bf16", "gelu_tanh", (1, 4, 16), (0.5, 0.7, 0.9),
        (3.0, 3.0), False,
        "GPT-2-medium-shaped GELU FFN, bf16, d=1024, d_ff=4096, E=64, 24 layers"),
    "llama2_7b_decode": Workload(
        "llama2_7b_decode", 4096, 11008, 172, 32, "bf16", "swiglu", (1,),
        (0.3, 0.5, 0.7, 0.9, 1.0), (2.0, 4.0), True,
        "Llama-2-7B-shaped SwiGLU FFN, bf16, d=4096, d_ff=11008, E=172, 32 layers, batch-1 decode"),
    "llama3_8b_batched": Workload(
        "llama3_8b_batched", 4096, 14336, 224, 32, "bf16", "swiglu", (1, 8, 32, 64),
        (0.3, 0.5, 0.7, 0.9, 0.95), (2.0, 4.0), True,
        "Llama-3-8B-shaped SwiGLU FFN, bf16, d=4096, d_ff=14336, E=224, 32 layers, batched decode"),
    "llama2_13b_prefill": Workload(
        "llama2_13b_prefill", 5120, 13824, 216, 40, "bf16", "swiglu", (8192,), (0.7,),
        (3.0, 3.0), False,
        "Llama-2-13B-shaped SwiGLU prefill, bf16, d=5120, d_ff=13824, E=216, 40 layers, "
        "4 sequences x 2048 tokens"),
}


def scaled(w: Workload, d_model: int, n_experts: int, name: Optional[str] = None) -> Workload:
    """Same recipe at a smaller shape (for fast parity cases)."""
    from dataclasses import replace
    return replace(w, name=name or (w.name + "_d%d_E%d" % (d_model, n_experts)),
                   d_model=d_model, n_experts=n_experts, d_ff=n_experts * w.d_expert)


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16, returned as uint16 bit patterns."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _rng(seed: int, layer: int, k: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, layer, k])))


def router_scale(w: Workload, seed: int, layer: int) -> float:
    lo, hi = w.router_std
    if lo == hi:
        return lo
    return float(_rng(seed, layer, 5).uniform(lo, hi))


def _cast(a32: np.ndarray, dtype: str) -> np.ndarray:
    return f32_to_bf16_bits(a32) if dtype == "bf16" else a32.astype(np.float32)


def host_tokens(w: Workload, T: int, seed: int = 0, layer: int = 0, stream: int = 4) -> np.ndarray:
    """x [T, d] in the workload's dtype (uint16 bits for bf16)."""
    x = _rng(seed, layer, stream).standard_normal((T, w.d_model), dtype=np.float32)
    if w.rms_norm_x:
        rms = np.sqrt(np.mean(x.astype(np.float64) ** 2, axis=1, keepdims=True))
        x = (x / rms).astype(np.float32)
    return _cast(x, w.dtype)


@dataclass
class HostLayer:
    x: np.ndarray
    Wr: np.ndarray
    Wg: Optional[np.ndarray]
    Wu: np.ndarray
    Wd: np.ndarray
    router_s: float
    workload: Workload = field(repr=False, default=None)


def host_layer(w: Workload, T: int, seed: int = 0, layer: int = 0) -> HostLayer:
    """All tensors of one layer, drawn on the host (see module docstring)."""
    d, dff, E = w.d_model, w.d_ff, w.n_experts
    s = router_scale(w, seed, layer)
    Wr = _rng(seed, layer, 0).standard_normal((E, d), dtype=np.float32) * np.float32(s / np.sqrt(d))
    Wg = None
    if w.gated:
        Wg = _rng(seed, layer, 1).standard_normal((dff, d), dtype=np.float32) * np.float32(0.02)
    Wu = _rng(seed, layer, 2).standard_normal((dff, d), dtype=np.float32) * np.float32(0.02)
    Wd = _rng(seed, layer, 3).standard_normal((d, dff), dtype=np.float32) * np.float32(0.02)
    x = host_tokens(w, T, seed, layer)
    return HostLayer(x=x, Wr=_cast(Wr, w.dtype), Wg=None if Wg is None else _cast(Wg, w.dtype),
                     Wu=_cast(Wu, w.dtype), Wd=_cast(Wd, w.dtype), router_s=s, workload=w)


def host_logits(T: int, E: int, std: float = 3.0, seed: int = 0, layer: int = 0) -> np.ndarray:
    """Synthetic router logits [T, E] (fp32), for the selection-only entry point."""
    return (_rng(seed, layer, 6).standard_normal((T, E), dtype=np.float32) * np.float32(std))


def to_torch(a: np.ndarray, device="cpu"):
    """numpy -> torch, reinterpreting uint16 arrays as bf16."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a))
    if a.dtype == np.uint16:
        t = t.view(torch.bfloat16)
    return t.to(device)


def device_layer(w: Workload, T: int, seed: int, layer: int, device, n_token_sets: int = 1):
    """Same distributions drawn on the GPU with torch's CUDA generator.

    Returns a dict of device tensors; ``x`` has shape [n_token_sets, T, d].
    """
    import torch
    d, dff, E = w.d_model, w.d_ff, w.n_experts
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    gen = torch.Generator(device=device)
    gen.manual_seed((seed * 1_000_003 + layer) & 0x7FFFFFFFFFFFFFFF)
    s = router_scale(w, seed, layer)

    def normal(shape, std):
        t = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
        return (t * std).to(tdt)

    out = {"Wr": normal((E, d), s / np.sqrt(d)),
           "Wg": normal((dff, d), 0.02) if w.gated else None,
           "Wu": normal((dff, d), 0.02),
           "Wd": normal((d, dff), 0.02)}
    x = torch.randn((n_token_sets, T, d), generator=gen, device=device, dtype=torch.float32)
    if w.rms_norm_x:
        x = x / x.pow(2).mean(dim=-1, keepdim=True).sqrt()
    out["x"] = x.to(tdt)
    out["router_s"] = s
    return out
