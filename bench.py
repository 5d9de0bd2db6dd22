#!/usr/bin/env python3
"""Sparse-FFN decode benchmark (PrunePath hot path on GB300).

Workload (default): the Llama-2-7B-shaped SwiGLU FFN, bf16, d=4096,
d_ff=11008, E=172 experts of 64 neurons, 32 stacked layers, batch-1 decode,
p = 0.7.  One step = one token through all 32 layers: for each layer one
``pp_layer`` call (router GEMV, softmax, sort, cumulative-mass cut, sparse
SwiGLU FFN over the selected experts).  Synthetic weights/inputs (seeded
torch CUDA generator, recipe in paper_2605_28283_gb300/workloads.py); each
layer cycles through a pool of pre-drawn token vectors so the expert choice
changes every step.  The 32 launches of a step are one CUDA graph; L2 is
flushed (256 MiB write) between steps, outside the timed events.

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle
instead (the reference arm of this build: a plain fp64 implementation).
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "sparse-FFN decode tokens/s; HBM GB/s on touched expert bytes vs peak"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama2_7b_decode")
    ap.add_argument("--p", type=float, default=0.7)
    ap.add_argument("--rule", default="min_prefix", choices=["min_prefix", "paper", "topk", "lte"],
                    help="activation rule of the headline timing (p is k for topk, delta for lte)")
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--pool", type=int, default=0,
                    help="distinct token sets per layer (default 64 for decode batches, 1 for prefill)")
    ap.add_argument("--sweep", default="0.3,0.5,0.7,0.9,1.0", help="p values for the sweep ('' = none)")
    ap.add_argument("--sweep-steps", type=int, default=400)
    ap.add_argument("--rules", default="topk:6,lte:0.995",
                    help="other activation rules timed on the same kernels, rule:param ('' = none)")
    ap.add_argument("--no-flush", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--layers", type=int, default=0, help="override the layer count (profiling runs)")
    ap.add_argument("--skip-extras", action="store_true",
                    help="only the headline timing (no warm/e2e/CPU legs); for profiler runs")
    ap.add_argument("--configs", default="llama3_8b_batched:64:0.7,llama2_13b_prefill:8192:0.7:1,gpt2m_gelu_bf16:4:0.7",
                    help="further workloads timed after the headline, workload:batch:p[:layers] ('' = none)")
    ap.add_argument("--config-steps", type=int, default=300)
    ap.add_argument("--timeline", action="store_true",
                    help="phase timeline of the fused decode kernel (B = 1) instead of the benchmark")
    return ap.parse_args()


def default_pool(batch):
    """Distinct token sets per layer that a step cycles through: 64 for
    decode batches (expert choice changes every step), 1 for prefill."""
    return 64 if batch <= 128 else 1


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(v, world, device):
    """The largest of the ranks' values (every rank gets it); v itself for one rank."""
    if world == 1:
        return v
    import torch
    t = torch.tensor([v], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(units_per_rank, seconds, world, device):
    """Whole-job throughput of `world` independent replicas that each
    processed units_per_rank units: all units over the slowest rank's time.
    Returns (units/s, slowest time)."""
    slowest = max_over_ranks(seconds, world, device)
    return world * units_per_rank / slowest, slowest


def load_peaks():
    """(HBM GB/s, dense bf16 TFLOP/s sustained, kind): measured copy and GEMM
    figures for this GPU pool, else the recipe's fallback numbers."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), float(pk.get("bf16_tflops_sustained", pk["bf16_tflops"])), "measured"
    except Exception:
        return 6800.0, 1700.0, "fallback"


# --------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "50"], stdout=self.out,
                stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.out.close()
        rows = []
        for line in open(self.path):
            parts = [s.strip() for s in line.split(",")]
            if len(parts) != 7:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[3:]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# -------------------------------------------------------------- workload
def make_layers(w, B, pool, seed, device):
    import torch
    from paper_2605_28283_gb300 import workloads as wl
    layers = []
    for l in range(w.n_layers):
        t = wl.device_layer(w, B, seed, l, device, n_token_sets=pool)
        t["y"] = torch.empty((B, w.d_model), dtype=t["x"].dtype, device=device)
        layers.append(t)
    return layers


def capture_graphs(pp, desc, layers, p, B, pool, ws, stream):
    import torch
    graphs = []
    with torch.cuda.stream(stream):
        for i in range(pool):  # warm the launch path once per pool entry outside capture
            for L in layers:
                pp.pp_layer(desc, L["x"][i], B, L["Wr"], L["Wg"], L["Wu"], L["Wd"], p, None, L["y"], ws,
                            stream=stream)
        stream.synchronize()
        for i in range(pool):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for L in layers:
                    pp.pp_layer(desc, L["x"][i], B, L["Wr"], L["Wg"], L["Wu"], L["Wd"], p, None, L["y"],
                                ws, stream=stream)
            graphs.append(g)
    return graphs


def time_graphs(graphs, steps, warmup, flush_buf, stream, profile_range=False):
    """Per-step CUDA-event timing on `stream`; L2 flushed between steps.
    With profile_range, the timed loop is bracketed by cudaProfilerStart/Stop
    so that `ncu --profile-from-start off` lists exactly its launches."""
    import torch
    with torch.cuda.stream(stream):
        for i in range(warmup):
            graphs[i % len(graphs)].replay()
        stream.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps)]
        if profile_range:
            torch.cuda.profiler.start()
        for i in range(steps):
            if flush_buf is not None:
                flush_buf.add_(1)
            ev[i][0].record(stream)
            graphs[i % len(graphs)].replay()
            ev[i][1].record(stream)
        stream.synchronize()
        if profile_range:
            torch.cuda.profiler.stop()
    return [a.elapsed_time(b) for a, b in ev]  # ms


def selection_stats(pp, desc, layers, w, p, B, pool, ws):
    """k per (pool entry, layer, token) and the union size |U| per (pool
    entry, layer) via pp_route on the same inputs, and the s_FFN accumulators
    (sum of k and its histogram, Sec. 4.1) from the library's own
    pp_sparsity_stats over the same counts."""
    import numpy as np
    import torch
    ks = torch.empty((pool, len(layers), B), dtype=torch.int64)
    union = torch.empty((pool, len(layers)), dtype=torch.int64)
    sel = pp.Selection.empty(B, w.n_experts, "cuda", with_logits=False)
    acc = torch.zeros(w.n_experts + 2, dtype=torch.int64, device="cuda")
    for i in range(pool):
        for l, L in enumerate(layers):
            pp.pp_route(desc, L["x"][i], B, L["Wr"], p, sel, ws)
            pp.pp_sparsity_stats(sel.counts, B, w.n_experts, acc)
            c = sel.counts.cpu()
            ks[i, l] = c.long()
            ids = sel.ids.cpu().numpy()
            cn = c.numpy()
            mask = np.arange(ids.shape[1])[None, :] < cn[:, None]
            union[i, l] = len(np.unique(ids[mask]))
    return ks, union, acc.cpu()


def layer_bytes(w, B, n_union):
    """Algorithmic HBM bytes of one pp_layer call: W_r, the union of the
    selected expert blocks (gate+up rows and down column block), x and y."""
    esz = 2 if w.dtype == "bf16" else 4
    mats = 3 if w.gated else 2
    router = w.n_experts * w.d_model * esz
    expert = mats * 64 * w.d_model * esz
    act = 2 * B * w.d_model * esz
    return router + n_union * expert + act, n_union * expert


def layer_flops(w, B, k_sum):
    """Algorithmic FLOPs of one pp_layer call: router GEMV/GEMM plus, per
    (token, activated expert), the gate/up and down products of a 64-wide block."""
    mats = 3 if w.gated else 2
    return 2.0 * B * w.n_experts * w.d_model + 2.0 * k_sum * mats * 64 * w.d_model


def path_kind(w, B):
    """Which kernels serve a pp_layer call: the fused decode kernel (bf16 up to
    4 tokens, every fp32 call) or the grouped tensor-core path."""
    return "decode" if (B <= 4 or w.dtype == "f32") else "grouped"


def kernel_traffic(workload, p, B, kind="decode"):
    """DRAM bytes per layer call measured by ncu (committed summary), valid
    only while the kernel's sources are unchanged; None otherwise."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        rec = json.load(open(path))
    except Exception:
        return None
    ent = rec.get("entries", {}).get("%s@p%g@B%d" % (workload, p, B))
    if ent is None or ent.get("sources_sha") != sources_sha(kind):
        return None
    return ent.get("dram_bytes_per_layer")


# source files each timed kernel is built from: a DRAM-traffic record stays
# valid while these are unchanged
KERNEL_SOURCES = {
    "decode": ["decode.cu", "pp_common.cuh", "pp_select.cuh", "pp_kernels.h", "api.cu"],
    "grouped": ["grouped.cu", "pp_common.cuh", "pp_select.cuh", "pp_tc.cuh", "pp_kernels.h", "api.cu"],
}


def sources_sha(kind="decode"):
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2605_28283_gb300", "csrc")
    for n in sorted(KERNEL_SOURCES[kind]):
        with open(os.path.join(d, n), "rb") as f:
            h.update(n.encode() + f.read())
    return h.hexdigest()[:16]


def roofline(w, B, p, bytes_per_launch, flops_per_launch, per_launch_ms):
    """Roofline record of one pp_layer call: the bound is whichever of HBM
    traffic and tensor work takes longer at the measured peaks; both
    fractions are reported."""
    hbm_peak, tc_peak, peak_kind = load_peaks()
    sec = per_launch_ms / 1e3
    hbm_gbs = bytes_per_launch / sec / 1e9
    tflops = flops_per_launch / sec / 1e12
    tensor_bound = flops_per_launch / (tc_peak * 1e12) > bytes_per_launch / (hbm_peak * 1e9)
    kind = path_kind(w, B)
    rec = {"bound": "tensor" if tensor_bound else "hbm",
           "unit": "TFLOP/s" if tensor_bound else "GB/s",
           "achieved": tflops if tensor_bound else hbm_gbs,
           "peak": tc_peak if tensor_bound else hbm_peak,
           "bytes_per_launch": bytes_per_launch, "flops_per_launch": flops_per_launch,
           "hbm_frac": hbm_gbs / hbm_peak, "tensor_frac": tflops / tc_peak,
           "traffic": kernel_traffic(w.name, p, B, kind), "peak_kind": peak_kind,
           "kernel": "decode_layer_kernel" if kind == "decode" else "pp_layer (grouped tcgen05 path, all kernels)",
           "per": "one pp_layer call (one layer)", "launch_ms": per_launch_ms}
    rec["frac"] = rec["achieved"] / rec["peak"]
    return rec


def measure(pp, w, B, p, steps, warmup, pool, seed, device, stream, flush, world, rule="min_prefix",
            gate="sigmoid", layers=None, profile_range=False, clocks=True):
    """Times `steps` steps (one token set through every layer, one CUDA graph
    per pool entry) and derives throughput, roofline and selection statistics
    from the actual selections of the pool entries."""
    import numpy as np
    import torch
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act, gate, rule)
    ws = pp.alloc_workspace(desc, B)
    if layers is None:
        layers = make_layers(w, B, pool, seed, device)
    # the workspace is zeroed and the inputs drawn on torch's current stream;
    # the library's launches go to `stream`
    torch.cuda.synchronize()
    pf = float(np.float32(p))
    graphs = capture_graphs(pp, desc, layers, pf, B, pool, ws, stream)
    sampler = ClockSampler(torch.cuda.current_device()) if clocks else None
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
    times = time_graphs(graphs, steps, warmup, flush, stream, profile_range=profile_range)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clk = sampler.stop() if sampler else None
    del graphs
    value, slowest_s = replica_throughput(B * steps, sum(times) / 1e3, world, device)
    status = pp.pp_get_device_status(ws)
    if status != pp.PP_OK:
        raise SystemExit("device status (%s B=%d p=%g): %s" % (w.name, B, p, pp.status_name(status)))
    ks, union, acc = selection_stats(pp, desc, layers, w, pf, B, pool, ws)
    step_ids = np.arange(steps) % pool
    tot_b = exp_b = tot_f = 0.0
    for i in range(pool):
        n_i = int((step_ids == i).sum())
        for l in range(w.n_layers):
            a, e = layer_bytes(w, B, int(union[i, l]))
            tot_b += n_i * a
            exp_b += n_i * e
            tot_f += n_i * layer_flops(w, B, int(ks[i, l].sum()))
    seconds = sum(times) / 1e3
    launches = steps * w.n_layers
    per_launch_ms = sum(times) / launches   # step time / L: includes the in-graph launch gaps
    hbm_peak = load_peaks()[0]
    n_sel = pool * w.n_layers * B
    k_sum = int(acc[0])
    return {"tokens_per_s": value, "ms_per_step": slowest_s * 1e3 / steps, "steps": steps, "seconds": seconds,
            "launches": launches, "per_launch_ms": per_launch_ms,
            "roofline": roofline(w, B, p, tot_b / launches, tot_f / launches, per_launch_ms),
            "expert_gbs": exp_b / seconds / 1e9, "total_gbs": tot_b / seconds / 1e9,
            "frac_of_hbm_peak": tot_b / seconds / 1e9 / hbm_peak, "tflops": tot_f / seconds / 1e12,
            "k_mean": k_sum / n_sel, "k_min": int(ks.min()), "k_max": int(ks.max()),
            "union_mean": float(union.float().mean()),
            "s_ffn": 1.0 - k_sum / (n_sel * w.n_experts),
            "s_ffn_from": "pp_sparsity_stats over the pool's pp_route counts (%d token-layers)" % n_sel,
            "clocks": clk, "ws": ws, "desc": desc, "layers": layers}


# ------------------------------------------------------------ CPU oracle
def cpu_env():
    """Host cores: all of them, the ones this process may run on, and the
    OpenMP threads the oracle's token loops may use."""
    aff = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    omp = int(os.environ.get("OMP_NUM_THREADS", aff))
    return {"cpu_count": os.cpu_count(), "affinity_cores": aff, "omp_threads": omp}


def oracle_sample_inputs(w, B, seed, n_layers=3, n_token_sets=8):
    """Host inputs of the bounded oracle sample: n_layers distinct layers,
    each with n_token_sets distinct token sets (the GPU arm likewise cycles
    distinct token sets through distinct layers)."""
    from paper_2605_28283_gb300 import workloads as wl
    n_layers = max(1, min(n_layers, w.n_layers))
    out = []
    for l in range(n_layers):
        L = wl.host_layer(w, B, seed=seed, layer=l)
        toks = [L.x] + [wl.host_tokens(w, B, seed, l, stream=16 + j) for j in range(n_token_sets - 1)]
        out.append((L, toks))
    return out


def oracle_calls(w, sample, p, B, seconds=None, calls=None):
    """Runs single-layer oracle calls (logits, selection, sparse FFN), call i
    on layer i mod n and on that layer's token set (i div n) mod m, until
    `seconds` have passed or `calls` calls are done.  Returns (calls, s)."""
    import numpy as np
    import oracle
    oracle.load()
    n, m = len(sample), len(sample[0][1])
    pf = float(np.float32(p))
    done = 0
    t0 = time.perf_counter()
    while True:
        L, toks = sample[done % n]
        oracle.layer(toks[(done // n) % m], L.Wr, L.Wg, L.Wu, L.Wd, pf, w.act, "sigmoid")
        done += 1
        el = time.perf_counter() - t0
        if (seconds is not None and el >= seconds) or (calls is not None and done >= calls):
            return done, el


def oracle_record(w, B, calls, el, n_layers, n_sets, what):
    env = cpu_env()
    per_layer = el / calls
    return {"value": B / (per_layer * w.n_layers), "unit": "tokens/s", "cores": max(1, min(env["omp_threads"], B)),
            "kind": "oracle", **env,
            "sample": "%s: %d single-layer calls x %d token(s), cycling %d distinct layers x %d distinct token "
                      "sets (%.1f s CPU), scaled to %d layers" % (what, calls, B, n_layers, n_sets, el, w.n_layers)}


def run_oracle_sample(w, seconds, seed, p=0.7, B=1):
    """The cpu_baseline leg: the oracle as it stands on a bounded sample of
    the workload, about `seconds` of CPU work."""
    sample = oracle_sample_inputs(w, B, seed)
    oracle_calls(w, sample, p, B, calls=1)   # load and first-touch
    calls, el = oracle_calls(w, sample, p, B, seconds=seconds)
    return oracle_record(w, B, calls, el, len(sample), len(sample[0][1]), "cpu_baseline leg")


def config_dict(w, B, p, pool, world, no_flush):
    return {"workload": w.name, "d_model": w.d_model, "d_ff": w.d_ff, "n_experts": w.n_experts,
            "d_expert": 64, "layers": w.n_layers, "batch": B, "p": p, "act": w.act, "token_pool": pool,
            "l2": "no flush (warm)" if no_flush else "flushed between steps (256 MiB write, untimed)",
            "parallelism": "replicas" if world > 1 else "single GPU"}


def run_reference(args):
    """Reference arm: the CPU oracle as it stands, timed on the host cores on
    the same workload, sampled exactly as the cpu_baseline leg samples it."""
    rank, world, _ = dist_env()
    from paper_2605_28283_gb300 import workloads as wl
    w = wl.WORKLOADS[args.workload]
    if rank != 0:
        return
    B = args.batch
    sample = oracle_sample_inputs(w, B, args.seed)
    oracle_calls(w, sample, args.p, B, calls=max(1, min(args.warmup, 3)))
    # each step is one single-layer call; the run is capped at about two minutes
    steps, el = oracle_calls(w, sample, args.p, B, calls=max(1, min(args.steps, 5000)), seconds=120.0)
    rec = oracle_record(w, B, steps, el, len(sample), len(sample[0][1]), "reference arm")
    value = rec["value"]
    out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus, "steps": steps,
           "warmup": args.warmup, "ms_per_step": el / steps * w.n_layers * 1e3, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
           "config": config_dict(w, B, args.p, args.pool, world, args.no_flush),
           "cpu_baseline": rec,
           "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out))


# -------------------------------------------------------------- timeline
STAMP_NAMES = ["entry", "released", "x", "router", "selected", "union", "issued4", "phase4", "first_h", "phase6",
               "end", "logits_in", "cut", "cand", "landed4"]


def timeline_summary(st):
    """st: [steps, layers, CTAs, 16] global-timer stamps (0 = phase skipped).
    Per launch, times are taken from the first CTA's release (the previous
    grid on the stream complete).  The timer advances in steps of a few
    hundred ns, so per phase the mean over CTAs (and the mean of the
    per-launch maximum) is reported, averaged over launches, in
    microseconds; also the gap from one launch's last CTA end to the next
    launch's release."""
    import numpy as np
    rows = {n: ([], []) for n in STAMP_NAMES}
    gaps = []
    S, L = st.shape[0], st.shape[1]
    for s in range(S):
        prev_end = None
        for l in range(L):
            a = st[s, l].astype(np.float64)
            rel = a[:, 1][a[:, 1] > 0]
            if rel.size == 0:
                continue
            t0 = rel.min()
            for i, n in enumerate(STAMP_NAMES):
                v = a[:, i][a[:, i] > 0]
                if v.size:
                    rows[n][0].append(np.mean(v - t0) / 1e3)
                    rows[n][1].append((v - t0).max() / 1e3)
            if prev_end is not None:
                gaps.append((t0 - prev_end) / 1e3)
            ends = a[:, 10][a[:, 10] > 0]
            prev_end = ends.max() if ends.size else None
    out = {n: {"mean_cta_us": float(np.mean(m)), "last_cta_us": float(np.mean(x))}
           for n, (m, x) in rows.items() if m}
    out["gap_last_end_to_next_release_us"] = float(np.mean(gaps)) if gaps else None
    return out


def run_timeline(args):
    """Headline workload (B = 1) through pp_debug_decode_timeline: the same
    kernel as pp_layer plus global-timer stamps at its phase boundaries; L
    layers per step back to back in one CUDA graph, as in the benchmark."""
    import numpy as np
    import torch
    from paper_2605_28283_gb300 import binding as pp
    from paper_2605_28283_gb300 import workloads as wl
    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    pp.load()
    w = wl.WORKLOADS[args.workload]
    if args.layers:
        from dataclasses import replace
        w = replace(w, n_layers=args.layers)
    pool = min(args.pool, 16)
    layers = make_layers(w, 1, pool, args.seed, device)
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    ws = pp.alloc_workspace(desc, 1)
    stamps = torch.zeros((w.n_layers, 256 * 16), dtype=torch.int64, device=device)
    flush = None if args.no_flush else torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=device)
    stream = torch.cuda.Stream()
    pf = float(np.float32(args.p))
    torch.cuda.synchronize()

    def step(i):
        for l, L in enumerate(layers):
            pp.pp_debug_decode_timeline(desc, L["x"][i], L["Wr"], L["Wg"], L["Wu"], L["Wd"], pf, L["y"], ws,
                                        stamps[l], stream=stream)
    graphs = []
    with torch.cuda.stream(stream):
        for i in range(pool):
            step(i)
        stream.synchronize()
        for i in range(pool):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                step(i)
            graphs.append(g)
        for i in range(args.warmup):
            graphs[i % pool].replay()
        out = []
        for i in range(args.steps):
            stamps.zero_()
            if flush is not None:
                flush.add_(1)
            graphs[i % pool].replay()
            stream.synchronize()
            out.append(stamps.view(w.n_layers, 256, 16).cpu().numpy())
    if pp.pp_get_device_status(ws) != pp.PP_OK:
        raise SystemExit("device status: %s" % pp.status_name(pp.pp_get_device_status(ws)))
    sm = torch.cuda.get_device_properties(0).multi_processor_count
    st = np.stack(out)[:, :, :sm, :]
    res = {"what": "decode_layer_kernel phase timeline (timeline instantiation, one stamp set per CTA)",
           "workload": w.name, "layers": w.n_layers, "p": args.p, "steps": args.steps, "token_pool": pool,
           "l2": "no flush" if args.no_flush else "flushed between steps", "phases": timeline_summary(st)}
    print(json.dumps(res))


# ------------------------------------------------------------------ main
def public(m):
    """A measurement record without its device objects."""
    return {k: v for k, v in m.items() if k not in ("ws", "desc", "layers")}


def main():
    args = parse()
    if args.pool <= 0:
        args.pool = default_pool(args.batch)
    if args.impl == "reference":
        return run_reference(args)
    if args.timeline:
        return run_timeline(args)
    import numpy as np
    import torch
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    device = torch.device("cuda", torch.cuda.current_device())
    from paper_2605_28283_gb300 import binding as pp
    from paper_2605_28283_gb300 import workloads as wl
    pp.load()
    w = wl.WORKLOADS[args.workload]
    if args.layers:
        from dataclasses import replace
        w = replace(w, n_layers=args.layers)
    B = args.batch
    stream = torch.cuda.Stream()
    flush = None if args.no_flush else torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=device)
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    # ---- headline: p = args.p
    pf = float(np.float32(args.p))
    head = measure(pp, w, B, args.p, args.steps, args.warmup, args.pool, args.seed, device, stream, flush, world,
                   rule=args.rule, gate="none" if args.rule == "lte" else "sigmoid", profile_range=True)
    desc, ws, layers = head["desc"], head["ws"], head["layers"]
    value, ms_per_step, roof = head["tokens_per_s"], head["ms_per_step"], head["roofline"]
    head_rec = public(head)
    kernels_per_layer = 1 if path_kind(w, B) == "decode" else 9

    if args.skip_extras:
        if rank == 0:
            print(json.dumps({"metric": METRIC, "value": value, "unit": "tokens/s", "ms_per_step": ms_per_step,
                              "workload": w.name, "layers": w.n_layers, "p": args.p, "batch": B,
                              "launch_ms": head["per_launch_ms"], "bytes_per_launch": roof["bytes_per_launch"],
                              "flops_per_launch": roof["flops_per_launch"], "roofline_bound": roof["bound"],
                              "achieved": roof["achieved"], "peak": roof["peak"], "frac": roof["frac"],
                              "sources_sha": sources_sha(path_kind(w, B))}))
        return

    # ---- p sweep (same kernels), speedup vs dense p >= 1
    sweep = {}
    for ps in [float(v) for v in args.sweep.split(",") if v]:
        m = measure(pp, w, B, ps, args.sweep_steps, 5, args.pool, args.seed, device, stream, flush, world,
                    layers=layers, clocks=False)
        sweep["%g" % ps] = {k: m[k] for k in ("tokens_per_s", "ms_per_step", "k_mean", "s_ffn", "expert_gbs",
                                              "total_gbs", "frac_of_hbm_peak")}
    dense = sweep.get("1")
    if dense:
        for v in sweep.values():
            v["speedup_vs_p1"] = v["tokens_per_s"] / dense["tokens_per_s"]

    # ---- the other activation rules (top-k, LTE's threshold) on the same kernels
    rules = {}
    for item in [v for v in args.rules.split(",") if v]:
        rname, rp = item.split(":")
        m = measure(pp, w, B, float(rp), args.sweep_steps, 5, args.pool, args.seed, device, stream, flush, world,
                    rule=rname, gate="none" if rname == "lte" else "sigmoid", layers=layers, clocks=False)
        rules[item] = {k: m[k] for k in ("tokens_per_s", "k_mean", "s_ffn", "total_gbs", "frac_of_hbm_peak")}

    # ---- chained decode step: layer l takes x_l = RMSNorm(x_{l-1} + y_{l-1}) (pp_layer_chained), so
    # every layer reads the previous layer's output; one CUDA graph per pool entry
    chained = None
    if B <= 4:
        xs_c = [torch.empty((B, w.d_model), dtype=layers[0]["x"].dtype, device=device) for _ in range(w.n_layers)]
        ys_c = [torch.empty_like(xs_c[0]) for _ in range(w.n_layers)]

        def chain_step(i):
            for l, L in enumerate(layers):
                x_prev = L["x"][i] if l == 0 else xs_c[l - 1]
                y_prev = None if l == 0 else ys_c[l - 1]
                pp.pp_layer_chained(desc, x_prev, y_prev, None, 1e-6, B, L["Wr"], L["Wg"], L["Wu"], L["Wd"], pf,
                                    None, xs_c[l], ys_c[l], ws, stream=stream)
        gs = []
        with torch.cuda.stream(stream):
            for i in range(args.pool):
                chain_step(i)
            stream.synchronize()
            for i in range(args.pool):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    chain_step(i)
                gs.append(g)
        tm = time_graphs(gs, args.sweep_steps, 5, flush, stream)
        if pp.pp_get_device_status(ws) != pp.PP_OK:
            raise SystemExit("device status after the chained leg: %s" % pp.status_name(pp.pp_get_device_status(ws)))
        chained = {"tokens_per_s": B * args.sweep_steps / (sum(tm) / 1e3), "ms_per_step": sum(tm) / args.sweep_steps,
                   "what": "%d layers chained through pp_layer_chained: x_l = RMSNorm(x_(l-1) + y_(l-1)) formed "
                           "in the fused decode kernel's prologue, layer 0 from the token input" % w.n_layers}
        del gs

    # ---- warm-L2 number (no flush), for context
    graphs = capture_graphs(pp, desc, layers, pf, B, args.pool, ws, stream)
    warm = time_graphs(graphs, min(args.steps, 500), 5, None, stream)
    warm_tok_s = B * len(warm) / (sum(warm) / 1e3)
    del graphs

    # ---- end to end through the public API with host buffers.  Every step
    # copies the L layer inputs from pinned host memory in one transfer,
    # replays a CUDA graph of the L pp_layer calls (captured once through
    # the binding) and reads the L outputs back; the host waits for them.
    esz = 2 if w.dtype == "bf16" else 4
    dt = layers[0]["x"].dtype
    npool = min(args.pool, 16)
    x_host = torch.empty((npool, w.n_layers, B, w.d_model), dtype=dt, pin_memory=True)
    for i in range(npool):
        for l, L in enumerate(layers):
            x_host[i, l].copy_(L["x"][i].cpu())
    y_host = torch.empty((w.n_layers, B, w.d_model), dtype=dt, pin_memory=True)
    x_dev = torch.empty((w.n_layers, B, w.d_model), dtype=dt, device=device)
    y_dev = torch.empty_like(x_dev)

    def e2e_layers():
        for l, L in enumerate(layers):
            pp.pp_layer(desc, x_dev[l], B, L["Wr"], L["Wg"], L["Wu"], L["Wd"], pf, None, y_dev[l], ws,
                        stream=stream)

    e2e_steps = min(args.steps, 500)
    with torch.cuda.stream(stream):
        e2e_layers()
        stream.synchronize()
        g_e2e = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_e2e, stream=stream):
            e2e_layers()
        timings = {}
        for mode in ("graph", "eager"):
            for rep in range(2):
                barrier()
                t0 = time.perf_counter()
                for i in range(e2e_steps if rep else 5):
                    x_dev.copy_(x_host[i % npool], non_blocking=True)
                    if mode == "graph":
                        g_e2e.replay()
                    else:
                        e2e_layers()
                    y_host.copy_(y_dev, non_blocking=True)
                    stream.synchronize()
                timings[mode] = time.perf_counter() - t0
    del g_e2e
    e2e = {"value": replica_throughput(B * e2e_steps, timings["graph"], world, device)[0],
           "unit": "tokens/s", "h2d_bytes_per_step": w.n_layers * B * w.d_model * esz,
           "d2h_bytes_per_step": w.n_layers * B * w.d_model * esz,
           "path": "pp_layer via the ctypes binding, %d calls captured once in a CUDA graph; per step one "
                   "pinned H2D copy of the %d layer inputs, graph replay, one D2H copy of the %d outputs, "
                   "host synchronisation" % (w.n_layers, w.n_layers, w.n_layers),
           "eager_value": replica_throughput(B * e2e_steps, timings["eager"], world, device)[0],
           "eager_path": "the same with the %d pp_layer calls made eagerly every step" % w.n_layers}

    # ---- router statistics (L_ent, L_bal, L_gate) over a batch of 8192 tokens' logits
    T_st = 8192
    g_st = torch.randn((T_st, w.n_experts), device=device) * 3.0
    ws_st = pp.alloc_workspace(desc, T_st)
    out_st = torch.empty(3, dtype=torch.float64, device=device)
    torch.cuda.synchronize()  # inputs and workspace were made on torch's current stream
    with torch.cuda.stream(stream):
        for _ in range(5):
            pp.pp_router_stats(desc, g_st, T_st, 1e-9, out_st, ws_st, stream=stream)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n_st = 200
        e0.record(stream)
        for _ in range(n_st):
            pp.pp_router_stats(desc, g_st, T_st, 1e-9, out_st, ws_st, stream=stream)
        e1.record(stream)
        stream.synchronize()
    us_st = e0.elapsed_time(e1) * 1e3 / n_st
    router_stats = {"tokens": T_st, "experts": w.n_experts, "us_per_call": us_st,
                    "gbs": T_st * w.n_experts * 4 / (us_st * 1e-6) / 1e9,
                    "note": "two launches (per-block parts, fixed-order final sum); logits L2-resident"}

    # ---- MoEfication repacking (Eq. permuted_weights) of one layer's weights by a random permutation
    L0 = layers[0]
    perm_d = torch.randperm(w.d_ff, device=device).to(torch.int32)
    outs = [None if L0["Wg"] is None else torch.empty_like(L0["Wg"]), torch.empty_like(L0["Wu"]),
            torch.empty_like(L0["Wd"])]
    ws_mp = pp.alloc_workspace(desc, 0)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for _ in range(3):
            pp.pp_moefy_permute(desc, perm_d, L0["Wg"], L0["Wu"], L0["Wd"], *outs, ws_mp, stream=stream)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n_mp = 20
        e0.record(stream)
        for _ in range(n_mp):
            pp.pp_moefy_permute(desc, perm_d, L0["Wg"], L0["Wu"], L0["Wd"], *outs, ws_mp, stream=stream)
        e1.record(stream)
        stream.synchronize()
    if pp.pp_get_device_status(ws_mp) != pp.PP_OK:
        raise SystemExit("device status after the repacking leg: %s" % pp.status_name(pp.pp_get_device_status(ws_mp)))
    pl = perm_d.long()
    ok = torch.equal(outs[1][:64], L0["Wu"][pl[:64]]) and torch.equal(outs[2][:, :64], L0["Wd"][:, pl[:64]])
    us_mp = e0.elapsed_time(e1) * 1e3 / n_mp
    n_mat = 3 if L0["Wg"] is not None else 2
    b_mp = 2 * n_mat * w.d_ff * w.d_model * L0["Wu"].element_size()
    moefy_permute = {"us_per_call": us_mp, "bytes": b_mp, "gbs": b_mp / (us_mp * 1e-6) / 1e9,
                     "frac_of_hbm_peak": b_mp / (us_mp * 1e-6) / 1e9 / load_peaks()[0], "spot_check": bool(ok),
                     "what": "pp_moefy_permute of one layer (W_gate/W_up rows, W_down columns) by a random "
                             "permutation; bytes = read + write of the three matrices"}
    del outs, ws_mp, head, layers, desc, ws
    torch.cuda.empty_cache()

    # ---- the other workload shapes: each timed on its own, with its own roofline and clocks
    configs = {}
    for item in [v for v in args.configs.split(",") if v]:
        parts = item.split(":")
        cw = wl.WORKLOADS[parts[0]]
        cB, cp = int(parts[1]), float(parts[2])
        if len(parts) > 3:
            from dataclasses import replace
            cw = replace(cw, n_layers=int(parts[3]))
        full_layers = wl.WORKLOADS[parts[0]].n_layers
        cpool = default_pool(cB)
        m = measure(pp, cw, cB, cp, args.config_steps, max(args.warmup, 5), cpool, args.seed, device, stream,
                    flush, world)
        rec = public(m)
        rec["config"] = config_dict(cw, cB, cp, cpool, world, args.no_flush)
        rec["gpu_launches"] = m["launches"] * (1 if path_kind(cw, cB) == "decode" else 9)
        if cw.n_layers != full_layers:
            rec["model_tokens_per_s"] = m["tokens_per_s"] * cw.n_layers / full_layers
            rec["scaling_note"] = ("timed on %d of the model's %d layers (same shape, independently drawn); "
                                   "model_tokens_per_s = tokens_per_s x %d / %d, layers running back to back"
                                   % (cw.n_layers, full_layers, cw.n_layers, full_layers))
        configs["%s@B%d@p%g" % (cw.name, cB, cp)] = rec
        del m
        torch.cuda.empty_cache()

    out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
           "config": config_dict(w, B, args.p, args.pool, world, args.no_flush),
           "roofline": roof,
           "expert_bytes": {"gbs": head_rec["expert_gbs"], "frac_of_peak": head_rec["expert_gbs"] / load_peaks()[0],
                            "frac_of_8tbs": head_rec["expert_gbs"] / 8000.0, "k_mean": head_rec["k_mean"],
                            "k_min": head_rec["k_min"], "k_max": head_rec["k_max"],
                            "union_mean": head_rec["union_mean"], "s_ffn": head_rec["s_ffn"],
                            "s_ffn_from": head_rec["s_ffn_from"]},
           "hbm_gbs_total": head_rec["total_gbs"], "tflops": head_rec["tflops"],
           "p_sweep": sweep, "rules": rules, "chained": chained, "router_stats": router_stats,
           "moefy_permute": moefy_permute, "warm_l2_tokens_per_s": warm_tok_s,
           "e2e": e2e, "gpu_launches": args.steps * w.n_layers * kernels_per_layer, "clocks": head_rec["clocks"],
           "configs": configs}
    if rank == 0 and world == 1:
        try:
            out["cpu_baseline"] = run_oracle_sample(w, args.cpu_seconds, args.seed, p=args.p, B=B)
        except Exception as ex:  # the oracle needs gcc; report rather than fail the bench
            out["cpu_baseline"] = {"value": None, "error": str(ex)[:200]}
    if rank == 0:
        print(json.dumps(out))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
