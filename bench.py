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
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--pool", type=int, default=0,
                    help="distinct token sets per layer (default 16 for decode batches, 1 for prefill)")
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
    return ap.parse_args()


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
def make_layers(w, args, device):
    import torch
    from paper_2605_28283_gb300 import workloads as wl
    layers = []
    for l in range(w.n_layers):
        t = wl.device_layer(w, args.batch, args.seed, l, device, n_token_sets=args.pool)
        t["y"] = torch.empty((args.batch, w.d_model), dtype=t["x"].dtype, device=device)
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
    """k per (pool entry, layer, token) via pp_route on the same inputs."""
    import numpy as np
    import torch
    ks = torch.empty((pool, len(layers), B), dtype=torch.int64)
    union = torch.empty((pool, len(layers)), dtype=torch.int64)
    sel = pp.Selection.empty(B, w.n_experts, "cuda", with_logits=False)
    for i in range(pool):
        for l, L in enumerate(layers):
            pp.pp_route(desc, L["x"][i], B, L["Wr"], p, sel, ws)
            c = sel.counts.cpu()
            ks[i, l] = c.long()
            ids = sel.ids.cpu().numpy()
            cn = c.numpy()
            mask = np.arange(ids.shape[1])[None, :] < cn[:, None]
            union[i, l] = len(np.unique(ids[mask]))
    return ks, union


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


# ------------------------------------------------------------ CPU oracle
def run_oracle_sample(w, seconds, seed, host_layers=None, p=0.7, B=1):
    """Times the oracle (as it stands) on a bounded sample of the workload:
    whole-layer calls (logits, selection, sparse FFN) for B tokens, over a
    few layers, repeated until `seconds` of CPU work; scaled to tokens/s of
    the full L-layer model."""
    import numpy as np
    import oracle
    from paper_2605_28283_gb300 import workloads as wl
    oracle.load()
    n_layers = 2 if host_layers is None else len(host_layers)
    if host_layers is None:
        host_layers = [wl.host_layer(w, B, seed=seed, layer=l) for l in range(n_layers)]
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    calls = 0
    t0 = time.perf_counter()
    while True:
        for L in host_layers:
            oracle.layer(L.x, L.Wr, L.Wg, L.Wu, L.Wd, float(np.float32(p)), w.act, "sigmoid")
            calls += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    per_layer = el / calls
    tok_s = B / (per_layer * w.n_layers)
    return {"value": tok_s, "unit": "tokens/s", "cores": min(threads, B) if B > 0 else 1, "kind": "oracle",
            "sample": "%d calls of one layer x %d token(s) over %d distinct layers (%.1f s CPU); "
                      "scaled to %d layers" % (calls, B, n_layers, el, w.n_layers)}


def run_reference(args):
    rank, world, _ = dist_env()
    from paper_2605_28283_gb300 import workloads as wl
    w = wl.WORKLOADS[args.workload]
    if rank != 0:
        return
    # Each step is one bounded sample (a single layer call), scaled to the
    # full model; the whole run stays within a few minutes.
    import numpy as np
    import oracle
    oracle.load()
    L = wl.host_layer(w, args.batch, seed=args.seed, layer=0)
    p = float(np.float32(args.p))
    for _ in range(max(1, min(args.warmup, 3))):
        oracle.layer(L.x, L.Wr, L.Wg, L.Wu, L.Wd, p, w.act, "sigmoid")
    steps = max(1, min(args.steps, 200))
    t0 = time.perf_counter()
    for _ in range(steps):
        oracle.layer(L.x, L.Wr, L.Wg, L.Wu, L.Wd, p, w.act, "sigmoid")
    el = time.perf_counter() - t0
    per_step_model = el / steps * w.n_layers
    value = args.batch / per_step_model
    # the oracle's OpenMP loops run over tokens
    cores = max(1, min(int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1)), args.batch))
    out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus, "steps": steps,
           "warmup": args.warmup, "ms_per_step": per_step_model * 1e3, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "impl": "reference",
           "config": {"workload": w.name, "d_model": w.d_model, "d_ff": w.d_ff, "n_experts": w.n_experts,
                      "layers": w.n_layers, "batch": args.batch, "p": args.p},
           "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                            "sample": "%d single-layer calls (layer 0) x %d token(s), scaled to %d layers"
                                      % (steps, args.batch, w.n_layers)},
           "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out))


# ------------------------------------------------------------------ main
def main():
    args = parse()
    if args.pool <= 0:
        args.pool = 16 if args.batch <= 128 else 1
    if args.impl == "reference":
        return run_reference(args)
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
    desc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act)
    stream = torch.cuda.Stream()
    ws = pp.alloc_workspace(desc, B)
    layers = make_layers(w, args, device)
    flush = None if args.no_flush else torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=device)
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    # ---- headline: p = args.p
    pf = float(np.float32(args.p))
    graphs = capture_graphs(pp, desc, layers, pf, B, args.pool, ws, stream)
    sampler = ClockSampler(local)
    barrier()
    sampler.start()
    times = time_graphs(graphs, args.steps, args.warmup, flush, stream, profile_range=True)
    barrier()
    clocks = sampler.stop()
    value, slowest_s = replica_throughput(B * args.steps, sum(times) / 1e3, world, device)
    total_ms = slowest_s * 1e3
    status = pp.pp_get_device_status(ws)
    if status != pp.PP_OK:
        raise SystemExit("device status: %s" % pp.status_name(status))
    ms_per_step = total_ms / args.steps

    # bytes per step from the actual selections of the pool entries
    ks, union = selection_stats(pp, desc, layers, w, pf, B, args.pool, ws)
    step_ids = np.arange(args.steps) % args.pool
    tot_b, exp_b, tot_f = 0.0, 0.0, 0.0
    for i in range(args.pool):
        n_i = int((step_ids == i).sum())
        for l in range(w.n_layers):
            a, e = layer_bytes(w, B, int(union[i, l]))
            tot_b += n_i * a
            exp_b += n_i * e
            tot_f += n_i * layer_flops(w, B, int(ks[i, l].sum()))
    seconds = sum(times) / 1e3
    launches = args.steps * w.n_layers
    # kernels of ours per layer call: the fused decode kernel (<= 4 bf16 / 8 fp32
    # tokens), else router, selection, 4 dispatch kernels, gate/up, down, combine
    kernels_per_layer = 1 if (B <= 4 or w.dtype == "f32") else 9
    per_launch_ms = sum(times) / launches   # step time / L: includes the in-graph launch gaps
    bytes_per_launch = tot_b / launches
    flops_per_launch = tot_f / launches
    hbm_peak, tc_peak, peak_kind = load_peaks()
    # the bound is whichever of HBM traffic and tensor work takes longer at peak
    tensor_bound = flops_per_launch / (tc_peak * 1e12) > bytes_per_launch / (hbm_peak * 1e9)
    if tensor_bound:
        achieved = flops_per_launch / (per_launch_ms / 1e3) / 1e12
        peak = tc_peak
        roof = {"bound": "tensor", "unit": "TFLOP/s", "flops_per_launch": flops_per_launch}
    else:
        achieved = bytes_per_launch / (per_launch_ms / 1e3) / 1e9
        peak = hbm_peak
        roof = {"bound": "hbm", "unit": "GB/s", "bytes_per_launch": bytes_per_launch}
    expert_gbs = exp_b / seconds / 1e9
    k_mean = float(ks.float().mean())
    s_ffn = 1.0 - k_mean / w.n_experts

    # ---- p sweep (same kernels), speedup vs dense p >= 1
    sweep = {}
    if args.sweep:
        for ps in [float(v) for v in args.sweep.split(",") if v]:
            psf = float(np.float32(ps))
            gs = capture_graphs(pp, desc, layers, psf, B, args.pool, ws, stream)
            tm = time_graphs(gs, args.sweep_steps, 5, flush, stream)
            kk, un = selection_stats(pp, desc, layers, w, psf, B, args.pool, ws)
            sid = np.arange(args.sweep_steps) % args.pool
            eb = sum(int((sid == i).sum()) * layer_bytes(w, B, int(un[i, l]))[1]
                     for i in range(args.pool) for l in range(w.n_layers))
            tb = sum(int((sid == i).sum()) * layer_bytes(w, B, int(un[i, l]))[0]
                     for i in range(args.pool) for l in range(w.n_layers))
            sec = sum(tm) / 1e3
            sweep["%g" % ps] = {"tokens_per_s": B * args.sweep_steps / sec, "ms_per_step": sum(tm) / args.sweep_steps,
                                "k_mean": float(kk.float().mean()), "s_ffn": 1 - float(kk.float().mean()) / w.n_experts,
                                "expert_gbs": eb / sec / 1e9, "total_gbs": tb / sec / 1e9,
                                "frac_of_hbm_peak": tb / sec / 1e9 / hbm_peak}
            del gs
        dense = sweep.get("1")
        if dense:
            for v in sweep.values():
                v["speedup_vs_p1"] = v["tokens_per_s"] / dense["tokens_per_s"]

    # ---- the other activation rules (top-k, LTE's threshold) on the same kernels
    rules = {}
    for item in [] if args.skip_extras else [v for v in args.rules.split(",") if v]:
        rname, rp = item.split(":")
        rpf = float(np.float32(float(rp)))
        rdesc = pp.make_desc(w.d_model, w.n_experts, w.dtype, w.act, "none" if rname == "lte" else "sigmoid", rname)
        gs = capture_graphs(pp, rdesc, layers, rpf, B, args.pool, ws, stream)
        tm = time_graphs(gs, args.sweep_steps, 5, flush, stream)
        kk, un = selection_stats(pp, rdesc, layers, w, rpf, B, args.pool, ws)
        sid = np.arange(args.sweep_steps) % args.pool
        tb = sum(int((sid == i).sum()) * layer_bytes(w, B, int(un[i, l]))[0]
                 for i in range(args.pool) for l in range(w.n_layers))
        sec = sum(tm) / 1e3
        rules[item] = {"tokens_per_s": B * args.sweep_steps / sec, "k_mean": float(kk.float().mean()),
                       "total_gbs": tb / sec / 1e9, "frac_of_hbm_peak": tb / sec / 1e9 / hbm_peak}
        del gs
    if pp.pp_get_device_status(ws) != pp.PP_OK:
        raise SystemExit("device status after the rule sweep: %s" % pp.status_name(pp.pp_get_device_status(ws)))

    # ---- chained decode step: layer l takes x_l = RMSNorm(x_{l-1} + y_{l-1}) (pp_layer_chained), so
    # every layer reads the previous layer's output; one CUDA graph per pool entry
    chained = None
    if not args.skip_extras and B <= 4:
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

    if args.skip_extras:
        if rank == 0:
            print(json.dumps({"metric": METRIC, "value": value, "unit": "tokens/s", "ms_per_step": ms_per_step,
                              "workload": w.name, "layers": w.n_layers, "p": args.p, "batch": B,
                              "launch_ms": per_launch_ms, "bytes_per_launch": bytes_per_launch,
                              "flops_per_launch": flops_per_launch, "roofline_bound": roof["bound"],
                              "achieved": achieved, "peak": peak, "frac": achieved / peak,
                              "sources_sha": sources_sha("decode" if B <= 4 or w.dtype == "f32" else "grouped")}))
        return

    # ---- warm-L2 number (no flush), for context
    warm = time_graphs(graphs, min(args.steps, 500), 5, None, stream)
    warm_tok_s = B * len(warm) / (sum(warm) / 1e3)

    # ---- end to end through the public API with host buffers.  Every step
    # copies the 32 layer inputs from pinned host memory in one transfer,
    # replays a CUDA graph of the 32 pp_layer calls (captured once through
    # the binding) and reads the 32 outputs back; the host waits for them.
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
    e2e = {"value": replica_throughput(B * e2e_steps, timings["graph"], world, device)[0],
           "unit": "tokens/s", "h2d_bytes_per_step": w.n_layers * B * w.d_model * esz,
           "d2h_bytes_per_step": w.n_layers * B * w.d_model * esz,
           "path": "pp_layer via the ctypes binding, 32 calls captured once in a CUDA graph; per step one "
                   "pinned H2D copy of the 32 layer inputs, graph replay, one D2H copy of the 32 outputs, "
                   "host synchronisation",
           "eager_value": replica_throughput(B * e2e_steps, timings["eager"], world, device)[0],
           "eager_path": "the same with the 32 pp_layer calls made eagerly every step"}

    # ---- router statistics (L_ent, L_bal, L_gate) over a batch of 8192 tokens' logits
    T_st = 8192
    g_st = torch.randn((T_st, w.n_experts), device=device) * 3.0
    ws_st = pp.alloc_workspace(desc, T_st)
    out_st = torch.empty(3, dtype=torch.float64, device=device)
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
                    "note": "two launches (per-256-token parts, fixed-order final sum); logits L2-resident"}

    # ---- MoEfication repacking (Eq. permuted_weights) of one layer's weights by a random permutation
    moefy_permute = None
    if not args.skip_extras:
        L0 = layers[0]
        perm_d = torch.randperm(w.d_ff, device=device).to(torch.int32)
        outs = [None if L0["Wg"] is None else torch.empty_like(L0["Wg"]), torch.empty_like(L0["Wu"]),
                torch.empty_like(L0["Wd"])]
        ws_mp = pp.alloc_workspace(desc, 0)
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
                         "frac_of_hbm_peak": b_mp / (us_mp * 1e-6) / 1e9 / hbm_peak, "spot_check": bool(ok),
                         "what": "pp_moefy_permute of one layer (W_gate/W_up rows, W_down columns) by a random "
                                 "permutation; bytes = read + write of the three matrices; 3 launches per call"}
        del outs, ws_mp

    out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
           "config": {"workload": w.name, "d_model": w.d_model, "d_ff": w.d_ff, "n_experts": w.n_experts,
                      "d_expert": 64, "layers": w.n_layers, "batch": B, "p": args.p, "act": w.act,
                      "token_pool": args.pool,
                      "l2": "no flush (warm)" if args.no_flush else "flushed between steps (256 MiB write, untimed)",
                      "parallelism": "replicas" if world > 1 else "single GPU"},
           "roofline": dict(roof, achieved=achieved, peak=peak, frac=achieved / peak,
                            traffic=kernel_traffic(w.name, args.p, B, "decode" if B <= 4 or w.dtype == "f32" else "grouped"),
                            peak_kind=peak_kind,
                            kernel="decode_layer_kernel" if B <= 4 else "pp_layer (grouped tcgen05 path)",
                            per="one pp_layer call (one layer)", launch_ms=per_launch_ms),
           "expert_bytes": {"gbs": expert_gbs, "frac_of_peak": expert_gbs / hbm_peak,
                            "frac_of_8tbs": expert_gbs / 8000.0, "k_mean": k_mean, "k_min": int(ks.min()),
                            "k_max": int(ks.max()), "s_ffn": s_ffn},
           "hbm_gbs_total": tot_b / seconds / 1e9, "tflops": tot_f / seconds / 1e12,
           "p_sweep": sweep, "rules": rules, "chained": chained, "router_stats": router_stats,
           "moefy_permute": moefy_permute, "warm_l2_tokens_per_s": warm_tok_s,
           "e2e": e2e, "gpu_launches": launches * kernels_per_layer, "clocks": clocks}
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
