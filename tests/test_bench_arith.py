"""The benchmark's roofline arithmetic (no GPU): algorithmic bytes and FLOPs
of one layer call for each workload shape, the validity rule of the stored
DRAM-traffic record, and the peak fallback.

Expected values are worked out by hand from the layer shapes: W_r is E x d,
an expert block is 64 rows of W_gate and W_up plus a 64-wide column block of
W_down (two matrices for the non-gated FFNs), x and y are B x d; the FLOPs
are 2 per multiply-add of the router and of every (token, selected expert)
block product."""
import json

import pytest

import bench
from paper_2605_28283_gb300 import workloads as wl

W = wl.WORKLOADS


@pytest.mark.parametrize("name,router,block", [
    ("tiny_relu_f32", 16 * 256 * 4, 128 * 1024),                # fp32, two matrices: 128 KiB
    ("gpt2m_gelu_bf16", 64 * 1024 * 2, 256 * 1024),             # bf16, two matrices: 256 KiB
    ("llama2_7b_decode", 1_409_024, 1_572_864),                 # 1.41 MB router, 1.5 MiB per expert
    ("llama3_8b_batched", 224 * 4096 * 2, 1_572_864),
    ("llama2_13b_prefill", 216 * 5120 * 2, 1_966_080),          # 1.875 MiB per expert
])
def test_layer_bytes(name, router, block):
    w = W[name]
    esz = 4 if w.dtype == "f32" else 2
    for B, union in [(1, 1), (1, 6), (64, 120)]:
        total, expert = bench.layer_bytes(w, B, union)
        assert expert == union * block
        assert total == router + union * block + 2 * B * w.d_model * esz


def test_dense_llama2_7b_layer():
    total, expert = bench.layer_bytes(W["llama2_7b_decode"], 1, 172)
    # all 172 experts = the three FFN matrices, 3 * 11008 * 4096 * 2 B = 270.5 MB; with the router and
    # x, y: 272.0 MB
    assert expert == 3 * 11008 * 4096 * 2 and round(expert / 1e6, 1) == 270.5
    assert round(total / 1e6, 1) == 272.0
    # 32 layers of FFN weights at the measured 6778 GB/s bound dense batch-1 decode at ~783 tokens/s
    assert round(6778e9 / (32 * expert)) == 783


def test_layer_flops_prefill():
    w = W["llama2_13b_prefill"]
    T, k = 8192, 6
    f = bench.layer_flops(w, T, T * k)
    router = 2.0 * T * 216 * 5120
    assert round(router / 1e9, 1) == 18.1
    assert round((f - router) / 1e9, 1) == 96.6      # sum_t k_t * 6 * 64 * d
    g = bench.layer_flops(W["gpt2m_gelu_bf16"], 1, 3)   # non-gated: 4 * 64 * d per expert
    assert g == 2.0 * 64 * 1024 + 2.0 * 3 * 2 * 64 * 1024


def test_traffic_record_only_for_unchanged_sources(tmp_path, monkeypatch):
    prof = tmp_path / "profiles"
    prof.mkdir()
    rec = {"entries": {"llama2_7b_decode@p0.7@B1": {"dram_bytes_per_layer": 123.0, "sources_sha": "abc"}}}
    (prof / "dram_traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "sources_sha", lambda kind="decode": "abc")
    assert bench.kernel_traffic("llama2_7b_decode", 0.7, 1) == 123.0
    assert bench.kernel_traffic("llama2_7b_decode", 0.9, 1) is None      # no record for this p
    monkeypatch.setattr(bench, "sources_sha", lambda kind="decode": "def")
    assert bench.kernel_traffic("llama2_7b_decode", 0.7, 1) is None      # kernel changed since


def test_committed_traffic_record_is_well_formed():
    import os
    path = os.path.join(os.path.dirname(bench.__file__), "profiles", "dram_traffic.json")
    rec = json.load(open(path))
    for key, ent in rec["entries"].items():
        name, p, b = key.split("@")
        assert name in W and p.startswith("p") and b.startswith("B")
        assert ent["dram_bytes_per_layer"] > 0 and len(ent["sources_sha"]) == 16


def test_peaks_fallback_without_measured_file(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.load_peaks() == (6800.0, 1700.0, "fallback")
    (tmp_path / "MEASURED_PEAKS.json").write_text(json.dumps({"hbm_gbs": 6778.0, "bf16_tflops": 1940.4,
                                                              "bf16_tflops_sustained": 1695.3}))
    assert bench.load_peaks() == (6778.0, 1695.3, "measured")


def test_default_benchmark_lines_have_current_traffic_records(monkeypatch):
    """Every workload the default bench run reports (the headline and its
    configs) has a DRAM-traffic record taken at the current kernel sources, so
    its roofline line carries measured traffic rather than null."""
    monkeypatch.setattr("sys.argv", ["bench.py"])
    args = bench.parse()
    runs = [(args.workload, args.p, args.batch)]
    for item in [v for v in args.configs.split(",") if v]:
        parts = item.split(":")
        runs.append((parts[0], float(parts[2]), int(parts[1])))
    for name, p, b in runs:
        kind = bench.path_kind(W[name], b)
        assert bench.kernel_traffic(name, p, b, kind) is not None, (name, p, b, kind)
