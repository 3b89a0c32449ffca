"""Host-side logic of bench.py on the CPU: the roofline traffic lookup (valid only while
the kernel source is unchanged), the clock-record parsing, the HBM-rate arithmetic and
the oracle sample."""
import hashlib
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
from paper_2607_18582_gb300 import workloads as wl  # noqa: E402


def _profile(tmp_path, src_text, sha, per_row=2000.0):
    (tmp_path / "profiles").mkdir(exist_ok=True)
    (tmp_path / "src.cu").write_text(src_text)
    (tmp_path / "profiles" / "k.md").write_text(
        f"# summary\n\n    dram_bytes_per_row: {per_row}\n    source_file: src.cu\n    source_sha256: {sha}\n")


def test_profiled_traffic_tracks_the_source(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    text = "kernel source\n"
    _profile(tmp_path, text, hashlib.sha256(text.encode()).hexdigest(), 2000.0)
    assert bench.profiled_traffic("k", 10.0) == 20000.0
    (tmp_path / "src.cu").write_text(text + "// changed\n")
    assert bench.profiled_traffic("k", 10.0) is None
    assert bench.profiled_traffic("missing", 10.0) is None


def test_clock_summary_parsing():
    cs = bench.ClockSampler(0)
    cs.lines = ["0, 2070, 2070, 900.0, 0x0, Not Active, Not Active, Not Active, Not Active",
                "0, 2040, 2070, 1390.0, 0x4, Not Active, Not Active, Not Active, Active",
                "0, 2070, 2070, 950.0, 0x0, Not Active, Not Active, Not Active, Not Active",
                "garbage line"]
    s = cs.summary()
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0 and s["samples"] == 3
    assert s["reasons"] == ["sw_power_cap"]
    empty = bench.ClockSampler(0)
    empty.lines = []
    assert empty.summary()["reasons"] == ["unsampled"]


def test_hbm_rates_arithmetic():
    w = wl.workload("lenet5", 4, 4)
    L = w.model.n_layers()
    rows = 1000
    macs = w.model.layer_macs(L - 1)
    results = [{"stats": {"bytes_gather": 6_799_300, "bytes_delta_values": 1_000_000,
                          "flops_layer": [0] * (L - 1) + [2 * macs * rows]}}]
    cls = {"delta": 0.75, "delta_values": 0.25, f"layer{L - 1}": 2.0}
    out = bench.hbm_rates(w, results, cls, {"hbm_gbs": 6799.3}, "measured")
    assert out["delta"]["achieved"] == pytest.approx(6.7993)            # 6.8 MB in 0.75 + 0.25 ms
    assert out["delta"]["frac"] == pytest.approx(6.7993 / 6799.3)
    assert out["cache_read"]["achieved"] == pytest.approx(4.0)          # 1 MB in 0.25 ms
    assert out["cache_read"]["frac"] == pytest.approx(4.0 / 6799.3)
    # no value kernels timed apart: no cache-read entry
    assert "cache_read" not in bench.hbm_rates(w, results, {"delta": 1.0}, {"hbm_gbs": 6799.3}, "measured")
    node = w.model.nodes[w.model.layers()[L - 1]]
    exp = rows * (node.cin * 4 + 1 / 8) / 2e-3 / 1e9
    assert out["output_layer"]["achieved"] == pytest.approx(exp)


@pytest.mark.parametrize("name", ["lenet5", "lenet5_modelwide", "lenet5_modelwide_5"])
def test_oracle_sample_is_stratified(name):
    w = wl.workload(name, 50, 400)
    sub, X, idx = bench.oracle_sample(w, 40, 20, with_index=True)
    assert len(sub) == 40 and len(X) == 20 and len(np.unique(idx)) == 40
    assert set(np.unique(sub.layer)) == set(np.unique(w.table.layer[:400]))
    if w.table.tagged is not None:
        assert np.array_equal(sub.tagged, w.table.tagged[idx])
        for j, i in enumerate(idx):
            a, n = int(w.table.neuron_off[i]), int(w.table.n_neurons[i])
            b = int(sub.neuron_off[j])
            assert np.array_equal(sub.pool[b:b + n], w.table.pool[a:a + n])


@pytest.mark.timeout(600)
def test_reference_arm_line_single_rank():
    """`bench.py --impl reference` at N = 1: one JSON line with every key of the
    contract; the oracle is timed on the host cores with no device copies."""
    import json
    import subprocess
    p = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "3",
                        "--workload", "mlp"], cwd=ROOT, capture_output=True, text=True, timeout=580)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "e2e", "cpu_baseline", "impl"):
        assert k in d, k
    assert d["impl"] == "reference" and d["n_gpus"] == 1 and d["steps"] == 1 and d["warmup"] == 3
    assert d["value"] > 0 and d["higher_is_better"] is True and d["vs_baseline"] is None
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert d["config"]["workload"].startswith("mlp")


def test_slices_flops_and_cache_bytes():
    """The step slices partition the table; the analytic FLOPs follow Lemma 4's cost
    model (vanilla - memo = the prefixes); the cache size counts every cached row."""
    w = wl.workload("vgg", 8, 400)
    sl = bench.table_slices(len(w.table), 20)
    assert sorted(np.concatenate(sl).tolist()) == list(range(400))
    assert max(len(x) for x in sl) - min(len(x) for x in sl) <= 1
    memo, van = bench.analytic_flops(w.model, w.table)
    L = w.model.n_layers()
    macs = [w.model.layer_macs(v) for v in range(L)]
    prefix = sum(2 * sum(macs[:int(l) + 1]) for l in w.table.layer)
    assert van - memo == pytest.approx(prefix)
    assert 0 < memo < van
    # a table of first-layer NEB mutants: the whole network but the first layer
    t = wl.table_from_rows([(0, "NEB", [0], 0.0, 0)])
    m1, v1 = bench.analytic_flops(w.model, t)
    assert m1 == 2 * sum(macs[1:]) and v1 == 2 * sum(macs)
    per = bench.cache_bytes(w.model, 64) / 64
    # input 3072 + z 65536 per 32x32x64 map ... at least the inputs and outputs of every layer
    assert per > 4 * sum(w.model.layer_width(v) for v in range(L))
    assert bench.cache_bytes(w.model, 1) == bench.cache_bytes(w.model, 64)   # inputs padded to 64
