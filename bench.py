"""Benchmark of memoized DNN mutation testing on GB300.

One step = the whole hot path over one batch of the workload: the prefix-activation
cache of ALL the workload's inputs (Algorithm 1 lines 10-12), descriptor expansion and
grouping, the delta and suffix kernels of every mutant group, the fused kill epilogue
and the score reduction, for one slice of the mutant table.  The table is cut into S
slices by a seeded random partition (each slice a uniform sample of the table's mix of
layers, operators and ratios); S consecutive steps cover the whole table once, so the
default 20 timed steps on the VGG workload (10,000 inputs x 5,000 mutants, S = 20) are
exactly one full job, with the cache rebuilt every step.  Default workload: the
VGG-style network, 10,000 inputs N(0,1), 5,000 mutants at 0.5 / 1 / 2 / 5 %.

  python bench.py [--gpus N --steps K --warmup W] [--impl reference] [--workload NAME]

Prints one JSON line (rank 0).  N > 1 runs N independent replicas (one per GPU,
launched by torchrun); the path has no cross-GPU exchange.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "mutant×input evals/sec at 1 GB300; suffix-GEMM tensor-pipe % of peak"
UNIT = "evals/s"
# CUDA-core fp32 peak of a GB300: 152 SMs x 128 FP32 lanes x 2 FLOP (FMA) x 2.07 GHz
SIMT_FP32_PEAK_TFLOPS = 152 * 128 * 2 * 2.070e9 / 1e12
L2_FLUSH_BYTES = 256 << 20

# slices of the mutant table per full job (one slice per step)
SLICES = {"vgg": 20, "vgg_stress": 20, "resnet20": 20}

WORKLOAD_TEXT = {
    "lenet5": "LeNet-5 28x28x1 (conv5x5 6 pad2, pool, conv5x5 16, pool, FC 400-120-84-10), 10,000 inputs U[0,1], "
              "2,000 single-layer mutants, 1% selection ratio, GF/NEB/NAI/NS, layer uniform over 5",
    "mlp": "MLP 784-128-64-10, 1,000 inputs U[0,1], 200 mutants, 1% ratio",
    "resnet20": "ResNet-20 32x32x3, 10,000 inputs N(0,1), 5,000 mutants, 1% ratio",
    "vgg": "VGG-style 32x32x3 (8 weighted layers), 10,000 inputs N(0,1), 5,000 mutants, ratios 0.5/1/2/5%",
    "vgg_stress": "VGG-style 32x32x3, 20,000 inputs N(0,1), 20,000 mutants, ratios 0.1/1/5/10%, 50% on the first conv",
    "lenet5_modelwide": "LeNet-5 28x28x1, 10,000 inputs U[0,1], 2,000 mutants over several layers: 1% of all 236 "
                        "neurons drawn model-wide per mutant (tagged descriptors), GF/NEB/NAI/NS",
    "mlp_modelwide": "MLP 784-128-64-10, 1,000 inputs U[0,1], 200 mutants, 1% of all neurons drawn model-wide",
    "lenet5_modelwide_3": "LeNet-5 28x28x1, 10,000 inputs U[0,1], 2,000 mutants over several layers: 3% of all 236 "
                          "neurons (7) drawn model-wide per mutant, GF/NEB/NAI/NS",
    "lenet5_modelwide_5": "LeNet-5 28x28x1, 10,000 inputs U[0,1], 2,000 mutants over several layers: 5% of all 236 "
                          "neurons (12) drawn model-wide per mutant, GF/NEB/NAI/NS",
}


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# ------------------------------------------------------------------- clocks --

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        self.device = device
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "200", "-i", str(self.device)],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for l in getattr(self, "lines", []):
            p = [x.strip() for x in l.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                mx.append(float(p[2]))
            except ValueError:
                continue
            for n, v in zip(names, p[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------- ncu traffic file --

def profiled_traffic(kernel_key, rows_per_launch):
    """DRAM bytes per launch of the dominant kernel from its committed ncu summary,
    scaled by rows; None when the summary is missing or the kernel source changed
    since the counters were taken."""
    path = os.path.join(ROOT, "profiles", f"{kernel_key}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    m_bytes = re.search(r"dram_bytes_per_row:\s*([0-9.eE+]+)", text)
    m_sha = re.search(r"source_sha256:\s*([0-9a-f]{64})", text)
    m_src = re.search(r"source_file:\s*(\S+)", text)
    if not (m_bytes and m_sha and m_src):
        return None
    try:
        cur = hashlib.sha256(open(os.path.join(ROOT, m_src.group(1)), "rb").read()).hexdigest()
    except OSError:
        return None
    if cur != m_sha.group(1):
        return None
    return float(m_bytes.group(1)) * rows_per_launch


def hbm_rates(w, results, cls_ms, pk, pk_kind):
    """Achieved HBM bandwidth of the memory-bound kernel classes against the measured
    copy bandwidth: the delta kernels (algorithmic bytes = the patch values they write
    and the cached z / x rows that each input of a batch stages once for all mutants)
    and the stand-alone output-layer kernel (its input rows read once, 1 bit written
    per row).  CUDA-event times of the timed steps."""
    out = {}
    peak = pk["hbm_gbs"]
    ms = cls_ms.get("delta", 0.0) + cls_ms.get("delta_values", 0.0)
    byts = sum(r["stats"]["bytes_gather"] for r in results)
    if ms > 0 and byts > 0:
        gbs = byts / (ms / 1e3) / 1e9
        out["delta"] = {"kernels": "every delta kernel (values and fan-in sums)", "bytes": byts, "ms": ms,
                        "achieved": gbs, "unit": "GB/s", "frac": gbs / peak,
                        "bytes_counted": "patch values written + cached z / x rows read once per input and batch"}
    # the value kernels alone (NEB / NAI / NS), timed apart where the fan-in sums run
    # in their own kernel: the cache read of the delta, memory-bound
    ms = cls_ms.get("delta_values", 0.0)
    byts = sum(r["stats"].get("bytes_delta_values", 0) for r in results)
    if ms > 0 and byts > 0:
        gbs = byts / (ms / 1e3) / 1e9
        out["cache_read"] = {"kernels": "k_patch_vals / k_patch_vals_staged (NEB / NAI / NS values of the mutated "
                                        "layer from the cached pre-activations)",
                             "bytes": byts, "ms": ms, "achieved": gbs, "unit": "GB/s", "frac": gbs / peak,
                             "bytes_counted": "cached z row of each input read once per batch + patch values written"}
    L = w.model.n_layers()
    last = f"layer{L - 1}"
    ms = cls_ms.get(last, 0.0)
    fl = sum(r["stats"]["flops_layer"][L - 1] for r in results)
    macs = w.model.layer_macs(L - 1)
    if ms > 0 and fl > 0:
        rows = fl / 2 / macs
        node = w.model.nodes[w.model.layers()[L - 1]]
        byts = rows * (node.cin * 4 + 1 / 8)
        gbs = byts / (ms / 1e3) / 1e9
        out["output_layer"] = {"kernels": "k_final_dense_rows / k_final_dense (output layer + kill, rows not fused into a dense epilogue)",
                               "bytes": byts, "ms": ms, "achieved": gbs, "unit": "GB/s", "frac": gbs / peak,
                               "bytes_counted": "input rows read once, kill bits written"}
    out["peak"] = peak
    out["peak_source"] = f"{pk_kind} (MEASURED_PEAKS.json hbm_gbs)"
    return out


# ------------------------------------------------------------- distributed --

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------- oracle leg --

def oracle_sample(w, n_mut, n_in, seed=0, with_index=False):
    from paper_2607_18582_gb300 import workloads as wl
    idx = wl.stratified(w.table, w.model, max(1, n_mut // (w.model.n_layers() * 4)))
    rng = np.random.default_rng(seed)
    if len(idx) < n_mut:
        rest = np.setdiff1d(np.arange(len(w.table)), idx)
        idx = np.sort(np.concatenate([idx, rng.choice(rest, min(len(rest), n_mut - len(idx)), replace=False)]))
    idx = idx[:n_mut]
    if with_index:
        return w.table.subset(idx), w.X[:n_in], idx
    return w.table.subset(idx), w.X[:n_in]


def cpu_oracle_rate(w, n_mut, n_in, threads, gpu_kill=None):
    """Oracle (memoized, Algorithm 1 on the CPU) evals/s on a bounded sample; with the
    GPU's kill matrix of the whole workload, also the agreement of the GPU's kill
    verdicts with the oracle's on that sample."""
    import oracle
    table, X, idx = oracle_sample(w, n_mut, n_in, with_index=True)
    t = time.perf_counter()
    res = oracle.memo(w.model, X, table, n_threads=threads, want_logits=False)
    dt = time.perf_counter() - t
    agree = None
    if gpu_kill is not None:
        n = len(X)
        cols = np.arange(n)
        ora = (np.asarray(res["kill_bits"], np.uint64)[:, cols // 64] >> (cols % 64).astype(np.uint64)) & np.uint64(1)
        g = np.asarray(gpu_kill, np.uint64)[idx]
        gpu = (g[:, cols // 64] >> (cols % 64).astype(np.uint64)) & np.uint64(1)
        diff = int((ora != gpu).sum())
        agree = {"verdicts": int(ora.size), "differ": diff, "agreement": 1.0 - diff / max(1, ora.size)}
    return (len(table) * len(X) / dt, dt, f"{len(table)} stratified mutants x first {len(X)} inputs, oracle memoized mode",
            agree)


def run_reference(args, world, rank):
    """The reference arm: the CPU oracle as it stands, on bounded samples."""
    if rank != 0:
        return 0
    from paper_2607_18582_gb300 import workloads as wl
    import oracle
    oracle.build()
    w = wl.workload(args.workload)
    threads = os.cpu_count() or 1
    n_mut, n_base = cpu_sample_size(w)
    n_in = max(1, n_base // 8)
    for _ in range(args.warmup):
        cpu_oracle_rate(w, n_mut, n_in, threads)
    t = time.perf_counter()
    for _ in range(args.steps):
        _, _, sample, _ = cpu_oracle_rate(w, n_mut, n_in, threads)
    dt = time.perf_counter() - t
    value = args.steps * n_mut * n_in / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32 (fp64 accumulation)",
            "data": "synthetic", "config": config_block(args, w),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def config_block(args, w):
    small = any(getattr(args, k, None) is not None for k in ("n_inputs", "n_mutants", "only_layer"))
    return {"workload": f"{args.workload}: {WORKLOAD_TEXT.get(args.workload, args.workload)}"
                        + (" [reduced profiling case]" if small else ""),
            "n_inputs": int(len(w.X)), "n_mutants": int(len(w.table)), "n_layers": w.model.n_layers(),
            "seeds": {"model": 0, "inputs": 1, "mutants": 2},
            "l2": "flushed between timed steps (256 MiB write, outside the step events)",
            "parallelism": f"{args.gpus} independent replica(s), no cross-GPU exchange"}


# ----------------------------------------------------------------- GPU leg --

def table_slices(n_mut, n_slices, seed=7):
    """A seeded random partition of the table's row indices into n_slices slices
    (sorted within each slice); slice k is step k's batch of mutants."""
    n_slices = max(1, min(n_slices, n_mut)) if n_mut else 1
    perm = np.random.default_rng(seed).permutation(n_mut)
    return [np.sort(perm[k::n_slices]) for k in range(n_slices)]


def analytic_flops(model, table):
    """FLOPs the method must spend on a table (per input), memoized and vanilla: the
    suffix layers after each mutant's first mutated layer l, the recomputed channels of
    layer l for GF / WS (k neurons x the layer's MACs per neuron) and, in vanilla mode,
    the prefix and the whole layer l (Lemma 4's cost model: vanilla - memo = the
    prefix every mutant of a cluster shares)."""
    L = model.n_layers()
    macs = np.array([model.layer_macs(v) for v in range(L)], np.float64)
    suffix = np.concatenate([np.cumsum(macs[::-1])[::-1][1:], [0.0]])   # sum over v > l
    prefix = np.cumsum(macs)                                            # sum over v <= l
    width = np.array([model.layer_width(v) for v in range(L)], np.float64)
    l = table.layer.astype(np.int64)
    dot = np.isin(table.op, [0, 4])          # GF, WS recompute their channels
    delta = np.where(dot, table.n_neurons * macs[l] / width[l], 0.0)
    memo = 2.0 * float((suffix[l] + delta).sum())
    vanilla = 2.0 * float((prefix[l] + suffix[l] + delta).sum())
    return memo, vanilla


def measure_tensor_peaks(dev):
    """Peaks of this GPU measured like the driver's bf16 figures: cuBLAS TF32 (fp32
    operands, TF32 tensor cores) and fp32 CUDA-core GEMMs of 8192^3 (2 N^3 FLOP), best
    of 10 back-to-back (burst), and TF32 back to back for about 2 s (sustained)."""
    import torch
    n = 8192
    a = torch.randn(n, n, device=f"cuda:{dev}")
    b = torch.randn(n, n, device=f"cuda:{dev}")
    old = torch.backends.cuda.matmul.allow_tf32

    def best(k):
        ts = []
        for _ in range(k):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            torch.matmul(a, b)
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1) / 1e3)
        return 2.0 * n ** 3 / min(ts) / 1e12
    try:
        torch.backends.cuda.matmul.allow_tf32 = True
        torch.matmul(a, b)
        tf32 = best(10)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = max(1, int(2.0 * tf32 * 1e12 / (2.0 * n ** 3)))
        e0.record()
        for _ in range(reps):
            torch.matmul(a, b)
        e1.record()
        torch.cuda.synchronize()
        tf32_sus = reps * 2.0 * n ** 3 / (e0.elapsed_time(e1) / 1e3) / 1e12
        torch.backends.cuda.matmul.allow_tf32 = False
        torch.matmul(a, b)
        fp32 = best(5)
    finally:
        torch.backends.cuda.matmul.allow_tf32 = old
    del a, b
    torch.cuda.empty_cache()
    return {"tf32_tflops": tf32, "tf32_tflops_sustained": tf32_sus, "fp32_tflops": fp32,
            "how": "torch.matmul fp32 8192^3 (2 N^3 FLOP): TF32 allowed best of 10 (burst) and back to back "
                   f"~2 s ({reps} GEMMs, sustained); TF32 disallowed (CUDA cores) best of 5"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="vgg")
    ap.add_argument("--slices", type=int, default=None,
                    help="slices of the mutant table (one per step); default per workload (VGG 20)")
    ap.add_argument("--skip-cpu-baseline", action="store_true")
    ap.add_argument("--skip-extras", action="store_true", help="no e2e / vanilla / stress / peaks legs")
    ap.add_argument("--n-inputs", type=int, default=None, help="smaller case (profiling): first n inputs")
    ap.add_argument("--n-mutants", type=int, default=None, help="smaller case (profiling): first n mutants")
    ap.add_argument("--only-layer", type=int, default=None, help="keep only the mutants of this layer")
    ap.add_argument("--precision", default="tf32x3", choices=["fp32", "tf32x3", "tf32"],
                    help="layer arithmetic: fp32 CUDA-core chains, tensor-core 3xTF32 (fp32-level), or one TF32 "
                         "product per MAC (the reduced-precision variant)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    world, rank, local = dist_setup()
    if args.impl == "reference":
        return run_reference(args, world, rank)

    import torch
    from paper_2607_18582_gb300 import mure, workloads as wl

    dev = local
    torch.cuda.set_device(dev)
    w = wl.workload(args.workload, args.n_inputs, args.n_mutants)
    if args.only_layer is not None:
        w.table = w.table.subset(np.nonzero(w.table.layer == args.only_layer)[0])
    n_slices = args.slices if args.slices is not None else SLICES.get(args.workload, 1)
    slices = table_slices(len(w.table), n_slices)
    tables = [w.table.subset(ix) for ix in slices]
    arrays = [mure.table_array(t) for t in tables]
    ctx = mure.mure_create(dev)
    model = mure.mure_model_load(ctx, w.model, precision=args.precision)
    X_dev = torch.from_numpy(w.X).to(f"cuda:{dev}")
    W64 = (len(w.X) + 63) // 64
    kill_dev = torch.empty((len(w.table), W64), dtype=torch.int64, device=f"cuda:{dev}")
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=f"cuda:{dev}")
    stream = torch.cuda.current_stream(dev)
    off = np.concatenate([[0], np.cumsum([len(t) for t in tables])])
    # step k evaluates slice k mod S; its kill rows go to their table positions afterwards
    kill_slices = [kill_dev[int(off[k]):int(off[k + 1])] for k in range(len(tables))]

    def step(k, timing=False):
        j = k % len(tables)
        cache = mure.mure_build_prefix_cache(model, X_dev)
        r = mure.mure_eval_mutants(cache, tables[j], outputs_on_device=True, kill_out=kill_slices[j],
                                   kernel_timing=timing, arrays=arrays[j])
        del cache
        return r

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    launches0 = mure.mure_kernel_launches(ctx)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    results = []
    with ClockSampler(dev) as clk:
        for i in range(args.steps):
            flush.zero_()                       # evict L2 between steps (not timed)
            evs[i][0].record(stream)
            results.append(step(i))
            evs[i][1].record(stream)
        torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    launches = mure.mure_kernel_launches(ctx) - launches0
    ms = [a.elapsed_time(b) for a, b in evs]
    t_total = max_over_ranks(sum(ms) / 1e3, world)
    step_evals = [len(tables[i % len(tables)]) * len(w.X) for i in range(args.steps)]
    n_evals = sum(step_evals)
    value = world * n_evals / t_total
    last = results[-1]

    # per-kernel device times from a separate pass with per-launch events (the timed
    # steps above run without them): the first min(S, 3) slices, scaled per step
    n_bd = min(len(tables), 3)
    bd = []
    cb_ms = []
    for i in range(n_bd):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        cache = mure.mure_build_prefix_cache(model, X_dev)
        e1.record(stream)
        bd.append(mure.mure_eval_mutants(cache, tables[i], outputs_on_device=True, kill_out=kill_slices[i],
                                         kernel_timing=True, arrays=arrays[i]))
        torch.cuda.synchronize()
        cb_ms.append(e0.elapsed_time(e1))
        del cache
    bd_evals = sum(len(tables[i]) * len(w.X) for i in range(n_bd))

    L = w.model.n_layers()
    cls_ms = {f"layer{v}": sum(r["stats"]["ms_layer"][v] for r in bd) for v in range(L)}
    cls_ms["delta"] = sum(r["stats"]["ms_delta"] for r in bd)
    cls_ms["delta_values"] = sum(r["stats"]["ms_delta_values"] for r in bd)
    cls_ms["epilogue"] = sum(r["stats"]["ms_epilogue"] for r in bd)
    top = max(cls_ms, key=cls_ms.get)
    pk, pk_kind = peaks()
    tp = None
    if not args.skip_extras:
        tp = measure_tensor_peaks(dev)
    # the step is long: the sustained TF32 figure applies when a step runs >= 1 s
    long_step = t_total / args.steps >= 1.0
    roof = None
    if top in ("delta", "delta_values"):
        byts = sum(r["stats"]["bytes_gather"] for r in bd)
        ms_d = cls_ms["delta"] + cls_ms["delta_values"]
        achieved = byts / (ms_d / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / pk["hbm_gbs"], "traffic": None, "kernel": "delta kernels (k_patch_*)",
                "ms_total": ms_d, "peak_source": f"{pk_kind} (MEASURED_PEAKS.json hbm_gbs)"}
    if top.startswith("layer"):
        v = int(top[5:])
        fl = sum(r["stats"]["flops_layer"][v] for r in bd)
        nl = sum(r["stats"]["launches_layer"][v] for r in bd)
        secs = cls_ms[top] / 1e3
        achieved = fl / secs / 1e12
        layer_node = w.model.nodes[w.model.layers()[v]]
        rows_total = fl / 2 / w.model.layer_macs(v)
        rows = rows_total / max(1, nl)   # rows per launch
        kname, macs_exec = model.layer_kernel(v)
        desc = f"layer {v}: {layer_node.kind} {layer_node.cin}->{layer_node.cout}"
        if kname in ("tc_gemm", "tc_window", "tc_conv"):
            # tensor cores: 3xTF32 spends three TF32 products per fp32 MAC, so its
            # fp32-equivalent peak is a third of the measured TF32 peak
            terms = 3 if args.precision == "tf32x3" else 1
            if tp:
                tf32_peak = tp["tf32_tflops_sustained"] if long_step else tp["tf32_tflops"]
                src = (f"measured here: cuBLAS TF32 {'sustained' if long_step else 'burst'} {tf32_peak:.1f} "
                       f"TFLOP/s / {terms} ({args.precision})")
            else:
                bf16 = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
                tf32_peak = bf16 * 1.1 / 2.25
                src = f"{pk_kind} bf16 sustained {bf16:.1f} TFLOP/s x 1.1/2.25 (TF32) / {terms} ({args.precision})"
            peak = tf32_peak / terms
            label = {"tc_window": "window GEMM", "tc_conv": "staged convolution", "tc_gemm": "implicit GEMM"}[kname]
            roof = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                    "traffic": profiled_traffic(f"{kname}_{args.workload}_layer{v}", rows), "rows_per_launch": rows,
                    "kernel": f"k_tc_gemm ({label}, {desc})", "launches": nl, "ms_total": cls_ms[top],
                    "peak_source": src + "; achieved counts the layer's useful fp32 MACs x 2",
                    "tensor_pipe_frac": terms * 2 * macs_exec * rows_total / secs / 1e12 / tf32_peak}
        else:
            key = "conv_small" if kname == "simt_small" else ("final_dense" if kname == "output" else "stage_simt")
            fp32_peak = tp["fp32_tflops"] if tp else SIMT_FP32_PEAK_TFLOPS
            roof = {"bound": "alu", "achieved": achieved, "peak": fp32_peak, "unit": "TFLOP/s",
                    "frac": achieved / fp32_peak,
                    "traffic": profiled_traffic(f"{key}_{args.workload}_layer{v}", rows), "rows_per_launch": rows,
                    "kernel": f"k_{key} ({desc})", "launches": nl, "ms_total": cls_ms[top],
                    "peak_source": ("measured here: cuBLAS fp32 (CUDA cores)" if tp else
                                    "derived: 152 SMs x 128 FP32 lanes x 2 x 2.07 GHz (CUDA cores)"),
                    "tensor_pipe_frac": 0.0}
    memo_fl, van_fl = analytic_flops(w.model, w.table)
    cfg = config_block(args, w)
    cfg["mutants_per_step"] = float(np.mean([len(tables[i % len(tables)]) for i in range(args.steps)]))
    cfg["slices"] = len(tables)
    cfg["step"] = (f"cache build over all {len(w.X):,} inputs + 1/{len(tables)} of the mutant table (a seeded random "
                   f"partition; {len(tables)} steps = the whole table once)" if len(tables) > 1 else
                   f"cache build over all {len(w.X):,} inputs + the whole mutant table")
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": 1e3 * t_total / args.steps, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": {"fp32": "f32", "tf32x3": "tf32x3", "tf32": "tf32"}[args.precision],
           "data": "synthetic",
           "config": cfg, "roofline": roof, "gpu_launches": int(launches),
           "kernel_ms_per_step": {k: v / n_bd * (n_evals / args.steps) / (bd_evals / n_bd) for k, v in cls_ms.items()},
           "kernel_breakdown": f"separate pass with per-launch events over slices 0..{n_bd - 1}, scaled to the mean "
                               "step; the timed steps run without per-launch events",
           "scores": {"killed_frac": last["scoreA"], "deepmutation": last["scoreB"],
                      "near_ties": last["stats"]["n_near_ties"]},
           "analytic_flops": {"memo_per_eval": memo_fl / len(w.table), "vanilla_per_eval": van_fl / len(w.table),
                              "memo_over_vanilla": memo_fl / van_fl,
                              "memo_tflops_achieved": memo_fl / len(w.table) * n_evals * world / t_total / 1e12}}

    if not args.skip_extras:
        out["clocks"] = clk.summary()
        # end to end through the C ABI with host buffers: pinned X in, kill bits out
        X_pin = torch.from_numpy(w.X).pin_memory()
        kill_host = [np.zeros((len(t), W64), np.uint64) for t in tables]
        k_e2e = max(3, min(args.steps, 5))

        def step_e2e(k):
            j = k % len(tables)
            cache = mure.mure_build_prefix_cache(model, X_pin.numpy())
            return mure.mure_eval_mutants(cache, tables[j], kill_out=kill_host[j], arrays=arrays[j])

        step_e2e(0)
        times, ev_e2e = [], 0
        for k in range(k_e2e):
            flush.zero_()
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            step_e2e(k)          # synchronous: returns with the kill bits in host memory
            times.append(time.perf_counter() - t0)
            ev_e2e += len(tables[k % len(tables)]) * len(w.X)
        e2e_t = max_over_ranks(sum(times), world)
        h2d = int(w.X.nbytes + np.mean([a[0].nbytes + a[1].nbytes for a in arrays]))
        d2h = int(np.mean([kh.nbytes for kh in kill_host]) + 32)
        out["e2e"] = {"value": world * ev_e2e / e2e_t, "unit": UNIT, "h2d_bytes_per_step": h2d,
                      "d2h_bytes_per_step": d2h, "steps": k_e2e}
        # the GPU vanilla mode (speed-up denominator), same kernels, no reuse: slice 0
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        van = mure.mure_eval_vanilla(model, X_dev, tables[0], outputs_on_device=True)
        torch.cuda.synchronize()
        tv = time.perf_counter() - t0
        same = bool(torch.equal(van["kill_bits"], kill_slices[0]))
        m0, v0 = analytic_flops(w.model, tables[0])
        van_rate = len(tables[0]) * len(w.X) / tv
        memo_rate = n_evals / t_total          # one replica's memoized rate
        out["gpu_vanilla"] = {"value": van_rate, "ms_per_step": 1e3 * tv, "slice": 0,
                              "speedup": memo_rate / van_rate, "gain": 1.0 - van_rate / memo_rate,
                              "kill_matrix_identical": same,
                              "achieved_tflops": v0 * len(w.X) / tv / 1e12,
                              "analytic_flops_per_eval": v0 / len(tables[0])}
        # exact unchanged-row elimination (rows whose first suffix input equals the
        # original are not run): the same steps' throughput counting every row, and the
        # share of rows dropped
        k_u = min(len(tables), 3)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        dropped = rows_u = 0
        t_u = 0.0
        for k in range(k_u):
            flush.zero_()
            e0.record(stream)
            cache = mure.mure_build_prefix_cache(model, X_dev)
            ru = mure.mure_eval_mutants(cache, tables[k], outputs_on_device=True, kill_out=kill_slices[k],
                                        arrays=arrays[k], skip_unchanged=True)
            e1.record(stream)
            torch.cuda.synchronize()
            del cache
            t_u += e0.elapsed_time(e1) / 1e3
            dropped += ru["stats"]["n_rows_unchanged"]
            rows_u += ru["stats"]["n_rows"]
        t_plain = sum(ms[i] for i in range(args.steps) if i % len(tables) < k_u) / 1e3
        n_plain = sum(1 for i in range(args.steps) if i % len(tables) < k_u)
        out["unchanged_rows"] = {"effective_value": rows_u / t_u, "unit": UNIT, "rows_dropped_frac": dropped / max(1, rows_u),
                                 "steps": k_u, "plain_value_same_slices": (n_plain and
                                     sum(len(tables[i % len(tables)]) * len(w.X) for i in range(args.steps)
                                         if i % len(tables) < k_u) / t_plain) or None,
                                 "counted": "every (mutant, input) row, dropped ones included, per second"}
        # the stress mix (half of the mutants on the first convolution, 0.1-10 %):
        # one slice of its table over all its inputs, after a warm-up on a few mutants
        if args.workload == "vgg" and args.n_inputs is None and args.n_mutants is None:
            ws_ = wl.workload("vgg_stress")
            st_sl = table_slices(len(ws_.table), SLICES["vgg_stress"])
            tab = ws_.table.subset(st_sl[0])
            Xs = torch.from_numpy(ws_.X).to(f"cuda:{dev}")
            mure.mure_eval_mutants(mure.mure_build_prefix_cache(model, Xs), tab.subset(np.arange(24)))
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            cs = mure.mure_build_prefix_cache(model, Xs)
            rs = mure.mure_eval_mutants(cs, tab, outputs_on_device=True)
            e1.record(stream)
            torch.cuda.synchronize()
            sm, sv = analytic_flops(ws_.model, tab)
            t_s = e0.elapsed_time(e1) / 1e3
            out["stress"] = {"workload": "vgg_stress: " + WORKLOAD_TEXT["vgg_stress"], "value": len(tab) * len(ws_.X) / t_s,
                             "unit": UNIT, "ms_per_step": 1e3 * t_s,
                             "step": f"cache build over all {len(ws_.X):,} inputs + 1/{SLICES['vgg_stress']} of the "
                                     f"table ({len(tab)} mutants)",
                             "memo_over_vanilla_flops": sm / sv, "killed_frac": rs["scoreA"]}
            del cs, Xs
    if rank == 0 and world == 1 and not args.skip_cpu_baseline:
        # the kill matrix of the whole table (slices the timed steps did not reach are
        # evaluated once, untimed) for the agreement check on the oracle's sample
        done = {i % len(tables) for i in range(args.warmup)} | {i % len(tables) for i in range(args.steps)}
        for j in range(len(tables)):
            if j not in done:
                step(j)
        torch.cuda.synchronize()
        import oracle
        oracle.build()
        threads = os.cpu_count() or 1
        n_mut, n_in = cpu_sample_size(w)
        # kill rows are stored slice after slice: put them back in table order
        kd = kill_dev.cpu().numpy()
        kill_table = np.empty_like(kd)
        for j, ix in enumerate(slices):
            kill_table[ix] = kd[int(off[j]):int(off[j + 1])]
        rate, dt, sample, agree = cpu_oracle_rate(w, n_mut, n_in, threads, gpu_kill=kill_table)
        out["cpu_baseline"] = {"value": rate, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample,
                               "seconds": dt}
        # kill verdicts of the timed GPU run against the oracle's on the same sample
        # (differences are expected only on near ties; the TF32 variant reports its rate)
        out["oracle_agreement"] = agree
    out["hbm"] = hbm_rates(w, bd, cls_ms, pk, pk_kind)
    # the cache build (a full forward over the inputs: tensor-bound), bytes for reference
    cb_bytes = w.X.nbytes + cache_bytes(w.model, len(w.X))
    cb_s = float(np.mean(cb_ms)) / 1e3
    out["hbm"]["cache_build"] = {"kernels": "the layer kernels over all inputs (mure_build_prefix_cache)",
                                 "bytes": cb_bytes, "ms": 1e3 * cb_s, "achieved": cb_bytes / cb_s / 1e9, "unit": "GB/s",
                                 "frac": cb_bytes / cb_s / 1e9 / pk["hbm_gbs"],
                                 "tflops": 2.0 * sum(w.model.layer_macs(v) for v in range(L)) * len(w.X) / cb_s / 1e12,
                                 "bytes_counted": "inputs read + every cached x_v and z_v row written once",
                                 "bound": "tensor (one forward pass over the inputs)"}
    # the batched suffix's activation rows written and read back through device memory
    # (not algorithmic bytes: ideally they would stay on chip)
    rows_b = sum(r["stats"].get("bytes_rows", 0) for r in bd)
    evals = sum(r["stats"]["n_rows"] for r in bd)
    if evals > 0:
        out["activation_rows"] = {"bytes_per_eval": rows_b / evals, "unit": "B",
                                  "counted": "suffix stage output rows, written once and read once"}
    out["peaks"] = {"source": pk_kind, "hbm_gbs": pk.get("hbm_gbs"), "bf16_tflops": pk.get("bf16_tflops")}
    if tp:
        out["peaks"].update(tp)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def cache_bytes(model, n_inputs):
    """Bytes of the prefix cache for n inputs: every weighted layer's input x_v and
    pre-activation z_v and the logits (rows rounded up to 4 floats, inputs to a
    multiple of 64), fp32."""
    shapes = model.shapes()
    n_pad = (n_inputs + 63) // 64 * 64
    r4 = lambda n: (n + 3) // 4 * 4
    per = r4(model.n_classes)
    for v in model.layers():
        nd = model.nodes[v]
        src = nd.inputs[0]
        ih, iw, ic = model.in_shape if src < 0 else shapes[src]
        h, ww, c = shapes[v]
        per += r4(ih * iw * ic) + r4(h * ww * c)
    return n_pad * per * 4


def cpu_sample_size(w):
    """(stratified mutants, inputs) of the CPU-baseline sample; the reference arm times
    the same mutants on fewer inputs per step (the oracle's rate is linear in the inputs
    and depends on the mutants per cluster, so both arms see the same rate)."""
    name = w.name
    if name.startswith("vgg"):
        return 128, 8
    if name.startswith("resnet"):
        return 160, 8
    if name.startswith("mlp"):
        return 200, 1000
    return 400, 2000


if __name__ == "__main__":
    sys.exit(main())
