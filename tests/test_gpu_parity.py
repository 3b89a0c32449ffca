"""Parity of the CUDA path (through the C ABI) with the CPU oracle on the same seeded
inputs: original logits, mutant logits, kill matrices and scores; memoized ==
vanilla bit for bit; expanded random patches bit for bit; batch invariance; edge
cases.  Rules in parity_util."""
import numpy as np
import pytest

from conftest import tiny_worked_example
from parity_util import bits, compare_kills, logits_close, margin_tie
from paper_2607_18582_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def M():
    from paper_2607_18582_gb300 import build
    build.build()
    from paper_2607_18582_gb300 import mure
    return mure


@pytest.fixture(scope="module")
def ctx(M):
    return M.mure_create(0)


def all_ops(model, per_layer, seed=5, ratios=(0.05,)):
    """Every operator on every layer (cycling the six operators)."""
    subs = []
    for l in range(model.n_layers()):
        ops = [wl.OPS[(l * per_layer + i) % 6] for i in range(per_layer)]
        subs.append(wl.mutants(model, per_layer, seed=seed + l, ratios=ratios, ops=tuple(ops), layers=[l]))
    return wl.concat(subs)


CASES = {
    # name: (n_inputs, table builder)
    "mlp": (200, lambda m: all_ops(m, 12)),
    "lenet5": (130, lambda m: all_ops(m, 8)),
    "resnet20": (66, lambda m: all_ops(m, 2)),
    "vgg": (65, lambda m: all_ops(m, 2)),
}


@pytest.fixture(scope="module")
def oracle_runs(oracle_mod):
    cache = {}

    def get(name):
        if name not in cache:
            n_in, mk = CASES[name]
            w = wl.workload(name, n_in, 1)
            table = mk(w.model)
            cache[name] = (w, table, oracle_mod.vanilla(w.model, w.X, table))
        return cache[name]
    return get


PRECISIONS = ["fp32", "tf32x3"]


@pytest.mark.parametrize("prec", PRECISIONS)
@pytest.mark.parametrize("name", list(CASES))
def test_cache_build_matches_oracle(M, ctx, oracle_runs, name, prec):
    w, table, ora = oracle_runs(name)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    lg, pred = M.mure_cache_outputs(cache)
    ok, worst = logits_close(lg, ora["orig_logits"])
    assert ok, worst
    ties = margin_tie(ora["orig_logits"])
    assert np.array_equal(pred[~ties], ora["orig_logits"].argmax(axis=1)[~ties])


@pytest.mark.parametrize("prec", PRECISIONS)
@pytest.mark.parametrize("name", list(CASES))
def test_memoized_matches_oracle(M, ctx, oracle_runs, name, prec):
    w, table, ora = oracle_runs(name)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    res = M.mure_eval_mutants(cache, table, logits=True)
    ok, worst = logits_close(res["logits"], ora["logits"])
    assert ok, worst
    bad, ties = compare_kills(res["kill_bits"], ora["kill_bits"], ora["orig_logits"], ora["logits"], len(w.X))
    assert bad == 0, (bad, ties)
    if ties == 0:
        assert res["scoreA"] == ora["scoreA"] and res["scoreB"] == pytest.approx(ora["scoreB"], abs=1e-12)
    assert res["stats"]["n_rows"] == len(table) * len(w.X)


@pytest.mark.parametrize("prec", PRECISIONS)
@pytest.mark.parametrize("name", list(CASES))
def test_memoized_equals_vanilla_bitwise(M, ctx, oracle_runs, name, prec):
    w, table, _ = oracle_runs(name)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    memo = M.mure_eval_mutants(cache, table, logits=True)
    van = M.mure_eval_vanilla(model, w.X, table, logits=True)
    assert np.array_equal(memo["kill_bits"], van["kill_bits"])
    assert np.array_equal(memo["logits"].view(np.uint32), van["logits"].view(np.uint32))
    assert memo["scoreA"] == van["scoreA"] and memo["scoreB"] == van["scoreB"]
    assert van["stats"]["flops"] > memo["stats"]["flops"]


def test_worked_example_gpu(M, ctx):
    m, X, labels, table, g = tiny_worked_example()
    model = M.mure_model_load(ctx, m)
    for lab, key in ((labels, "labels"), (None, "nolabels")):
        cache = M.mure_build_prefix_cache(model, X, labels=lab)
        r = M.mure_eval_mutants(cache, table)
        assert r["kill_bits"][:, 0].tolist() == [int(v) for v in g["kill_" + key][0]]
        assert r["scoreA"] == pytest.approx(float(g["scoreA_" + key][0][0]), abs=1e-15)
        assert r["scoreB"] == pytest.approx(float(g["scoreB_" + key][0][0]), abs=1e-15)
        v = M.mure_eval_vanilla(model, X, table, labels=lab)
        assert np.array_equal(v["kill_bits"], r["kill_bits"])


def test_labels_given(M, ctx, oracle_mod):
    w = wl.workload("lenet5", 190, 1)
    table = all_ops(w.model, 4, seed=11)
    labels = np.random.default_rng(3).integers(0, 10, 190).astype(np.int32)
    ora = oracle_mod.vanilla(w.model, w.X, table, labels=labels)
    model = M.mure_model_load(ctx, w.model)
    cache = M.mure_build_prefix_cache(model, w.X, labels=labels)
    res = M.mure_eval_mutants(cache, table, logits=True)
    bad, ties = compare_kills(res["kill_bits"], ora["kill_bits"], ora["orig_logits"], ora["logits"], 190)
    assert bad == 0
    if ties == 0:
        assert res["scoreB"] == pytest.approx(ora["scoreB"], abs=1e-12)


def test_expanded_patches_bitexact(M, ctx, oracle_mod):
    """GF noise and WS shuffles from the library equal the oracle's generator."""
    for name in ("lenet5", "vgg"):
        w = wl.workload(name, 1, 1)
        rows = []
        for l in range(w.model.n_layers()):
            N = w.model.layer_width(l)
            rows.append((l, "GF", [0, N - 1], 0.1, 1000 + l))
            rows.append((l, "WS", [N // 2], 0.0, 2000 + l))
        table = wl.table_from_rows(rows)
        model = M.mure_model_load(ctx, w.model)
        vals, offs = M.mure_expand_patches(model, table)
        mism = total = 0
        for i, (l, op, ids, param, seed) in enumerate(rows):
            nd = w.model.nodes[w.model.layers()[l]]
            F = nd.W.size // nd.cout
            if op == "GF":
                sigma = float(np.float32(param)) * oracle_mod.layer_std(w.model, l)
                for q in range(len(ids)):
                    s = oracle_mod.sm64(seed, q)
                    exp = np.array([np.float32(sigma * oracle_mod.gauss(s, f)) for f in range(F)], np.float32)
                    got = vals[offs[i] + q * F: offs[i] + (q + 1) * F]
                    mism += int((got.view(np.uint32) != exp.view(np.uint32)).sum())
                    total += F
            else:
                Wm, _, _ = oracle_mod.mutant_layer(w.model, table, i)
                got = vals[offs[i]: offs[i] + F]
                exp = Wm.reshape(nd.cout, -1)[ids[0]]
                assert np.array_equal(got, exp)
        # fp64 libm results may differ in their last bit between host and device;
        # after scaling and rounding to fp32 that almost never shows
        assert mism <= max(1, total // 1_000_000), (mism, total)


@pytest.mark.parametrize("prec", PRECISIONS)
def test_batch_invariance(M, ctx, prec):
    """Tiny workspaces force many batches (input tiles, mutant chunks): results are
    bitwise identical to one large batch."""
    w = wl.workload("lenet5", 300, 1)
    table = all_ops(w.model, 6, seed=21)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    big = M.mure_eval_mutants(cache, table, logits=True)
    small = M.mure_eval_mutants(cache, table, logits=True, workspace_bytes=64 * 8 * 1024)
    assert small["stats"]["n_batches"] > big["stats"]["n_batches"]
    assert np.array_equal(big["kill_bits"], small["kill_bits"])
    assert np.array_equal(big["logits"].view(np.uint32), small["logits"].view(np.uint32))
    # a cache built over a subset of the inputs gives the same rows
    cache2 = M.mure_build_prefix_cache(model, w.X[:70])
    sub = M.mure_eval_mutants(cache2, table, logits=True)
    assert np.array_equal(sub["logits"].view(np.uint32), big["logits"][:, :70].view(np.uint32))


def test_repeat_and_vanilla_bitwise_at_scale(M, ctx):
    """A larger LeNet-5 run (many tiles per CTA, every copy ring wrapping many times):
    two memoized evaluations and the vanilla one give the same bits.  Catches races
    between the copy engines and the threads that read their buffers."""
    w = wl.workload("lenet5", 4096, 400)
    model = M.mure_model_load(ctx, w.model, precision="tf32x3")
    cache = M.mure_build_prefix_cache(model, w.X)
    a = M.mure_eval_mutants(cache, w.table)
    b = M.mure_eval_mutants(cache, w.table)
    assert np.array_equal(a["kill_bits"], b["kill_bits"])
    van = M.mure_eval_vanilla(model, w.X, w.table)
    assert np.array_equal(a["kill_bits"], van["kill_bits"])


@pytest.mark.parametrize("prec", ["tf32x3", "tf32"])
def test_batch_invariance_tensor_core_delta(M, ctx, prec):
    """GF / WS deltas of the generic convolutions run as one tensor-core GEMM per batch
    whose output channels are the batch's slots: a slot's values must not depend on
    how many other slots share its batch (many small batches vs one)."""
    w = wl.workload("vgg", 64, 1)
    rows = []
    for l in range(1, w.model.n_layers() - 2):
        for i in range(6):
            rows.append((l, "GF" if i % 2 == 0 else "WS", [i, i + 7], 1.0 if i % 2 == 0 else 0.0, 100 + 7 * l + i))
    table = wl.table_from_rows(rows)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    big = M.mure_eval_mutants(cache, table, logits=True)
    small = M.mure_eval_mutants(cache, table, logits=True, workspace_bytes=32 << 20)
    assert small["stats"]["n_batches"] > big["stats"]["n_batches"]
    assert np.array_equal(big["logits"].view(np.uint32), small["logits"].view(np.uint32))
    van = M.mure_eval_vanilla(model, w.X, table, logits=True)
    assert np.array_equal(big["logits"].view(np.uint32), van["logits"].view(np.uint32))


@pytest.mark.parametrize("prec", ["tf32x3", "tf32"])
def test_batch_invariance_windows_pairs_residual_delta(M, ctx, prec):
    """ResNet-20 on the tensor cores: its 16-channel convolutions run as 2x2 output
    windows, its 16- to 64-channel ones in pairs of tiles, and the GF / WS deltas of the
    convolutions with a residual add as the slot GEMM with each slot's skip channel:
    every operator on every layer gives the same bits in many small batches as in a few
    large ones, and memoized == vanilla bit for bit."""
    w = wl.workload("resnet20", 128, 1)
    table = all_ops(w.model, 6, seed=61)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    big = M.mure_eval_mutants(cache, table, logits=True)
    small = M.mure_eval_mutants(cache, table, logits=True, workspace_bytes=64 << 20)
    assert small["stats"]["n_batches"] > big["stats"]["n_batches"]
    assert np.array_equal(big["kill_bits"], small["kill_bits"])
    assert np.array_equal(big["logits"].view(np.uint32), small["logits"].view(np.uint32))
    van = M.mure_eval_vanilla(model, w.X, table, logits=True)
    assert np.array_equal(big["logits"].view(np.uint32), van["logits"].view(np.uint32))


@pytest.mark.parametrize("name,prec", [("resnet20", "fp32"), ("mlp", "tf32x3"), ("lenet5", "tf32x3")])
def test_identity_mutants_never_killed(M, ctx, name, prec):
    w = wl.workload(name, 96, 1)
    rows = []
    for l in range(w.model.n_layers()):
        rows.append((l, "IDENTITY", [], 0.0, 0))
        rows.append((l, "GF", [0, 3], 0.0, 7))   # sigma multiplier 0
    table = wl.table_from_rows(rows)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    lg0, _ = M.mure_cache_outputs(cache)
    r = M.mure_eval_mutants(cache, table, logits=True)
    assert not r["kill_bits"].any() and r["scoreA"] == 0.0
    for i in range(len(rows)):
        assert np.array_equal(r["logits"][i].view(np.uint32), lg0.view(np.uint32))


@pytest.mark.parametrize("n_in", [1, 63, 64, 65, 129])
def test_ragged_inputs(M, ctx, oracle_mod, n_in):
    w = wl.workload("mlp", n_in, 1)
    table = all_ops(w.model, 6, seed=31)
    ora = oracle_mod.vanilla(w.model, w.X, table)
    model = M.mure_model_load(ctx, w.model)
    cache = M.mure_build_prefix_cache(model, w.X)
    r = M.mure_eval_mutants(cache, table, logits=True)
    bad, _ = compare_kills(r["kill_bits"], ora["kill_bits"], ora["orig_logits"], ora["logits"], n_in)
    assert bad == 0
    assert r["kill_bits"].shape == (len(table), (n_in + 63) // 64)
    # padding bits beyond n_in are zero
    assert not (bits(np.asarray(r["kill_bits"]), ((n_in + 63) // 64) * 64)[:, n_in:]).any()


def test_empty_and_invalid(M, ctx):
    w = wl.workload("mlp", 10, 6)
    model = M.mure_model_load(ctx, w.model)
    cache = M.mure_build_prefix_cache(model, w.X)
    r = M.mure_eval_mutants(cache, w.table.subset([]))
    assert r["scoreA"] == 0.0 and r["scoreB"] == 0.0
    empty = M.mure_build_prefix_cache(model, w.X[:0])
    r = M.mure_eval_mutants(empty, w.table)
    assert r["scoreA"] == 0.0 and r["kill_bits"].shape[1] == 0
    bad_rows = [[(5, "GF", [0], 0.1, 1)], [(0, "NEB", [128], 0.0, 1)], [(0, "NAI", [3, 3], 0.0, 1)],
                [(0, "NS", [1, 2, 3], 0.0, 1)]]
    for rows in bad_rows:
        kill = np.full((1, 1), 0xDEADBEEF, np.uint64)
        with pytest.raises(M.MureError) as ei:
            M.mure_eval_mutants(cache, wl.table_from_rows(rows), kill_out=kill)
        assert ei.value.status == 1
        assert kill[0, 0] == 0xDEADBEEF   # outputs untouched on a validation error
    with pytest.raises(M.MureError):
        M.mure_build_prefix_cache(model, w.X, labels=np.full(10, 12, np.int32))


def test_device_inputs_and_outputs(M, ctx):
    import torch
    w = wl.workload("lenet5", 128, 40)
    model = M.mure_model_load(ctx, w.model)
    host = M.mure_eval_mutants(M.mure_build_prefix_cache(model, w.X), w.table)
    Xd = torch.from_numpy(w.X).cuda()
    dev = M.mure_eval_mutants(M.mure_build_prefix_cache(model, Xd), w.table, outputs_on_device=True)
    torch.cuda.synchronize()
    assert np.array_equal(dev["kill_bits"].cpu().numpy().view(np.uint64), host["kill_bits"])
    assert dev["scoreA"] == host["scoreA"]


@pytest.mark.slow
@pytest.mark.parametrize("prec", PRECISIONS)
def test_full_size_lenet_sampled(M, ctx, oracle_mod, prec):
    """The LeNet-5 configuration at full size (10,000 inputs, 2,000 mutants, one
    batch geometry as the benchmark runs it) in both fp32-level modes (CUDA-core fp32
    chains and the benchmarked 3xTF32 tensor-core path), checked on a sample of
    mutants x inputs that the oracle computes one by one."""
    w = wl.workload("lenet5")
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    r = M.mure_eval_mutants(cache, w.table)
    rng = np.random.default_rng(0)
    mi = np.sort(rng.choice(len(w.table), 48, replace=False))
    ti = np.sort(rng.choice(len(w.X), 256, replace=False))
    sub = w.table.subset(mi)
    ora = oracle_mod.vanilla(w.model, w.X[ti], sub)
    g = bits(r["kill_bits"], len(w.X))[mi][:, ti]
    o = bits(ora["kill_bits"], len(ti))
    ties = margin_tie(ora["logits"]) | margin_tie(ora["orig_logits"])[None, :]
    assert int(((g != o) & ~ties).sum()) == 0
    assert 0.0 <= r["scoreA"] <= 1.0 and 0.0 <= r["scoreB"] <= 1.0


def test_kernel_variants_agree_bitwise(M, ctx, monkeypatch):
    """The shared-memory direct convolution and the implicit-GEMM kernel compute the
    same fp32 chains: a model forced onto the generic kernel gives identical bits."""
    w = wl.workload("lenet5", 200, 1)
    table = all_ops(w.model, 6, seed=41)
    fast = M.mure_model_load(ctx, w.model)
    monkeypatch.setenv("MURE_FORCE_GENERIC", "1")
    generic = M.mure_model_load(ctx, w.model)
    monkeypatch.delenv("MURE_FORCE_GENERIC")
    r1 = M.mure_eval_mutants(M.mure_build_prefix_cache(fast, w.X), table, logits=True)
    r2 = M.mure_eval_mutants(M.mure_build_prefix_cache(generic, w.X), table, logits=True)
    assert np.array_equal(r1["logits"].view(np.uint32), r2["logits"].view(np.uint32))
    assert np.array_equal(r1["kill_bits"], r2["kill_bits"])
    v1 = M.mure_eval_vanilla(fast, w.X, table, logits=True)
    assert np.array_equal(v1["logits"].view(np.uint32), r1["logits"].view(np.uint32))


@pytest.mark.parametrize("name", list(CASES))
def test_tf32_variant_verdicts(M, ctx, oracle_runs, name):
    """The reduced-precision variant (one TF32 product per MAC on the tensor cores):
    memoized == vanilla bit for bit, and its kill verdicts agree with the fp32 oracle
    on nearly every (mutant, input) pair; the agreement rate is what is reported."""
    w, table, ora = oracle_runs(name)
    model = M.mure_model_load(ctx, w.model, precision="tf32")
    cache = M.mure_build_prefix_cache(model, w.X)
    memo = M.mure_eval_mutants(cache, table, logits=True)
    van = M.mure_eval_vanilla(model, w.X, table, logits=True)
    assert np.array_equal(memo["kill_bits"], van["kill_bits"])
    assert np.array_equal(memo["logits"].view(np.uint32), van["logits"].view(np.uint32))
    agree = (bits(memo["kill_bits"], len(w.X)) == bits(ora["kill_bits"], len(w.X))).mean()
    assert agree >= 0.98, agree


@pytest.mark.parametrize("mode", ["small", "generic"])
@pytest.mark.parametrize("prec", ["tf32x3", "tf32"])
def test_tensor_core_conv_on_small_layers(M, ctx, oracle_mod, monkeypatch, prec, mode):
    """LeNet's conv 6->16 on the tensor cores, in the small-image mode (a GEMM row per
    pooling window, N = 4 positions x 16 channels, maps staged in shared memory) and
    through the implicit-GEMM producers: memoized == vanilla bit for bit, 3xTF32 within
    the fp32 tolerance of the oracle, the TF32 variant's verdicts nearly all agree.
    With 25 windows per map, 128-row tiles straddle up to seven maps."""
    w = wl.workload("lenet5", 130, 1)
    table = all_ops(w.model, 6, seed=51)
    ora = oracle_mod.vanilla(w.model, w.X, table)
    monkeypatch.setenv("MURE_TC_CONV", mode)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    monkeypatch.delenv("MURE_TC_CONV")
    r = M.mure_eval_mutants(M.mure_build_prefix_cache(model, w.X), table, logits=True)
    v = M.mure_eval_vanilla(model, w.X, table, logits=True)
    assert np.array_equal(v["logits"].view(np.uint32), r["logits"].view(np.uint32))
    assert np.array_equal(v["kill_bits"], r["kill_bits"])
    if prec == "tf32x3":
        ok, worst = logits_close(r["logits"], ora["logits"])
        assert ok, worst
        bad, _ = compare_kills(r["kill_bits"], ora["kill_bits"], ora["orig_logits"], ora["logits"], len(w.X))
        assert bad == 0
    else:
        agree = (bits(r["kill_bits"], len(w.X)) == bits(ora["kill_bits"], len(w.X))).mean()
        assert agree >= 0.98, agree


@pytest.mark.parametrize("name", ["vgg", "resnet20"])
def test_gather_mode_convolutions_match_oracle(M, ctx, oracle_runs, monkeypatch, name):
    """Stride-1 convolutions with 32k input channels run by default on input rows
    staged in shared memory (K order: 32-channel chunk, tap, channel); with
    MURE_TC_CONV=gather they keep the per-row gathers from device memory (K order: tap,
    channel).  Both orders are fixed per model, so each mode is memoized == vanilla bit
    for bit and within the fp32 tolerance of the oracle; the model reports which kernel
    each layer uses."""
    w, table, ora = oracle_runs(name)
    staged = M.mure_model_load(ctx, w.model, precision="tf32x3")
    kinds = [staged.layer_kernel(l)[0] for l in range(w.model.n_layers())]
    assert "tc_conv" in kinds, kinds
    monkeypatch.setenv("MURE_TC_CONV", "gather")
    gather = M.mure_model_load(ctx, w.model, precision="tf32x3")
    monkeypatch.delenv("MURE_TC_CONV")
    assert "tc_conv" not in [gather.layer_kernel(l)[0] for l in range(w.model.n_layers())]
    for model in (staged, gather):
        r = M.mure_eval_mutants(M.mure_build_prefix_cache(model, w.X), table, logits=True)
        ok, worst = logits_close(r["logits"], ora["logits"])
        assert ok, worst
        bad, _ = compare_kills(r["kill_bits"], ora["kill_bits"], ora["orig_logits"], ora["logits"], len(w.X))
        assert bad == 0
        v = M.mure_eval_vanilla(model, w.X, table, logits=True)
        assert np.array_equal(v["logits"].view(np.uint32), r["logits"].view(np.uint32))
