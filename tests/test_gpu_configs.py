"""Parity of the benchmarked path (3xTF32 tensor cores, the default precision of the
benchmark) with the CPU oracle at the workloads' own scale: the VGG-style network at
each of its four selection ratios, ResNet-20, and the VGG stress mix (half of the
mutants on the first convolution, ratios 0.1% to 10%).

The GPU evaluates a stratified set of each workload's mutant table (every layer x
operator x selection ratio, at least 25 mutants per layer) over ALL of the workload's
inputs (10,000, or 20,000 for the stress mix) with the default batch geometry.  The
oracle computes a sample of those (mutant, input) pairs one by one: every sampled
mutant on inputs spread over the whole input range (first, last and in between).
Logits and kill bits are compared with the rules of parity_util; memoized == vanilla
bit for bit on the stress mix, the memoization floor (the paper's soundness theorem,
Sec. 4).  The oracle's time (a few hundred evaluations per second on the VGG family)
bounds the sample: 8 inputs per mutant."""
import numpy as np
import pytest

from parity_util import bits, logits_close, margin_tie
from paper_2607_18582_gb300 import workloads as wl

N_SAMPLE_INPUTS = 8


@pytest.fixture(scope="module")
def M():
    from paper_2607_18582_gb300 import build
    build.build()
    from paper_2607_18582_gb300 import mure
    return mure


@pytest.fixture(scope="module")
def ctx(M):
    return M.mure_create(0)


def stratified_by_ratio(table, n_layers, per_class, min_per_layer):
    """Indices of the first `per_class` mutants of every (layer, operator, ratio) class
    in table order, topped up in table order until every layer has at least
    `min_per_layer` of its mutants."""
    picked, seen = [], {}
    for i in range(len(table)):
        key = (int(table.layer[i]), int(table.op[i]), float(table.ratio[i]))
        if seen.get(key, 0) < per_class:
            seen[key] = seen.get(key, 0) + 1
            picked.append(i)
    chosen = set(picked)
    per_layer = np.bincount(table.layer[picked], minlength=n_layers)
    for i in range(len(table)):
        l = int(table.layer[i])
        if per_layer[l] >= min_per_layer:
            continue
        if i not in chosen:
            chosen.add(i)
            per_layer[l] += 1
    return np.array(sorted(chosen), np.int64)


def sample_inputs(n):
    """Inputs spread over the whole range, the first and the last included."""
    return np.unique(np.linspace(0, n - 1, N_SAMPLE_INPUTS).round().astype(np.int64))


CONFIGS = {
    # workload: (mutants per (layer, op, ratio) class, minimum per layer)
    "vgg": (2, 25),
    "resnet20": (7, 25),
    "vgg_stress": (2, 25),
}


@pytest.mark.gpu
@pytest.mark.slow
@pytest.mark.parametrize("name", list(CONFIGS))
def test_config_scale_matches_oracle(M, ctx, oracle_mod, name):
    per_class, min_per_layer = CONFIGS[name]
    w = wl.workload(name)
    L = w.model.n_layers()
    idx = stratified_by_ratio(w.table, L, per_class, min_per_layer)
    sub = w.table.subset(idx)
    # coverage of the stratified set: every layer, every operator and every ratio
    assert np.bincount(sub.layer, minlength=L).min() >= min_per_layer
    assert set(np.unique(sub.op).tolist()) == {wl.OP_INDEX[o] for o in wl.CONFIG_OPS}
    assert set(np.unique(sub.ratio).tolist()) == set(wl.CONFIGS[name][3])

    model = M.mure_model_load(ctx, w.model, precision="tf32x3")
    cache = M.mure_build_prefix_cache(model, w.X)
    res = M.mure_eval_mutants(cache, sub, logits=True)
    lg0, pred0 = M.mure_cache_outputs(cache)
    n = len(w.X)
    assert 0.0 <= res["scoreA"] <= 1.0 and 0.0 <= res["scoreB"] <= 1.0
    assert res["stats"]["n_rows"] == len(sub) * n

    ti = sample_inputs(n)
    ora = oracle_mod.vanilla(w.model, w.X[ti], sub)
    ok, worst = logits_close(lg0[ti], ora["orig_logits"])
    assert ok, ("original logits", worst)
    ok, worst = logits_close(res["logits"][:, ti], ora["logits"])
    assert ok, ("mutant logits", worst)
    g = bits(res["kill_bits"], n)[:, ti]
    o = bits(ora["kill_bits"], len(ti))
    ties = margin_tie(ora["logits"]) | margin_tie(ora["orig_logits"])[None, :]
    assert int(((g != o) & ~ties).sum()) == 0, int(ties.sum())

    if name == "vgg_stress":
        van = M.mure_eval_vanilla(model, w.X, sub)
        assert np.array_equal(van["kill_bits"], res["kill_bits"])
        assert van["scoreA"] == res["scoreA"] and van["scoreB"] == res["scoreB"]


def test_stratified_sets_cover_the_skewed_mix():
    """The stress mix's sample holds the first convolution's share and the extreme
    ratios (0.1% and 10%) on every layer (host-side check of the sampling)."""
    w = wl.workload("vgg_stress", 64)
    idx = stratified_by_ratio(w.table, w.model.n_layers(), *CONFIGS["vgg_stress"])
    sub = w.table.subset(idx)
    for l in range(w.model.n_layers()):
        rs = set(sub.ratio[sub.layer == l].tolist())
        assert {0.001, 0.10} <= rs, (l, rs)
