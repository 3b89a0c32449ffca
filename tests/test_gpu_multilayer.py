"""Mutants over several layers (tagged descriptors, model-wide selection ratio) on the
CUDA path: parity with the oracle, memoized == vanilla bit for bit, a mutant's bits
independent of the batch it shares with single-layer mutants, tagged single-layer
descriptors equal to untagged ones, and the descriptor checks.  Rules in parity_util."""
import numpy as np
import pytest

from parity_util import compare_kills, logits_close
from paper_2607_18582_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

PRECISIONS = ["fp32", "tf32x3"]


@pytest.fixture(scope="module")
def M():
    from paper_2607_18582_gb300 import build
    build.build()
    from paper_2607_18582_gb300 import mure
    return mure


@pytest.fixture(scope="module")
def ctx(M):
    return M.mure_create(0)


def _case(name):
    """(workload, table): model-wide tables that mutate several layers per mutant."""
    if name == "lenet5":
        w = wl.workload("lenet5_modelwide", 130, 80)
        return w, w.table
    if name == "mlp":
        w = wl.workload("mlp_modelwide", 200, 60)
        return w, w.table
    if name == "resnet20":
        w = wl.workload("resnet20", 66, 1)
        return w, wl.modelwide_mutants(w.model, 16, seed=7, ratio=0.004)
    w = wl.workload("vgg", 65, 1)
    return w, wl.modelwide_mutants(w.model, 12, seed=8, ratio=0.002)


@pytest.fixture(scope="module")
def runs(oracle_mod):
    cache = {}

    def get(name):
        if name not in cache:
            w, table = _case(name)
            spans = [len({int(e) >> 20 for e in table.pool[a:a + n]})
                     for a, n in zip(table.neuron_off, table.n_neurons)]
            assert max(spans) >= 2
            cache[name] = (w, table, oracle_mod.vanilla(w.model, w.X, table))
        return cache[name]
    return get


@pytest.mark.parametrize("prec", PRECISIONS)
@pytest.mark.parametrize("name", ["lenet5", "mlp", "resnet20", "vgg"])
def test_modelwide_matches_oracle_and_vanilla(M, ctx, runs, name, prec):
    w, table, ora = runs(name)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    res = M.mure_eval_mutants(cache, table, logits=True)
    ok, worst = logits_close(res["logits"], ora["logits"])
    assert ok, worst
    bad, ties = compare_kills(res["kill_bits"], ora["kill_bits"], ora["orig_logits"], ora["logits"], len(w.X))
    assert bad == 0, (bad, ties)
    if ties == 0:
        assert res["scoreA"] == ora["scoreA"] and res["scoreB"] == pytest.approx(ora["scoreB"], abs=1e-12)
    van = M.mure_eval_vanilla(model, w.X, table, logits=True)
    assert np.array_equal(res["kill_bits"], van["kill_bits"])
    assert np.array_equal(res["logits"].view(np.uint32), van["logits"].view(np.uint32))


@pytest.mark.parametrize("prec", PRECISIONS)
def test_mixed_tables_batch_invariance(M, ctx, prec):
    """Single-layer and model-wide mutants in one table: every mutant's bits equal
    those of the same mutant evaluated alone in its kind's table and under a small
    workspace (many batches)."""
    w = wl.workload("lenet5", 260, 120)
    mw = wl.modelwide_mutants(w.model, 60, seed=9)
    single = w.table
    tag1 = np.zeros(len(single), np.int32)
    single_t = wl.MutantTable(single.layer, single.op, single.n_neurons, single.neuron_off, single.param,
                              single.seed, single.pool, single.ratio, tag1)
    mixed = wl.concat([single_t, mw])
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    both = M.mure_eval_mutants(cache, mixed, logits=True)
    a = M.mure_eval_mutants(cache, single_t, logits=True)
    b = M.mure_eval_mutants(cache, mw, logits=True)
    small = M.mure_eval_mutants(cache, mixed, logits=True, workspace_bytes=64 * 8 * 1024)
    n1 = len(single_t)
    assert np.array_equal(both["logits"][:n1].view(np.uint32), a["logits"].view(np.uint32))
    assert np.array_equal(both["logits"][n1:].view(np.uint32), b["logits"].view(np.uint32))
    assert np.array_equal(both["logits"].view(np.uint32), small["logits"].view(np.uint32))
    assert np.array_equal(both["kill_bits"], small["kill_bits"])


def test_tagged_single_layer_equals_untagged(M, ctx):
    w = wl.workload("lenet5", 140, 100)
    t = w.table
    pool = t.pool.copy()
    for i in range(len(t)):
        a, n = int(t.neuron_off[i]), int(t.n_neurons[i])
        pool[a:a + n] = (int(t.layer[i]) << 20) | t.pool[a:a + n]
    tag = wl.MutantTable(t.layer, t.op, t.n_neurons, t.neuron_off, t.param, t.seed, pool, t.ratio,
                         np.ones(len(t), np.int32))
    model = M.mure_model_load(ctx, w.model, precision="tf32x3")
    cache = M.mure_build_prefix_cache(model, w.X)
    r0 = M.mure_eval_mutants(cache, t, logits=True)
    r1 = M.mure_eval_mutants(cache, tag, logits=True)
    assert np.array_equal(r0["logits"].view(np.uint32), r1["logits"].view(np.uint32))
    assert np.array_equal(r0["kill_bits"], r1["kill_bits"])


def test_invalid_tagged_descriptors(M, ctx):
    w = wl.workload("lenet5", 10, 1)
    model = M.mure_model_load(ctx, w.model)
    cache = M.mure_build_prefix_cache(model, w.X)

    def tagged(entries, op, layer):
        ent = np.array([(l << 20) | j for l, j in entries], np.int32)
        return wl.MutantTable(np.array([layer], np.int32), np.array([wl.OP_INDEX[op]], np.int32),
                              np.array([len(ent)], np.int32), np.array([0], np.int64), np.array([0.1], np.float32),
                              np.array([1], np.uint64), ent, np.zeros(1), np.ones(1, np.int32))
    bad = [tagged([(1, 3), (2, 5)], "NEB", 2), tagged([(1, 3), (2, 5)], "NS", 1), tagged([(1, 3), (1, 3)], "GF", 1),
           tagged([(1, 16)], "GF", 1), tagged([(5, 0)], "GF", 5)]
    for t in bad:
        kill = np.full((1, 1), 0xDEADBEEF, np.uint64)
        with pytest.raises(M.MureError) as ei:
            M.mure_eval_mutants(cache, t, kill_out=kill)
        assert ei.value.status == 1
        assert kill[0, 0] == 0xDEADBEEF
    # the expansion entry points take untagged descriptors only
    with pytest.raises(M.MureError):
        M.mure_expand_patches(model, tagged([(1, 3), (3, 5)], "GF", 1))
