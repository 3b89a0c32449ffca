"""Graphs whose skip branch holds a weighted layer (Algorithm 2's dependence graph is
not a chain): ResNet-10 of Table 1 with 1x1 projection shortcuts.  The GPU compiles a
projection as a stage that reads the block input (an earlier stage input) and adds the
previous stage's output in its epilogue.  Every operator on every layer, projections
included, against the oracle (which runs Algorithm 2's graph literally), memoized ==
vanilla bit for bit, identity mutants never killed, in both fp32-level modes."""
import numpy as np
import pytest

from parity_util import compare_kills, logits_close
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


@pytest.fixture(scope="module")
def case(oracle_mod):
    model = wl.resnet10()
    X = wl.inputs(model, 80, 1)
    subs = []
    for l in range(model.n_layers()):
        ops = tuple(wl.OPS[(l + i) % 6] for i in range(3))
        subs.append(wl.mutants(model, 3, seed=40 + l, ratios=(0.05,), ops=ops, layers=[l]))
    table = wl.concat(subs)
    return model, X, table, oracle_mod.vanilla(model, X, table)


def projection_layers(model):
    """The projections: 1x1 convolutions that read the same block input as the
    convolution two layers before them."""
    lay = model.layers()
    return [l for l, v in enumerate(lay)
            if model.nodes[v].kind == "conv" and model.nodes[v].kh == 1 and l >= 2
            and model.nodes[v].inputs[0] == model.nodes[lay[l - 2]].inputs[0]]


@pytest.mark.parametrize("prec", ["fp32", "tf32x3"])
def test_projection_shortcuts_match_oracle(M, ctx, case, prec):
    model, X, table, ora = case
    proj = projection_layers(model)
    assert len(proj) == 3 and set(proj) <= set(table.layer.tolist())
    m = M.mure_model_load(ctx, model, precision=prec)
    cache = M.mure_build_prefix_cache(m, X)
    lg0, _ = M.mure_cache_outputs(cache)
    ok, worst = logits_close(lg0, ora["orig_logits"])
    assert ok, worst
    r = M.mure_eval_mutants(cache, table, logits=True)
    ok, worst = logits_close(r["logits"], ora["logits"])
    assert ok, worst
    bad, _ = compare_kills(r["kill_bits"], ora["kill_bits"], ora["orig_logits"], ora["logits"], len(X))
    assert bad == 0
    v = M.mure_eval_vanilla(m, X, table, logits=True)
    assert np.array_equal(v["kill_bits"], r["kill_bits"])
    assert np.array_equal(v["logits"].view(np.uint32), r["logits"].view(np.uint32))
    u = M.mure_eval_mutants(cache, table, logits=True, skip_unchanged=True)
    assert np.array_equal(u["logits"].view(np.uint32), r["logits"].view(np.uint32))


def test_projection_identity_mutants(M, ctx):
    model = wl.resnet10()
    X = wl.inputs(model, 64, 1)
    rows = []
    for l in range(model.n_layers()):
        rows.append((l, "IDENTITY", [], 0.0, 0))
        rows.append((l, "GF", [0, 1], 0.0, 3))
    m = M.mure_model_load(ctx, model, precision="tf32x3")
    cache = M.mure_build_prefix_cache(m, X)
    lg0, _ = M.mure_cache_outputs(cache)
    r = M.mure_eval_mutants(cache, wl.table_from_rows(rows), logits=True)
    assert not r["kill_bits"].any()
    for i in range(len(rows)):
        assert np.array_equal(r["logits"][i].view(np.uint32), lg0.view(np.uint32))
