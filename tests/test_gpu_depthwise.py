"""Depthwise convolutions and ReLU6 (the paper's MobileNetV2 family, Table 1): a
MobileNetV2-style network (inverted residual blocks: 1x1 expansion + ReLU6, 3x3
depthwise + ReLU6, linear 1x1 projection, residual add where the shape is kept).  A
depthwise neuron is one channel whose fan-in is its own 3x3 filter, so GF / WS
recompute it from that channel of the cached input alone.  Every operator on every
layer against the oracle, memoized == vanilla bit for bit, the unchanged-row
elimination exact, identity mutants never killed, in both fp32-level modes."""
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
    model = wl.mobilenetv2_tiny()
    X = wl.inputs(model, 72, 1)
    subs = []
    for l in range(model.n_layers()):
        ops = tuple(wl.OPS[(l + i) % 6] for i in range(3))
        subs.append(wl.mutants(model, 3, seed=60 + l, ratios=(0.05,), ops=ops, layers=[l]))
    table = wl.concat(subs)
    return model, X, table, oracle_mod.vanilla(model, X, table)


@pytest.mark.parametrize("prec", ["fp32", "tf32x3"])
def test_depthwise_network_matches_oracle(M, ctx, case, prec):
    model, X, table, ora = case
    dw = [l for l, v in enumerate(model.layers()) if model.nodes[v].kind == "dwconv"]
    assert len(dw) == 3 and set(dw) <= set(table.layer.tolist())
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


def test_depthwise_identity_mutants(M, ctx):
    model = wl.mobilenetv2_tiny()
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
