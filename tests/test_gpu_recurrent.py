"""The recurrent family on the GPU (the paper's RNN models, Sec. 5.3 / Table 1):
embedding + two LSTM layers (the first returning every step) + dense.  A mutant of an
embedding channel changes that channel at every step (its delta is the table entry of
the step's id); a mutant of an LSTM unit changes the whole layer from the first step on
(the recurrence), so the layer is recomputed for the mutant's rows with the unit's rows
rewritten.  Every operator on every layer against the oracle (logits within the fp32
rule, kill bits exact outside near ties), memoized == vanilla bit for bit, the
unchanged-row elimination exact, identity mutants never killed; the IMDB-sized model of
Table 1 (vocabulary 20,000, width 128, 64 units, 80 steps) on a sample; an id outside the
table is refused."""
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


def small_rnn(seed=0):
    return wl.rnn(seed, n_classes=2, vocab=50, dim=8, units=(6, 5), steps=12, name="rnn_small")


def every_operator(model, per_layer, seed):
    subs = []
    for l in range(model.n_layers()):
        ops = tuple(wl.OPS[(l + i) % 6] for i in range(per_layer))
        subs.append(wl.mutants(model, per_layer, seed=seed + l, ratios=(0.3,), ops=ops, layers=[l]))
    return wl.concat(subs)


@pytest.mark.parametrize("size", ["small", "imdb", "reuters"])
def test_recurrent_network_matches_oracle(M, ctx, oracle_mod, size):
    if size == "small":
        model, n_in, per_layer = small_rnn(), 160, 12
    elif size == "imdb":
        model, n_in, per_layer = wl.rnn(), 64, 6
    else:
        # 90 classes: the 96-accumulator output layer and 96-label score sets
        model, n_in, per_layer = wl.rnn_reuters(), 64, 6
    X = wl.inputs(model, n_in, 1)
    table = every_operator(model, per_layer, 70)
    ora = oracle_mod.vanilla(model, X, table)
    m = M.mure_model_load(ctx, model, precision="tf32x3")
    assert [m.layer_kernel(l)[0] for l in range(model.n_layers())][-1] == "output"
    cache = M.mure_build_prefix_cache(m, X)
    lg0, _ = M.mure_cache_outputs(cache)
    ok, worst = logits_close(lg0, ora["orig_logits"])
    assert ok, worst
    r = M.mure_eval_mutants(cache, table, logits=True)
    ok, worst = logits_close(r["logits"], ora["logits"])
    assert ok, worst
    bad, _ = compare_kills(r["kill_bits"], ora["kill_bits"], ora["orig_logits"], ora["logits"], n_in)
    assert bad == 0
    assert r["kill_bits"].any()          # the table kills something
    v = M.mure_eval_vanilla(m, X, table, logits=True)
    assert np.array_equal(v["kill_bits"], r["kill_bits"])
    assert np.array_equal(v["logits"].view(np.uint32), r["logits"].view(np.uint32))
    u = M.mure_eval_mutants(cache, table, logits=True, skip_unchanged=True)
    assert np.array_equal(u["logits"].view(np.uint32), r["logits"].view(np.uint32))
    assert np.array_equal(u["kill_bits"], r["kill_bits"])


def test_recurrent_identity_mutants_and_bad_ids(M, ctx):
    model = small_rnn()
    X = wl.inputs(model, 64, 1)
    rows = []
    for l in range(model.n_layers()):
        rows.append((l, "IDENTITY", [], 0.0, 0))
        rows.append((l, "GF", [0, 1], 0.0, 3))
    m = M.mure_model_load(ctx, model)
    cache = M.mure_build_prefix_cache(m, X)
    lg0, _ = M.mure_cache_outputs(cache)
    r = M.mure_eval_mutants(cache, wl.table_from_rows(rows), logits=True)
    assert not r["kill_bits"].any()
    for i in range(len(rows)):
        assert np.array_equal(r["logits"][i].view(np.uint32), lg0.view(np.uint32))
    bad = X.copy()
    bad[3, 0, 5, 0] = 50.0                 # one id past the table
    with pytest.raises(M.MureError) as ei:
        M.mure_build_prefix_cache(m, bad)
    assert ei.value.status == 1
    # the context stays usable
    again = M.mure_eval_mutants(M.mure_build_prefix_cache(m, X), wl.table_from_rows(rows), logits=True)
    assert np.array_equal(again["logits"].view(np.uint32), r["logits"].view(np.uint32))
