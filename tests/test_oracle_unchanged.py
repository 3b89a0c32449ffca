"""Pins of the oracle's exact unchanged-row reference (a (mutant, input) row whose mutated
layers all give the original outputs bit for bit): soundness against the vanilla run,
closed characterisations for NEB (the channel was all +0) and NS (the two channels were
equal), identity mutants, and mutants over several layers."""
import numpy as np
import pytest

from parity_util import bits
from paper_2607_18582_gb300 import workloads as wl


def _sound(oracle_mod, model, X, table):
    ub = bits(oracle_mod.unchanged_rows(model, X, table), len(X))
    r = oracle_mod.vanilla(model, X, table)
    kb = bits(r["kill_bits"], len(X))
    for i, t in zip(*np.nonzero(ub)):
        assert np.array_equal(r["logits"][i, t].view(np.uint32), r["orig_logits"][t].view(np.uint32))
        assert not kb[i, t]
    return ub


@pytest.mark.parametrize("name", ["lenet5", "lenet5_modelwide", "mlp_modelwide"])
def test_unchanged_rows_are_sound(oracle_mod, name):
    w = wl.workload(name, 40, 80)
    ub = _sound(oracle_mod, w.model, w.X, w.table)
    assert ub.shape == (80, 40)


def test_neb_and_ns_characterisations(oracle_mod):
    w = wl.workload("lenet5", 30, 1)
    m = w.model
    rows = []
    for layer in range(m.n_layers()):
        for j in range(min(6, m.layer_width(layer))):
            rows.append((layer, "NEB", [j], 0.0, 0))
        rows.append((layer, "NS", [0, 1], 0.0, 0))
    table = wl.table_from_rows(rows)
    ub = _sound(oracle_mod, m, w.X, table)
    nodes = [oracle_mod.forward_nodes(m, x) for x in w.X]
    for i, (layer, op, ids, _, _) in enumerate(rows):
        v = m.layers()[layer]
        for t in range(len(w.X)):
            out = nodes[t][v].reshape(-1, m.layer_width(layer))
            if op == "NEB":
                exp = bool(np.all(out[:, ids[0]].view(np.uint32) == 0))        # every value +0
            else:
                exp = bool(np.array_equal(out[:, 0].view(np.uint32), out[:, 1].view(np.uint32)))
            assert ub[i, t] == exp, (layer, op, ids, t)
    assert ub.any()   # LeNet-5 has dead channels for some inputs


def test_identity_rows_all_unchanged(oracle_mod):
    w = wl.workload("lenet5", 20, 1)
    t = wl.table_from_rows([(1, "IDENTITY", [2], 0.0, 1), (3, "GF", [4, 5], 0.0, 7), (2, "GF", [1], 0.1, 7)])
    ub = bits(oracle_mod.unchanged_rows(w.model, w.X, t), 20)
    assert ub[0].all() and ub[1].all() and not ub[2].any()
