"""The library's host-side validation on the CPU (mure_check_descriptors: no context,
no device): every named workload is accepted; descriptor tables corrupted one field
at a time are rejected exactly when the oracle rejects them; graphs and settings
outside the supported shape are refused with UNSUPPORTED; inconsistent descriptions
with INVALID_ARG; the reason string is NUL-terminated within the caller's buffer."""
import ctypes

import numpy as np
import pytest

from paper_2607_18582_gb300 import mure
from paper_2607_18582_gb300 import workloads as wl

OK, INVALID, UNSUPPORTED = 0, 1, 2


@pytest.mark.parametrize("name", sorted(wl.CONFIGS))
@pytest.mark.parametrize("precision", ["fp32", "tf32x3", "tf32"])
def test_named_workloads_accepted(name, precision):
    w = wl.workload(name, 1, 300)
    assert mure.mure_check_descriptors(w.model, w.table, precision) == (OK, "")


def _copy(t):
    return wl.MutantTable(t.layer.copy(), t.op.copy(), t.n_neurons.copy(), t.neuron_off.copy(), t.param.copy(),
                          t.seed.copy(), t.pool.copy(), t.ratio.copy(),
                          None if t.tagged is None else t.tagged.copy())


def _corrupt(t, model, rng):
    """One field of one descriptor changed at random (often, not always, invalid)."""
    t = _copy(t)
    i = int(rng.integers(len(t)))
    L = model.n_layers()
    a, n = int(t.neuron_off[i]), int(t.n_neurons[i])
    tagged = t.tagged is not None and t.tagged[i] == 1
    kind = int(rng.integers(10))
    if kind == 0:
        t.layer[i] = int(rng.choice([-1, L, L + 3, int(rng.integers(L))]))
    elif kind == 1:
        t.op[i] = int(rng.choice([-1, 6, 7, int(rng.integers(6))]))
    elif kind == 2 and n:
        q = int(rng.integers(n))
        l = int(t.pool[a + q]) >> 20 if tagged else int(t.layer[i])
        j = int(rng.choice([model.layer_width(l), model.layer_width(l) + 5, -1]))
        t.pool[a + q] = ((l << 20) | j) if tagged and j >= 0 else j
    elif kind == 3 and n >= 2:
        t.pool[a + 1] = t.pool[a]                              # a repeated neuron
    elif kind == 4:
        t.n_neurons[i] = n + int(rng.choice([-1, 1, len(t.pool)]))
    elif kind == 5:
        t.neuron_off[i] = int(rng.choice([-1, len(t.pool), len(t.pool) - n + 1]))
    elif kind == 6:
        t.op[i] = wl.OP_INDEX["NS"]                            # NS with whatever count it has
    elif kind == 7 and tagged and n:
        t.layer[i] = int(rng.integers(L))                      # maybe no longer the smallest layer
    elif kind == 8:
        if t.tagged is None:
            t.tagged = np.zeros(len(t), np.int32)
        t.tagged[i] = int(rng.choice([2, -1, 1]))
    elif kind == 9 and tagged and n >= 2:
        q = 1 + 2 * int(rng.integers(n // 2)) if n >= 2 else 1
        l = (int(t.pool[a + q]) >> 20) + 1                     # move one entry to another layer
        if l < L:
            t.pool[a + q] = (l << 20) | (int(t.pool[a + q]) & 0xFFFFF) % model.layer_width(l)
    return t


@pytest.mark.parametrize("name", ["lenet5", "lenet5_modelwide", "mlp_modelwide", "resnet20"])
def test_table_validation_agrees_with_oracle(oracle_mod, name):
    w = wl.workload(name, 1, 12)
    X = w.X[:1]
    rng = np.random.default_rng(77)
    rejected = 0
    for _ in range(60):
        t = _corrupt(w.table, w.model, rng)
        st, msg = mure.mure_check_descriptors(w.model, t)
        try:
            oracle_mod.vanilla(w.model, X, t, n_threads=1, want_logits=False)
            oracle_ok = True
        except oracle_mod.OracleError:
            oracle_ok = False
        assert (st == OK) == oracle_ok, (st, msg)
        assert st in (OK, INVALID)
        assert (msg == "") == (st == OK)
        rejected += st != OK
    assert 20 <= rejected < 60   # both outcomes are exercised


def test_unsupported_graphs_and_settings():
    # a weighted layer in a skip branch (ResNet-10's projection shortcuts) is a stage
    # that reads an earlier stage input, its add taking the previous stage's output
    for prec in ("fp32", "tf32x3", "tf32"):
        assert mure.mure_check_descriptors(wl.resnet10(), precision=prec) == (OK, "")
    # depthwise convolutions and ReLU6 (MobileNetV2)
    for prec in ("fp32", "tf32x3"):
        assert mure.mure_check_descriptors(wl.mobilenetv2_tiny(), precision=prec) == (OK, "")
    # ... but not when that add skips the layer just before it (a dead branch)
    m = wl.resnet10()
    adds = [i for i, n in enumerate(m.nodes) if n.kind == "add"]
    add = m.nodes[adds[1]]                      # the second block's add: (conv_b, projection)
    conv_a = m.nodes[add.inputs[0]].inputs[0]
    add.inputs = (conv_a, add.inputs[1])
    st, msg = mure.mure_check_descriptors(m)
    assert st == UNSUPPORTED and "earlier stage input" in msg
    # more classes than the output-layer kernel keeps accumulators for
    st, msg = mure.mure_check_descriptors(wl.mlp(widths=(784, 64, 100)))
    assert st == UNSUPPORTED and "n_classes" in msg
    # up to 96 classes: the Reuters-sized recurrent model (90)
    assert mure.mure_check_descriptors(wl.mlp(widths=(784, 64, 40))) == (OK, "")
    assert mure.mure_check_descriptors(wl.rnn_reuters()) == (OK, "")
    st, msg = mure.mure_check_descriptors(wl.lenet5(), precision="bf16")
    assert st == UNSUPPORTED and "precision" in msg


def _broken(edit):
    m = wl.lenet5()
    edit(m)
    return mure.mure_check_descriptors(m)


def test_inconsistent_descriptions():
    st, msg = _broken(lambda m: setattr(m.nodes[2], "cin", 5))           # conv channels
    assert st == INVALID and "conv" in msg
    st, msg = _broken(lambda m: setattr(m.nodes[5], "cin", 399))         # dense fan-in
    assert st == INVALID and "fan-in" in msg
    st, msg = _broken(lambda m: setattr(m, "n_classes", 11))
    assert st == INVALID and "n_classes" in msg
    st, msg = _broken(lambda m: setattr(m.nodes[1], "inputs", (3,)))     # a later node as input
    assert st == INVALID and "earlier" in msg
    st, msg = _broken(lambda m: setattr(m, "in_shape", (0, 28, 1)))
    assert st == INVALID and "input shape" in msg


def test_reason_fits_the_buffer():
    w = wl.workload("lenet5", 1, 4)
    t = _copy(w.table)
    t.layer[2] = 99
    desc, keep = mure._model_desc(w.model, "fp32")
    arr, pool, plen = mure.table_array(t)
    for size in (1, 8, 512):
        buf = ctypes.create_string_buffer(b"\xff" * size, size)
        st = mure.lib().mure_check_descriptors(ctypes.byref(desc), mure._ptr(arr), len(t), mure._ptr(pool), plen,
                                               buf, size)
        assert st == INVALID
        raw = buf.raw
        assert raw.index(b"\0") <= size - 1
        assert raw[:raw.index(b"\0")].decode() == "mutant 2: layer 99 out of range"[:size - 1]
    # a NULL buffer is allowed; a NULL description is an argument error
    assert mure.lib().mure_check_descriptors(ctypes.byref(desc), None, 0, None, 0, None, 0) == OK
    assert mure.lib().mure_check_descriptors(None, None, 0, None, 0, None, 0) == INVALID


def _corrupt_model(model, rng):
    """A copy of the network with one geometry field of one node changed."""
    m = wl.Model(model.name, model.in_shape, model.n_classes,
                 [wl.Node(n.kind, n.inputs, n.act, n.kh, n.kw, n.stride, n.pad, n.cin, n.cout, n.W, n.b)
                  for n in model.nodes])
    v = int(rng.integers(len(m.nodes)))
    n = m.nodes[v]
    field = str(rng.choice(["kh", "kw", "stride", "pad", "cin", "cout", "inputs", "n_classes"]))
    if field == "inputs":
        n.inputs = (int(rng.integers(-1, len(m.nodes))),) + tuple(n.inputs[1:])
    elif field == "n_classes":
        m.n_classes = int(rng.choice([model.n_classes - 1, model.n_classes + 1]))
    else:
        setattr(n, field, max(-1, getattr(n, field) + int(rng.choice([-2, -1, 1, 3]))))
    return m


@pytest.mark.parametrize("name", ["lenet5", "resnet20", "mlp"])
def test_description_checks_cover_the_oracles(oracle_mod, name):
    """A description the oracle's graph checks refuse is refused by the library too
    (the library also refuses supported-shape violations the oracle can run)."""
    base = wl.MODELS[name](0)
    rng = np.random.default_rng(5)
    refused_by_oracle = 0
    for _ in range(80):
        m = _corrupt_model(base, rng)
        try:
            sh = oracle_mod.OModel(m).shapes()
            oracle_ok = int(np.prod(sh[-1])) == m.n_classes
        except oracle_mod.OracleError:
            oracle_ok = False
        st, msg = mure.mure_check_descriptors(m)
        if not oracle_ok:
            refused_by_oracle += 1
            assert st != OK, msg
        assert (msg == "") == (st == OK)
    assert refused_by_oracle >= 10
