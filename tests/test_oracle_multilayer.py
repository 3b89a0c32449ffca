"""Pins of the oracle's mutants over several layers (the paper's set mu(M') of mutated
layers; DeepMutation's model-wide selection ratio): hand-expanded brute force on a
tiny MLP with neurons mutated in both of its layers, equivalence with single-layer
descriptors, the per-layer materialisation, Theorem 1 (memo == vanilla) and the
descriptor checks."""
import numpy as np
import pytest

from paper_2607_18582_gb300 import workloads as wl

OPS = wl.OP_INDEX


def _tiny_mlp(sizes, seed):
    rng = np.random.default_rng(seed)
    m = wl.Model("tiny", (1, 1, sizes[0]), sizes[-1])
    for i in range(len(sizes) - 1):
        W = rng.standard_normal((sizes[i + 1], sizes[i])).astype(np.float32)
        b = rng.uniform(-0.5, 0.5, sizes[i + 1]).astype(np.float32)
        m.nodes.append(wl.Node("dense", (i - 1,), "relu" if i < len(sizes) - 2 else "none",
                               cin=sizes[i], cout=sizes[i + 1], W=W, b=b))
    return m


def _tagged(entries, op, param=0.0, seed=1):
    """One tagged mutant from (layer, neuron) entries."""
    ent = np.array([(l << 20) | j for l, j in entries], np.int32)
    return wl.MutantTable(np.array([min(l for l, _ in entries)], np.int32), np.array([OPS[op]], np.int32),
                          np.array([len(ent)], np.int32), np.array([0], np.int64), np.array([param], np.float32),
                          np.array([seed], np.uint64), ent, np.zeros(1), np.ones(1, np.int32))


def _brute_4_3_2(W0, b0, W1, b1, x, blk0=(), blk1=()):
    """Hand-expanded 4-3-2 MLP: ReLU hidden layer, linear output, fp64 sums rounded to
    fp32 once per neuron; blocked neurons output 0."""
    r = lambda v: max(float(np.float32(v)), 0.0)
    h = [r(b0[j] + W0[j][0] * x[0] + W0[j][1] * x[1] + W0[j][2] * x[2] + W0[j][3] * x[3]) for j in range(3)]
    h = [0.0 if j in blk0 else h[j] for j in range(3)]
    y = [float(np.float32(b1[c] + W1[c][0] * h[0] + W1[c][1] * h[1] + W1[c][2] * h[2])) for c in range(2)]
    return [0.0 if c in blk1 else y[c] for c in range(2)]


def _as64(a):
    return np.asarray(a, np.float64).tolist()


def test_two_layer_mutants_bruteforce(oracle_mod):
    m = _tiny_mlp((4, 3, 2), 31)
    X = np.random.default_rng(32).standard_normal((6, 1, 1, 4)).astype(np.float32)
    W0, b0 = _as64(m.nodes[0].W), _as64(m.nodes[0].b)
    W1, b1 = _as64(m.nodes[1].W), _as64(m.nodes[1].b)
    cases = []
    # NAI on hidden neuron 2 and output neuron 0
    W0n = [row[:] for row in W0]; b0n = b0[:]
    W0n[2] = [-v for v in W0[2]]; b0n[2] = -b0[2]
    W1n = [row[:] for row in W1]; b1n = b1[:]
    W1n[0] = [-v for v in W1[0]]; b1n[0] = -b1[0]
    cases.append(("NAI", [(0, 2), (1, 0)], 0.0, 3, (W0n, b0n, W1n, b1n, (), ())))
    # NEB on hidden neuron 1 and output neuron 1
    cases.append(("NEB", [(0, 1), (1, 1)], 0.0, 4, (W0, b0, W1, b1, (1,), (1,))))
    # NS: the pair (0, 2) in the hidden layer and the pair (0, 1) in the output layer
    W0s = [W0[2][:], W0[1][:], W0[0][:]]; b0s = [b0[2], b0[1], b0[0]]
    W1s = [W1[1][:], W1[0][:]]; b1s = [b1[1], b1[0]]
    cases.append(("NS", [(0, 0), (0, 2), (1, 0), (1, 1)], 0.0, 5, (W0s, b0s, W1s, b1s, (), ())))
    # GF on hidden neuron 1 (slot 0) and output neuron 1 (slot 1): each layer's own
    # sigma, each slot its own stream
    sig0 = float(np.float32(0.1)) * float(np.std(np.asarray(W0)))
    sig1 = float(np.float32(0.1)) * float(np.std(np.asarray(W1)))
    s0, s1 = oracle_mod.sm64(6, 0), oracle_mod.sm64(6, 1)
    W0g = [row[:] for row in W0]; W1g = [row[:] for row in W1]
    W0g[1] = [float(np.float32(W0[1][f]) + np.float32(sig0 * oracle_mod.gauss(s0, f))) for f in range(4)]
    W1g[1] = [float(np.float32(W1[1][f]) + np.float32(sig1 * oracle_mod.gauss(s1, f))) for f in range(3)]
    cases.append(("GF", [(0, 1), (1, 1)], 0.1, 6, (W0g, b0, W1g, b1, (), ())))
    # WS on output neuron 0 (slot 0) and hidden neuron 2 (slot 1): list order decides
    # the streams, not the layer order
    p0 = oracle_mod.fisher_yates(oracle_mod.sm64(7, 0), 3)
    p1 = oracle_mod.fisher_yates(oracle_mod.sm64(7, 1), 4)
    W0w = [row[:] for row in W0]; W1w = [row[:] for row in W1]
    W1w[0] = [W1[0][p0[f]] for f in range(3)]
    W0w[2] = [W0[2][p1[f]] for f in range(4)]
    cases.append(("WS", [(1, 0), (0, 2)], 0.0, 7, (W0w, b0, W1w, b1, (), ())))
    for op, entries, param, seed, (a, b, c, d, k0, k1) in cases:
        t = _tagged(entries, op, param, seed)
        for fn in (oracle_mod.vanilla, oracle_mod.memo):
            res = fn(m, X, t)
            for i in range(6):
                exp = _brute_4_3_2(a, b, c, d, _as64(X[i].ravel()), k0, k1)
                assert res["logits"][0, i].tolist() == exp, (op, i)


def test_tagged_single_layer_equals_untagged(oracle_mod):
    w = wl.workload("lenet5", 12, 40)
    t = w.table
    tag = wl.MutantTable(t.layer.copy(), t.op.copy(), t.n_neurons.copy(), t.neuron_off.copy(), t.param.copy(),
                         t.seed.copy(), np.zeros_like(t.pool), t.ratio.copy(), np.ones(len(t), np.int32))
    for i in range(len(t)):
        a, n = int(t.neuron_off[i]), int(t.n_neurons[i])
        tag.pool[a:a + n] = (int(t.layer[i]) << 20) | t.pool[a:a + n]
    r0 = oracle_mod.vanilla(w.model, w.X, t)
    r1 = oracle_mod.vanilla(w.model, w.X, tag)
    assert np.array_equal(r0["logits"], r1["logits"])
    assert np.array_equal(r0["kill_bits"], r1["kill_bits"])


def test_per_layer_materialisation(oracle_mod):
    w = wl.workload("lenet5", 1, 1)
    m = w.model
    t = _tagged([(1, 3), (1, 7), (3, 10), (3, 50)], "NAI")
    for layer in range(m.n_layers()):
        nd = m.nodes[m.layers()[layer]]
        Wm, bm, blk = oracle_mod.mutant_layer(m, t, 0, layer)
        W2, Wm2 = nd.W.reshape(nd.cout, -1), Wm.reshape(nd.cout, -1)
        ids = {1: [3, 7], 3: [10, 50]}.get(layer, [])
        other = np.setdiff1d(np.arange(nd.cout), ids)
        assert np.array_equal(Wm2[other], W2[other]) and np.array_equal(bm[other], nd.b[other])
        if ids:
            assert np.array_equal(Wm2[ids], -W2[ids]) and np.array_equal(bm[ids], -nd.b[ids])
        assert not blk.any()


@pytest.mark.parametrize("name,n_in,n_mut", [("lenet5_modelwide", 16, 40), ("mlp_modelwide", 24, 40),
                                            ("lenet5_modelwide_5", 12, 40)])
def test_theorem1_memo_equals_vanilla_modelwide(oracle_mod, name, n_in, n_mut):
    w = wl.workload(name, n_in, n_mut)
    assert (w.table.tagged == 1).all()
    spans = [len({int(e) >> 20 for e in w.table.pool[a:a + n]})
             for a, n in zip(w.table.neuron_off, w.table.n_neurons)]
    assert max(spans) >= 2   # the table does exercise several layers per mutant
    r0 = oracle_mod.vanilla(w.model, w.X, w.table)
    r1 = oracle_mod.memo(w.model, w.X, w.table)
    assert np.array_equal(r0["logits"], r1["logits"])
    assert np.array_equal(r0["kill_bits"], r1["kill_bits"])
    assert r0["scoreA"] == r1["scoreA"] and r0["scoreB"] == r1["scoreB"]


def test_modelwide_resnet_theorem1(oracle_mod):
    w = wl.workload("resnet20", 2, 1)
    t = wl.modelwide_mutants(w.model, 10, seed=3, ratio=0.005)
    r0 = oracle_mod.vanilla(w.model, w.X, t)
    r1 = oracle_mod.memo(w.model, w.X, t)
    assert np.array_equal(r0["logits"], r1["logits"])


def test_invalid_tagged_mutants_rejected(oracle_mod):
    w = wl.workload("lenet5", 2, 1)
    bad = [
        ([(1, 3), (2, 5)], "NEB", 2),        # layer is not the smallest listed
        ([(1, 3), (2, 5)], "NS", 1),         # an NS pair across two layers
        ([(1, 3), (1, 3)], "GF", 1),         # repeated entry
        ([(1, 16)], "GF", 1),                # neuron out of range for its layer
        ([(5, 0)], "GF", 5),                 # layer out of range
    ]
    for entries, op, layer in bad:
        t = _tagged(entries, op)
        t.layer[0] = layer
        with pytest.raises(oracle_mod.OracleError):
            oracle_mod.vanilla(w.model, w.X, t)


@pytest.mark.parametrize("name", ["lenet5", "vgg", "resnet20", "mlp"])
def test_modelwide_generator_structure(name):
    """The model-wide tables are well formed: distinct (layer, neuron) entries in range,
    `layer` the smallest listed one, NS pairs inside one layer, k from the ratio."""
    w = wl.workload(name, 1, 1)
    m = w.model
    widths = [m.layer_width(l) for l in range(m.n_layers())]
    t = wl.modelwide_mutants(m, 64, seed=13, ratio=0.01)
    k = max(1, int(np.floor(0.01 * sum(widths) + 0.5)))
    for i in range(len(t)):
        a, n = int(t.neuron_off[i]), int(t.n_neurons[i])
        ent = [(int(e) >> 20, int(e) & 0xFFFFF) for e in t.pool[a:a + n]]
        assert len(set(ent)) == n
        assert all(0 <= l < len(widths) and 0 <= j < widths[l] for l, j in ent)
        assert int(t.layer[i]) == min(l for l, _ in ent)
        if wl.OPS[int(t.op[i])] == "NS":
            assert n == 2 * max(1, k // 2)
            assert all(ent[q][0] == ent[q + 1][0] for q in range(0, n, 2))
        else:
            assert n == min(k, sum(widths))
