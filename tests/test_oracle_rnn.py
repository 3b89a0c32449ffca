"""Pins of the oracle's recurrent family (Sec. 5.3, Table 1: an embedding, two LSTM
layers, a dense output): the architecture against Table 1's parameter counts, the
embedding against PyTorch's lookup, the LSTM layer and the whole network against
PyTorch fp64 LSTM cells, NEB and NAI against networks whose weights were changed
instead (bit for bit), the operators' rewrites of an LSTM unit, Theorem 1 and identity
mutants.  The GPU library has no recurrent layer yet: these pin the oracle side."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_2607_18582_gb300 import workloads as wl

OPS = wl.OP_INDEX


def _small(seed=0, n_classes=3):
    return wl.rnn(seed, n_classes=n_classes, vocab=50, dim=8, units=(6, 5), steps=12, name="rnn_small")


def _cell(nd):
    """A PyTorch fp64 LSTM cell with the node's weights (PyTorch's gate order i, f, g, o
    is the node's; PyTorch's second bias set to 0)."""
    H, c = nd.cout, nd.cin
    cell = torch.nn.LSTMCell(c, H, bias=True, dtype=torch.float64)
    W = nd.W.astype(np.float64)
    with torch.no_grad():
        cell.weight_ih.copy_(torch.from_numpy(W[:, :, :c].transpose(1, 0, 2).reshape(4 * H, c)))
        cell.weight_hh.copy_(torch.from_numpy(W[:, :, c:].transpose(1, 0, 2).reshape(4 * H, H)))
        cell.bias_ih.copy_(torch.from_numpy(nd.b.astype(np.float64).T.reshape(4 * H)))
        cell.bias_hh.zero_()
    return cell


def _torch_lstm(nd, xs):
    """xs [T][cin] -> outputs [T][H] (or the last [1][H]); the state is stored in fp32
    between steps, as the network stores every activation."""
    cell = _cell(nd)
    h = torch.zeros(1, nd.cout, dtype=torch.float64)
    c = torch.zeros(1, nd.cout, dtype=torch.float64)
    outs = []
    with torch.no_grad():
        for t in range(xs.shape[0]):
            h, c = cell(torch.from_numpy(xs[t:t + 1].astype(np.float64)), (h, c))
            h, c = h.float().double(), c.float().double()
            outs.append(h[0].numpy().astype(np.float32))
    return np.stack(outs) if nd.kh else outs[-1][None]


def _torch_rnn(model, X):
    """The network composed from PyTorch routines, activations stored in fp32."""
    out = []
    for x in X:
        a = x.reshape(-1)
        for n in model.nodes:
            if n.kind == "embed":
                a = F.embedding(torch.from_numpy(a.astype(np.int64)), torch.from_numpy(n.W.T.copy())).numpy()
            elif n.kind == "lstm":
                a = _torch_lstm(n, a)
            elif n.kind == "dense":
                a = F.linear(torch.from_numpy(a.reshape(-1).astype(np.float64)), torch.from_numpy(n.W).double(),
                             torch.from_numpy(n.b).double()).float().numpy()
            else:
                raise AssertionError(n.kind)
        out.append(a.reshape(-1))
    return np.stack(out)


def test_table1_sizes():
    """Vocabulary 20,000, width 128 and two 64-unit LSTMs reproduce Table 1's sizes."""
    count = lambda m: sum(n.W.size + (0 if n.b is None else n.b.size) for n in m.nodes)
    assert count(wl.rnn()) == 2642562          # IMDB, 2 classes
    assert count(wl.rnn_reuters()) == 2648282  # Reuters, 90 classes
    m = wl.rnn()
    assert [n.kind for n in m.nodes] == ["embed", "lstm", "lstm", "dense"] and m.n_layers() == 4


def test_token_recipe():
    m = wl.rnn()
    X = wl.inputs(m, 64)
    assert X.shape == (64, 1, 80, 1)
    assert np.array_equal(X, np.floor(X)) and X.min() >= 0 and X.max() < 20000
    lengths = (X[:, 0, :, 0] > 0).sum(axis=1)
    for t in range(64):   # pre-padded: zeros only before the first word
        assert (X[t, 0, :80 - lengths[t], 0] == 0).all() and (X[t, 0, 80 - lengths[t]:, 0] > 0).all()
    assert lengths.min() >= 8 and len(np.unique(lengths)) > 10


def test_embedding_matches_torch(oracle_mod):
    m = _small()
    x = wl.inputs(m, 1, seed=4)[0]
    got = oracle_mod.node_forward(m, 0, x)
    ref = F.embedding(torch.from_numpy(x.reshape(-1).astype(np.int64)), torch.from_numpy(m.nodes[0].W.T.copy()))
    assert np.array_equal(got.reshape(-1, 8), ref.numpy())


@pytest.mark.parametrize("bad", [50.0, -1.0, 2.5, float("nan")])
def test_invalid_tokens_rejected(oracle_mod, bad):
    m = _small()
    X = wl.inputs(m, 3, seed=4)
    X[1, 0, 5, 0] = bad
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.forward(m, X)
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.vanilla(m, X, wl.table_from_rows([(1, "NAI", [0], 0.0, 1)]))


def test_recurrent_node_checks(oracle_mod):
    m = _small()
    m.nodes[1].act = "relu"          # an LSTM has its own activations
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.OModel(m).shapes()
    m = _small()
    m.nodes[1].inputs = (-1,)        # an LSTM on raw token ids of width 1 != cin
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.OModel(m).shapes()


@pytest.mark.parametrize("sequences,T,cin,H", [(True, 15, 7, 5), (False, 9, 3, 11), (True, 1, 4, 4)])
def test_lstm_layer_matches_torch_fp64(oracle_mod, sequences, T, cin, H):
    rng = np.random.default_rng(T * 100 + cin)
    m = wl.Model("t", (1, T, cin), H)
    W = rng.standard_normal((H, 4, cin + H)).astype(np.float32)          # saturates some gates
    b = rng.standard_normal((H, 4)).astype(np.float32)
    m.nodes.append(wl.Node("lstm", (-1,), "none", 1 if sequences else 0, 1, 1, 0, cin, H, W, b))
    x = rng.standard_normal((1, T, cin)).astype(np.float32)
    got = oracle_mod.node_forward(m, 0, x).reshape(-1, H)
    ref = _torch_lstm(m.nodes[0], x[0])
    assert got.shape == ref.shape
    assert np.max(np.abs(got - ref)) <= 2e-6   # h in (-1, 1); fp32 rounding of the stored gates


def test_rnn_network_matches_torch(oracle_mod):
    m = _small()
    X = wl.inputs(m, 5, seed=7)
    lg, _ = oracle_mod.forward(m, X)
    ref = _torch_rnn(m, X)
    assert np.max(np.abs(lg - ref)) <= 1e-5 * max(1.0, np.abs(ref).max())


def _with(model, edits):
    """A copy of the model whose weights were changed by edits(nodes)."""
    m = wl.Model(model.name, model.in_shape, model.n_classes,
                 [wl.Node(n.kind, n.inputs, n.act, n.kh, n.kw, n.stride, n.pad, n.cin, n.cout,
                          None if n.W is None else n.W.copy(), None if n.b is None else n.b.copy())
                  for n in model.nodes])
    edits(m.nodes)
    return m


def test_neb_equals_zeroed_outgoing_weights(oracle_mod):
    """NEB holds a neuron's output at 0 at every step: bit for bit the network whose
    weights reading that output (the next layer's input weights, and for an LSTM unit
    its layer's recurrent weights) are zero."""
    m = _small()
    X = wl.inputs(m, 6, seed=8)
    c1 = m.nodes[1].cin                      # 8
    c2 = m.nodes[2].cin                      # 6
    cases = [
        (0, 3, lambda N: N[1].W[:, :, 3].__setitem__(Ellipsis, 0.0)),
        (1, 2, lambda N: (N[1].W[:, :, c1 + 2].__setitem__(Ellipsis, 0.0),
                          N[2].W[:, :, 2].__setitem__(Ellipsis, 0.0))),
        (2, 4, lambda N: (N[2].W[:, :, c2 + 4].__setitem__(Ellipsis, 0.0),
                          N[3].W[:, 4].__setitem__(Ellipsis, 0.0))),
    ]
    for layer, j, edit in cases:
        r = oracle_mod.vanilla(m, X, wl.table_from_rows([(layer, "NEB", [j], 0.0, 1)]))
        lg, _ = oracle_mod.forward(_with(m, edit), X)
        assert np.array_equal(r["logits"][0].view(np.uint32), lg.view(np.uint32)), layer
        assert not np.array_equal(lg, r["orig_logits"])


def test_nai_on_embedding_equals_negated_input_column(oracle_mod):
    m = _small()
    X = wl.inputs(m, 6, seed=9)
    r = oracle_mod.vanilla(m, X, wl.table_from_rows([(0, "NAI", [5], 0.0, 1)]))

    def edit(N):
        N[1].W[:, :, 5] *= -1.0
    lg, _ = oracle_mod.forward(_with(m, edit), X)
    assert np.array_equal(r["logits"][0].view(np.uint32), lg.view(np.uint32))


def test_operators_on_an_lstm_unit(oracle_mod):
    m = _small()
    layer, nd = 1, m.nodes[1]
    H, Fi = nd.cout, 4 * (nd.cin + nd.cout)
    ids = np.array([4, 1], np.int32)
    W2 = nd.W.reshape(H, Fi)
    for op in ("GF", "WS", "NAI", "NS", "NEB"):
        t = wl.MutantTable(np.array([layer], np.int32), np.array([OPS[op]], np.int32), np.array([2], np.int32),
                           np.array([0], np.int64), np.array([0.1], np.float32), np.array([11], np.uint64),
                           ids, np.zeros(1))
        Wm, bm, blk = oracle_mod.mutant_layer(m, t, 0)
        Wm2 = Wm.reshape(H, Fi)
        other = np.setdiff1d(np.arange(H), ids)
        assert np.array_equal(Wm2[other], W2[other]) and np.array_equal(bm[other], nd.b[other])
        if op == "GF":
            sig = float(np.float32(0.1)) * float(np.std(nd.W.astype(np.float64)))
            for q, j in enumerate(ids):
                s = oracle_mod.sm64(11, q)
                exp = [np.float32(W2[j][f]) + np.float32(sig * oracle_mod.gauss(s, f)) for f in range(Fi)]
                assert np.array_equal(Wm2[j], np.array(exp, np.float32))
            assert np.array_equal(bm, nd.b)
        elif op == "WS":
            for q, j in enumerate(ids):
                assert np.array_equal(Wm2[j], W2[j][oracle_mod.fisher_yates(oracle_mod.sm64(11, q), Fi)])
        elif op == "NAI":
            assert np.array_equal(Wm2[ids], -W2[ids]) and np.array_equal(bm[ids], -nd.b[ids])
        elif op == "NS":
            assert np.array_equal(Wm2[4], W2[1]) and np.array_equal(Wm2[1], W2[4])
            assert np.array_equal(bm[4], nd.b[1]) and np.array_equal(bm[1], nd.b[4])
        assert blk.tolist() == [op == "NEB" and c in ids for c in range(H)]
    # an embedding neuron has no bias
    t = wl.table_from_rows([(0, "NAI", [2], 0.0, 1)])
    Wm, bm, _ = oracle_mod.mutant_layer(m, t, 0)
    assert bm is None and np.array_equal(Wm[2], -m.nodes[0].W[2])


@pytest.mark.parametrize("op", ["GF", "WS", "NAI", "NS"])
def test_mutated_lstm_matches_torch(oracle_mod, op):
    """A mutant's logits are the PyTorch network run with its materialised weights."""
    m = _small()
    X = wl.inputs(m, 4, seed=10)
    for layer in (1, 2):
        t = wl.table_from_rows([(layer, op, [0, 3], 0.2, 21)])
        Wm, bm, _ = oracle_mod.mutant_layer(m, t, 0)
        r = oracle_mod.vanilla(m, X, t)
        v = m.layers()[layer]

        def edit(N):
            N[v].W[...] = Wm
            N[v].b[...] = bm
        ref = _torch_rnn(_with(m, edit), X)
        assert np.max(np.abs(r["logits"][0] - ref)) <= 1e-5 * max(1.0, np.abs(ref).max())


@pytest.mark.parametrize("full", [False, True])
def test_rnn_theorem1_and_boundaries(oracle_mod, full):
    m = wl.rnn() if full else _small()
    X = wl.inputs(m, 2 if full else 8, seed=12)
    ops = ("GF", "NEB", "NAI", "NS", "WS")
    subs = [wl.mutants(m, 5 if full else 10, seed=30 + l, ratios=(0.05,), layers=[l], ops=ops)
            for l in range(m.n_layers())]
    subs.append(wl.modelwide_mutants(m, 4 if full else 10, seed=41, ratio=0.05))
    table = wl.concat(subs)
    r0 = oracle_mod.vanilla(m, X, table)
    r1 = oracle_mod.memo(m, X, table)
    assert np.array_equal(r0["logits"], r1["logits"])
    assert np.array_equal(r0["kill_bits"], r1["kill_bits"])
    # a chain: the boundary of layer l is the node that feeds it
    for l, v in enumerate(m.layers()):
        assert oracle_mod.boundary(m, l) == [m.nodes[v].inputs[0]]


def test_rnn_identity_mutants(oracle_mod):
    m = _small()
    X = wl.inputs(m, 6, seed=13)
    t = wl.table_from_rows([(1, "IDENTITY", [1, 2], 0.0, 1), (2, "GF", [0, 1, 2], 0.0, 2),
                            (0, "GF", [3], 0.0, 3)])
    r = oracle_mod.vanilla(m, X, t)
    for i in range(3):
        assert np.array_equal(r["logits"][i], r["orig_logits"])
    assert not r["kill_bits"].any()
    assert oracle_mod.unchanged_rows(m, X, t).astype(bool).any(axis=1).all()
