"""Pins of the oracle's depthwise convolution and ReLU6 (the MobileNetV2 family of the
paper's Table 1): the layer against PyTorch's grouped convolution in fp64, a whole
MobileNetV2-style network against a PyTorch fp64 composition, the operators on a
depthwise layer (a neuron is a channel with its own filter), Theorem 1 and identity
mutants.  The GPU library has no depthwise layer yet: these pin the oracle side."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_2607_18582_gb300 import workloads as wl

OPS = wl.OP_INDEX


def _act(y, act):
    if act == "relu":
        return y.clamp_min(0)
    if act == "relu6":
        return y.clamp(0, 6)
    return y


def _torch_forward(model, X):
    """The network composed from PyTorch fp64 routines, activations stored in fp32."""
    outs = {-1: torch.from_numpy(X).double().permute(0, 3, 1, 2)}
    for v, n in enumerate(model.nodes):
        a = outs[n.inputs[0]]
        if n.kind == "conv":
            y = F.conv2d(a, torch.from_numpy(n.W).double().permute(0, 3, 1, 2), torch.from_numpy(n.b).double(),
                         stride=n.stride, padding=n.pad)
        elif n.kind == "dwconv":
            y = F.conv2d(a, torch.from_numpy(n.W).double()[:, None], torch.from_numpy(n.b).double(),
                         stride=n.stride, padding=n.pad, groups=n.cout)
        elif n.kind == "dense":
            flat = a.permute(0, 2, 3, 1).reshape(a.shape[0], -1)
            y = F.linear(flat, torch.from_numpy(n.W).double(), torch.from_numpy(n.b).double())[:, :, None, None]
        elif n.kind == "add":
            y = a + outs[n.inputs[1]]
        elif n.kind == "gap":
            y = a.mean(dim=(2, 3), keepdim=True)
        else:
            raise AssertionError(n.kind)
        outs[v] = _act(y, n.act).float().double()
    return outs[len(model.nodes) - 1].reshape(X.shape[0], -1).float().numpy()


@pytest.mark.parametrize("k,stride,pad,act", [(3, 1, 1, "relu6"), (3, 2, 1, "none"), (5, 1, 0, "relu"),
                                              (3, 2, 0, "relu6")])
def test_depthwise_layer_matches_torch_fp64(oracle_mod, k, stride, pad, act):
    rng = np.random.default_rng(k * 10 + stride)
    c = 7
    m = wl.Model("t", (9, 11, c), 1)
    W = (rng.standard_normal((c, k, k)) * 2.0).astype(np.float32)
    b = rng.standard_normal(c).astype(np.float32)
    m.nodes.append(wl.Node("dwconv", (-1,), act, k, k, stride, pad, c, c, W, b))
    x = (rng.standard_normal((9, 11, c)) * 2.0).astype(np.float32)
    got = oracle_mod.node_forward(m, 0, x)
    ref = F.conv2d(torch.from_numpy(x).double().permute(2, 0, 1)[None], torch.from_numpy(W).double()[:, None],
                   torch.from_numpy(b).double(), stride=stride, padding=pad, groups=c)
    ref = _act(ref, act)[0].permute(1, 2, 0).float().numpy()
    assert got.shape == ref.shape
    assert np.array_equal(got, ref)   # one fp64 sum rounded once on both sides
    if act == "relu6":
        assert got.max() <= 6.0 and got.min() >= 0.0


def test_mobilenet_forward_matches_torch(oracle_mod):
    m = wl.mobilenetv2_tiny()
    X = wl.inputs(m, 3)
    lg, _ = oracle_mod.forward(m, X)
    ref = _torch_forward(m, X)
    scale = np.abs(ref).max(axis=1, keepdims=True)
    assert np.all(np.abs(lg - ref) <= 1e-5 * scale)


def test_operators_on_a_depthwise_layer(oracle_mod):
    m = wl.mobilenetv2_tiny()
    layer = [m.nodes[v].kind for v in m.layers()].index("dwconv")
    nd = m.nodes[m.layers()[layer]]
    ids = np.array([3, 40], np.int32)
    for op in ("GF", "WS", "NAI", "NS", "NEB"):
        t = wl.MutantTable(np.array([layer], np.int32), np.array([OPS[op]], np.int32), np.array([2], np.int32),
                           np.array([0], np.int64), np.array([0.1], np.float32), np.array([5], np.uint64),
                           ids, np.zeros(1))
        Wm, bm, blk = oracle_mod.mutant_layer(m, t, 0)
        W2, Wm2 = nd.W.reshape(nd.cout, -1), Wm.reshape(nd.cout, -1)
        other = np.setdiff1d(np.arange(nd.cout), ids)
        assert np.array_equal(Wm2[other], W2[other]) and np.array_equal(bm[other], nd.b[other])
        if op == "GF":
            # fp32(w + fp32(sigma n)), sigma from the layer's weights, a stream per slot
            sig = float(np.float32(0.1)) * float(np.std(nd.W.astype(np.float64)))
            for q, j in enumerate(ids):
                s = oracle_mod.sm64(5, q)
                exp = [np.float32(W2[j][f]) + np.float32(sig * oracle_mod.gauss(s, f)) for f in range(9)]
                assert np.array_equal(Wm2[j], np.array(exp, np.float32))
        elif op == "WS":
            for q, j in enumerate(ids):
                p = oracle_mod.fisher_yates(oracle_mod.sm64(5, q), 9)
                assert np.array_equal(Wm2[j], W2[j][p])
        elif op == "NAI":
            assert np.array_equal(Wm2[ids], -W2[ids]) and np.array_equal(bm[ids], -nd.b[ids])
        elif op == "NS":
            assert np.array_equal(Wm2[ids[0]], W2[ids[1]]) and np.array_equal(Wm2[ids[1]], W2[ids[0]])
        assert blk.tolist() == [op == "NEB" and c in ids for c in range(nd.cout)]


def test_mobilenet_theorem1_and_identity(oracle_mod):
    m = wl.mobilenetv2_tiny()
    X = wl.inputs(m, 6)
    subs = [wl.mutants(m, 6, seed=20 + l, ratios=(0.05,), layers=[l],
                      ops=tuple(wl.OPS[(l + i) % 5] for i in range(6))) for l in range(m.n_layers())]
    subs.append(wl.modelwide_mutants(m, 8, seed=31, ratio=0.01))
    table = wl.concat(subs)
    r0 = oracle_mod.vanilla(m, X, table)
    r1 = oracle_mod.memo(m, X, table)
    assert np.array_equal(r0["logits"], r1["logits"])
    assert np.array_equal(r0["kill_bits"], r1["kill_bits"])
    # identity mutants on a depthwise layer reproduce the original logits
    layer = [m.nodes[v].kind for v in m.layers()].index("dwconv")
    ident = wl.table_from_rows([(layer, "IDENTITY", [1, 2], 0.0, 1), (layer, "GF", [1, 2], 0.0, 2)])
    r = oracle_mod.vanilla(m, X, ident)
    assert np.array_equal(r["logits"][0], r["orig_logits"]) and np.array_equal(r["logits"][1], r["orig_logits"])
    assert not r["kill_bits"].any()
