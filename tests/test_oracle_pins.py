"""Pins of the CPU oracle against things other than itself: published generator
outputs, library routines (PyTorch CPU fp64, numpy, scipy), a hand-worked example,
brute-force hand-expanded dot products, closed forms and the paper's theorems."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from conftest import load_golden, tiny_worked_example
from paper_2607_18582_gb300 import workloads as wl

OPS = wl.OP_INDEX


# ------------------------------------------------------------- random numbers --

def test_splitmix64_published_outputs(oracle_mod):
    g = load_golden("splitmix64.txt")
    rows = [(int(k), int(v[0]), int(v[1])) for k, vals in g.items() for v in vals]
    assert len(rows) == 8
    for seed, i, out in rows:
        assert oracle_mod.sm64(seed, i) == out


def test_gauss_is_standard_normal(oracle_mod):
    from scipy import stats
    xs = np.array([oracle_mod.gauss(0xABCDEF, f) for f in range(20000)])
    assert abs(xs.mean()) < 0.03 and abs(xs.std() - 1.0) < 0.03
    assert stats.kstest(xs, "norm").pvalue > 1e-3
    # the cos and sin halves of a Box-Muller pair are uncorrelated
    assert abs(np.corrcoef(xs[0::2], xs[1::2])[0, 1]) < 0.03


def test_fisher_yates_uniform(oracle_mod):
    from scipy import stats
    n, trials = 5, 12000
    counts = np.zeros((n, n))
    perms = {}
    for s in range(trials):
        p = oracle_mod.fisher_yates(oracle_mod.sm64(77, s), n)
        assert sorted(p.tolist()) == list(range(n))
        counts[np.arange(n), p] += 1
        perms[tuple(p)] = perms.get(tuple(p), 0) + 1
    assert len(perms) == 120
    assert stats.chisquare(counts.ravel(), np.full(n * n, trials / n)).pvalue > 1e-3
    assert stats.chisquare(list(perms.values())).pvalue > 1e-3


# ------------------------------------------------------------ layer functions --

def _rand_model(kind, rng, **kw):
    """One-node network around `kind` for the layer-function pins."""
    h, w, c = kw.get("in_shape", (7, 9, 3))
    m = wl.Model("t", (h, w, c), 1)
    if kind == "conv":
        k, s, p, co = kw["k"], kw["stride"], kw["pad"], kw["cout"]
        W = rng.standard_normal((co, k, k, c)).astype(np.float32)
        b = rng.standard_normal(co).astype(np.float32)
        m.nodes.append(wl.Node("conv", (-1,), kw.get("act", "none"), k, k, s, p, c, co, W, b))
    elif kind == "dense":
        co = kw["cout"]
        W = rng.standard_normal((co, h * w * c)).astype(np.float32)
        b = rng.standard_normal(co).astype(np.float32)
        m.nodes.append(wl.Node("dense", (-1,), kw.get("act", "none"), 1, 1, 1, 0, h * w * c, co, W, b))
    return m


def _close32(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    # fp64 accumulations in different orders may straddle one fp32 rounding boundary
    assert np.all(np.abs(a - b) <= 2.0 ** -22 * np.maximum(np.abs(b), 1e-30) + 1e-37), np.max(np.abs(a - b))


@pytest.mark.parametrize("k,stride,pad,cout,act", [(3, 1, 1, 4, "none"), (5, 1, 2, 6, "relu"), (5, 1, 0, 2, "none"),
                                                  (3, 2, 1, 5, "relu"), (1, 1, 0, 3, "none")])
def test_conv_matches_torch_fp64(oracle_mod, k, stride, pad, cout, act):
    rng = np.random.default_rng(k * 100 + stride * 10 + pad)
    m = _rand_model("conv", rng, k=k, stride=stride, pad=pad, cout=cout, act=act)
    x = rng.standard_normal((7, 9, 3)).astype(np.float32)
    got = oracle_mod.node_forward(m, 0, x)
    nd = m.nodes[0]
    ref = F.conv2d(torch.from_numpy(x).double().permute(2, 0, 1)[None],
                   torch.from_numpy(nd.W).double().permute(0, 3, 1, 2), torch.from_numpy(nd.b).double(),
                   stride=stride, padding=pad)[0].permute(1, 2, 0).numpy().astype(np.float32)
    if act == "relu":
        ref = np.maximum(ref, 0)
    assert got.shape == ref.shape
    _close32(got, ref)


def test_dense_matches_torch_fp64(oracle_mod):
    rng = np.random.default_rng(3)
    m = _rand_model("dense", rng, cout=11, act="relu", in_shape=(1, 1, 37))
    x = rng.standard_normal((1, 1, 37)).astype(np.float32)
    got = oracle_mod.node_forward(m, 0, x)
    nd = m.nodes[0]
    ref = F.linear(torch.from_numpy(x.reshape(-1)).double(), torch.from_numpy(nd.W).double(),
                   torch.from_numpy(nd.b).double()).clamp_min(0).numpy().astype(np.float32)
    _close32(got.reshape(-1), ref)


def test_pool_gap_shortcut_add_flatten(oracle_mod):
    rng = np.random.default_rng(4)
    x = rng.standard_normal((6, 8, 5)).astype(np.float32)
    y = rng.standard_normal((6, 8, 5)).astype(np.float32)
    m = wl.Model("t", (6, 8, 5), 1)
    m.nodes = [wl.Node("maxpool", (-1,), "none", 2, 2, 2), wl.Node("gap", (-1,)),
               wl.Node("shortcut", (-1,), "none", 1, 1, 2, 0, 5, 9), wl.Node("flatten", (-1,))]
    pooled = oracle_mod.node_forward(m, 0, x)
    ref = F.max_pool2d(torch.from_numpy(x).permute(2, 0, 1)[None], 2, 2)[0].permute(1, 2, 0).numpy()
    assert np.array_equal(pooled, ref)
    g = oracle_mod.node_forward(m, 1, x)
    _close32(g.reshape(-1), x.astype(np.float64).mean(axis=(0, 1)).astype(np.float32))
    sc = oracle_mod.node_forward(m, 2, x)
    ref_sc = np.zeros((3, 4, 9), np.float32)
    ref_sc[:, :, :5] = x[::2, ::2, :]
    assert np.array_equal(sc, ref_sc)
    assert np.array_equal(oracle_mod.node_forward(m, 3, x).reshape(-1), x.reshape(-1))
    m2 = wl.Model("t", (6, 8, 5), 1)
    m2.nodes = [wl.Node("add", (-1, -1), "relu")]
    assert np.array_equal(oracle_mod.node_forward(m2, 0, x, x), np.maximum(x + x, 0))


def _torch_forward(model, X):
    """The same network composed from PyTorch fp64 library routines."""
    outs = {-1: torch.from_numpy(X).double().permute(0, 3, 1, 2)}
    for v, n in enumerate(model.nodes):
        a = outs[n.inputs[0]]
        if n.kind == "conv":
            y = F.conv2d(a, torch.from_numpy(n.W).double().permute(0, 3, 1, 2), torch.from_numpy(n.b).double(),
                         stride=n.stride, padding=n.pad)
        elif n.kind == "dense":
            flat = a.permute(0, 2, 3, 1).reshape(a.shape[0], -1)
            y = F.linear(flat, torch.from_numpy(n.W).double(), torch.from_numpy(n.b).double())[:, :, None, None]
        elif n.kind == "maxpool":
            y = F.max_pool2d(a, n.kh, n.stride)
        elif n.kind == "flatten":
            y = a.permute(0, 2, 3, 1).reshape(a.shape[0], -1)[:, :, None, None]
        elif n.kind == "add":
            y = a + outs[n.inputs[1]]
        elif n.kind == "gap":
            y = a.mean(dim=(2, 3), keepdim=True)
        elif n.kind == "shortcut":
            s = a[:, :, ::n.stride, ::n.stride]
            y = F.pad(s, (0, 0, 0, 0, 0, n.cout - s.shape[1]))
        if n.act == "relu":
            y = y.clamp_min(0)
        # the oracle stores every activation in fp32
        outs[v] = y.float().double()
    return outs[len(model.nodes) - 1].reshape(X.shape[0], -1).float().numpy()


@pytest.mark.parametrize("name,n", [("mlp", 8), ("lenet5", 4), ("resnet20", 2), ("vgg", 1)])
def test_network_forward_matches_torch(oracle_mod, name, n):
    w = wl.workload(name, n, 1)
    lg, pred = oracle_mod.forward(w.model, w.X)
    ref = _torch_forward(w.model, w.X)
    scale = np.abs(ref).max(axis=1, keepdims=True)
    assert np.all(np.abs(lg - ref) <= 1e-5 * scale)
    assert np.array_equal(pred, ref.argmax(axis=1))


# ------------------------------------------------- brute force on tiny MLPs --

def _tiny_mlp(sizes, seed):
    rng = np.random.default_rng(seed)
    m = wl.Model("tiny", (1, 1, sizes[0]), sizes[-1])
    for i in range(len(sizes) - 1):
        W = rng.standard_normal((sizes[i + 1], sizes[i])).astype(np.float32)
        b = rng.uniform(-0.5, 0.5, sizes[i + 1]).astype(np.float32)
        m.nodes.append(wl.Node("dense", (i - 1,), "relu" if i < len(sizes) - 2 else "none",
                               cin=sizes[i], cout=sizes[i + 1], W=W, b=b))
    return m


def _brute_4_3_2(W0, b0, W1, b1, x, blocked=()):
    """Hand-expanded 4-3-2 MLP (ReLU hidden layer), fp64 sums rounded to fp32 per layer."""
    r = lambda v: max(float(np.float32(v)), 0.0)
    h0 = r(b0[0] + W0[0][0] * x[0] + W0[0][1] * x[1] + W0[0][2] * x[2] + W0[0][3] * x[3])
    h1 = r(b0[1] + W0[1][0] * x[0] + W0[1][1] * x[1] + W0[1][2] * x[2] + W0[1][3] * x[3])
    h2 = r(b0[2] + W0[2][0] * x[0] + W0[2][1] * x[1] + W0[2][2] * x[2] + W0[2][3] * x[3])
    h = [0.0 if 0 in blocked else h0, 0.0 if 1 in blocked else h1, 0.0 if 2 in blocked else h2]
    y0 = float(np.float32(b1[0] + W1[0][0] * h[0] + W1[0][1] * h[1] + W1[0][2] * h[2]))
    y1 = float(np.float32(b1[1] + W1[1][0] * h[0] + W1[1][1] * h[1] + W1[1][2] * h[2]))
    return [y0, y1]


def _as64(a):
    return np.asarray(a, np.float64).tolist()


def test_tiny_mlp_logits_bruteforce_every_operator(oracle_mod):
    m = _tiny_mlp((4, 3, 2), 11)
    rng = np.random.default_rng(12)
    X = rng.standard_normal((6, 1, 1, 4)).astype(np.float32)
    W0, b0 = _as64(m.nodes[0].W), _as64(m.nodes[0].b)
    W1, b1 = _as64(m.nodes[1].W), _as64(m.nodes[1].b)
    lg, _ = oracle_mod.forward(m, X)
    for t in range(6):
        assert lg[t].tolist() == _brute_4_3_2(W0, b0, W1, b1, _as64(X[t].ravel()))
    # one mutant per operator on the hidden layer, each expected value hand-expanded
    sig = float(np.float32(0.1)) * float(np.std(np.asarray(W0)))  # the descriptor holds param in fp32
    cases = []
    # NAI on neuron 1: w_1 -> -w_1, b_1 -> -b_1
    W0n = [row[:] for row in W0]; b0n = b0[:]
    W0n[1] = [-v for v in W0[1]]; b0n[1] = -b0[1]
    cases.append(("NAI", [1], 0.0, 5, W0n, b0n, ()))
    # NS on (0, 2): swap filters and biases
    W0s = [W0[2][:], W0[1][:], W0[0][:]]; b0s = [b0[2], b0[1], b0[0]]
    cases.append(("NS", [0, 2], 0.0, 6, W0s, b0s, ()))
    # NEB on neuron 2: its output forced to 0
    cases.append(("NEB", [2], 0.0, 7, W0, b0, (2,)))
    # GF on neuron 0: w_0f += fl32(sigma * n_f) with n from the slot-0 stream
    s0 = oracle_mod.sm64(8, 0)
    W0g = [row[:] for row in W0]
    W0g[0] = [float(np.float32(W0[0][f]) + np.float32(sig * oracle_mod.gauss(s0, f))) for f in range(4)]
    cases.append(("GF", [0], 0.1, 8, W0g, b0, ()))
    # WS on neuron 1: w_1f -> w_1,perm(f)
    perm = oracle_mod.fisher_yates(oracle_mod.sm64(9, 0), 4)
    W0w = [row[:] for row in W0]
    W0w[1] = [W0[1][perm[f]] for f in range(4)]
    cases.append(("WS", [1], 0.0, 9, W0w, b0, ()))
    for op, ids, param, seed, Wm, bm, blk in cases:
        table = wl.MutantTable(np.array([0], np.int32), np.array([OPS[op]], np.int32), np.array([len(ids)], np.int32),
                               np.array([0], np.int64), np.array([param], np.float32), np.array([seed], np.uint64),
                               np.array(ids, np.int32), np.zeros(1))
        res = oracle_mod.vanilla(m, X, table)
        for t in range(6):
            exp = _brute_4_3_2(Wm, bm, W1, b1, _as64(X[t].ravel()), blk)
            assert res["logits"][0, t].tolist() == exp, (op, t)


def test_neb_equals_zeroed_outgoing_weights(oracle_mod):
    """NEB read as 'output forced to 0' equals DeepMutation's 'zero the neuron's
    outgoing weights' when the consumer is a dense layer."""
    m = _tiny_mlp((5, 4, 3), 21)
    X = np.random.default_rng(22).standard_normal((9, 1, 1, 5)).astype(np.float32)
    table = wl.MutantTable(np.array([0], np.int32), np.array([OPS["NEB"]], np.int32), np.array([2], np.int32),
                           np.array([0], np.int64), np.zeros(1, np.float32), np.zeros(1, np.uint64),
                           np.array([1, 3], np.int32), np.zeros(1))
    got = oracle_mod.vanilla(m, X, table)["logits"][0]
    m2 = _tiny_mlp((5, 4, 3), 21)
    m2.nodes[1].W = m2.nodes[1].W.copy()
    m2.nodes[1].W[:, [1, 3]] = 0.0
    ref, _ = oracle_mod.forward(m2, X)
    assert np.array_equal(got, ref)


def test_worked_example(oracle_mod):
    m, X, labels, table, g = tiny_worked_example()
    lg, _ = oracle_mod.forward(m, X)
    assert lg.ravel().tolist() == [float(v) for v in g["logits"][0]]
    for lab, key in ((labels, "labels"), (None, "nolabels")):
        for fn in (oracle_mod.vanilla, oracle_mod.memo):
            r = fn(m, X, table, labels=lab)
            assert r["kill_bits"][:, 0].tolist() == [int(v) for v in g["kill_" + key][0]]
            assert r["scoreA"] == pytest.approx(float(g["scoreA_" + key][0][0]), abs=1e-15)
            assert r["scoreB"] == pytest.approx(float(g["scoreB_" + key][0][0]), abs=1e-15)


# ---------------------------------------------------------------- operators --

def test_operator_weight_rewrites(oracle_mod):
    w = wl.workload("lenet5", 1, 1)
    m = w.model
    rng = np.random.default_rng(5)
    for layer in range(m.n_layers()):
        nd = m.nodes[m.layers()[layer]]
        W2 = nd.W.reshape(nd.cout, -1)
        assert oracle_mod.layer_std(m, layer) == pytest.approx(float(np.std(nd.W.astype(np.float64))), rel=1e-12)
        for op in ("GF", "WS", "NAI", "NS", "NEB", "IDENTITY"):
            k = 2
            ids = rng.choice(nd.cout, size=k, replace=False).astype(np.int32)
            t = wl.MutantTable(np.array([layer], np.int32), np.array([OPS[op]], np.int32),
                               np.array([k], np.int32), np.array([0], np.int64), np.array([0.1], np.float32),
                               np.array([99 + layer], np.uint64), ids, np.zeros(1))
            Wm, bm, blk = oracle_mod.mutant_layer(m, t, 0)
            Wm = Wm.reshape(nd.cout, -1)
            other = np.setdiff1d(np.arange(nd.cout), ids)
            assert np.array_equal(Wm[other], W2[other]) and np.array_equal(bm[other], nd.b[other])
            if op == "NAI":
                assert np.array_equal(Wm[ids], -W2[ids]) and np.array_equal(bm[ids], -nd.b[ids])
            elif op == "NS":
                assert np.array_equal(Wm[ids[0]], W2[ids[1]]) and np.array_equal(Wm[ids[1]], W2[ids[0]])
                assert bm[ids[0]] == nd.b[ids[1]] and bm[ids[1]] == nd.b[ids[0]]
            elif op == "WS":
                for j in ids:
                    assert np.array_equal(np.sort(Wm[j]), np.sort(W2[j]))
                assert np.array_equal(bm, nd.b)
            elif op == "GF":
                sig = 0.1 * np.std(nd.W.astype(np.float64))
                d = (Wm[ids].astype(np.float64) - W2[ids]) / sig
                assert abs(d.mean()) < 0.5 and 0.5 < d.std() < 1.5
            else:
                assert np.array_equal(Wm, W2)
            assert blk.tolist() == [op == "NEB" and c in ids for c in range(nd.cout)]


def test_gf_noise_distribution(oracle_mod):
    from scipy import stats
    w = wl.workload("vgg", 1, 1)
    m = w.model
    layer = 7 - 1  # FC 4096 -> 512: 4096 noise values per neuron
    nd = m.nodes[m.layers()[layer]]
    t = wl.MutantTable(np.array([layer], np.int32), np.array([OPS["GF"]], np.int32), np.array([3], np.int32),
                       np.array([0], np.int64), np.array([0.1], np.float32), np.array([123], np.uint64),
                       np.array([5, 77, 300], np.int32), np.zeros(1))
    Wm, _, _ = oracle_mod.mutant_layer(m, t, 0)
    sig = 0.1 * np.std(nd.W.astype(np.float64))
    d = ((Wm[[5, 77, 300]].astype(np.float64) - nd.W[[5, 77, 300]]) / sig).ravel()
    assert stats.kstest(d, "norm").pvalue > 1e-3


def test_invalid_mutants_rejected(oracle_mod):
    w = wl.workload("mlp", 4, 1)
    bad = [(5, "GF", [0]), (0, "GF", [128]), (0, "NEB", [3, 3]), (0, "NS", [1, 2, 3]), (0, "GF", [-1])]
    for layer, op, ids in bad:
        t = wl.MutantTable(np.array([layer], np.int32), np.array([OPS[op]], np.int32), np.array([len(ids)], np.int32),
                           np.array([0], np.int64), np.array([0.1], np.float32), np.array([1], np.uint64),
                           np.array(ids, np.int32), np.zeros(1))
        with pytest.raises(oracle_mod.OracleError):
            oracle_mod.vanilla(w.model, w.X, t)
