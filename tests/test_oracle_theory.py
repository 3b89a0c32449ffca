"""The oracle against what the paper fixes: Theorem 1 (memoized = vanilla), the
memoization boundary of Algorithm 1, the cost accounting of Lemma 4, the kill
predicate and mutation score of Sec. 5.2, identity mutants, score bounds and
monotonicity, and closed forms for mutants of the output layer."""
import numpy as np
import pytest

from paper_2607_18582_gb300 import workloads as wl

OPS = wl.OP_INDEX


def _all_ops_table(model, per=2, seed=3):
    """Every operator (GF, NEB, NAI, NS, WS, IDENTITY) on every layer."""
    subs = [wl.mutants(model, per * 6, seed=seed + l, ratios=(0.05,), ops=wl.OPS, layers=[l])
            for l in range(model.n_layers())]
    return wl.concat(subs)


@pytest.mark.parametrize("name,n_in,per", [("mlp", 40, 2), ("lenet5", 12, 1), ("resnet20", 3, 1), ("vgg", 2, 1)])
def test_theorem1_memo_equals_vanilla(oracle_mod, name, n_in, per):
    w = wl.workload(name, n_in, 1)
    table = _all_ops_table(w.model, per)
    v = oracle_mod.vanilla(w.model, w.X, table)
    m = oracle_mod.memo(w.model, w.X, table)
    assert np.array_equal(v["logits"], m["logits"])      # bit-for-bit
    assert np.array_equal(v["kill_bits"], m["kill_bits"])
    assert v["scoreA"] == m["scoreA"] and v["scoreB"] == m["scoreB"]


def test_boundary_structure(oracle_mod):
    # Sequential networks: K = {the node right before the mutated layer} (Lemma 2,
    # case 1); a mutation of the first node leaves only the input (Alg. 3, p = []).
    le = wl.lenet5()
    for layer, node in enumerate(le.layers()):
        assert oracle_mod.boundary(le, layer) == [node - 1]
    # ResNet: a block's second conv needs the first conv's output and the block input
    # (the skip edge), i.e. two memo tensors.
    rn = wl.resnet20()
    L = rn.layers()
    # layer 2 = conv_b of the first block; its block input is the stem (node 0)
    assert oracle_mod.boundary(rn, 2) == [0, L[1]]
    # conv_a of a block: only the block input
    assert oracle_mod.boundary(rn, 1) == [0]
    # the FC after global average pooling: only the GAP output
    assert oracle_mod.boundary(rn, len(L) - 1) == [len(rn.nodes) - 2]


def test_cost_accounting_lemma4(oracle_mod):
    """Lemma 4 with MACs as the cost: for a cluster C with shared prefix P,
    vanilla - memo = (|C| - 1) cost(P), where memo pays P once."""
    le = wl.lenet5()
    macs = [oracle_mod.node_macs(le, v) for v in range(len(le.nodes))]
    # LeNet-5 layer costs (closed form: Ho*Wo*Cout*kh*kw*Cin and in*out)
    assert [macs[v] for v in le.layers()] == [28 * 28 * 6 * 25, 10 * 10 * 16 * 150, 400 * 120, 120 * 84, 84 * 10]
    total = sum(macs)
    table = wl.mutants(le, 50, seed=4)
    van = memo = 0
    clusters = {}
    for i in range(len(table)):
        mmi = le.layers()[int(table.layer[i])]
        clusters.setdefault(tuple(oracle_mod.boundary(le, int(table.layer[i]))), []).append(mmi)
    saving = 0
    for K, mmis in clusters.items():
        P = sum(macs[:mmis[0]])
        S = sum(macs[mmis[0]:])
        assert all(x == mmis[0] for x in mmis)
        van += len(mmis) * (P + S)
        memo += P + len(mmis) * S
        saving += (len(mmis) - 1) * P
    assert van == len(table) * total
    assert van - memo == saving >= 0


def _lemma4_gain(oracle_mod, model, table):
    """1 - memo / vanilla in MACs: memo computes each group's prefix once and every
    mutant's suffix from its first mutated layer on; vanilla runs every mutant whole."""
    macs = [oracle_mod.node_macs(model, v) for v in range(len(model.nodes))]
    L = model.layers()
    counts = np.bincount(table.layer, minlength=len(L))
    memo = sum(sum(macs[:L[l]]) + c * sum(macs[L[l]:]) for l, c in enumerate(counts) if c)
    return 1.0 - memo / (len(table) * sum(macs))


@pytest.mark.parametrize("name", ["lenet5", "mlp"])
def test_modelwide_ratio_trend(oracle_mod, name):
    """RQ2 (Sec. 5.5): with neurons drawn over the whole model, a larger selection ratio
    moves the first mutated layer earlier and shrinks the shared prefix, so the gain
    falls as the ratio grows (1 %, 3 %, 5 %)."""
    m = wl.MODELS[name](0)
    tables = [wl.modelwide_mutants(m, 400, seed=2, ratio=r) for r in (0.01, 0.03, 0.05)]
    first = [float(np.mean(t.layer)) for t in tables]
    gains = [_lemma4_gain(oracle_mod, m, t) for t in tables]
    assert first[0] > first[1] >= first[2]
    assert gains[0] > gains[1] >= gains[2] >= 0.0
    if name == "lenet5":
        assert gains[0] > gains[1] > gains[2] > 0.3


def test_identity_mutants_never_killed(oracle_mod):
    w = wl.workload("lenet5", 64, 1)
    m = w.model
    rows = []
    for layer in range(m.n_layers()):
        rows.append((layer, "IDENTITY", [], 0.0))
        rows.append((layer, "GF", [0, 1], 0.0))          # sigma multiplier 0
    # NEB on a channel that is dead (ReLU output 0) on every input
    lg, _ = oracle_mod.forward(m, w.X)
    outs = [oracle_mod.forward_nodes(m, x) for x in w.X]
    for layer in range(m.n_layers() - 1):
        v = m.layers()[layer]
        act = np.stack([o[v] for o in outs])
        dead = np.where(act.reshape(-1, act.shape[-1]).max(axis=0) <= 0)[0]
        if dead.size:
            rows.append((layer, "NEB", [int(dead[0])], 0.0))
    pool, off, nn = [], [], []
    for r in rows:
        off.append(len(pool)); nn.append(len(r[2])); pool += r[2]
    n = len(rows)
    t = wl.MutantTable(np.array([r[0] for r in rows], np.int32), np.array([OPS[r[1]] for r in rows], np.int32),
                       np.array(nn, np.int32), np.array(off, np.int64), np.array([r[3] for r in rows], np.float32),
                       np.arange(n, dtype=np.uint64), np.array(pool, np.int32), np.zeros(n))
    res = oracle_mod.vanilla(m, w.X, t)
    assert not res["kill_bits"].any()
    assert res["scoreA"] == 0.0 and res["scoreB"] == 0.0
    for i in range(n):
        assert np.array_equal(res["logits"][i], lg)


def test_scores_bounded_and_kills_monotone(oracle_mod):
    w = wl.workload("mlp", 200, 60)
    small = oracle_mod.vanilla(w.model, w.X[:70], w.table)
    big = oracle_mod.vanilla(w.model, w.X, w.table)
    for r in (small, big):
        assert 0.0 <= r["scoreA"] <= 1.0 and 0.0 <= r["scoreB"] <= 1.0
    # adding inputs never un-kills a mutant: the first 70 bits agree
    mask = np.uint64((1 << 6) - 1)
    assert np.array_equal(big["kill_bits"][:, 0], small["kill_bits"][:, 0])
    assert np.array_equal(big["kill_bits"][:, 1] & mask, small["kill_bits"][:, 1] & mask)
    assert big["scoreA"] >= small["scoreA"]


def test_kill_predicate_with_labels(oracle_mod):
    w = wl.workload("mlp", 150, 40)
    labels = np.random.default_rng(9).integers(0, 10, 150).astype(np.int32)
    r = oracle_mod.vanilla(w.model, w.X, w.table, labels=labels)
    pred0 = r["orig_logits"].argmax(axis=1)
    pred = r["logits"].argmax(axis=2)
    kill = (pred0 == labels)[None, :] & (pred != labels[None, :])
    bits = np.zeros_like(r["kill_bits"])
    for i, t in zip(*np.nonzero(kill)):
        bits[i, t // 64] |= np.uint64(1) << np.uint64(t % 64)
    assert np.array_equal(bits, r["kill_bits"])
    # score B brute force: distinct labels of the killing inputs
    L = len(set(labels.tolist()))
    sb = sum(len(set(labels[kill[i]].tolist())) for i in range(len(w.table))) / (len(w.table) * L)
    assert r["scoreB"] == pytest.approx(sb, abs=1e-15)
    assert r["scoreA"] == pytest.approx(kill.any(axis=1).mean(), abs=1e-15)


def test_output_layer_closed_forms(oracle_mod):
    """Mutants of the output layer: NEB sets logit j to 0, NAI negates it, NS swaps
    two logits, so each kill follows from the original logits alone."""
    w = wl.workload("lenet5", 80, 1)
    m = w.model
    last = m.n_layers() - 1
    rows = [("NEB", [3]), ("NAI", [7]), ("NS", [2, 5]), ("NEB", [0, 9]), ("NAI", [1, 4, 8])]
    pool, off = [], []
    for r in rows:
        off.append(len(pool)); pool += r[1]
    n = len(rows)
    t = wl.MutantTable(np.full(n, last, np.int32), np.array([OPS[r[0]] for r in rows], np.int32),
                       np.array([len(r[1]) for r in rows], np.int32), np.array(off, np.int64),
                       np.zeros(n, np.float32), np.zeros(n, np.uint64), np.array(pool, np.int32), np.zeros(n))
    res = oracle_mod.vanilla(m, w.X, t)
    z = res["orig_logits"]
    pred0 = z.argmax(axis=1)
    for i, (op, ids) in enumerate(rows):
        zz = z.copy()
        if op == "NEB":
            zz[:, ids] = 0.0
        elif op == "NAI":
            zz[:, ids] = -zz[:, ids]
        else:
            zz[:, [ids[0], ids[1]]] = zz[:, [ids[1], ids[0]]]
        assert np.array_equal(res["logits"][i], zz)
        kill = zz.argmax(axis=1) != pred0
        got = [(int(res["kill_bits"][i, tt // 64]) >> (tt % 64)) & 1 for tt in range(80)]
        assert got == kill.astype(int).tolist()


def test_empty_inputs_and_mutants(oracle_mod):
    w = wl.workload("mlp", 10, 5)
    r = oracle_mod.vanilla(w.model, w.X[:0], w.table)
    assert r["scoreA"] == 0.0 and r["scoreB"] == 0.0 and r["kill_bits"].size == 0
    r = oracle_mod.vanilla(w.model, w.X, w.table.subset([]))
    assert r["scoreA"] == 0.0 and r["scoreB"] == 0.0
    r = oracle_mod.memo(w.model, w.X, w.table.subset([]))
    assert r["scoreA"] == 0.0
