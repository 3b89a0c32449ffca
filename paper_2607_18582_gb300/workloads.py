"""Seeded synthetic workloads: networks, test inputs and mutant descriptor tables.

This module only *generates data*.  It holds none of the method's arithmetic (no
layer function, no mutation operator, no kill rule) and imports neither the GPU
binding nor the oracle, so both can be fed the very same arrays.

The paper's trained models and datasets (Table 1: LeNet-5, ResNet, MobileNetV2, FCNN,
RNN on MNIST-family, SVHN, CIFAR-10, Caltech-101, IMDB, Reuters) are not available
here.  Random-initialised networks of the same shapes and random inputs of the
datasets' shapes (28x28x1 / 32x32x3, 10 classes) stand in for them.

Recipe (every choice is seeded):
  * weights  He-normal, W ~ N(0, 2 / fan_in), numpy PCG64 seeded with `model_seed`
    (default 0); biases ~ U(-0.05, 0.05).
  * inputs   U[0,1] for the MLP and LeNet (MNIST-like), N(0,1) per channel for the
    32x32x3 networks (CIFAR-like); PCG64 seeded with `input_seed` (default 1).
  * mutants  PCG64 seeded with `mutant_seed` (default 2).  Mutant i: layer uniform over
    the weighted layers (stress mix: half on layer 0, the rest uniform over the
    others); operator [GF, NEB, NAI, NS][i % 4]; selection ratio
    ratios[(i // 4) % len(ratios)]; k = max(1, floor(r * N_l + 0.5)) neurons of layer
    l drawn without replacement (NS: 2 * max(1, k // 2) neurons, paired in order);
    GF sigma multiplier 0.1; a 63-bit seed for the operator's random numbers.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

OPS = ("GF", "NEB", "NAI", "NS", "WS", "IDENTITY")
WEIGHTED = ("conv", "dense", "dwconv", "embed", "lstm")
OP_INDEX = {name: i for i, name in enumerate(OPS)}
CONFIG_OPS = ("GF", "NEB", "NAI", "NS")


@dataclass
class Node:
    kind: str                 # conv | dense | maxpool | flatten | add | gap | shortcut | dwconv | embed | lstm
    inputs: tuple             # node ids; -1 = the model input
    act: str = "none"         # none | relu | relu6
    kh: int = 1               # lstm: 1 = every step's output, 0 = the last step's
    kw: int = 1
    stride: int = 1
    pad: int = 0
    cin: int = 0
    cout: int = 0
    # conv [cout][kh][kw][cin], dense [cout][cin], dwconv [c][kh][kw], embed [cout][vocabulary]
    # (channel-major), lstm [units][4][cin + units] (gates i, f, g, o; input then recurrent), fp32
    W: np.ndarray | None = None
    b: np.ndarray | None = None   # [cout]; lstm [units][4]; embed None


@dataclass
class Model:
    name: str
    in_shape: tuple           # (H, W, C), NHWC
    n_classes: int
    nodes: list = field(default_factory=list)

    def layers(self):
        """Node ids of the weighted nodes in node order."""
        return [v for v, n in enumerate(self.nodes) if n.kind in WEIGHTED]

    def n_layers(self):
        return len(self.layers())

    def layer_width(self, layer):
        return self.nodes[self.layers()[layer]].cout

    def shapes(self):
        """Output shape (H, W, C) of every node."""
        out = []
        for n in self.nodes:
            h, w, c = self.in_shape if n.inputs[0] < 0 else out[n.inputs[0]]
            if n.kind in ("conv", "dwconv"):
                out.append(((h + 2 * n.pad - n.kh) // n.stride + 1, (w + 2 * n.pad - n.kw) // n.stride + 1, n.cout))
            elif n.kind == "dense":
                out.append((1, 1, n.cout))
            elif n.kind == "maxpool":
                out.append(((h - n.kh) // n.stride + 1, (w - n.kw) // n.stride + 1, c))
            elif n.kind in ("flatten",):
                out.append((1, 1, h * w * c))
            elif n.kind == "gap":
                out.append((1, 1, c))
            elif n.kind == "shortcut":
                out.append(((h - 1) // n.stride + 1, (w - 1) // n.stride + 1, n.cout))
            elif n.kind == "embed":
                out.append((h, w, n.cout))
            elif n.kind == "lstm":
                out.append((1, w if n.kh else 1, n.cout))
            else:
                out.append((h, w, c))
        return out

    def layer_macs(self, layer):
        """Multiply-accumulates of weighted layer `layer` on one input."""
        v = self.layers()[layer]
        n = self.nodes[v]
        h, w, c = self.shapes()[v]
        if n.kind == "dwconv":
            return h * w * c * n.kh * n.kw
        if n.kind == "embed":
            return 0   # a table lookup
        if n.kind == "lstm":
            steps = (self.in_shape if n.inputs[0] < 0 else self.shapes()[n.inputs[0]])[1]
            return steps * n.cout * 4 * (n.cin + n.cout)
        return h * w * c * (n.kh * n.kw * n.cin if n.kind == "conv" else n.cin)


@dataclass
class MutantTable:
    layer: np.ndarray        # int32 [n]
    op: np.ndarray           # int32 [n], index into OPS
    n_neurons: np.ndarray    # int32 [n]
    neuron_off: np.ndarray   # int64 [n]
    param: np.ndarray        # float32 [n]
    seed: np.ndarray         # uint64 [n]
    pool: np.ndarray         # int32 [sum n_neurons]
    ratio: np.ndarray        # float64 [n] (bookkeeping only)
    # int32 [n] or None (all 0): 1 = the pool entries are (layer << 20 | neuron), the
    # mutant spans several layers and `layer` is the smallest of them
    tagged: np.ndarray = None

    def __len__(self):
        return int(self.layer.shape[0])

    def subset(self, idx):
        idx = np.asarray(idx, dtype=np.int64)
        pools, offs, off = [], [], 0
        for i in idx:
            a = int(self.neuron_off[i])
            n = int(self.n_neurons[i])
            pools.append(self.pool[a:a + n])
            offs.append(off)
            off += n
        pool = np.concatenate(pools).astype(np.int32) if pools else np.zeros(0, np.int32)
        return MutantTable(self.layer[idx].copy(), self.op[idx].copy(), self.n_neurons[idx].copy(),
                           np.asarray(offs, np.int64), self.param[idx].copy(), self.seed[idx].copy(),
                           pool, self.ratio[idx].copy(),
                           None if self.tagged is None else self.tagged[idx].copy())


# ----------------------------------------------------------------- networks --

class _Builder:
    def __init__(self, name, in_shape, n_classes, seed):
        self.m = Model(name, tuple(in_shape), n_classes)
        self.rng = np.random.default_rng(seed)
        self.shape = {-1: tuple(in_shape)}

    def _add(self, node, shape):
        self.m.nodes.append(node)
        v = len(self.m.nodes) - 1
        self.shape[v] = shape
        return v

    def _init(self, fan_in, shape_w, cout):
        W = (self.rng.standard_normal(shape_w) * np.sqrt(2.0 / fan_in)).astype(np.float32)
        b = self.rng.uniform(-0.05, 0.05, size=cout).astype(np.float32)
        return W, b

    def conv(self, x, cout, k, stride=1, pad=0, act="relu"):
        h, w, c = self.shape[x]
        W, b = self._init(k * k * c, (cout, k, k, c), cout)
        oh = (h + 2 * pad - k) // stride + 1
        ow = (w + 2 * pad - k) // stride + 1
        return self._add(Node("conv", (x,), act, k, k, stride, pad, c, cout, W, b), (oh, ow, cout))

    def dwconv(self, x, k, stride=1, pad=0, act="relu6"):
        h, w, c = self.shape[x]
        W = (self.rng.standard_normal((c, k, k)) * np.sqrt(2.0 / (k * k))).astype(np.float32)
        b = self.rng.uniform(-0.05, 0.05, size=c).astype(np.float32)
        oh = (h + 2 * pad - k) // stride + 1
        ow = (w + 2 * pad - k) // stride + 1
        return self._add(Node("dwconv", (x,), act, k, k, stride, pad, c, c, W, b), (oh, ow, c))

    def dense(self, x, cout, act="relu"):
        h, w, c = self.shape[x]
        W, b = self._init(h * w * c, (cout, h * w * c), cout)
        return self._add(Node("dense", (x,), act, 1, 1, 1, 0, h * w * c, cout, W, b), (1, 1, cout))

    def maxpool(self, x, k=2, stride=2):
        h, w, c = self.shape[x]
        return self._add(Node("maxpool", (x,), "none", k, k, stride), ((h - k) // stride + 1, (w - k) // stride + 1, c))

    def embed(self, x, vocab, dim):
        """Keras Embedding initialiser: U(-0.05, 0.05); stored channel-major."""
        h, w, _ = self.shape[x]
        W = self.rng.uniform(-0.05, 0.05, size=(dim, vocab)).astype(np.float32)
        return self._add(Node("embed", (x,), "none", 1, 1, 1, 0, vocab, dim, W, None), (h, w, dim))

    def lstm(self, x, units, sequences):
        """Keras LSTM initialisers: Glorot-uniform input weights, orthogonal recurrent
        weights, forget-gate bias 1; the other biases ~ U(-0.05, 0.05) so that every
        bias path is exercised."""
        _, T, c = self.shape[x]
        lim = np.sqrt(6.0 / (c + 4 * units))
        Wx = self.rng.uniform(-lim, lim, size=(c, 4 * units))
        q, r = np.linalg.qr(self.rng.standard_normal((4 * units, units)))
        Wh = (q * np.sign(np.diag(r))).T                        # [units][4 units], orthonormal rows
        W = np.zeros((units, 4, c + units), np.float32)
        for g in range(4):
            W[:, g, :c] = Wx[:, g * units:(g + 1) * units].T
            W[:, g, c:] = Wh[:, g * units:(g + 1) * units].T
        b = self.rng.uniform(-0.05, 0.05, size=(units, 4)).astype(np.float32)
        b[:, 1] = 1.0
        return self._add(Node("lstm", (x,), "none", 1 if sequences else 0, 1, 1, 0, c, units, W, b),
                         (1, T if sequences else 1, units))

    def flatten(self, x):
        h, w, c = self.shape[x]
        return self._add(Node("flatten", (x,)), (1, 1, h * w * c))

    def add(self, a, b, act="relu"):
        return self._add(Node("add", (a, b), act), self.shape[a])

    def gap(self, x):
        return self._add(Node("gap", (x,)), (1, 1, self.shape[x][2]))

    def shortcut(self, x, stride, cout):
        h, w, c = self.shape[x]
        return self._add(Node("shortcut", (x,), "none", 1, 1, stride, 0, c, cout),
                         ((h - 1) // stride + 1, (w - 1) // stride + 1, cout))


def mlp(seed=0, widths=(784, 128, 64, 10)):
    """Fully connected 784-128-64-10, ReLU (the paper's FCNN family, Table 1)."""
    bld = _Builder("mlp", (1, 1, widths[0]), widths[-1], seed)
    x = -1
    for i, w in enumerate(widths[1:]):
        x = bld.dense(x, w, act="relu" if i < len(widths) - 2 else "none")
    return bld.m


def lenet5(seed=0):
    """LeNet-5 style CNN on 28x28x1 (Table 1): conv5x5(6, pad 2)+ReLU+pool,
    conv5x5(16, valid)+ReLU+pool, FC 400-120-84-10."""
    bld = _Builder("lenet5", (28, 28, 1), 10, seed)
    x = bld.conv(-1, 6, 5, pad=2)
    x = bld.maxpool(x)
    x = bld.conv(x, 16, 5, pad=0)
    x = bld.maxpool(x)
    x = bld.flatten(x)
    x = bld.dense(x, 120)
    x = bld.dense(x, 84)
    bld.dense(x, 10, act="none")
    return bld.m


def vgg(seed=0):
    """VGG-style CNN on 32x32x3 with BN folded into the conv biases:
    [64,64,P][128,128,P][256,256,P], FC 4096-512-10 (8 weighted layers, 3,248,202
    parameters)."""
    bld = _Builder("vgg", (32, 32, 3), 10, seed)
    x = -1
    for c in (64, 128, 256):
        x = bld.conv(x, c, 3, pad=1)
        x = bld.conv(x, c, 3, pad=1)
        x = bld.maxpool(x)
    x = bld.flatten(x)
    x = bld.dense(x, 512)
    bld.dense(x, 10, act="none")
    return bld.m


def resnet20(seed=0):
    """ResNet-20 on 32x32x3: stem conv, 3 stages x 3 basic blocks (16/32/64
    channels, BN folded), parameter-free option-A shortcuts (stride-2 subsampling,
    zero channels appended), global average pooling, FC 64-10.  19 convs + 1 FC."""
    bld = _Builder("resnet20", (32, 32, 3), 10, seed)
    x = bld.conv(-1, 16, 3, pad=1)
    cin = 16
    for s, c in enumerate((16, 32, 64)):
        for blk in range(3):
            stride = 2 if (s > 0 and blk == 0) else 1
            a = bld.conv(x, c, 3, stride=stride, pad=1, act="relu")
            bb = bld.conv(a, c, 3, stride=1, pad=1, act="none")
            sc = x if (stride == 1 and cin == c) else bld.shortcut(x, stride, c)
            x = bld.add(bb, sc, act="relu")
            cin = c
    x = bld.gap(x)
    bld.dense(x, 10, act="none")
    return bld.m


def resnet10(seed=0):
    """ResNet-10 on 32x32x3 (the paper's ResNet family, Table 1): stem conv, four
    stages of one basic block each (16/32/64/128 channels), projection shortcuts (a
    1x1 convolution of stride 2 in the skip branch where the shape changes), global
    average pooling, FC 128-10.  The skip branch holds a weighted layer, so the
    memoization boundary of a mutant depends on Algorithm 2's graph, not on a chain.
    Oracle only: the GPU stage compiler takes option-A shortcuts."""
    bld = _Builder("resnet10", (32, 32, 3), 10, seed)
    x = bld.conv(-1, 16, 3, pad=1)
    cin = 16
    for s, c in enumerate((16, 32, 64, 128)):
        stride = 1 if s == 0 else 2
        a = bld.conv(x, c, 3, stride=stride, pad=1, act="relu")
        bb = bld.conv(a, c, 3, stride=1, pad=1, act="none")
        sc = x if (stride == 1 and cin == c) else bld.conv(x, c, 1, stride=stride, pad=0, act="none")
        x = bld.add(bb, sc, act="relu")
        cin = c
    x = bld.gap(x)
    bld.dense(x, 10, act="none")
    return bld.m


def mobilenetv2_tiny(seed=0):
    """A small MobileNetV2-style network on 32x32x3 (the paper's MobileNetV2 family,
    Table 1): conv3x3(16)+ReLU6, three inverted residual blocks (1x1 expansion x4 +
    ReLU6, 3x3 depthwise + ReLU6, linear 1x1 projection; a residual add where the shape
    is kept), conv1x1(64)+ReLU6, global average pooling, dense 10.  Oracle only: the
    GPU library has no depthwise layer yet."""
    bld = _Builder("mobilenetv2_tiny", (32, 32, 3), 10, seed)
    x = bld.conv(-1, 16, 3, stride=1, pad=1, act="relu6")
    for cout, stride in ((16, 1), (24, 2), (24, 1)):
        cin = bld.shape[x][2]
        h = bld.conv(x, 4 * cin, 1, act="relu6")
        h = bld.dwconv(h, 3, stride=stride, pad=1, act="relu6")
        h = bld.conv(h, cout, 1, act="none")
        x = bld.add(h, x, act="none") if stride == 1 and cin == cout else h
    x = bld.conv(x, 64, 1, act="relu6")
    x = bld.gap(x)
    bld.dense(x, 10, act="none")
    return bld.m


def rnn(seed=0, n_classes=2, vocab=20000, dim=128, units=(64, 64), steps=80, name="rnn_imdb"):
    """The paper's RNN family (Sec. 5.3, Table 1): embedding, two LSTM layers (the
    first returns every step), dense output.  Vocabulary 20,000, width 128 and 64
    units per LSTM give exactly Table 1's sizes: 2,642,562 parameters with 2 classes
    (IMDB) and 2,648,282 with 90 (Reuters).  Sequences of `steps` tokens.  Oracle
    only: the GPU library has no recurrent layer yet."""
    bld = _Builder(name, (1, steps, 1), n_classes, seed)
    x = bld.embed(-1, vocab, dim)
    x = bld.lstm(x, units[0], sequences=True)
    for u in units[1:-1]:
        x = bld.lstm(x, u, sequences=True)
    x = bld.lstm(x, units[-1], sequences=False)
    bld.dense(x, n_classes, act="none")
    return bld.m


def rnn_reuters(seed=0):
    return rnn(seed, n_classes=90, name="rnn_reuters")


MODELS = {"mlp": mlp, "lenet5": lenet5, "vgg": vgg, "resnet20": resnet20, "resnet10": resnet10,
          "mobilenetv2_tiny": mobilenetv2_tiny, "rnn_imdb": rnn, "rnn_reuters": rnn_reuters}


# ------------------------------------------------------------------- inputs --

def inputs(model: Model, n: int, seed: int = 1, dist: str | None = None) -> np.ndarray:
    """n inputs of the model's shape, [n][H][W][C] float32."""
    if model.nodes and model.nodes[0].kind == "embed":
        return token_sequences(model, n, seed)
    if dist is None:
        dist = "uniform" if model.in_shape[2] == 1 else "normal"
    rng = np.random.default_rng(seed)
    shape = (n,) + tuple(model.in_shape)
    if dist == "uniform":
        return rng.random(shape, dtype=np.float32)
    return rng.standard_normal(shape, dtype=np.float32)


def token_sequences(model: Model, n: int, seed: int = 1) -> np.ndarray:
    """n token sequences for a model that starts with an embedding (IMDB / Reuters
    stand-ins), [n][1][T][1] float32 holding integer ids: review lengths
    ~ lognormal (median T / 2) clipped to [8, T], word ids 1 + Zipf(1.3) clipped to the
    vocabulary (word frequencies in text are heavy-tailed), pre-padded with id 0 as
    Keras' pad_sequences does."""
    rng = np.random.default_rng(seed)
    T, V = model.in_shape[1], model.nodes[0].cin
    out = np.zeros((n, 1, T, 1), np.float32)
    for t in range(n):
        length = int(np.clip(np.round(np.exp(rng.normal(np.log(T / 2), 0.6))), min(8, T), T))
        ids = np.minimum(rng.zipf(1.3, size=length), V - 1)
        out[t, 0, T - length:, 0] = ids
    return out


# ------------------------------------------------------------------ mutants --

def mutants(model: Model, n: int, seed: int = 2, ratios=(0.01,), ops=CONFIG_OPS,
            first_layer_share: float | None = None, layers=None) -> MutantTable:
    """Descriptor table of n single-layer mutants (recipe in the module docstring)."""
    rng = np.random.default_rng(seed)
    L = model.n_layers()
    cand = list(range(L)) if layers is None else list(layers)
    lay = np.zeros(n, np.int32)
    opv = np.zeros(n, np.int32)
    nn = np.zeros(n, np.int32)
    off = np.zeros(n, np.int64)
    par = np.zeros(n, np.float32)
    sd = np.zeros(n, np.uint64)
    rat = np.zeros(n, np.float64)
    pool = []
    pos = 0
    for i in range(n):
        if first_layer_share is not None:
            l = 0 if rng.random() < first_layer_share else int(rng.integers(1, L))
        else:
            l = cand[int(rng.integers(0, len(cand)))]
        op = ops[i % len(ops)]
        r = ratios[(i // len(ops)) % len(ratios)]
        N = model.layer_width(l)
        k = max(1, int(np.floor(r * N + 0.5)))
        if op == "NS":
            k = min(2 * max(1, k // 2), N - (N % 2))
        k = min(k, N)
        ids = rng.choice(N, size=k, replace=False).astype(np.int32)
        lay[i] = l
        opv[i] = OP_INDEX[op]
        nn[i] = k
        off[i] = pos
        par[i] = 0.1 if op == "GF" else 0.0
        sd[i] = np.uint64(int(rng.integers(0, 2 ** 63 - 1)))
        rat[i] = r
        pool.append(ids)
        pos += k
    return MutantTable(lay, opv, nn, off, par, sd,
                       np.concatenate(pool).astype(np.int32) if pool else np.zeros(0, np.int32), rat)


def modelwide_mutants(model: Model, n: int, seed: int = 2, ratio: float = 0.01, ops=CONFIG_OPS) -> MutantTable:
    """Descriptor table of n mutants whose neurons are drawn over the whole model
    (DeepMutation's model-wide selection ratio; the paper's set mu(M') of mutated
    layers): k = max(1, round(ratio x all neurons)) distinct (layer, neuron) pairs,
    uniform over the model's neurons; NS draws k / 2 pairs, each inside one layer
    chosen with probability proportional to its width.  Entries are encoded
    (layer << 20 | neuron) in layer order ("tagged"); `layer` is the smallest."""
    rng = np.random.default_rng(seed)
    L = model.n_layers()
    widths = np.array([model.layer_width(l) for l in range(L)], np.int64)
    total = int(widths.sum())
    starts = np.concatenate([[0], np.cumsum(widths)])
    lay = np.zeros(n, np.int32)
    opv = np.zeros(n, np.int32)
    nn = np.zeros(n, np.int32)
    off = np.zeros(n, np.int64)
    par = np.zeros(n, np.float32)
    sd = np.zeros(n, np.uint64)
    rat = np.full(n, ratio, np.float64)
    pool = []
    pos = 0
    k = max(1, int(np.floor(ratio * total + 0.5)))
    pair_w = np.where(widths >= 2, widths, 0).astype(np.float64)
    for i in range(n):
        op = ops[i % len(ops)]
        if op == "NS":
            chosen = set()
            ent = []
            for _ in range(max(1, k // 2)):
                while True:
                    l = int(rng.choice(L, p=pair_w / pair_w.sum()))
                    a, b = (int(v) for v in rng.choice(int(widths[l]), size=2, replace=False))
                    if (l, a) not in chosen and (l, b) not in chosen:
                        break
                chosen.update({(l, a), (l, b)})
                ent.append((l, a, b))
            ent.sort()
            entries = [(l << 20) | j for l, a, b in ent for j in (a, b)]
        else:
            flat = np.sort(rng.choice(total, size=min(k, total), replace=False))
            ls = np.searchsorted(starts, flat, side="right") - 1
            entries = [(int(l) << 20) | int(f - starts[l]) for f, l in zip(flat, ls)]
        lay[i] = min(e >> 20 for e in entries)
        opv[i] = OP_INDEX[op]
        nn[i] = len(entries)
        off[i] = pos
        par[i] = 0.1 if op == "GF" else 0.0
        sd[i] = np.uint64(int(rng.integers(0, 2 ** 63 - 1)))
        pool.append(np.array(entries, np.int32))
        pos += len(entries)
    return MutantTable(lay, opv, nn, off, par, sd,
                       np.concatenate(pool).astype(np.int32) if pool else np.zeros(0, np.int32), rat,
                       np.ones(n, np.int32))


def concat(tables) -> MutantTable:
    """One table holding the rows of several, in order."""
    tables = list(tables)
    offs, pos = [], 0
    for t in tables:
        offs.append(t.neuron_off + pos)
        pos += t.pool.size
    cat = lambda f, dt: np.concatenate([getattr(t, f) for t in tables]).astype(dt) if tables else np.zeros(0, dt)
    tagged = None
    if any(t.tagged is not None for t in tables):
        tagged = np.concatenate([t.tagged if t.tagged is not None else np.zeros(len(t), np.int32)
                                 for t in tables]).astype(np.int32)
    return MutantTable(cat("layer", np.int32), cat("op", np.int32), cat("n_neurons", np.int32),
                       np.concatenate(offs).astype(np.int64) if tables else np.zeros(0, np.int64),
                       cat("param", np.float32), cat("seed", np.uint64), cat("pool", np.int32),
                       cat("ratio", np.float64), tagged)


def table_from_rows(rows) -> MutantTable:
    """Build a table from (layer, op_name, neuron_ids, param, seed) tuples."""
    pool, off, nn = [], [], []
    for r in rows:
        off.append(len(pool))
        nn.append(len(r[2]))
        pool += list(r[2])
    n = len(rows)
    return MutantTable(np.array([r[0] for r in rows], np.int32), np.array([OP_INDEX[r[1]] for r in rows], np.int32),
                       np.array(nn, np.int32), np.array(off, np.int64),
                       np.array([r[3] for r in rows], np.float32), np.array([r[4] for r in rows], np.uint64),
                       np.array(pool, np.int32), np.zeros(n))


def stratified(table: MutantTable, model: Model, per_layer_op: int) -> np.ndarray:
    """Indices of a stratified subsample: the first `per_layer_op` mutants of every
    (layer, operator) pair, in table order."""
    picked = []
    seen = {}
    for i in range(len(table)):
        key = (int(table.layer[i]), int(table.op[i]))
        if seen.get(key, 0) < per_layer_op:
            seen[key] = seen.get(key, 0) + 1
            picked.append(i)
    return np.asarray(picked, np.int64)


# ------------------------------------------------------------ named configs --

@dataclass
class Workload:
    name: str
    model: Model
    X: np.ndarray
    table: MutantTable
    labels: np.ndarray | None = None


CONFIGS = {
    # name: (model, n_inputs, n_mutants, ratios, first-layer share)
    "mlp": ("mlp", 1000, 200, (0.01,), None),
    "lenet5": ("lenet5", 10000, 2000, (0.01,), None),
    "vgg": ("vgg", 10000, 5000, (0.005, 0.01, 0.02, 0.05), None),
    "resnet20": ("resnet20", 10000, 5000, (0.01,), None),
    "vgg_stress": ("vgg", 20000, 20000, (0.001, 0.01, 0.05, 0.10), 0.5),
    # model-wide selection: each mutant's neurons drawn over all layers (1 % of them)
    "lenet5_modelwide": ("lenet5", 10000, 2000, (0.01,), "model"),
    # the paper's RQ2 ratios (Sec. 5.5): 3 % and 5 % of all neurons per mutant
    "lenet5_modelwide_3": ("lenet5", 10000, 2000, (0.03,), "model"),
    "lenet5_modelwide_5": ("lenet5", 10000, 2000, (0.05,), "model"),
    "mlp_modelwide": ("mlp", 1000, 200, (0.01,), "model"),
}


def workload(name: str, n_inputs: int | None = None, n_mutants: int | None = None,
             model_seed: int = 0, input_seed: int = 1, mutant_seed: int = 2) -> Workload:
    """A named configuration, optionally truncated to its first inputs / mutants
    (the truncated table equals the prefix of the full one)."""
    mname, n_in, n_mut, ratios, skew = CONFIGS[name]
    model = MODELS[mname](model_seed)
    n_in = n_in if n_inputs is None else n_inputs
    n_mut = n_mut if n_mutants is None else n_mutants
    X = inputs(model, n_in, input_seed)
    if skew == "model":
        table = modelwide_mutants(model, n_mut, mutant_seed, ratio=ratios[0])
    else:
        table = mutants(model, n_mut, mutant_seed, ratios=ratios, first_layer_share=skew)
    return Workload(name, model, X, table)
