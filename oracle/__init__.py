"""ctypes front end of the CPU oracle (mure_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, by __graft_entry__.smoke() and by the
CPU-baseline leg of bench.py.  The GPU library and its Python binding never import
this package.  It accepts the plain arrays of paper_2607_18582_gb300.workloads (or
any object with the same fields) and converts them to its own C structures.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mure_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libmure_oracle.so")

KINDS = {"conv": 0, "dense": 1, "maxpool": 2, "flatten": 3, "add": 4, "gap": 5, "shortcut": 6, "dwconv": 7, "embed": 8,
         "lstm": 9}
ACTS = {"none": 0, "relu": 1, "relu6": 2}
OPS = {"GF": 0, "NEB": 1, "NAI": 2, "NS": 3, "WS": 4, "IDENTITY": 5}


class OracleError(RuntimeError):
    pass


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C11, -O2, pthreads)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-Wall", "-fPIC", "-shared", "-o", tmp, _SRC,
                               "-lm", "-lpthread"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Node(C.Structure):
    _fields_ = [("kind", C.c_int32), ("act", C.c_int32), ("in0", C.c_int32), ("in1", C.c_int32),
                ("kh", C.c_int32), ("kw", C.c_int32), ("stride", C.c_int32), ("pad", C.c_int32),
                ("cin", C.c_int32), ("cout", C.c_int32),
                ("W", C.POINTER(C.c_float)), ("b", C.POINTER(C.c_float))]


class _Model(C.Structure):
    _fields_ = [("in_h", C.c_int32), ("in_w", C.c_int32), ("in_c", C.c_int32), ("n_classes", C.c_int32),
                ("n_nodes", C.c_int32), ("nodes", C.POINTER(_Node))]


class _Mutant(C.Structure):
    _fields_ = [("layer", C.c_int32), ("op", C.c_int32), ("n_neurons", C.c_int32), ("tagged", C.c_int32),
                ("neuron_off", C.c_int64), ("param", C.c_float), ("reserved2", C.c_float), ("seed", C.c_uint64)]


_lib = None
_lock = threading.Lock()
_FP = C.POINTER(C.c_float)
_I32P = C.POINTER(C.c_int32)
_U64P = C.POINTER(C.c_uint64)
_U8P = C.POINTER(C.c_uint8)
_DP = C.POINTER(C.c_double)


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            L.or_sm64.restype = C.c_uint64
            L.or_sm64.argtypes = [C.c_uint64, C.c_uint64]
            L.or_gauss.restype = C.c_double
            L.or_gauss.argtypes = [C.c_uint64, C.c_int64]
            L.or_fisher_yates.restype = None
            L.or_fisher_yates.argtypes = [C.c_uint64, C.c_int32, _I32P]
            L.or_shapes.argtypes = [C.POINTER(_Model), _I32P]
            L.or_node_forward.argtypes = [C.POINTER(_Model), C.c_int32, _FP, _FP, _FP]
            L.or_n_layers.argtypes = [C.POINTER(_Model)]
            L.or_layer_std.restype = C.c_double
            L.or_layer_std.argtypes = [C.POINTER(_Model), C.c_int32]
            L.or_mutant_layer.argtypes = [C.POINTER(_Model), C.POINTER(_Mutant), _I32P, C.c_int64, _FP, _FP, _U8P]
            L.or_mutant_layer_at.argtypes = [C.POINTER(_Model), C.POINTER(_Mutant), _I32P, C.c_int64, C.c_int32,
                                             _FP, _FP, _U8P]
            L.or_unchanged_rows.argtypes = [C.POINTER(_Model), _FP, C.c_int64, C.POINTER(_Mutant), C.c_int64,
                                            _I32P, C.c_int64, C.c_int32, _U64P]
            L.or_forward.argtypes = [C.POINTER(_Model), _FP, C.c_int64, _FP, _I32P]
            L.or_forward_nodes.argtypes = [C.POINTER(_Model), _FP, _FP]
            L.or_scores.argtypes = [_U64P, C.c_int64, C.c_int64, _I32P, C.c_int32, _DP, _DP, C.POINTER(C.c_int64)]
            L.or_vanilla.argtypes = [C.POINTER(_Model), _FP, C.c_int64, _I32P, C.POINTER(_Mutant), C.c_int64,
                                     _I32P, C.c_int64, C.c_int32, _FP, _FP, _U64P, _DP, _DP]
            L.or_memo.argtypes = [C.POINTER(_Model), _FP, C.c_int64, _I32P, C.POINTER(_Mutant), C.c_int64,
                                  _I32P, C.c_int64, C.c_int32, _FP, _U64P, _DP, _DP, _I32P]
            L.or_node_macs.restype = C.c_int64
            L.or_node_macs.argtypes = [C.POINTER(_Model), C.c_int32]
            L.or_boundary.argtypes = [C.POINTER(_Model), C.c_int32, _U8P]
            _lib = L
    return _lib


def _ptr(a, t):
    return a.ctypes.data_as(t) if a is not None else None


class OModel:
    """The oracle's own C view of a network description (keeps arrays alive)."""

    def __init__(self, model):
        self.model = model
        self._keep = []
        nodes = (_Node * len(model.nodes))()
        for v, n in enumerate(model.nodes):
            W = None if n.W is None else np.ascontiguousarray(n.W, np.float32)
            b = None if n.b is None else np.ascontiguousarray(n.b, np.float32)
            self._keep += [W, b]
            ins = list(n.inputs) + [-1] * (2 - len(n.inputs))
            nodes[v] = _Node(KINDS[n.kind], ACTS[n.act], ins[0], ins[1], n.kh, n.kw, n.stride, n.pad, n.cin, n.cout,
                             _ptr(W, _FP), _ptr(b, _FP))
        self._nodes = nodes
        h, w, c = model.in_shape
        self.c = _Model(h, w, c, model.n_classes, len(model.nodes), nodes)
        self.in_size = h * w * c

    def shapes(self):
        out = np.zeros((len(self.model.nodes), 3), np.int32)
        _check(lib().or_shapes(C.byref(self.c), _ptr(out, _I32P)))
        return out


def _check(rc):
    if rc != 0:
        raise OracleError(f"oracle returned status {rc}")


def _mutants(table):
    n = len(table)
    arr = (_Mutant * max(n, 1))()
    tagged = getattr(table, "tagged", None)
    for i in range(n):
        arr[i] = _Mutant(int(table.layer[i]), int(table.op[i]), int(table.n_neurons[i]),
                         int(tagged[i]) if tagged is not None else 0,
                         int(table.neuron_off[i]), float(table.param[i]), 0.0, int(table.seed[i]))
    pool = np.ascontiguousarray(table.pool, np.int32)
    if pool.size == 0:
        pool = np.zeros(1, np.int32)
    return arr, pool, int(table.pool.size)


def sm64(seed: int, i: int) -> int:
    return int(lib().or_sm64(seed, i))


def gauss(stream_seed: int, f: int) -> float:
    return float(lib().or_gauss(stream_seed, f))


def fisher_yates(stream_seed: int, n: int) -> np.ndarray:
    p = np.zeros(n, np.int32)
    lib().or_fisher_yates(stream_seed, n, _ptr(p, _I32P))
    return p


def node_forward(model, v, in0, in1=None):
    om = OModel(model)
    shp = om.shapes()
    out = np.zeros(tuple(shp[v]), np.float32)
    a0 = np.ascontiguousarray(in0, np.float32)
    a1 = None if in1 is None else np.ascontiguousarray(in1, np.float32)
    _check(lib().or_node_forward(C.byref(om.c), v, _ptr(a0, _FP), _ptr(a1, _FP), _ptr(out, _FP)))
    return out


def forward(model, X):
    """Original network: (logits [n][C], predictions [n])."""
    om = OModel(model)
    X = np.ascontiguousarray(X, np.float32)
    n = X.shape[0]
    lg = np.zeros((n, model.n_classes), np.float32)
    pr = np.zeros(n, np.int32)
    _check(lib().or_forward(C.byref(om.c), _ptr(X, _FP), n, _ptr(lg, _FP), _ptr(pr, _I32P)))
    return lg, pr


def forward_nodes(model, x):
    """Every node's output for one input, as a list of arrays shaped (H, W, C)."""
    om = OModel(model)
    shp = om.shapes()
    tot = int(np.prod(shp, axis=1).sum())
    buf = np.zeros(tot, np.float32)
    x = np.ascontiguousarray(x, np.float32)
    _check(lib().or_forward_nodes(C.byref(om.c), _ptr(x, _FP), _ptr(buf, _FP)))
    outs, off = [], 0
    for s in shp:
        k = int(np.prod(s))
        outs.append(buf[off:off + k].reshape(tuple(s)))
        off += k
    return outs


def layer_std(model, layer):
    return float(lib().or_layer_std(C.byref(OModel(model).c), layer))


def mutant_layer(model, table, i, layer=None):
    """Materialised parameters of weighted layer `layer` of mutant i (default: its
    first mutated layer): (W', b', blocked)."""
    om = OModel(model)
    layer = int(table.layer[i]) if layer is None else int(layer)
    v = model.layers()[layer]
    nd = model.nodes[v]
    W = np.zeros_like(nd.W)
    b = np.zeros_like(nd.b) if nd.b is not None else np.zeros(1, np.float32)   # an embedding has no bias
    blk = np.zeros(nd.cout, np.uint8)
    arr, pool, plen = _mutants(table)
    _check(lib().or_mutant_layer_at(C.byref(om.c), C.byref(arr[i]), _ptr(pool, _I32P), plen, layer,
                                    _ptr(W, _FP), _ptr(b, _FP), _ptr(blk, _U8P)))
    return W, (b if nd.b is not None else None), blk.astype(bool)


def _run(fn, model, X, table, labels, n_threads, want_logits, memo):
    om = OModel(model)
    X = np.ascontiguousarray(X, np.float32)
    n_in = X.shape[0]
    n_mut = len(table)
    arr, pool, plen = _mutants(table)
    W64 = (n_in + 63) // 64
    kill = np.zeros((max(n_mut, 1), max(W64, 1)), np.uint64)
    lg = np.zeros((n_mut, n_in, model.n_classes), np.float32) if want_logits else None
    sa, sb = C.c_double(0), C.c_double(0)
    lab = None if labels is None else np.ascontiguousarray(labels, np.int32)
    if n_threads is None:
        n_threads = os.cpu_count() or 1
    Xp = _ptr(X, _FP) if X.size else None
    if memo:
        ncl = C.c_int32(0)
        _check(fn(C.byref(om.c), Xp, n_in, _ptr(lab, _I32P), arr, n_mut, _ptr(pool, _I32P), plen, n_threads,
                  _ptr(lg, _FP), _ptr(kill, _U64P), C.byref(sa), C.byref(sb), C.byref(ncl)))
        extra = {"n_clusters": ncl.value}
    else:
        orig = np.zeros((n_in, model.n_classes), np.float32)
        _check(fn(C.byref(om.c), Xp, n_in, _ptr(lab, _I32P), arr, n_mut, _ptr(pool, _I32P), plen, n_threads,
                  _ptr(lg, _FP), _ptr(orig, _FP), _ptr(kill, _U64P), C.byref(sa), C.byref(sb)))
        extra = {"orig_logits": orig}
    res = {"kill_bits": kill[:n_mut, :W64], "scoreA": sa.value, "scoreB": sb.value, "logits": lg}
    res.update(extra)
    return res


def vanilla(model, X, table, labels=None, n_threads=None, want_logits=True):
    """Vanilla mutation testing (every mutant built and run end to end)."""
    return _run(lib().or_vanilla, model, X, table, labels, n_threads, want_logits, memo=False)


def unchanged_rows(model, X, table, n_threads=None):
    """Bits [n_mut][ceil(n_in/64)]: every layer the mutant changes gives, on that input,
    the original output bit for bit (the row's suffix and prediction are the original's)."""
    om = OModel(model)
    X = np.ascontiguousarray(X, np.float32)
    n_in, n_mut = X.shape[0], len(table)
    arr, pool, plen = _mutants(table)
    W64 = (n_in + 63) // 64
    bits = np.zeros((max(n_mut, 1), max(W64, 1)), np.uint64)
    _check(lib().or_unchanged_rows(C.byref(om.c), _ptr(X, _FP) if X.size else None, n_in, arr, n_mut,
                                   _ptr(pool, _I32P), plen, n_threads or (os.cpu_count() or 1), _ptr(bits, _U64P)))
    return bits[:n_mut, :W64]


def memo(model, X, table, labels=None, n_threads=None, want_logits=True):
    """Memoized mutation testing (Algorithm 1 with Algorithms 2-4)."""
    return _run(lib().or_memo, model, X, table, labels, n_threads, want_logits, memo=True)


def scores(kill_bits, labels, n_classes):
    kb = np.ascontiguousarray(kill_bits, np.uint64)
    n_mut = kb.shape[0]
    n_in = labels.shape[0]
    sa, sb = C.c_double(0), C.c_double(0)
    killed = np.zeros(max(n_mut, 1), np.int64)
    lab = np.ascontiguousarray(labels, np.int32)
    _check(lib().or_scores(_ptr(kb, _U64P), n_mut, n_in, _ptr(lab, _I32P), n_classes, C.byref(sa), C.byref(sb),
                           killed.ctypes.data_as(C.POINTER(C.c_int64))))
    return sa.value, sb.value, killed[:n_mut]


def node_macs(model, v):
    return int(lib().or_node_macs(C.byref(OModel(model).c), v))


def boundary(model, layer):
    """Memoization boundary K of a mutant at weighted layer `layer`: sorted node ids
    (-1 = the model input)."""
    inK = np.zeros(len(model.nodes) + 1, np.uint8)
    _check(lib().or_boundary(C.byref(OModel(model).c), layer, _ptr(inK, _U8P)))
    return [p - 1 for p in range(len(inK)) if inK[p]]
