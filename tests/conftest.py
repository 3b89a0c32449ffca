import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running GPU case at full configuration size")


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.build()
    return oracle


def load_golden(name):
    """Parse a golden fixture: '#' lines are comments; other lines are 'key v1 v2 ...'
    (repeated keys collect into a list)."""
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *vals = line.split()
            out.setdefault(key, []).append(vals)
    return out


def tiny_worked_example():
    """The network, inputs and mutants of tests/golden/tiny_mlp_worked_example.txt."""
    from paper_2607_18582_gb300 import workloads as wl
    g = load_golden("tiny_mlp_worked_example.txt")
    f = lambda k: np.array([float(v) for v in g[k][0]], np.float32)
    m = wl.Model("tiny", (1, 1, 2), 2)
    m.nodes.append(wl.Node("dense", (-1,), "relu", cin=2, cout=2, W=f("W0").reshape(2, 2), b=f("b0")))
    m.nodes.append(wl.Node("dense", (0,), "none", cin=2, cout=2, W=f("W1").reshape(2, 2), b=f("b1")))
    X = f("X").reshape(4, 1, 1, 2)
    labels = np.array([int(v) for v in g["labels"][0]], np.int32)
    rows = g["mutant"]
    pool, off, lay, op, nn = [], [], [], [], []
    for r in rows:
        lay.append(int(r[0]))
        op.append(wl.OP_INDEX[r[1]])
        ids = [int(v) for v in r[2:]]
        if r[1] == "IDENTITY":
            ids = []
        off.append(len(pool))
        nn.append(len(ids))
        pool += ids
    n = len(rows)
    table = wl.MutantTable(np.array(lay, np.int32), np.array(op, np.int32), np.array(nn, np.int32),
                           np.array(off, np.int64), np.zeros(n, np.float32), np.arange(n, dtype=np.uint64),
                           np.array(pool, np.int32), np.zeros(n))
    return m, X, labels, table, g
