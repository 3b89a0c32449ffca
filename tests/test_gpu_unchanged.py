"""Exact unchanged-row elimination on the GPU (beyond the paper; sound by its soundness
theorem's argument): a single-layer mutant's row whose input to the first suffix layer
equals the original bit for bit repeats the original forward pass, so it is not run;
its kill bit is 0 and its logits are the original logits.  Checked against a run
without the elimination (identical kill matrices, logits and scores, bit for bit),
against the GPU vanilla mode, and against the oracle's unchanged-row reference
(or_unchanged_rows: the mutated layer's output equal to the original).  The GPU
compares the layer's output after its pooling and residual add, which every row equal
before them also is, so it drops at least the oracle's rows (exactly them where
nothing follows the activation, as in the MLP)."""
import numpy as np
import pytest

from parity_util import bits
from paper_2607_18582_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def M():
    from paper_2607_18582_gb300 import build
    build.build()
    from paper_2607_18582_gb300 import mure
    return mure


@pytest.fixture(scope="module")
def ctx(M):
    return M.mure_create(0)


def dead_heavy_table(model, seed):
    """Every operator on every layer, with NEB and NS on many neurons so that dead
    ReLU units (NEB) and equal channels (NS) give unchanged rows."""
    rng = np.random.default_rng(seed)
    rows = []
    for l in range(model.n_layers()):
        N = model.layer_width(l)
        for i in range(8):
            ids = rng.choice(N, size=min(2, N), replace=False).tolist()
            op = ("NEB", "NS", "GF", "NAI", "WS", "IDENTITY", "NEB", "NEB")[i]
            if op == "IDENTITY":
                rows.append((l, op, [], 0.0, 0))
            elif op == "GF":
                rows.append((l, op, ids, 0.0 if i == 2 else 0.1, 10 + i))   # sigma 0: unchanged everywhere
            elif op == "WS":
                rows.append((l, op, ids[:1], 0.0, 20 + i))
            else:
                rows.append((l, op, ids, 0.0, 0))
    return wl.table_from_rows(rows)


CASES = [("mlp", 160, "fp32"), ("lenet5", 140, "tf32x3"), ("vgg", 48, "tf32x3"), ("resnet20", 48, "tf32x3"),
         ("resnet20", 40, "fp32")]


@pytest.mark.parametrize("name,n_in,prec", CASES)
def test_elimination_is_exact(M, ctx, oracle_mod, name, n_in, prec):
    w = wl.workload(name, n_in, 1)
    table = dead_heavy_table(w.model, 3)
    model = M.mure_model_load(ctx, w.model, precision=prec)
    cache = M.mure_build_prefix_cache(model, w.X)
    full = M.mure_eval_mutants(cache, table, logits=True)
    skip = M.mure_eval_mutants(cache, table, logits=True, skip_unchanged=True)
    assert np.array_equal(full["kill_bits"], skip["kill_bits"])
    assert np.array_equal(full["logits"].view(np.uint32), skip["logits"].view(np.uint32))
    assert full["scoreA"] == skip["scoreA"] and full["scoreB"] == skip["scoreB"]
    assert full["stats"]["n_near_ties"] == skip["stats"]["n_near_ties"]
    assert full["stats"]["n_rows_unchanged"] == 0
    n_skip = skip["stats"]["n_rows_unchanged"]
    van = M.mure_eval_vanilla(model, w.X, table, logits=True)
    assert np.array_equal(van["kill_bits"], skip["kill_bits"])
    # the oracle's unchanged rows (the mutated layer's output equal before its post-ops)
    ora = bits(oracle_mod.unchanged_rows(w.model, w.X, table), n_in)
    # rows of the output layer's mutants are never dropped (their suffix is the epilogue),
    # nor those whose first suffix layer stages whole consecutive rows (the window GEMM,
    # the CUDA-core small convolution)
    L = w.model.n_layers()
    eligible = [l for l in range(L - 1)
                if l + 1 == L - 1 or model.layer_kernel(l + 1)[0] not in ("tc_window", "simt_small")]
    ora_eligible = int(ora[np.isin(table.layer, eligible)].sum())
    assert n_skip >= ora_eligible > 0, (n_skip, ora_eligible)
    if name == "mlp":
        assert n_skip == ora_eligible
    # a dropped row is never killed
    assert not (bits(skip["kill_bits"], n_in) & ora).any()


def test_elimination_with_small_batches(M, ctx):
    """Many batches (input tiles and mutant chunks), each compacted on its own, give
    the same bits as one batch."""
    w = wl.workload("lenet5", 300, 1)
    table = dead_heavy_table(w.model, 5)
    model = M.mure_model_load(ctx, w.model, precision="tf32x3")
    cache = M.mure_build_prefix_cache(model, w.X)
    big = M.mure_eval_mutants(cache, table, logits=True, skip_unchanged=True)
    small = M.mure_eval_mutants(cache, table, logits=True, skip_unchanged=True, workspace_bytes=64 * 8 * 1024)
    assert small["stats"]["n_batches"] > big["stats"]["n_batches"]
    assert np.array_equal(big["kill_bits"], small["kill_bits"])
    assert np.array_equal(big["logits"].view(np.uint32), small["logits"].view(np.uint32))
    assert big["stats"]["n_rows_unchanged"] == small["stats"]["n_rows_unchanged"] > 0
