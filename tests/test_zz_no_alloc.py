"""The allocation-free expansion entry point (for callers that cannot allocate device
memory, e.g. when another allocator owns the device's memory) against the ordinary
one.  The file name makes pytest collect it after every other test file."""
import numpy as np
import pytest

from paper_2607_18582_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def M():
    from paper_2607_18582_gb300 import build
    build.build()
    from paper_2607_18582_gb300 import mure
    return mure


def _table(model, seed):
    rows = []
    rng = np.random.default_rng(seed)
    for l in range(model.n_layers()):
        N = model.layer_width(l)
        ids = rng.choice(N, size=min(3, N), replace=False).tolist()
        rows.append((l, "GF", ids[:2], 0.1, 100 + seed + l))
        rows.append((l, "WS", ids[:1], 0.0, 200 + seed + l))
        rows.append((l, "NEB", ids[:1], 0.0, 0))
        rows.append((l, "NS", ids[:2], 0.0, 0))
    return wl.table_from_rows(rows)


def test_noalloc_expansion_matches_allocating_entry_point(M):
    import torch
    ctx = M.mure_create(0)
    for name, seed in (("lenet5", 1), ("vgg", 2)):
        model = M.mure_model_load(ctx, wl.MODELS[name]())
        out = torch.full((600_000,), float("nan"), dtype=torch.float32, device="cuda")
        for call in range(2):                      # two calls in a row, different tables
            table = _table(model.src, seed + 10 * call)
            ref_vals, ref_offs = M.mure_expand_patches(model, table)
            offs = M.mure_expand_patches_noalloc(model, table, out)
            torch.cuda.synchronize()
            got = out[:ref_vals.size].cpu().numpy()
            assert np.array_equal(offs, ref_offs)
            # the same kernel on the same inputs: identical bits
            assert np.array_equal(got.view(np.uint32), ref_vals.view(np.uint32))


def test_noalloc_rejects_tables_beyond_its_scratch(M):
    import torch
    ctx = M.mure_create(0)
    model = M.mure_model_load(ctx, wl.vgg())
    # WS on the 4096-input dense layer needs 16 KiB of permutation scratch per neuron;
    # 600 of them exceed the 8 MiB array
    rows = [(6, "WS", list(range((q % 85) * 6, (q % 85) * 6 + 6)), 0.0, q) for q in range(100)]
    table = wl.table_from_rows(rows)
    out = torch.empty(600 * 4096, dtype=torch.float32, device="cuda")
    with pytest.raises(M.MureError) as ei:
        M.mure_expand_patches_noalloc(model, table, out)
    assert ei.value.status == 1 and "scratch" in str(ei.value)


def test_noalloc_short_output_and_tables_without_patches(M):
    """An output buffer one value short is refused with the needed count (nothing is
    launched); a table whose operators have no patch (NEB, NS, NAI, IDENTITY) returns
    offsets of -1 without touching the device; a tagged table is refused as the
    allocating entry point refuses it."""
    import torch
    ctx = M.mure_create(0)
    model = M.mure_model_load(ctx, wl.lenet5())
    table = _table(model.src, 3)
    ref_vals, _ = M.mure_expand_patches(model, table)
    out = torch.zeros(ref_vals.size - 1, dtype=torch.float32, device="cuda")
    with pytest.raises(M.MureError) as ei:
        M.mure_expand_patches_noalloc(model, table, out)
    assert ei.value.status == 1 and "needed" in str(ei.value)
    rows = [(l, op, [0, 1] if op == "NS" else [0], 0.0, 0)
            for l in range(model.src.n_layers()) for op in ("NEB", "NS", "NAI", "IDENTITY")]
    rows = [(l, op, [] if op == "IDENTITY" else ids, p, s) for l, op, ids, p, s in rows]
    offs = M.mure_expand_patches_noalloc(model, wl.table_from_rows(rows), out)
    assert offs.tolist() == [-1] * len(rows)
    tagged = wl.workload("lenet5_modelwide", 1, 4).table
    with pytest.raises(M.MureError) as ei:
        M.mure_expand_patches_noalloc(model, tagged, out)
    assert ei.value.status == 2
