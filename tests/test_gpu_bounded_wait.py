"""Failure detection without a GPU fault: the tensor-core kernels' device-side waits
are bounded.  A wait limit far below the kernels' normal waits (one SM cycle) makes
them give up; the call must return TIMEOUT (the kernels stop their roles, let their
own copies and MMAs land, free their tensor memory and return), and the next call on
the same context, with the default limit back, must give the same bits as before."""
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


@pytest.mark.parametrize("name", ["lenet5", "vgg"])
def test_expired_waits_return_timeout_and_the_context_recovers(M, name):
    ctx = M.mure_create(0)
    w = wl.workload(name, 256, 24)
    model = M.mure_model_load(ctx, w.model, precision="tf32x3")
    cache = M.mure_build_prefix_cache(model, w.X)
    ref = M.mure_eval_mutants(cache, w.table, logits=True)
    M.mure_set_wait_limit(ctx, 1)
    with pytest.raises(M.MureError) as ei:
        M.mure_eval_mutants(cache, w.table)
    assert ei.value.status == 5, ei.value
    with pytest.raises(M.MureError) as ei:
        M.mure_eval_vanilla(model, w.X, w.table)
    assert ei.value.status == 5, ei.value
    M.mure_set_wait_limit(ctx, 0)
    again = M.mure_eval_mutants(cache, w.table, logits=True)
    assert np.array_equal(again["kill_bits"], ref["kill_bits"])
    assert np.array_equal(again["logits"].view(np.uint32), ref["logits"].view(np.uint32))
    van = M.mure_eval_vanilla(model, w.X, w.table, logits=True)
    assert np.array_equal(van["logits"].view(np.uint32), ref["logits"].view(np.uint32))


def test_wait_limit_argument_checks(M):
    ctx = M.mure_create(0)
    with pytest.raises(M.MureError) as ei:
        M.mure_set_wait_limit(ctx, -1)
    assert ei.value.status == 1
    M.mure_set_wait_limit(ctx, 0)
