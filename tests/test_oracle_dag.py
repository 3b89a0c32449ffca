"""Pins of the oracle on a graph whose skip branch holds a weighted layer (ResNet-10 with
1x1 projection shortcuts, Table 1): the forward against a PyTorch fp64 composition, the
memoization boundary from Algorithm 2's dependence graph, and Theorem 1 with mutants of
every layer (the projections included) and model-wide ones."""
import numpy as np
import torch
import torch.nn.functional as F

from paper_2607_18582_gb300 import workloads as wl


def _torch_forward(model, X):
    outs = {-1: torch.from_numpy(X).double().permute(0, 3, 1, 2)}
    for v, n in enumerate(model.nodes):
        a = outs[n.inputs[0]]
        if n.kind == "conv":
            y = F.conv2d(a, torch.from_numpy(n.W).double().permute(0, 3, 1, 2), torch.from_numpy(n.b).double(),
                         stride=n.stride, padding=n.pad)
        elif n.kind == "dense":
            y = F.linear(a.permute(0, 2, 3, 1).reshape(a.shape[0], -1), torch.from_numpy(n.W).double(),
                         torch.from_numpy(n.b).double())[:, :, None, None]
        elif n.kind == "add":
            y = a + outs[n.inputs[1]]
        elif n.kind == "gap":
            y = a.mean(dim=(2, 3), keepdim=True)
        else:
            raise AssertionError(n.kind)
        if n.act == "relu":
            y = y.clamp_min(0)
        outs[v] = y.float().double()
    return outs[len(model.nodes) - 1].reshape(X.shape[0], -1).float().numpy()


def test_resnet10_forward_matches_torch(oracle_mod):
    m = wl.resnet10()
    X = wl.inputs(m, 3)
    lg, _ = oracle_mod.forward(m, X)
    ref = _torch_forward(m, X)
    assert np.all(np.abs(lg - ref) <= 1e-5 * np.abs(ref).max(axis=1, keepdims=True))


def test_projection_boundary(oracle_mod):
    """A mutant of a block's first convolution needs the block input (read by the
    projection after it) in K; a mutant of the projection needs the main branch's
    output, computed before it in node order."""
    m = wl.resnet10()
    kinds = [m.nodes[v].kind for v in m.layers()]
    proj = [l for l, v in enumerate(m.layers()) if m.nodes[v].kind == "conv" and m.nodes[v].kh == 1]
    assert len(proj) == 3 and kinds.count("conv") == 12
    p = proj[0]
    v_proj = m.layers()[p]
    block_in = m.nodes[v_proj].inputs[0]
    v_a = m.layers()[p - 2]                     # the block's first convolution
    assert oracle_mod.boundary(m, p - 2) == [block_in]
    main = m.layers()[p - 1]                    # the block's second convolution
    assert oracle_mod.boundary(m, p) == sorted([main, block_in])
    assert m.nodes[v_a].inputs[0] == block_in


def test_resnet10_theorem1(oracle_mod):
    m = wl.resnet10()
    X = wl.inputs(m, 4)
    subs = [wl.mutants(m, 5, seed=40 + l, ratios=(0.05,), layers=[l],
                      ops=tuple(wl.OPS[(l + i) % 6] for i in range(5))) for l in range(m.n_layers())]
    subs.append(wl.modelwide_mutants(m, 6, seed=41, ratio=0.005))
    table = wl.concat(subs)
    r0 = oracle_mod.vanilla(m, X, table)
    r1 = oracle_mod.memo(m, X, table)
    assert np.array_equal(r0["logits"], r1["logits"])
    assert np.array_equal(r0["kill_bits"], r1["kill_bits"])
