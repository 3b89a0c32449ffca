"""Comparison rules between the CUDA path and the oracle.

Logits (fp32 path): |gpu - oracle| <= 1e-4 * max_c |oracle logit| for every row.
Kill bits: identical, except entries that are near ties in the oracle (top-2 logit
margin < 1e-4 |max logit| in the original's or the mutant's logits): those may differ
and are counted.
"""
import numpy as np

REL = 1e-4


def bits(kill_bits, n_in):
    """[n_mut][ceil(n_in/64)] uint64 -> bool [n_mut][n_in]."""
    kb = np.asarray(kill_bits).astype(np.uint64)
    if kb.size == 0:
        return np.zeros((kb.shape[0], n_in), bool)
    by = kb.view(np.uint8).reshape(kb.shape[0], -1)
    return np.unpackbits(by, axis=1, bitorder="little")[:, :n_in].astype(bool)


def margin_tie(lg):
    """Near-tie mask of logit vectors [..., C]."""
    s = np.sort(lg.astype(np.float64), axis=-1)
    top, second = s[..., -1], s[..., -2]
    return (top - second) < REL * np.abs(top)


def logits_close(gpu, ora):
    scale = np.abs(ora.astype(np.float64)).max(axis=-1, keepdims=True)
    err = np.abs(gpu.astype(np.float64) - ora)
    return bool(np.all(err <= REL * np.maximum(scale, 1e-30))), float((err / np.maximum(scale, 1e-30)).max())


def compare_kills(gpu_bits, ora_bits, orig_logits, mut_logits, n_in):
    """(number of mismatches outside near ties, number of near-tie entries)."""
    g = bits(gpu_bits, n_in)
    o = bits(ora_bits, n_in)
    ties = margin_tie(mut_logits) | margin_tie(orig_logits)[None, :]
    bad = (g != o) & ~ties
    return int(bad.sum()), int(ties.sum())
