"""Brute-force NumPy twins used to pin the C oracle (test infrastructure).

These materialise everything the oracle streams: the whole joint-attention
matrix with a library softmax (Eq. 5), a full stable sort for TopK (Eq. 9).
They are independent re-statements, not copies of the C loops, and are
only practical on small inputs.
"""
from __future__ import annotations

import numpy as np


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def as_f64(a: np.ndarray) -> np.ndarray:
    return bf16_to_f64(a) if a.dtype == np.uint16 else np.asarray(a, np.float64)


def spatial_full_softmax(q_img, k_all, L, scale, text_mask=None):
    """A [B,M] and mass [B,H,M]: softmax(Q K^T * scale) over all keys
    (scipy's softmax), text columns summed, mean over heads (Eq. 3).  The
    text columns are the first L, or those where text_mask [B,Nk] is set."""
    from scipy.special import softmax
    q = as_f64(q_img)
    k = as_f64(k_all)
    P = np.einsum("bhmd,bhnd->bhmn", q, k) * scale
    alpha = softmax(P, axis=-1)
    if text_mask is None:
        mass = alpha[..., :L].sum(-1)
    else:
        w = (np.asarray(text_mask) != 0).astype(np.float64)[:, None, None, :]
        mass = (alpha * w).sum(-1)
    return mass.mean(axis=1), mass


def topk_full_sort(S, k):
    """Selected index sets by a full stable sort on (-S, index); NaN last."""
    S = np.asarray(S, np.float64)
    out = []
    for row in S:
        key = np.where(np.isnan(row), np.inf, -row)
        order = np.lexsort((np.arange(len(row)), key))
        out.append(np.sort(order[:k]))
    return np.stack(out) if out else np.zeros((0, k), np.int64)
