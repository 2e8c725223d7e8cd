"""Oracle of the branch-isolating attention of the packed lookahead forward pass
(Sec. 3.1 "Lookahead scoring"; Fig. 2, right).

TEST INFRASTRUCTURE. Only the test-suite uses this module; the library never
imports it.

The lookahead forward pass scores every candidate branch in one pass over a
packed sequence: the shared context, then the generation region once per
branch. Branch 0 is the anchor (the normal sequence's own generation region),
branches 1..NB-1 the candidate assignments. Each branch is isolated from the
others, so that it sees what the model would see if only its own token were
assigned at the pivot:

* a query of branch j attends to the context and to branch j;
* a query of the context attends to the normal sequence: the context and
  branch 0.

Per (batch, head): out_i = sum_{k in A(i)} softmax_k(scale q_i . k_k) v_k over the
allowed keys A(i), in fp64 from the exact bf16 inputs (a library matmul for the
products).

Layout (numpy arrays of bf16 bit patterns, uint16): q, k, v are
[batch][heads][tokens][head_dim], tokens = n_context + n_branch * branch_len in
packed order. Returns fp64 [batch][heads][tokens][head_dim].
"""
from __future__ import annotations

import numpy as np


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def segments(n_context: int, n_branch: int, branch_len: int):
    """(start, length) of the context and of each branch in the packed order."""
    segs = [(0, n_context)]
    for j in range(n_branch):
        segs.append((n_context + j * branch_len, branch_len))
    return segs


def allowed_keys(n_context: int, n_branch: int, branch_len: int, segment: int) -> np.ndarray:
    """Key token indices a query of `segment` attends to (0 = context, 1 + j = branch j)."""
    ctx = np.arange(n_context)
    j = 0 if segment == 0 else segment - 1
    start = n_context + j * branch_len
    return np.concatenate([ctx, np.arange(start, start + branch_len)])


def softmax_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float) -> np.ndarray:
    """Plain attention of queries q [n][D] over keys k [m][D] and values v [m][D] (fp64)."""
    s = scale * (q @ k.T)
    s -= s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p /= p.sum(axis=1, keepdims=True)
    return p @ v


def packed_attention(q, k, v, n_context: int, n_branch: int, branch_len: int, scale: float) -> np.ndarray:
    """Branch-isolating attention of the packed sequence (see the module header)."""
    qf, kf, vf = bf16_to_f64(q), bf16_to_f64(k), bf16_to_f64(v)
    n_b, n_h, n_tok, _ = qf.shape
    if n_tok != n_context + n_branch * branch_len:
        raise ValueError("tokens must be n_context + n_branch * branch_len")
    out = np.zeros_like(qf)
    for b in range(n_b):
        for h in range(n_h):
            for seg, (start, length) in enumerate(segments(n_context, n_branch, branch_len)):
                if length == 0:
                    continue
                keys = allowed_keys(n_context, n_branch, branch_len, seg)
                rows = slice(start, start + length)
                out[b, h, rows] = softmax_attention(qf[b, h, rows], kf[b, h, keys], vf[b, h, keys], scale)
    return out
