"""Oracle of the LM-head contraction followed by the row statistics: the logits
of a row are its hidden state times the unembedding matrix transposed,
z = h W^T (W: one row of d weights per token), and the row statistics of Sec. 2,
Eq. 1 and Eq. 3 follow from z as for stored logits.

TEST INFRASTRUCTURE. Only the test-suite uses this module; the library never
imports it.

Inputs are bf16 bit patterns (numpy uint16). The product is taken in fp64 (a
library matmul) and rounded once to fp32, the precision of a tensor-core
accumulator, before the statistics; the statistics themselves are the
row-statistics oracle's (fp64 arithmetic on the fp32 logits).
"""
from __future__ import annotations

import numpy as np


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def lmhead_logits(hidden_bits: np.ndarray, unembed_bits: np.ndarray) -> np.ndarray:
    """[n][V] fp32 logits of hidden [n][d] and unembedding [V][d] (bf16 bits)."""
    h = bf16_to_f64(hidden_bits)
    w = bf16_to_f64(unembed_bits)
    if h.ndim != 2 or w.ndim != 2 or h.shape[1] != w.shape[1]:
        raise ValueError("hidden is [n][d] and the unembedding [V][d]")
    return (h @ w.T).astype(np.float32)


def lmhead_row_stats(o, hidden_bits: np.ndarray, unembed_bits: np.ndarray, k: int):
    """Row statistics (top-k mode for k > 0) of the rows' logits h W^T."""
    return o.row_stats(lmhead_logits(hidden_bits, unembed_bits), k)
