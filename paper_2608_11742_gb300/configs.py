"""Synthetic workloads shaped like the paper's decoding steps.

The paper decodes LLaDA-8B-Instruct (vocab 126,464) and Dream-v0-7B (vocab
151,936) with generation length L = 256 and semi-autoregressive block B = 32
(Sec. 4 "Setup"), on GSM8K / MATH500 / HumanEval / MBPP. No model, dataset or
weight is used here: each workload is a seeded logit tensor of the same shape
(``synth.py``), standing in for one denoising step's base prediction plus its
packed lookahead branches (Sec. 3.1, Fig. 2).

Hyper-parameters follow Sec. 4 "Implementation details" and Appendix C:
k_max = 10, r = 0.1, tau_pivot = 0.9 (LLaDA) / 0.95 (Dream), lambda in
[0.1, 0.5], confidence threshold tau = 0.9.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional, Tuple

import numpy as np

from . import synth


@dataclass(frozen=True)
class Params:
    """RPS hyper-parameters (the ``rps_params`` struct of the C ABI)."""
    k_max: int = 10            # |T_i|, Eq. 3
    r: float = 0.1             # reachability ratio of the candidate set, Sec. 3.1
    tau_pivot: float = 0.9     # probability-mass constraint, Eq. 3
    tau: float = 0.9           # confidence threshold, Eq. 2 (third rule)
    lam: float = 0.1           # plausibility weight lambda, Eq. 4
    n_pivots: int = 4          # pivot slots P per step
    tokens_per_pivot: int = 2  # candidate tokens K per pivot
    pivot_rule: int = 0        # 0: truncated entropy under the mass constraint (Eq. 3);
                               # 1: max confidence, 2: max entropy (ablation strategies, Sec. 4.3)
    commit_rule: int = 0       # 0: confidence threshold tau (Eq. 2, third rule, with the fallback);
                               # 1: top-k confidence, 2: top-k lowest entropy (Eq. 2, first two rules)
    commit_k: int = 0          # k of the top-k commit rules

    @property
    def n_branch(self) -> int:
        return self.n_pivots * self.tokens_per_pivot


# Paper defaults (LLaDA) with the four-pivot, top-2 layout of the workloads.
PAPER = Params()
# Setting under which every stage of the step runs on the synthetic logits. With
# the paper's tau_pivot = 0.9 no synthetic row at vocab 126,464 reaches the mass
# constraint and every step takes the skip path of Algorithm 1. With every row
# feasible but tau = 0.9, the truncated-entropy argmax lands on the one-spike
# rows, whose second token is ~8 nats down (a single candidate: skip again).
# tau = 0.05 commits those rows in the standard commit, so the pivots come from
# the flatter rows, which have several candidates, and the lookahead branches are
# scored every step.
EXERCISE = Params(tau=0.05, tau_pivot=0.0)


@dataclass(frozen=True)
class Workload:
    name: str
    n_req: int
    L: int                     # positions per request in the logit tensor
    V: int
    dtype: str                 # "bf16" or "f32"
    n_pivots: int
    tokens_per_pivot: int
    mixture: Tuple[float, float, float]   # (low, mid, high) regime probabilities
    masked_frac: float = 1.0   # fraction of the L positions that are masked
    ragged: Optional[Tuple[int, int]] = None  # per-request masked count range
    pad_nan: bool = False      # unmasked rows are NaN (must never be read)
    seed: int = 0
    steps: int = 1             # decode steps replayed (multi-step workloads)

    @property
    def n_branch(self) -> int:
        return self.n_pivots * self.tokens_per_pivot

    @property
    def elem_bytes(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    def params(self, base: Params = EXERCISE) -> Params:
        return Params(base.k_max, base.r, base.tau_pivot, base.tau, base.lam,
                      self.n_pivots, self.tokens_per_pivot, base.pivot_rule, base.commit_rule, base.commit_k)

    def mask_counts(self) -> np.ndarray:
        if self.ragged is not None:
            lo, hi = self.ragged
            return np.array([synth.ragged_count(self.seed, q, lo, hi) for q in range(self.n_req)],
                            dtype=np.int32)
        c = int(np.floor(self.masked_frac * self.L + 0.5))  # round half up
        return np.full(self.n_req, c, dtype=np.int32)

    def mask(self):
        """(mask_pos [n_req][L] int32 padded with -1, mask_cnt [n_req] int32)."""
        cnt = self.mask_counts()
        pos = np.full((self.n_req, self.L), -1, dtype=np.int32)
        for q in range(self.n_req):
            if cnt[q] == self.L:
                pos[q, :] = np.arange(self.L, dtype=np.int32)
            else:
                sel = synth.masked_positions(self.seed, q, self.L, int(cnt[q]))
                pos[q, :len(sel)] = sel
        return pos, cnt

    def valid_rows(self) -> Optional[np.ndarray]:
        """[n_req][L] uint8: 1 where the row holds logits, 0 for NaN padding."""
        if not self.pad_nan:
            return None
        pos, cnt = self.mask()
        valid = np.zeros((self.n_req, self.L), dtype=np.uint8)
        for q in range(self.n_req):
            valid[q, pos[q, :cnt[q]]] = 1
        return valid

    def tensor_bytes(self) -> int:
        return self.n_req * (1 + self.n_branch) * self.L * self.V * self.elem_bytes

    def thresholds(self):
        return synth.regime_thresholds(self.mixture)

    def scaled(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


MIX_A = (0.4, 0.3, 0.3)

# 1 sequence, 32 masked positions, vocab 4,096, fp32, 1 base + 8 branches.
TINY = Workload("tiny", 1, 32, 4096, "f32", 4, 2, MIX_A)
# One generation step: 256 masked positions, vocab 126,464 (LLaDA), bf16.
STEP = Workload("step", 1, 256, 126464, "bf16", 4, 2, MIX_A)
STEP_50 = STEP.scaled(name="step-50", masked_frac=0.5)
STEP_10 = STEP.scaled(name="step-10", masked_frac=0.1)
# Long generation: 512 positions, 1 base + 16 branches, 64-step replay.
LONG = Workload("long", 1, 512, 126464, "bf16", 8, 2, (0.3, 0.4, 0.3), steps=64)
# Batched serving: 8 requests x 256 positions, vocab 151,936 (Dream), ragged masks.
SERVE = Workload("serve", 8, 256, 151936, "bf16", 8, 2, MIX_A, ragged=(16, 256), pad_nan=True)
# KV-cache block mode: 64 requests, only the current 32-position block masked.
BLOCK = Workload("block", 64, 32, 126464, "bf16", 4, 2, (0.5, 0.3, 0.2))

ALL = {w.name: w for w in (TINY, STEP, STEP_50, STEP_10, LONG, SERVE, BLOCK)}
