"""Multi-step replay of a synthetic decode (host state only, no scoring arithmetic).

Algorithm 1 runs the scoring step again and again on one block until nothing is
masked. A replay needs the logits of every step, and these depend on what
the previous step decided:

* a committed lookahead branch b becomes the next base prediction: the spike
  strength of every position is multiplied by that branch's factor f_b,i of
  the step (the generator's branch perturbation);
* "skip" (no feasible pivot, or no pivot with two candidates) means that the
  next step needs a fresh forward pass: every position draws new noise (the
  noise epoch advances);
* "anchor" (every searched pivot kept [MASK]) reuses the base;
* the mask of the next step is the mask the commit decision leaves.

The lookahead branch factors of step s are drawn with step index s, so the
branches differ from step to step even when the base does not.
"""
from __future__ import annotations

import numpy as np

from paper_2608_11742_gb300 import synth

WIN_ANCHOR, WIN_SKIP, WIN_DONE = -1, -2, -3


class ReplayState:
    def __init__(self, w):
        self.w = w
        self.scale = np.ones((w.n_req, w.L), dtype=np.float32)
        self.epoch = np.zeros((w.n_req, w.L), dtype=np.int32)
        self.mask_pos, self.mask_cnt = w.mask()
        self.step = 0

    def logits(self) -> np.ndarray:
        w = self.w
        return synth.make_logits(w.seed, w.n_req, w.n_branch, w.L, w.V, w.mixture, w.dtype, valid=w.valid_rows(),
                                 scale=self.scale, epoch=self.epoch, step=self.step)

    def row(self, q: int, branch: int, pos: int) -> np.ndarray:
        w = self.w
        return synth.row_logits(w.seed, w.V, q, branch, pos, w.mixture, w.dtype, float(self.scale[q, pos]),
                                int(self.epoch[q, pos]), self.step)

    def done(self) -> bool:
        return bool((self.mask_cnt == 0).all())

    def advance(self, winner, mask_pos, mask_cnt) -> None:
        """Apply one step's decisions (winner code per request, mask after the step)."""
        w = self.w
        for q in range(w.n_req):
            win = int(winner[q])
            if win >= 0:
                f = np.array([synth.branch_factor(w.seed, q, 1 + win, p, self.step) for p in range(w.L)],
                             dtype=np.float32)
                self.scale[q] = (self.scale[q] * f).astype(np.float32)
            elif win == WIN_SKIP:
                self.epoch[q] += 1
        cnt = np.asarray(mask_cnt, dtype=np.int32).copy()
        pos = np.full((w.n_req, w.L), -1, dtype=np.int32)
        for q in range(w.n_req):
            pos[q, :cnt[q]] = np.asarray(mask_pos)[q, :cnt[q]]
        self.mask_pos, self.mask_cnt = pos, cnt
        self.step += 1
