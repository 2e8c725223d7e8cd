"""Algorithm 1 on the device: a whole response decoded step after step with no
host round trip.

The response of ``L_total`` positions is decoded in semi-autoregressive blocks
of ``B`` positions, left to right (Sec. 2 "Decoding"; Algorithm 1). One step:

1. the denoiser forward pass -- here the seeded generator, which stands in for
   the model: the base prediction and the lookahead branches of every request's
   current block (``synth.device_fill_blocks``);
2. the scoring path: row statistics of the masked rows, standard commit and
   pivots, row statistics of the lookahead rows, scores and the commit decision
   (``rps.Step``);
3. the generator's view of the decision: a committed branch becomes the next
   base, a skip draws a fresh forward pass (``synth.device_advance``);
4. ``rps_decode_advance``: the committed tokens go into the response, and a
   request whose block is decoded moves to its next block.

Every step reads its state (step index, blocks, masks) from device memory, so
it can be captured once as a CUDA graph and replayed.
"""
from __future__ import annotations

import torch

from . import rps, synth


class DecodeLoop:
    def __init__(self, n_req: int, B: int, L_total: int, V: int, prm, seed: int, mixture, device,
                 dtype=torch.bfloat16):
        self.n_req, self.B, self.L_total, self.V = n_req, B, L_total, V
        self.prm, self.seed, self.mixture = prm, seed, mixture
        self.device = torch.device(device)
        self.logits = torch.empty((n_req, 1 + prm.n_pivots * prm.tokens_per_pivot, B, V), dtype=dtype,
                                  device=self.device)
        self.step = rps.Step(n_req, B, V, prm, self.device, dtype)
        i32 = dict(dtype=torch.int32, device=self.device)
        self.tokens = torch.full((n_req, L_total), -1, **i32)
        self.block = torch.zeros(n_req, **i32)
        self.mask_pos = torch.full((n_req, B), -1, **i32)
        n0 = min(B, L_total)
        self.mask_pos[:, :n0] = torch.arange(n0, **i32)
        self.mask_cnt = torch.full((n_req,), n0, **i32)
        self.done = torch.zeros(n_req, **i32)
        self.scale = torch.ones((n_req, L_total), dtype=torch.float32, device=self.device)
        self.epoch = torch.zeros((n_req, L_total), **i32)
        self.d_step = torch.zeros(1, **i32)
        self.steps = torch.zeros(n_req, **i32)  # steps each request took
        self.graph = None

    # launches of one step: the scoring step, the generator's advance (two kernels) and the
    # decode advance (the generator's fill runs in the denoiser stub's graph)
    LAUNCHES = rps.Step.LAUNCHES + 3

    def forward_stub(self, stream=None):
        synth.device_fill_blocks(self.logits, self.seed, self.mixture, self.d_step, self.block, self.L_total,
                                 self.scale, self.epoch, stream)

    def score(self, stream=None):
        self.step.run(self.logits, self.mask_pos, self.mask_cnt, stream)

    def advance(self, stream=None):
        st = self.step
        synth.device_advance(st.commit.winner, self.B, self.L_total, self.block, self.d_step, self.scale,
                             self.epoch, self.seed, stream)
        rps.rps_decode_advance(st.piv, st.commit, self.n_req, self.B, self.L_total, self.tokens, self.block,
                               self.mask_pos, self.mask_cnt, self.done, self.steps, stream)

    def score_and_advance(self, stream=None):
        self.score(stream)
        self.advance(stream)

    def step_once(self, stream=None):
        self.forward_stub(stream)
        self.score_and_advance(stream)

    def capture(self, stream) -> None:
        """One step as a CUDA graph on ``stream`` (its state lives in device memory)."""
        with torch.cuda.stream(stream):
            self.step_once(stream)  # warm-up outside capture (loads kernels, sets attributes)
        stream.synchronize()
        self.reset()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph, stream=stream):
            self.step_once(stream)

    def reset(self) -> None:
        n0 = min(self.B, self.L_total)
        self.tokens.fill_(-1)
        self.block.zero_()
        self.mask_pos.fill_(-1)
        self.mask_pos[:, :n0] = torch.arange(n0, dtype=torch.int32, device=self.device)
        self.mask_cnt.fill_(n0)
        self.done.zero_()
        self.scale.fill_(1.0)
        self.epoch.zero_()
        self.d_step.zero_()
        self.steps.zero_()

    def run_split(self, stream, check_every: int = 8, max_steps: int | None = None, between=None, after=None):
        """Decode to the end (or for max_steps steps) with the forward stub, the
        scoring step and the state's advance captured as three graphs, timing each
        scoring replay (the five launches of ``rps.Step.run``) with CUDA events on
        ``stream``. ``between`` and ``after`` (optional) run on ``stream`` outside
        the timed region, after each stub replay and after each scoring replay (an
        L2 flush, a row count).
        Returns (steps, per-step scoring ms, total ms)."""
        with torch.cuda.stream(stream):
            self.step_once(stream)
        stream.synchronize()
        self.reset()
        g_fwd, g_score, g_adv = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_fwd, stream=stream):
            self.forward_stub(stream)
        with torch.cuda.graph(g_score, stream=stream):
            self.score(stream)
        with torch.cuda.graph(g_adv, stream=stream):
            self.advance(stream)
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev = []
        with torch.cuda.stream(stream):
            t0.record(stream)
        steps = 0
        limit = self.L_total if max_steps is None else min(max_steps, self.L_total)
        while steps < limit:
            for _ in range(min(check_every, limit - steps)):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                with torch.cuda.stream(stream):
                    g_fwd.replay()
                    if between is not None:
                        between()
                    e0.record(stream)
                    g_score.replay()
                    e1.record(stream)
                    if after is not None:
                        after()
                    g_adv.replay()
                ev.append((e0, e1))
            steps += min(check_every, limit - steps)
            stream.synchronize()
            if bool(self.done.all()):
                break
        with torch.cuda.stream(stream):
            t1.record(stream)
        stream.synchronize()
        taken = min(int(self.steps.max().item()), steps) if bool(self.done.all()) else steps
        score_ms = [a.elapsed_time(b) for a, b in ev[:taken]]
        return taken, score_ms, t0.elapsed_time(t1)

    def run(self, stream, max_steps: int | None = None, check_every: int = 16) -> int:
        """Replay the step graph until every request is done; returns the steps taken.
        Each step commits at least one position, so L_total steps always suffice."""
        if self.graph is None:
            self.capture(stream)
        limit = self.L_total if max_steps is None else max_steps
        steps = 0
        while steps < limit:
            n = min(check_every, limit - steps)
            with torch.cuda.stream(stream):
                for _ in range(n):
                    self.graph.replay()
            steps += n
            stream.synchronize()
            if bool(self.done.all()):
                break
        return int(self.steps.max().item())
