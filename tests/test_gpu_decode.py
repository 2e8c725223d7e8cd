"""Algorithm 1 decoded on the device (paper_2608_11742_gb300.decode): every step of
a whole response checked against the oracle and against a host mirror of the
decode state.

At each step the host regenerates the current blocks' logits from its mirror
of the state (step index, blocks, spike scale, noise epoch), and checks:
* the device generator wrote the same bits;
* the GPU's row statistics match the oracle on those logits;
* the GPU's decisions are the oracle's on the GPU's own statistics;
* after the step, the device state (response tokens, blocks, masks, done
  flags, generator state) equals the mirror advanced by the GPU's decisions.
The captured step graph, replayed to the end, must give the same response.
"""
import numpy as np
import pytest
import torch

from gpu_harness import (MAX_EXCUSED, assert_close, commit_np, compare_commit, compare_scores, compare_select, piv_np, scores_np,
                         stats_np)
from oracle import default as oracle_default
from paper_2608_11742_gb300 import configs, synth
from paper_2608_11742_gb300.decode import DecodeLoop

pytestmark = pytest.mark.gpu

N_REQ, B, L_TOTAL, V = 2, 16, 40, 1024  # two full blocks and a partial one
MIX = (0.4, 0.3, 0.3)
SEED = 3


class Mirror:
    def __init__(self, prm):
        self.prm = prm
        self.nb = prm.n_pivots * prm.tokens_per_pivot
        self.tokens = np.full((N_REQ, L_TOTAL), -1, np.int32)
        self.block = np.zeros(N_REQ, np.int32)
        self.mask_pos = np.full((N_REQ, B), -1, np.int32)
        self.mask_pos[:, :B] = np.arange(B)
        self.mask_cnt = np.full(N_REQ, B, np.int32)
        self.done = np.zeros(N_REQ, np.int32)
        self.scale = np.ones((N_REQ, L_TOTAL), np.float32)
        self.epoch = np.zeros((N_REQ, L_TOTAL), np.int32)
        self.step = 0

    def logits(self):
        out = np.full((N_REQ, 1 + self.nb, B, V), 0x7FC0, np.uint16)
        for q in range(N_REQ):
            for p in range(B):
                pos = int(self.block[q]) * B + p
                if pos >= L_TOTAL:
                    continue
                for b in range(1 + self.nb):
                    out[q, b, p] = synth.row_logits(SEED, V, q, b, pos, MIX, "bf16", float(self.scale[q, pos]),
                                                    int(self.epoch[q, pos]), self.step)
        return out

    def advance(self, piv, cm):
        for q in range(N_REQ):
            if self.done[q]:
                continue
            first = int(self.block[q]) * B
            w = int(cm["winner"][q])
            for p in range(min(B, L_TOTAL - first)):
                pos = first + p
                if w >= 0:
                    f = synth.branch_factor(SEED, q, 1 + w, pos, self.step)
                    self.scale[q, pos] = np.float32(self.scale[q, pos] * f)
                elif w == -2:
                    self.epoch[q, pos] += 1
            for i in range(int(piv["n_commit"][q])):
                self.tokens[q, first + piv["commit_pos"][q, i]] = piv["commit_tok"][q, i]
            if cm["commit_pos"][q] >= 0:
                self.tokens[q, first + cm["commit_pos"][q]] = cm["commit_tok"][q]
            n = int(cm["mask_cnt"][q])
            if n > 0:
                self.mask_pos[q, :n] = cm["mask_pos"][q, :n]
                self.mask_cnt[q] = n
            elif first + B < L_TOTAL:
                self.block[q] += 1
                nn = min(B, L_TOTAL - first - B)
                self.mask_pos[q, :nn] = np.arange(nn)
                self.mask_cnt[q] = nn
            else:
                self.done[q] = 1
                self.mask_cnt[q] = 0
        self.step += 1


def _run_checked(prm):
    o = oracle_default()
    loop = DecodeLoop(N_REQ, B, L_TOTAL, V, prm, SEED, MIX, "cuda")
    m = Mirror(prm)
    stream = torch.cuda.current_stream()
    winners = []
    for s in range(L_TOTAL + 1):
        if m.done.all():
            break
        z = m.logits()
        loop.forward_stub(stream)
        zg = loop.logits.view(torch.int16).cpu().numpy().view(np.uint16)
        for q in range(N_REQ):
            n = int(m.mask_cnt[q])
            rows = m.mask_pos[q, :n]
            assert np.array_equal(zg[q][:, rows], z[q][:, rows]), f"step {s}: generator rows of request {q}"
        loop.score_and_advance(stream)
        torch.cuda.synchronize()
        st = loop.step
        base, piv, br = stats_np(st.base), piv_np(st.piv), stats_np(st.branch)
        ref = o.base_stats(z, m.mask_pos, m.mask_cnt, prm.k_max)
        slots = [q * B + k for q in range(N_REQ) for k in range(int(m.mask_cnt[q]))]
        for name in ("zmax", "lse", "H", "pmax", "mu", "htrunc"):
            assert_close(getattr(base, name)[slots], getattr(ref, name)[slots], f"step {s} base {name}")
        assert (base.argmax[slots] == ref.argmax[slots]).all()
        piv_o = o.select_pivots(m.mask_pos, m.mask_cnt, base, prm)
        compare_select(piv, piv_o, m.mask_cnt, B, prm.n_pivots, prm.tokens_per_pivot, {}, f"step {s} select")
        sc_o = o.score_branches(piv, br, base, z[:, 0], prm)
        sc_g = scores_np(st.scores)
        compare_scores(sc_g, sc_o, prm, f"step {s} scores")
        cm = commit_np(st.commit)
        assert len(compare_commit(cm, o.commit(piv, sc_o, prm), sc_g, sc_o, piv, prm, f"step {s} commit")) <= MAX_EXCUSED
        winners += [int(w) for q, w in enumerate(cm["winner"]) if not m.done[q]]
        m.advance(piv, cm)
        assert np.array_equal(loop.tokens.cpu().numpy(), m.tokens), f"step {s}: response tokens"
        assert np.array_equal(loop.block.cpu().numpy(), m.block) and np.array_equal(loop.done.cpu().numpy(), m.done)
        gc = loop.mask_cnt.cpu().numpy()
        assert np.array_equal(gc, m.mask_cnt)
        for q in range(N_REQ):
            assert np.array_equal(loop.mask_pos.cpu().numpy()[q, :gc[q]], m.mask_pos[q, :gc[q]])
        assert np.array_equal(loop.scale.cpu().numpy(), m.scale) and np.array_equal(loop.epoch.cpu().numpy(), m.epoch)
        assert int(loop.d_step.item()) == m.step
    assert m.done.all() and (m.tokens >= 0).all(), "every position of the response is decoded"
    assert int(loop.steps.max().item()) <= L_TOTAL
    return m, winners


@pytest.mark.parametrize("prm", [configs.EXERCISE, configs.Params(tau=0.5, tau_pivot=0.003, lam=0.3)],
                         ids=["exercise", "mid"])
def test_decode_loop_every_step(prm):
    m, winners = _run_checked(prm)
    assert any(w >= 0 for w in winners), winners


def test_decode_graph_replays_the_same_response():
    prm = configs.EXERCISE
    m, _ = _run_checked(prm)
    loop = DecodeLoop(N_REQ, B, L_TOTAL, V, prm, SEED, MIX, "cuda")
    stream = torch.cuda.Stream()
    steps = loop.run(stream, check_every=4)
    assert bool(loop.done.all())
    assert np.array_equal(loop.tokens.cpu().numpy(), m.tokens)
    assert steps == int(loop.steps.max().item()) and steps <= L_TOTAL
