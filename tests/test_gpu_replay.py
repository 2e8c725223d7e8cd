"""Long-generation replay on the GPU: 64 decode steps in which the mask and the
logits follow each step's decisions (see replay.py), checked against the oracle
at every step.

* A reduced long workload (vocab 2,048, 64 positions) is compared element by
  element at every step; the replay follows the oracle's own decisions.
* The full long workload (512 positions, vocab 126,464, 1 + 16 branches) runs in
  the benchmark's launch configuration; each step's decisions must be exactly
  those the oracle derives from the GPU's statistics, and sampled rows match the
  oracle on host-generated logits.
"""
import numpy as np
import pytest
import torch

from gpu_harness import (MAX_EXCUSED, GpuStep, assert_close, commit_np, compare_commit, compare_scores, compare_select, piv_np,
                         scores_np, stats_np)
from oracle import default as oracle_default
from paper_2608_11742_gb300 import configs, rps, synth
from replay import ReplayState

pytestmark = pytest.mark.gpu
STEPS = 64


def test_long_replay_reduced():
    w = configs.LONG.scaled(V=2048, L=64)
    prm = w.params(configs.EXERCISE)
    o = oracle_default()
    st = ReplayState(w)
    winners = []
    for s in range(STEPS):
        if st.done():
            break
        z = st.logits()
        GpuStep(z, st.mask_pos, st.mask_cnt, prm).run_and_compare(f"replay step {s}")
        ref = o.step(z, st.mask_pos, st.mask_cnt, prm)["commit"]
        winners.append(int(ref["winner"][0]))
        st.advance(ref["winner"], ref["mask_pos"], ref["mask_cnt"])
    assert len(winners) >= 8 and any(x >= 0 for x in winners), winners


def test_long_replay_full_size():
    w = configs.LONG
    prm = w.params(configs.EXERCISE)
    o = oracle_default()
    st = ReplayState(w)
    dev = torch.device("cuda")
    logits = torch.empty((w.n_req, 1 + w.n_branch, w.L, w.V), dtype=torch.bfloat16, device=dev)
    step = rps.Step(w.n_req, w.L, w.V, prm, dev, torch.bfloat16)
    rng = np.random.default_rng(1)
    winners = []
    for s in range(STEPS):
        if st.done():
            break
        synth.device_fill(logits, w.seed, w.mixture, step=st.step, scale=torch.from_numpy(st.scale).to(dev),
                          epoch=torch.from_numpy(st.epoch).to(dev))
        mpos, mcnt = st.mask_pos.copy(), st.mask_cnt.copy()
        step.run(logits, torch.from_numpy(mpos).to(dev), torch.from_numpy(mcnt).to(dev))
        status, detail = rps.rps_poll_device_status()
        assert status == rps.RPS_OK, hex(detail)
        base, piv, br = stats_np(step.base), piv_np(step.piv), stats_np(step.branch)

        # sampled rows against the oracle on host-generated rows of this step
        k = int(rng.integers(0, int(mcnt[0])))
        ref = o.row_stats(st.row(0, 0, int(mpos[0, k]))[None], prm.k_max)
        for name in ("zmax", "lse", "H", "pmax", "mu", "htrunc"):
            assert_close(getattr(base, name)[[k]], getattr(ref, name), f"step {s} base {name}")
        assert base.argmax[k] == ref.argmax[0] and (base.topk_idx[k] == ref.topk_idx[0]).all()
        if piv["n_branch_rows"][0] > 0:
            i = int(rng.integers(0, int(piv["n_branch_rows"][0])))
            rq, rb, rp = (int(x) for x in piv["branch_rows"][0, i])
            ref = o.row_stats(st.row(rq, rb, rp)[None], 0)
            for name in ("zmax", "lse", "H", "pmax"):
                assert_close(getattr(br, name)[[i]], getattr(ref, name), f"step {s} branch {name}")

        # the decisions are the oracle's on the GPU's statistics
        piv_o = o.select_pivots(mpos, mcnt, base, prm)
        compare_select(piv, piv_o, mcnt, w.L, prm.n_pivots, prm.tokens_per_pivot, {}, f"step {s} select")
        anchor = logits[:, 0].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        sc_o = o.score_branches(piv, br, base, anchor, prm)
        sc_g = scores_np(step.scores)
        compare_scores(sc_g, sc_o, prm, f"step {s} scores")
        cm_o = o.commit(piv, sc_o, prm)
        cm = commit_np(step.commit)
        assert len(compare_commit(cm, cm_o, sc_g, sc_o, piv, prm, f"step {s} commit")) <= MAX_EXCUSED
        winners.append(int(cm["winner"][0]))
        st.advance(cm["winner"], cm["mask_pos"], cm["mask_cnt"])
    assert len(winners) == STEPS, "512 positions outlast 64 steps"
    assert int(st.mask_cnt[0]) < w.L
    assert any(x >= 0 for x in winners), winners
