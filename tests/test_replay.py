"""Multi-step replay with the oracle alone (CPU): the host replay state and the
oracle's decisions over a whole block.

Algorithm 1 commits at least one position per step (the standard commit falls
back to the most confident row when no position passes tau, Eq. 2), so a block
of L masked positions is decoded in at most L steps, and a committed position
never returns to the mask. The positions leaving the mask in a step are the
standard commit S plus at most the one committed pivot.
"""
import numpy as np

from paper_2608_11742_gb300 import configs
from replay import ReplayState, WIN_ANCHOR, WIN_DONE, WIN_SKIP


def run_block(o, w, prm):
    st = ReplayState(w)
    start = set(st.mask_pos[0, :st.mask_cnt[0]].tolist())
    committed, winners = set(), []
    for _ in range(w.L + 1):
        if st.done():
            break
        before = set(st.mask_pos[0, :st.mask_cnt[0]].tolist())
        ref = o.step(st.logits(), st.mask_pos, st.mask_cnt, prm)
        cm, piv = ref["commit"], ref["pivots"]
        after = set(cm["mask_pos"][0, :cm["mask_cnt"][0]].tolist())
        assert after < before, "every step commits at least one position"
        gone = before - after
        assert not gone & committed
        n_s = int(piv["n_commit"][0])
        assert len(gone) == n_s + (1 if cm["commit_pos"][0] >= 0 else 0)
        assert set(piv["commit_pos"][0, :n_s].tolist()) <= gone
        if cm["commit_pos"][0] >= 0:
            assert cm["winner"][0] >= 0 and cm["commit_pos"][0] in gone
        committed |= gone
        winners.append(int(cm["winner"][0]))
        st.advance(cm["winner"], cm["mask_pos"], cm["mask_cnt"])
    assert st.done() and committed == start
    return winners


def test_oracle_replay_decodes_the_block(oracle):
    w = configs.LONG.scaled(V=512, L=40)
    winners = run_block(oracle, w, w.params(configs.EXERCISE))
    assert len(winners) <= w.L
    assert any(x >= 0 for x in winners), "a lookahead commit occurs"


def test_oracle_replay_with_the_paper_parameters(oracle):
    # tau_pivot = 0.9: at this vocabulary some rows are feasible, some steps skip
    w = configs.LONG.scaled(V=512, L=24)
    winners = run_block(oracle, w, w.params(configs.PAPER))
    assert set(winners) <= {WIN_SKIP, WIN_ANCHOR, WIN_DONE} | set(range(w.n_branch))


def test_replay_state_rules():
    w = configs.LONG.scaled(V=64, L=8, n_pivots=2)
    st = ReplayState(w)
    base_before = st.row(0, 0, 3)
    st.advance([WIN_SKIP], st.mask_pos, st.mask_cnt)
    assert (st.epoch[0] == 1).all() and (st.scale[0] == 1).all() and st.step == 1
    assert not np.array_equal(st.row(0, 0, 3), base_before), "a skip draws fresh noise"
    st.advance([WIN_ANCHOR], st.mask_pos, st.mask_cnt)
    assert (st.epoch[0] == 1).all() and (st.scale[0] == 1).all() and st.step == 2
    from paper_2608_11742_gb300 import synth
    f = synth.branch_factor(w.seed, 0, 1 + 2, 5, 2)
    st.advance([2], st.mask_pos, st.mask_cnt)
    assert st.scale[0, 5] == np.float32(f) and 0.8 <= f < 1.6
