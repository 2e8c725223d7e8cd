"""GPU-vs-oracle comparison helpers for the ``-m gpu`` parity tests.

Tolerances (from the target statement of the scoring path): entropies,
confidences, masses and scores within 1e-3 nats absolute plus 1e-4 relative;
argmax, top-k indices, pivots, candidates and commit decisions bit-exact,
except where the oracle's deciding quantity lies within BAND of its threshold
(or of its competitor), where either outcome is accepted.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import default as oracle_default
from oracle.oracle import RowStats
from paper_2608_11742_gb300 import rps, synth

ATOL = 1e-3
RTOL = 1e-4
BAND = 1e-4
# near-threshold differences a single step may excuse (each one is printed)
MAX_EXCUSED = 1


def to_device(logits_np: np.ndarray, device="cuda") -> torch.Tensor:
    if logits_np.dtype == np.uint16:
        return torch.from_numpy(logits_np.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(logits_np).to(device)


def padded_tensor(logits_np: np.ndarray, device="cuda") -> torch.Tensor:
    """Device copy whose rows start 16-byte aligned even when V is not a multiple of the unit."""
    V = logits_np.shape[-1]
    unit = 8 if logits_np.dtype == np.uint16 else 4
    Vp = (V + unit - 1) // unit * unit
    if Vp == V:
        return to_device(np.ascontiguousarray(logits_np), device)
    pad = np.zeros(logits_np.shape[:-1] + (Vp,), dtype=logits_np.dtype)
    pad[..., :V] = logits_np
    return to_device(pad, device)[..., :V]


def stats_np(buf: rps.RowStatsBuf) -> RowStats:
    g = lambda t: None if t is None else t.detach().cpu().numpy().astype(np.float64)
    gi = lambda t: None if t is None else t.detach().cpu().numpy()
    return RowStats(g(buf.zmax), g(buf.lse), g(buf.H), g(buf.pmax), g(buf.mu), g(buf.htrunc), gi(buf.argmax),
                    gi(buf.topk_idx), g(buf.topk_logit))


def assert_close(gpu, ref, what, atol=ATOL, rtol=RTOL):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    bad = ~(np.abs(gpu - ref) <= atol + rtol * np.abs(ref))
    bad &= ~(np.isnan(gpu) & np.isnan(ref))
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{what}: {bad.sum()} entries out of tolerance, e.g. {idx.tolist()} "
                             f"gpu={gpu[bad][:5]} oracle={ref[bad][:5]}")


def compare_stats(g: RowStats, o: RowStats, slots, k: int, what: str):
    slots = np.asarray(slots, dtype=np.int64)
    for name in ("zmax", "lse", "H", "pmax"):
        assert_close(getattr(g, name)[slots], getattr(o, name)[slots], f"{what} {name}")
    assert (g.argmax[slots] == o.argmax[slots]).all(), f"{what} argmax"
    if k:
        assert_close(g.mu[slots], o.mu[slots], f"{what} mu")
        assert_close(g.htrunc[slots], o.htrunc[slots], f"{what} htrunc")
        assert (g.topk_idx[slots, :k] == o.topk_idx[slots, :k]).all(), f"{what} top-k indices"
        assert (g.topk_logit[slots, :k] == o.topk_logit[slots, :k]).all(), f"{what} top-k logits"


def piv_np(buf: rps.PivotsBuf) -> dict:
    return {f: getattr(buf, f).detach().cpu().numpy() for f in rps._PIVOT_FIELDS}


def _top_gap(values, i):
    """Gap between the i-th and (i + 1)-th largest finite values (inf when there is no such pair)."""
    v = np.sort(np.asarray(values, np.float64)[~np.isnan(values)])[::-1]
    return v[i] - v[i + 1] if len(v) > i + 1 else np.inf


def near_threshold_requests(o: RowStats, piv_o: dict, mask_cnt, L, prm) -> dict:
    """Requests whose selection hinges on an oracle quantity within BAND of its threshold.

    Only the comparison that decides the outcome counts, each with its reason:
    - threshold commit rule: some P^max within BAND of tau (that row's
      membership of S), or, only when no row reaches tau so that the fallback
      of Eq. 2 decides, the two largest P^max within BAND of each other;
    - top-k commit rules: the commit_k-th and (commit_k + 1)-th values (the
      boundary of the set; the order inside S does not matter);
    - pivots: mu within BAND of tau_pivot for a row of M', or two adjacent
      values among the P + 1 best keys (the slot order of the pivots matters).
    """
    commit_rule = getattr(prm, "commit_rule", 0)
    pivot_rule = getattr(prm, "pivot_rule", 0)
    out = {}
    tau, tau_p = np.float32(prm.tau), np.float32(prm.tau_pivot)
    for q in range(len(mask_cnt)):
        s = slice(q * L, q * L + int(mask_cnt[q]))
        pm, H = o.pmax[s], o.H[s]
        if commit_rule == 0:
            if np.any(np.abs(pm - tau) < BAND):
                out[q] = "P^max within the band of tau"
                continue
            if not np.any(pm >= tau) and _top_gap(pm, 0) < BAND:
                out[q] = "fallback commit: the two largest P^max tie"
                continue
        elif _top_gap(pm if commit_rule == 1 else -H, prm.commit_k - 1) < BAND:
            out[q] = "top-k commit: tie at the commit_k boundary"
            continue
        rem = piv_o["rem_k"][q, :piv_o["rem_cnt"][q]]
        if pivot_rule == 0:
            mu = np.array([o.mu[q * L + k] for k in rem])
            if np.any(np.abs(mu - tau_p) < BAND):
                out[q] = "mu within the band of tau_pivot"
                continue
            vals = [o.htrunc[q * L + k] for k in rem if o.mu[q * L + k] >= tau_p]
        else:
            src = o.pmax if pivot_rule == 1 else o.H
            vals = [src[q * L + k] for k in rem]
        if any(_top_gap(np.array(vals, np.float64), i) < BAND for i in range(prm.n_pivots)):
            out[q] = "pivot keys tie among the P + 1 best"
    return out


SELECT_KEYS = ("n_commit", "rem_cnt", "state")


def compare_select(g: dict, o: dict, mask_cnt, L, P, K, exempt: dict, what: str):
    """Every integer output of pivot selection, per request. Returns the
    differing requests that `exempt` excused, as (request, reason)."""
    n_req = len(mask_cnt)
    diff = []
    for q in range(n_req):
        same = all(g[k][q] == o[k][q] for k in SELECT_KEYS)
        if same:
            nc, nr = int(o["n_commit"][q]), int(o["rem_cnt"][q])
            same &= (g["commit_pos"][q, :nc] == o["commit_pos"][q, :nc]).all()
            same &= (g["commit_tok"][q, :nc] == o["commit_tok"][q, :nc]).all()
            same &= (g["rem_pos"][q, :nr] == o["rem_pos"][q, :nr]).all()
            same &= (g["rem_k"][q, :nr] == o["rem_k"][q, :nr]).all()
        if same and o["state"][q] in (0, 3):
            same &= (g["pivot_pos"][q] == o["pivot_pos"][q]).all() and (g["n_cand"][q] == o["n_cand"][q]).all()
            same &= (g["cand_tok"][q] == o["cand_tok"][q]).all()
        if same and o["state"][q] == 0:
            same &= (g["branch_valid"][q] == o["branch_valid"][q]).all()
            same &= (g["branch_off"][q] == o["branch_off"][q]).all()
            same &= (g["branch_cnt"][q] == o["branch_cnt"][q]).all()
            n = int(o["n_branch_rows"][q])
            same &= g["n_branch_rows"][q] == n and (g["branch_rows"][q, :n] == o["branch_rows"][q, :n]).all()
        if not same:
            diff.append(q)
    unexplained = [q for q in diff if q not in exempt]
    assert not unexplained, f"{what}: selection differs from the oracle for requests {unexplained}"
    return [(q, exempt[q]) for q in diff]


def scores_np(buf: rps.ScoresBuf) -> dict:
    return {f: getattr(buf, f).detach().cpu().numpy() for f in ("mean_H", "n_tau", "log_a", "score")}


def commit_np(buf: rps.CommitBuf) -> dict:
    return {f: getattr(buf, f).detach().cpu().numpy() for f in
            ("best_slot", "gain", "winner", "commit_pos", "commit_tok", "margin", "mask_pos", "mask_cnt")}


class SlotRows:
    """P^max of the rows each score slot counts in N_tau (Proposition 1), from
    the GPU's and the oracle's statistics: D_j in branch b = j K + c for a
    token slot (compact lookahead layout), the anchor's rows of D_j for the
    [MASK] slot c = K."""

    def __init__(self, piv: dict, branch_g: RowStats, branch_o: RowStats, anchor_g: RowStats, anchor_o: RowStats,
                 L: int, prm):
        self.piv, self.L, self.P, self.K = piv, L, prm.n_pivots, prm.tokens_per_pivot
        self.bg, self.bo, self.ag, self.ao = branch_g, branch_o, anchor_g, anchor_o

    def __call__(self, q: int, j: int, c: int):
        piv, L, K = self.piv, self.L, self.K
        NB = self.P * K
        if c < K:
            b = j * K + c
            first = q * NB * L + int(piv["branch_off"][q, b])
            idx = np.arange(first, first + int(piv["branch_cnt"][q, b]))
            return self.bg.pmax[idx], self.bo.pmax[idx]
        rem = piv["rem_k"][q, :int(piv["rem_cnt"][q])]
        idx = np.array([q * L + k for k in rem if k != piv["pivot_k"][q, j]], dtype=np.int64)
        return self.ag.pmax[idx], self.ao.pmax[idx]


def compare_scores(g: dict, o: dict, prm, what: str, slot_rows: SlotRows = None):
    """Eq. 4 scores within tolerance; N_tau exactly.

    With `slot_rows` (the oracle scored the oracle's statistics) an N_tau
    difference in slot (q, j, c) is excused only row by row: the GPU's count
    must equal the number of that slot's rows whose GPU P^max reaches tau, and
    every row on which the GPU's and the oracle's P^max fall on different sides
    of tau must lie within BAND of it. Without it (the oracle scored the GPU's
    own statistics) N_tau must match exactly. Returns the excused slots."""
    valid = ~np.isnan(o["score"])
    assert (np.isnan(g["score"]) == ~valid).all(), f"{what}: scored slots differ"
    for k in ("mean_H", "log_a", "score"):
        assert_close(g[k][valid], o[k][valid], f"{what} {k}")
    mism = (g["n_tau"] != o["n_tau"]) & valid
    if slot_rows is None:
        assert not mism.any(), f"{what}: N_tau differs at slots {np.argwhere(mism)[:5].tolist()}"
        return []
    tau = np.float32(prm.tau)
    excused = []
    for q, j, c in np.argwhere(valid):
        pg, po = slot_rows(q, j, c)
        assert g["n_tau"][q, j, c] == int(np.sum(pg >= tau)), f"{what}: N_tau({q},{j},{c}) miscounts the GPU's rows"
        assert o["n_tau"][q, j, c] == int(np.sum(po >= tau)), f"{what}: oracle N_tau({q},{j},{c}) miscounts"
        if mism[q, j, c]:
            flips = (pg >= tau) != (po >= tau)
            assert np.all(np.abs(po[flips] - tau) < BAND), \
                f"{what}: N_tau({q},{j},{c}) differs on rows away from tau: {po[flips][:5]}"
            excused.append(((int(q), int(j), int(c)), int(flips.sum())))
    return excused


def compare_commit(g: dict, o: dict, scores_g: dict, scores_o: dict, piv: dict, prm, what: str):
    """Commit decisions.

    1. The oracle's decision logic run on the GPU's own scores gives the GPU's
       decisions exactly (the only latitude: two pivots whose fp32 gains are
       equal, where the fp64 comparison may still order them).
    2. Against the oracle's decisions on its own scores, a difference is
       excused only where the two choices' oracle scores (or gains) lie within
       BAND plus the measured GPU-oracle error of the scores involved.
    Returns the excused requests, as (request, reason)."""
    oracle = oracle_default()
    on_g = oracle.commit(piv, {"score": np.ascontiguousarray(scores_g["score"], np.float64)}, prm)
    K = prm.tokens_per_pivot
    for q in range(len(o["winner"])):
        same = all(np.array_equal(np.asarray(g[k][q]), np.asarray(on_g[k][q]))
                   for k in ("winner", "commit_pos", "commit_tok", "best_slot", "mask_cnt"))
        n = int(on_g["mask_cnt"][q])
        same = same and (g["mask_pos"][q, :n] == on_g["mask_pos"][q, :n]).all()
        if not same:
            wg, wo = int(g["winner"][q]), int(on_g["winner"][q])
            gains = g["gain"][q]
            tie = wg >= 0 and wo >= 0 and np.float32(gains[wg // K]) == np.float32(gains[wo // K])
            assert tie, f"{what}: commit of request {q} is not the oracle's decision on the GPU's scores"
    excused = []
    for q in range(len(o["winner"])):
        same = all(np.array_equal(np.asarray(g[k][q]), np.asarray(o[k][q]))
                   for k in ("winner", "commit_pos", "commit_tok", "best_slot", "mask_cnt"))
        n = int(o["mask_cnt"][q])
        same = same and (g["mask_pos"][q, :n] == o["mask_pos"][q, :n]).all()
        if same:
            continue
        sg, so = scores_g["score"][q].astype(np.float64), scores_o["score"][q]
        ok = ~np.isnan(so)
        err = float(np.max(np.abs(sg[ok] - so[ok]))) if ok.any() else 0.0
        band = BAND + 2 * err
        for j in range(prm.n_pivots):
            bg, bo = int(g["best_slot"][q, j]), int(o["best_slot"][q, j])
            if bg != bo:
                assert bg >= 0 and bo >= 0 and abs(so[j, bg] - so[j, bo]) <= band, \
                    f"{what}: pivot {j} of request {q} picks slot {bg} against the oracle's {bo} away from a tie"
        wg, wo = int(g["winner"][q]), int(o["winner"][q])
        if wg != wo:
            gain_o = o["gain"][q]
            if wg >= 0 and wo >= 0:
                assert abs(gain_o[wg // K] - gain_o[wo // K]) <= 2 * band or wg // K == wo // K, \
                    f"{what}: request {q} commits branch {wg} against the oracle's {wo} away from a tie"
            else:
                b = wg if wg >= 0 else wo
                assert b >= 0 and abs(gain_o[b // K]) <= 2 * band, \
                    f"{what}: request {q} winner {wg} against the oracle's {wo} away from a zero gain"
        excused.append((q, f"near-tied scores (band {band:.2e})"))
    return excused


def assert_same_step(a: rps.Step, b: rps.Step, what: str) -> None:
    """Every output buffer of two steps is bit-identical (NaN matches NaN)."""
    from dataclasses import fields
    for part in ("base", "branch", "piv", "scores", "commit"):
        x, y = getattr(a, part), getattr(b, part)
        for f in fields(x):
            tx, ty = getattr(x, f.name), getattr(y, f.name)
            if tx is None:
                assert ty is None
                continue
            same = torch.equal(tx.nan_to_num(-7.0), ty.nan_to_num(-7.0)) if tx.is_floating_point() else \
                torch.equal(tx, ty)
            assert same, f"{what}: {part}.{f.name} differs between rps_run_step and the separate calls"


class GpuStep:
    """Runs one step through the C ABI and compares every stage with the oracle."""

    def __init__(self, logits_np: np.ndarray, mask_pos: np.ndarray, mask_cnt: np.ndarray, prm, device="cuda"):
        self.o = oracle_default()
        self.logits_np = logits_np
        self.mask_pos, self.mask_cnt, self.prm = mask_pos, mask_cnt, prm
        n_req, nb1, L, V = logits_np.shape
        self.n_req, self.L, self.V = n_req, L, V
        self.t = padded_tensor(logits_np, device)
        self.d_mask_pos = torch.from_numpy(mask_pos).to(device)
        self.d_mask_cnt = torch.from_numpy(mask_cnt).to(device)
        self.step = rps.Step(n_req, L, V, prm, device, self.t.dtype)

    def run_and_compare(self, what: str = ""):
        prm, o, st = self.prm, self.o, self.step
        P, K = prm.n_pivots, prm.tokens_per_pivot
        # stage 1: base row statistics
        st.score_base(self.t, self.d_mask_pos, self.d_mask_cnt)
        st.select(self.d_mask_pos, self.d_mask_cnt)
        st.score_branch_rows(self.t)
        st.score(self.t)
        st.decide()
        # the fused launch must give exactly the results of the two separate calls
        fused_sc = rps.ScoresBuf.alloc(self.n_req, P, K, self.t.device)
        fused_cm = rps.CommitBuf.alloc(self.n_req, self.L, P, self.t.device)
        rps.rps_score_and_commit(self.t, 0, st.base, st.branch, self.n_req, self.L, st.piv, prm, fused_sc, fused_cm)
        status, detail = rps.rps_poll_device_status()
        assert status == rps.RPS_OK, f"{what}: device error bits {detail:#x}"
        for name in ("mean_H", "n_tau", "log_a", "score"):
            assert torch.equal(getattr(fused_sc, name).nan_to_num(-7.0), getattr(st.scores, name).nan_to_num(-7.0)), name
        for name in ("best_slot", "winner", "commit_pos", "commit_tok", "mask_cnt"):
            assert torch.equal(getattr(fused_cm, name), getattr(st.commit, name)), name
        # rps_run_step (the same four kernels, two of them waiting later) gives
        # exactly the results of the separate calls
        one = rps.Step(self.n_req, self.L, self.V, prm, self.t.device, self.t.dtype)
        one.run(self.t, self.d_mask_pos, self.d_mask_cnt)
        status, detail = rps.rps_poll_device_status()
        assert status == rps.RPS_OK, f"{what}: device error bits {detail:#x} (rps_run_step)"
        assert_same_step(one, st, what)

        base_o = o.base_stats(self.logits_np, self.mask_pos, self.mask_cnt, prm.k_max)
        base_g = stats_np(st.base)
        slots = [q * self.L + k for q in range(self.n_req) for k in range(int(self.mask_cnt[q]))]
        compare_stats(base_g, base_o, slots, prm.k_max, f"{what} base")

        # stage 2: selection
        piv_o = o.select_pivots(self.mask_pos, self.mask_cnt, base_o, prm)
        piv_g = piv_np(st.piv)
        near = near_threshold_requests(base_o, piv_o, self.mask_cnt, self.L, prm)
        excused = {"select": compare_select(piv_g, piv_o, self.mask_cnt, self.L, P, K, near, f"{what} select")}
        # the decision logic itself on the GPU's own statistics must agree exactly
        piv_on_g = o.select_pivots(self.mask_pos, self.mask_cnt, base_g, prm)
        compare_select(piv_g, piv_on_g, self.mask_cnt, self.L, P, K, {}, f"{what} select(gpu stats)")

        # stage 3: lookahead rows, scored for the rows the GPU listed
        br_o = o.branch_stats(self.logits_np, piv_g, prm.n_branch)
        br_g = stats_np(st.branch)
        bslots = [q * prm.n_branch * self.L + i for q in range(self.n_req) for i in range(int(piv_g["n_branch_rows"][q]))]
        if bslots:
            compare_stats(br_g, br_o, bslots, 0, f"{what} branch")

        # stage 4: Eq. 4 scores on the GPU's pivots; exactly the oracle's
        # integers on the GPU's own statistics, row-by-row excuses against the
        # oracle's statistics
        anchor_np = self.logits_np[:, 0]
        sc_g = scores_np(st.scores)
        sc_on_g = o.score_branches(piv_g, br_g, base_g, anchor_np, prm)
        compare_scores(sc_g, sc_on_g, prm, f"{what} scores(gpu stats)")
        sc_o = o.score_branches(piv_g, br_o, base_o, anchor_np, prm)
        rows = SlotRows(piv_g, br_g, br_o, base_g, base_o, self.L, prm)
        excused["n_tau"] = compare_scores(sc_g, sc_o, prm, f"{what} scores", rows)

        # stage 5: commit
        cm_o = o.commit(piv_g, sc_o, prm)
        cm_g = commit_np(st.commit)
        excused["commit"] = compare_commit(cm_g, cm_o, sc_g, sc_o, piv_g, prm, f"{what} commit")
        n_exc = sum(len(v) for v in excused.values())
        if n_exc:
            print(f"{what}: excused near-threshold differences {excused}")
        assert n_exc <= MAX_EXCUSED, f"{what}: {n_exc} near-threshold differences excused: {excused}"
        return dict(base=base_g, piv=piv_g, branch=br_g, scores=sc_g, commit=cm_g, piv_o=piv_o, excused=excused)


def workload_inputs(w, **overrides):
    """Host logits (numpy) and the mask of a workload, optionally shrunk (V, L, n_req, ...)."""
    w = w.scaled(**overrides) if overrides else w
    mask_pos, mask_cnt = w.mask()
    logits = synth.make_logits(w.seed, w.n_req, w.n_branch, w.L, w.V, w.mixture, w.dtype, valid=w.valid_rows())
    return w, logits, mask_pos, mask_cnt
