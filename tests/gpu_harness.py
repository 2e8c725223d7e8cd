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


def near_threshold_requests(o: RowStats, piv_o: dict, mask_cnt, L, prm) -> set:
    """Requests whose selection hinges on an oracle quantity within BAND of its threshold.

    Only the comparisons that decide the outcome count. Commit set: P^max
    against tau and the two most confident rows (threshold rule and its
    fallback), or adjacent values among the k + 1 best of M (top-k rules).
    Pivots: mu against tau_pivot and adjacent truncated entropies among the
    P + 1 highest feasible rows of M' (Eq. 3), or adjacent confidences /
    entropies among the P + 1 highest rows of M' (the other pivot rules).
    """
    def close_pair(values, n):
        v = np.sort(np.asarray(values, np.float64))[::-1][:n]
        return len(v) > 1 and np.min(-np.diff(v)) < BAND

    commit_rule = getattr(prm, "commit_rule", 0)
    pivot_rule = getattr(prm, "pivot_rule", 0)
    out = set()
    tau, tau_p = np.float32(prm.tau), np.float32(prm.tau_pivot)
    for q in range(len(mask_cnt)):
        s = slice(q * L, q * L + int(mask_cnt[q]))
        pm, mu, H = o.pmax[s], o.mu[s], o.H[s]
        if commit_rule == 0:
            if np.any(np.abs(pm - tau) < BAND) or close_pair(pm, 2):
                out.add(q)
                continue
        elif close_pair(pm if commit_rule == 1 else -H, prm.commit_k + 1):
            out.add(q)
            continue
        rem = piv_o["rem_k"][q, :piv_o["rem_cnt"][q]]
        if pivot_rule == 0:
            if np.any(np.abs(np.array([o.mu[q * L + k] for k in rem]) - tau_p) < BAND):
                out.add(q)
                continue
            vals = [o.htrunc[q * L + k] for k in rem if o.mu[q * L + k] >= tau_p]
        else:
            src = o.pmax if pivot_rule == 1 else o.H
            vals = [src[q * L + k] for k in rem]
        if close_pair(vals, prm.n_pivots + 1):
            out.add(q)
    return out


SELECT_KEYS = ("n_commit", "rem_cnt", "state")


def compare_select(g: dict, o: dict, mask_cnt, L, P, K, exempt: set, what: str):
    """Every integer output of pivot selection, per request."""
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
    return diff


def scores_np(buf: rps.ScoresBuf) -> dict:
    return {f: getattr(buf, f).detach().cpu().numpy() for f in ("mean_H", "n_tau", "log_a", "score")}


def commit_np(buf: rps.CommitBuf) -> dict:
    return {f: getattr(buf, f).detach().cpu().numpy() for f in
            ("best_slot", "gain", "winner", "commit_pos", "commit_tok", "margin", "mask_pos", "mask_cnt")}


def compare_scores(g: dict, o: dict, branch_pmax_o: np.ndarray, prm, what: str):
    valid = ~np.isnan(o["score"])
    assert (np.isnan(g["score"]) == ~valid).all(), f"{what}: scored slots differ"
    for k in ("mean_H", "log_a", "score"):
        assert_close(g[k][valid], o[k][valid], f"{what} {k}")
    # N_tau is an integer decided by P^max >= tau; a difference needs a row in the band
    mism = (g["n_tau"] != o["n_tau"]) & valid
    if mism.any():
        near = np.any(np.abs(branch_pmax_o[~np.isnan(branch_pmax_o)] - np.float32(prm.tau)) < BAND)
        assert near, f"{what}: N_tau differs with no confidence near tau"


def compare_commit(g: dict, o: dict, scores_o: dict, mask_L: int, what: str):
    n_req = len(o["winner"])
    for q in range(n_req):
        same = g["winner"][q] == o["winner"][q] and g["commit_pos"][q] == o["commit_pos"][q] \
            and g["commit_tok"][q] == o["commit_tok"][q]
        n = int(o["mask_cnt"][q])
        same &= g["mask_cnt"][q] == n and (g["mask_pos"][q, :n] == o["mask_pos"][q, :n]).all()
        same &= (g["best_slot"][q] == o["best_slot"][q]).all()
        if not same:
            near = False
            for row, gain in zip(scores_o["score"][q], o["gain"][q]):
                v = np.sort(row[~np.isnan(row)])[::-1]
                if len(v) > 1 and v[0] - v[1] < BAND:
                    near = True
                if not np.isnan(gain) and abs(gain) < BAND:
                    near = True
            gains = np.sort(o["gain"][q][~np.isnan(o["gain"][q])])[::-1]
            if len(gains) > 1 and gains[0] - gains[1] < BAND:
                near = True
            assert near, f"{what}: commit of request {q} differs from the oracle away from any tie"


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
        exempt = near_threshold_requests(base_o, piv_o, self.mask_cnt, self.L, prm)
        compare_select(piv_g, piv_o, self.mask_cnt, self.L, P, K, exempt, f"{what} select")
        # the decision logic itself on the GPU's own statistics must agree exactly
        piv_on_g = o.select_pivots(self.mask_pos, self.mask_cnt, base_g, prm)
        compare_select(piv_g, piv_on_g, self.mask_cnt, self.L, P, K, set(), f"{what} select(gpu stats)")

        # stage 3: lookahead rows, scored for the rows the GPU listed
        br_o = o.branch_stats(self.logits_np, piv_g, prm.n_branch)
        br_g = stats_np(st.branch)
        bslots = [q * prm.n_branch * self.L + i for q in range(self.n_req) for i in range(int(piv_g["n_branch_rows"][q]))]
        if bslots:
            compare_stats(br_g, br_o, bslots, 0, f"{what} branch")

        # stage 4: Eq. 4 scores on the GPU's pivots
        sc_o = o.score_branches(piv_g, br_o, base_o, self.logits_np[:, 0], prm)
        sc_g = scores_np(st.scores)
        compare_scores(sc_g, sc_o, br_o.pmax, prm, f"{what} scores")

        # stage 5: commit
        cm_o = o.commit(piv_g, sc_o, prm)
        cm_g = commit_np(st.commit)
        compare_commit(cm_g, cm_o, sc_o, self.L, f"{what} commit")
        return dict(base=base_g, piv=piv_g, branch=br_g, scores=sc_g, commit=cm_g, piv_o=piv_o)


def workload_inputs(w, **overrides):
    """Host logits (numpy) and the mask of a workload, optionally shrunk (V, L, n_req, ...)."""
    w = w.scaled(**overrides) if overrides else w
    mask_pos, mask_cnt = w.mask()
    logits = synth.make_logits(w.seed, w.n_req, w.n_branch, w.L, w.V, w.mixture, w.dtype, valid=w.valid_rows())
    return w, logits, mask_pos, mask_cnt
