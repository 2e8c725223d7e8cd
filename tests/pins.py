"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Every ``pin_*`` function takes an ``Oracle`` instance and raises AssertionError
on a mismatch. ``test_oracle_pins.py`` runs them against the oracle;
``test_oracle_mutants.py`` runs them against copies of the oracle with planted
mistakes and requires each mistake to fail at least one pin.

Sources of truth used here:
  * closed forms of the definitions (uniform, one-spike and two-level rows),
  * invariants (0 <= truncated entropy <= H <= log V, 1/V <= P^max <= mu <= 1, ...),
  * fp64 library routines (torch.log_softmax, numpy lexsort / sort),
  * brute-force enumeration of pivot, candidate and commit decisions on tiny
    inputs, with probabilities computed by numpy,
  * Propositions 1 and 2 of the paper as invariants of the scores,
  * the control-flow cases of Algorithm 1 on hand-built inputs.
"""
from __future__ import annotations

import math
from dataclasses import replace

import numpy as np

from paper_2608_11742_gb300 import synth
from paper_2608_11742_gb300.configs import Params

TOL = 1e-10


def close(a, b, tol=TOL, what=""):
    a, b = np.broadcast_arrays(np.asarray(a, dtype=np.float64), np.asarray(b, dtype=np.float64))
    ok = np.isclose(a, b, rtol=tol, atol=tol, equal_nan=True)
    assert ok.all(), f"{what}: {a[~ok][:5]} != {b[~ok][:5]}"


# --------------------------------------------------------------------------
# Row statistics (Sec. 2 notation, Eq. 1, Eq. 3)
# --------------------------------------------------------------------------

def pin_uniform_rows(o):
    """Uniform logits: H = ln V, P^max = 1/V, mu = k/V, truncated entropy = (k/V) ln V."""
    for V in (1, 2, 5, 64, 4096):
        for c in (0.0, 80.0, -30.5):
            k = min(10, V)
            st = o.row_stats(np.full((1, V), c, np.float32), k)
            close(st.H, math.log(V), what=f"H V={V}")
            close(st.pmax, 1.0 / V, what="pmax")
            close(st.mu, k / V, what="mu")
            close(st.htrunc, (k / V) * math.log(V), what="htrunc")
            close(st.lse, c + math.log(V), what="lse")
            close(st.zmax, c, what="zmax")
            assert st.argmax[0] == 0
            assert list(st.topk_idx[0]) == list(range(k)), "ties must rank the lower token first"


def _spike_expect(V, t, a, k):
    """Closed form of a row of zeros with z_t = a."""
    if a > 0:
        lnZ = a + math.log1p((V - 1) * math.exp(-a))
    else:
        lnZ = math.log((V - 1) + math.exp(a))
    lp1, lp0 = a - lnZ, -lnZ
    p1, p0 = math.exp(lp1), math.exp(lp0)
    H = -(p1 * lp1) - (V - 1) * p0 * lp0
    others = [v for v in range(V) if v != t]
    if a > 0:
        top = [t] + others[:k - 1]
        mu = p1 + (k - 1) * p0
        ht = -(p1 * lp1) - (k - 1) * p0 * lp0
        pmax, amax = p1, t
    else:
        top = others[:k]
        mu = k * p0
        ht = -k * p0 * lp0
        pmax, amax = p0, others[0]
    return dict(lse=lnZ, H=H, pmax=pmax, mu=mu, htrunc=ht, argmax=amax, top=top)


def pin_spike_rows(o):
    """One token raised by a over zeros: exact entropy, confidence, mass and support."""
    for V in (16, 4096):
        for t in (0, 5, V - 1):
            for a in (0.5, 3.0, 12.0, 50.0, -2.0):
                for k in (1, 3, 10):
                    row = np.zeros((1, V), np.float32)
                    row[0, t] = a
                    st = o.row_stats(row, k)
                    e = _spike_expect(V, t, float(np.float32(a)), k)
                    what = f"V={V} t={t} a={a} k={k}"
                    close(st.lse, e["lse"], what="lse " + what)
                    close(st.H, e["H"], what="H " + what)
                    close(st.pmax, e["pmax"], what="pmax " + what)
                    close(st.mu, e["mu"], what="mu " + what)
                    close(st.htrunc, e["htrunc"], what="htrunc " + what)
                    assert st.argmax[0] == e["argmax"], what
                    assert list(st.topk_idx[0]) == e["top"], what


def pin_two_level_rows(o):
    """m tokens raised by a: H = ln Z - m a e^a / Z with Z = m e^a + V - m."""
    rng = np.random.default_rng(1)
    for V, m, a in ((64, 3, 2.0), (4096, 5, 4.0), (1000, 2, 7.5)):
        spikes = np.sort(rng.choice(V, m, replace=False))
        row = np.zeros((1, V), np.float32)
        row[0, spikes] = a
        Z = m * math.exp(a) + (V - m)
        k = 10
        st = o.row_stats(row, k)
        close(st.H, math.log(Z) - m * a * math.exp(a) / Z, what="two-level H")
        close(st.pmax, math.exp(a) / Z, what="two-level pmax")
        close(st.mu, (m * math.exp(a) + (k - m)) / Z, what="two-level mu")
        rest = [v for v in range(V) if v not in set(spikes)]
        assert list(st.topk_idx[0]) == list(spikes) + rest[:k - m]
        assert st.argmax[0] == spikes[0]


def pin_rank_order(o):
    """Top-k ranks by logit, then by lower token id (Eq. 3 support T_i)."""
    row = np.array([[1.0, 3.0, 3.0, 2.0, 3.0, -1.0, 2.0]], np.float32)
    st = o.row_stats(row, 7)
    assert list(st.topk_idx[0]) == [1, 2, 4, 3, 6, 0, 5]
    close(st.topk_logit[0], [3, 3, 3, 2, 2, 1, -1], what="topk logits")
    assert st.argmax[0] == 1


def _torch_reference(rows_f64, k):
    import torch
    z = torch.from_numpy(rows_f64)
    ls = torch.log_softmax(z, dim=-1)
    p = ls.exp()
    H = -(torch.where(p > 0, p * ls, torch.zeros_like(p))).sum(-1).numpy()
    pmax = p.max(-1).values.numpy()
    lse = torch.logsumexp(z, dim=-1).numpy()
    top = []
    for r in rows_f64:
        order = np.lexsort((np.arange(r.shape[0]), -r))
        top.append(order[:k])
    top = np.array(top)
    pt = np.take_along_axis(p.numpy(), top, axis=1)
    lt = np.take_along_axis(ls.numpy(), top, axis=1)
    mu = pt.sum(1)
    ht = -(np.where(pt > 0, pt * lt, 0.0)).sum(1)
    return H, pmax, lse, top, mu, ht


def _random_rows(rng, n, V, bf16):
    z = rng.standard_normal((n, V)).astype(np.float32) * rng.uniform(0.5, 3.0, (n, 1)).astype(np.float32)
    for i in range(n):
        z[i, rng.integers(0, V, 3)] += np.float32(rng.uniform(0, 10))
    if bf16:
        bits = synth.bf16_round(z)
        return bits, synth.bf16_to_f32(bits).astype(np.float64)
    return z, z.astype(np.float64)


def pin_library_crosscheck(o):
    """fp64 torch.log_softmax / logsumexp and numpy lexsort agree with the oracle."""
    rng = np.random.default_rng(7)
    for V, bf16 in ((50, False), (4096, True), (3001, True), (777, False)):
        stored, z64 = _random_rows(rng, 6, V, bf16)
        k = 10
        st = o.row_stats(stored, k)
        H, pmax, lse, top, mu, ht = _torch_reference(z64, k)
        close(st.H, H, 1e-9, "H vs torch")
        close(st.pmax, pmax, 1e-9, "pmax vs torch")
        close(st.lse, lse, 1e-9, "lse vs torch")
        close(st.mu, mu, 1e-9, "mu vs torch")
        close(st.htrunc, ht, 1e-9, "htrunc vs torch")
        assert (st.topk_idx == top).all(), "top-k vs lexsort"
        close(st.topk_logit, np.take_along_axis(z64, top, 1), 0, "top-k logits")
        assert (st.argmax == top[:, 0]).all()


def pin_synth_rows_crosscheck(o):
    """The generator's bf16 rows, scored by the oracle and by fp64 torch."""
    for pos in (0, 1, 2, 3, 4, 5):
        bits = synth.row_logits(0, 5000, 0, 0, pos, (0.4, 0.3, 0.3), "bf16")
        st = o.row_stats(bits[None], 10)
        z64 = synth.bf16_to_f32(bits).astype(np.float64)[None]
        H, pmax, lse, top, mu, ht = _torch_reference(z64, 10)
        close(st.H, H, 1e-9, "synth H")
        close(st.pmax, pmax, 1e-9, "synth pmax")
        assert (st.topk_idx == top).all()


def pin_invariants(o):
    """0 <= truncated entropy <= H <= ln V; 1/V <= P^max <= mu <= 1; nesting in k."""
    rng = np.random.default_rng(11)
    for V in (7, 300, 4096):
        stored, _ = _random_rows(rng, 8, V, V > 100)
        prev_mu = prev_ht = None
        for k in range(1, min(V, 12) + 1):
            st = o.row_stats(stored, k)
            eps = 1e-12
            assert (st.htrunc >= -eps).all() and (st.htrunc <= st.H + eps).all()
            assert (st.H <= math.log(V) + eps).all()
            assert (st.pmax >= 1.0 / V - eps).all() and (st.pmax <= st.mu + eps).all()
            assert (st.mu <= 1 + eps).all()
            assert (st.argmax == st.topk_idx[:, 0]).all()
            if k == 1:
                close(st.mu, st.pmax, 1e-12, "mu(k=1) = P^max")
            if prev_mu is not None:
                assert (st.mu >= prev_mu - eps).all() and (st.htrunc >= prev_ht - eps).all()
            prev_mu, prev_ht = st.mu, st.htrunc
        full = o.row_stats(stored, V) if V <= 300 else None
        if full is not None:
            close(full.mu, 1.0, 1e-12, "mu(k=V) = 1")
            close(full.htrunc, full.H, 1e-9, "htrunc(k=V) = H")


def pin_neg_inf_entries(o):
    """-inf logits carry zero probability: the row equals the row without them."""
    rng = np.random.default_rng(3)
    z = rng.standard_normal(40).astype(np.float32)
    drop = np.array([0, 7, 8, 39])
    zi = z.copy()
    zi[drop] = -np.inf
    keep = np.setdiff1d(np.arange(40), drop)
    a = o.row_stats(zi[None], 5)
    b = o.row_stats(z[keep][None], 5)
    close(a.H, b.H, 1e-12, "H with -inf")
    close(a.lse, b.lse, 1e-12, "lse with -inf")
    close(a.pmax, b.pmax, 1e-12, "pmax with -inf")
    assert list(a.topk_idx[0]) == list(keep[b.topk_idx[0]])


# --------------------------------------------------------------------------
# Decisions: brute force on tiny inputs
# --------------------------------------------------------------------------

def _softmax64(z):
    z = np.asarray(z, np.float64)
    e = np.exp(z - z.max())
    return e / e.sum()


def _entropy64(p):
    nz = p > 0
    return float(-(p[nz] * np.log(p[nz])).sum())


def brute_select(logits, mask_pos, mask_cnt, prm: Params):
    """Selection decisions recomputed from numpy probabilities, by enumeration."""
    n_req = logits.shape[0]
    out = []
    for q in range(n_req):
        M = [int(x) for x in mask_pos[q, :mask_cnt[q]]]
        probs = {i: _softmax64(logits[q, 0, i]) for i in M}
        if not M:
            out.append(dict(state=1, commit=[], rem=[], pivots=[], cands=[]))
            continue
        if prm.commit_rule == 0:  # confidence threshold with the fallback (Eq. 2, Algorithm 1)
            S = [i for i in M if probs[i].max() >= np.float32(prm.tau)]
            if not S:
                S = [max(M, key=lambda i: (probs[i].max(), -i))]
        elif prm.commit_rule == 1:  # top-k confidence (Eq. 2, first rule)
            S = sorted(M, key=lambda i: (-probs[i].max(), i))[:prm.commit_k]
        else:  # top-k lowest entropy (Eq. 2, second rule)
            S = sorted(M, key=lambda i: (_entropy64(probs[i]), i))[:prm.commit_k]
        commit = [(i, int(np.argmax(logits[q, 0, i]))) for i in M if i in S]
        rem = [i for i in M if i not in S]
        if not rem:
            out.append(dict(state=1, commit=commit, rem=rem, pivots=[], cands=[]))
            continue

        def top(i):
            z = np.asarray(logits[q, 0, i], np.float64)
            return list(np.lexsort((np.arange(z.shape[0]), -z))[:prm.k_max])

        mu = {i: float(probs[i][top(i)].sum()) for i in rem}
        # -sum p log p over T_i only (probabilities not renormalised)
        ht = {i: float(-sum(probs[i][v] * math.log(probs[i][v]) for v in top(i) if probs[i][v] > 0))
              for i in rem}
        if prm.pivot_rule == 0:  # Eq. 3: mass constraint, then truncated entropy
            feas = [i for i in rem if mu[i] >= np.float32(prm.tau_pivot)]
            key = lambda i: (-ht[i], i)
        elif prm.pivot_rule == 1:  # max confidence over M'
            feas, key = list(rem), lambda i: (-probs[i].max(), i)
        else:  # max entropy over M', unconstrained
            feas, key = list(rem), lambda i: (-_entropy64(probs[i]), i)
        if not feas:
            out.append(dict(state=2, commit=commit, rem=rem, pivots=[], cands=[]))
            continue
        ranked = sorted(feas, key=key)
        pivots = ranked[:prm.n_pivots]
        cands = []
        for i in pivots:
            pm = probs[i].max()
            c = [v for v in top(i) if probs[i][v] >= np.float32(prm.r) * pm][:prm.tokens_per_pivot]
            cands.append(c)
        state = 0 if any(len(c) >= 2 for c in cands) else 3
        out.append(dict(state=state, commit=commit, rem=rem, pivots=pivots, cands=cands))
    return out


def _tiny_case(rng, n_req, L, V, spread):
    z = rng.standard_normal((n_req, 1, L, V)) * spread
    for q in range(n_req):
        for i in range(L):
            kind = rng.integers(0, 4)
            if kind == 0:
                z[q, 0, i, rng.integers(0, V)] += rng.uniform(3, 8)
            elif kind == 1:
                z[q, 0, i, rng.choice(V, 2, replace=False)] += rng.uniform(1, 3)
    z = z.astype(np.float32)
    if L >= 3:  # duplicate rows exercise position tie-breaks
        z[:, 0, 2] = z[:, 0, 1]
    return z


def pin_select_brute_force(o):
    """Commit set, fallback, feasibility, pivots and candidates match enumeration,
    for the paper's rules (Eq. 2 threshold, Eq. 3) and for the other commit rules
    of Eq. 2 and the ablation pivot strategies."""
    rng = np.random.default_rng(5)
    grid = [Params(k_max=k, r=r, tau_pivot=tp, tau=tau, lam=0.2, n_pivots=P, tokens_per_pivot=K, pivot_rule=pr,
                   commit_rule=cr, commit_k=ck)
            for (k, r, tp, tau, P, K, pr, cr, ck) in [
                (4, 0.1, 0.0, 0.9, 1, 2, 0, 0, 0), (4, 0.3, 0.5, 0.5, 2, 2, 0, 0, 0), (6, 0.05, 0.9, 0.9, 3, 3, 0, 0, 0),
                (3, 0.5, 0.3, 0.3, 2, 1, 0, 0, 0), (5, 0.2, 0.6, 0.7, 1, 5, 0, 0, 0), (4, 0.1, 0.2, 0.99, 4, 2, 0, 0, 0),
                (4, 0.1, 0.9, 0.9, 2, 2, 1, 0, 0), (4, 0.1, 0.9, 0.9, 3, 2, 2, 0, 0),
                (4, 0.2, 0.3, 0.9, 2, 2, 0, 1, 2), (4, 0.2, 0.3, 0.9, 2, 2, 0, 2, 3),
                (5, 0.1, 0.0, 0.5, 2, 3, 2, 1, 1), (5, 0.1, 0.0, 0.5, 3, 2, 1, 2, 4)]]
    for trial in range(72):
        prm = grid[trial % len(grid)]
        n_req, L, V = 2, 7, 12
        z = _tiny_case(rng, n_req, L, V, rng.uniform(0.3, 2.0))
        cnt = rng.integers(0, L + 1, n_req).astype(np.int32)
        mpos = np.full((n_req, L), -1, np.int32)
        for q in range(n_req):
            mpos[q, :cnt[q]] = np.sort(rng.choice(L, cnt[q], replace=False))
        base = o.base_stats(z, mpos, cnt, prm.k_max)
        got = o.select_pivots(mpos, cnt, base, prm)
        want = brute_select(z, mpos, cnt, prm)
        for q in range(n_req):
            w = want[q]
            assert got["state"][q] == w["state"], (trial, q, got["state"][q], w["state"])
            nc = got["n_commit"][q]
            assert [(int(a), int(b)) for a, b in zip(got["commit_pos"][q, :nc], got["commit_tok"][q, :nc])] \
                == w["commit"], (trial, q)
            assert list(got["rem_pos"][q, :got["rem_cnt"][q]]) == w["rem"]
            if w["state"] in (0, 3):
                piv = [int(x) for x in got["pivot_pos"][q] if x >= 0]
                assert piv == w["pivots"], (trial, q, piv, w["pivots"])
                for j, c in enumerate(w["cands"]):
                    assert list(got["cand_tok"][q, j, :got["n_cand"][q, j]]) == c, (trial, q, j)
            if w["state"] == 0:
                # branch rows: every searched branch lists M' without its pivot
                K = prm.tokens_per_pivot
                for j, c in enumerate(w["cands"]):
                    for s in range(K):
                        b = j * K + s
                        valid = len(c) >= 2 and s < len(c)
                        assert bool(got["branch_valid"][q, b]) == valid
                        if valid:
                            off, n = got["branch_off"][q, b], got["branch_cnt"][q, b]
                            rows = got["branch_rows"][q, off:off + n]
                            assert list(rows[:, 2]) == [i for i in w["rem"] if i != w["pivots"][j]]
                            assert (rows[:, 0] == q).all() and (rows[:, 1] == 1 + b).all()


def _lookahead_case(rng, n_req, L, V, prm, spread=1.0):
    """Tiny base + branch logits where pivots are searched."""
    NB = prm.n_branch
    z = rng.standard_normal((n_req, 1 + NB, L, V)) * spread
    for q in range(n_req):
        for i in range(L):
            toks = rng.choice(V, 3, replace=False)
            z[q, 0, i, toks] += rng.uniform(0.5, 2.5, 3)
            for b in range(1, 1 + NB):
                z[q, b, i] = z[q, 0, i] + rng.standard_normal(V) * 0.3
                z[q, b, i, toks] *= rng.uniform(0.5, 3.0)
    return z.astype(np.float32)


def brute_score_commit(o, z, mpos, cnt, prm, piv):
    """Eq. 4 scores and the commit decision by enumeration over numpy probabilities."""
    n_req = z.shape[0]
    K, P = prm.tokens_per_pivot, prm.n_pivots
    res = []
    for q in range(n_req):
        rem = [int(x) for x in piv["rem_pos"][q, :piv["rem_cnt"][q]]]
        scores = {}
        if piv["state"][q] == 0:
            for j in range(P):
                ip = int(piv["pivot_pos"][q, j])
                nc = int(piv["n_cand"][q, j])
                if ip < 0 or nc < 2:
                    continue
                D = [i for i in rem if i != ip]
                pa = _softmax64(z[q, 0, ip])
                for c in range(nc):
                    b = 1 + j * K + c
                    Hs = [_entropy64(_softmax64(z[q, b, i])) for i in D]
                    ntau = sum(_softmax64(z[q, b, i]).max() >= np.float32(prm.tau) for i in D)
                    hbar = float(np.mean(Hs)) if D else 0.0
                    la = math.log(pa[int(piv["cand_tok"][q, j, c])])
                    scores[(j, c)] = (hbar, ntau, la, -hbar + float(np.float32(prm.lam)) * la)
                Hs = [_entropy64(_softmax64(z[q, 0, i])) for i in D]
                ntau = sum(_softmax64(z[q, 0, i]).max() >= np.float32(prm.tau) for i in D)
                hbar = float(np.mean(Hs)) if D else 0.0
                la = math.log(pa.max())
                scores[(j, K)] = (hbar, ntau, la, -hbar + float(np.float32(prm.lam)) * la)
        # decision: per pivot the best slot (ties: [MASK], then candidate rank)
        best = {}
        for j in sorted({j for (j, _) in scores}):
            slots = [c for (jj, c) in scores if jj == j]
            order = sorted(slots, key=lambda c: (-scores[(j, c)][3], 0 if c == K else 1, c))
            b = order[0]
            best[j] = (b, scores[(j, b)][3] - scores[(j, K)][3])
        winners = [(g, -int(piv["pivot_pos"][q, j]), j) for j, (b, g) in best.items() if b != K and g > 0]
        if piv["state"][q] == 1:
            win = -3
        elif piv["state"][q] != 0:
            win = -2
        elif not winners:
            win = -1
        else:
            g, _, j = max(winners)
            win = j * K + best[j][0]
        res.append(dict(scores=scores, best=best, winner=win))
    return res


def pin_score_commit_brute_force(o):
    """Eq. 4 (mean entropy, N_tau, log a, score) and the commit decision by enumeration."""
    rng = np.random.default_rng(9)
    grid = [Params(k_max=6, r=0.05, tau_pivot=0.0, tau=0.5, lam=lam, n_pivots=P, tokens_per_pivot=K)
            for lam, P, K in ((0.0, 1, 2), (0.1, 2, 2), (0.5, 3, 2), (2.0, 2, 3), (0.3, 1, 4))]
    n_search = 0
    for trial in range(30):
        prm = grid[trial % len(grid)]
        n_req, L, V = 2, 6, 10
        z = _lookahead_case(rng, n_req, L, V, prm, spread=rng.uniform(0.3, 1.5))
        cnt = rng.integers(1, L + 1, n_req).astype(np.int32)
        mpos = np.full((n_req, L), -1, np.int32)
        for q in range(n_req):
            mpos[q, :cnt[q]] = np.sort(rng.choice(L, cnt[q], replace=False))
        out = o.step(z, mpos, cnt, prm)
        piv, sc, cm = out["pivots"], out["scores"], out["commit"]
        want = brute_score_commit(o, z, mpos, cnt, prm, piv)
        K = prm.tokens_per_pivot
        for q in range(n_req):
            w = want[q]
            n_search += piv["state"][q] == 0
            for (j, c), (hbar, ntau, la, s) in w["scores"].items():
                close(sc["mean_H"][q, j, c], hbar, 1e-9, f"mean_H {trial} {q} {j} {c}")
                assert sc["n_tau"][q, j, c] == ntau, (trial, q, j, c)
                close(sc["log_a"][q, j, c], la, 1e-9, "log a")
                close(sc["score"][q, j, c], s, 1e-9, "score")
            assert cm["winner"][q] == w["winner"], (trial, q, cm["winner"][q], w["winner"])
            for j, (b, g) in w["best"].items():
                assert cm["best_slot"][q, j] == b
                close(cm["gain"][q, j], g, 1e-9, "gain")
            rem = [int(x) for x in piv["rem_pos"][q, :piv["rem_cnt"][q]]]
            if w["winner"] >= 0:
                j, c = divmod(w["winner"], K)
                assert cm["commit_pos"][q] == piv["pivot_pos"][q, j]
                assert cm["commit_tok"][q] == piv["cand_tok"][q, j, c]
                rem = [i for i in rem if i != piv["pivot_pos"][q, j]]
            assert list(cm["mask_pos"][q, :cm["mask_cnt"][q]]) == rem
    assert n_search >= 10, "the brute-force cases must reach the lookahead search"


# --------------------------------------------------------------------------
# Closed-form scores and Algorithm 1 control flow
# --------------------------------------------------------------------------

def _uniform(V, c=0.0):
    return np.full(V, c, np.float32)


def _spike(V, t, a):
    r = np.zeros(V, np.float32)
    r[t] = a
    return r


def pin_score_closed_form(o):
    """Eq. 4 on rows with closed-form entropies; n = |M| - 1 excludes the pivot.

    Request: 4 masked positions, V = 8. Base rows: positions 0 and 1 one-spike
    (not committed: P^max < tau), position 2 uniform, position 3 two-level; the
    pivot (largest truncated entropy, k_max = 8, tau_pivot = 0) is position 2.
    Branch (token c) rows: uniform at 0, spike at 1, spike at 3.
    """
    V, a, b = 8, 1.5, 0.75
    prm = Params(k_max=8, r=0.5, tau_pivot=0.0, tau=0.95, lam=0.3, n_pivots=1, tokens_per_pivot=2)
    z = np.zeros((1, 3, 4, V), np.float32)
    z[0, 0, 0] = _spike(V, 1, a)
    z[0, 0, 1] = _spike(V, 2, b)
    z[0, 0, 2] = _uniform(V)
    two = np.zeros(V, np.float32)
    two[[4, 5]] = np.float32(0.25)
    z[0, 0, 3] = two
    for br in (1, 2):
        z[0, br, 0] = _uniform(V)
        z[0, br, 1] = _spike(V, 3, a * br)
        z[0, br, 3] = _spike(V, 6, b * br)
    mpos = np.array([[0, 1, 2, 3]], np.int32)
    cnt = np.array([4], np.int32)
    out = o.step(z, mpos, cnt, prm)
    piv = out["pivots"]
    assert piv["state"][0] == 0 and piv["pivot_pos"][0, 0] == 2
    # S is empty, so the fallback commits the most confident row: position 0 (spike a > b, two-level).
    assert piv["n_commit"][0] == 1 and piv["commit_pos"][0, 0] == 0 and piv["commit_tok"][0, 0] == 1
    # uniform pivot row: candidates are tokens 0 and 1 (ties to lower id), p = 1/8 each
    assert list(piv["cand_tok"][0, 0]) == [0, 1]

    def H_spike(V, h):
        Z = math.exp(h) + V - 1
        return math.log(Z) - h * math.exp(h) / Z

    def H_two(V, m, h):
        Z = m * math.exp(h) + V - m
        return math.log(Z) - m * h * math.exp(h) / Z

    # D = M' \ {pivot} = {1, 3}; n = 2
    sc = out["scores"]
    for c in (0, 1):
        br = 1 + c
        hbar = (H_spike(V, float(np.float32(a * br))) + H_spike(V, float(np.float32(b * br)))) / 2
        la = math.log(1.0 / V)
        close(sc["mean_H"][0, 0, c], hbar, 1e-12, "closed-form mean_H")
        close(sc["log_a"][0, 0, c], la, 1e-12, "closed-form log a")
        close(sc["score"][0, 0, c], -hbar + float(np.float32(0.3)) * la, 1e-12, "closed-form score")
    hbar_mask = (H_spike(V, b) + H_two(V, 2, 0.25)) / 2
    close(sc["mean_H"][0, 0, 2], hbar_mask, 1e-12, "closed-form mean_H [MASK]")
    close(sc["log_a"][0, 0, 2], math.log(1.0 / V), 1e-12, "closed-form log a [MASK]")


def _one_request(rows_base, rows_branch, prm, mask=None):
    L = len(rows_base)
    V = rows_base[0].shape[0]
    z = np.zeros((1, 1 + prm.n_branch, L, V), np.float32)
    for i, r in enumerate(rows_base):
        z[0, 0, i] = r
    for b, rows in enumerate(rows_branch):
        for i, r in enumerate(rows):
            z[0, 1 + b, i] = r
    mpos = np.array([mask if mask is not None else list(range(L))], np.int32)
    cnt = np.array([mpos.shape[1]], np.int32)
    return z, mpos, cnt


def pin_control_flow(o):
    """Algorithm 1 cases: fallback, done, no feasible row, no candidates, abstain, commit."""
    V = 6
    P1 = Params(k_max=3, r=0.5, tau_pivot=0.0, tau=0.9, lam=0.0, n_pivots=1, tokens_per_pivot=2)

    # fallback: no row reaches tau; two identical rows tie -> lower position committed
    base = [_spike(V, 2, 1.0), _spike(V, 2, 1.0), _uniform(V)]
    z, m, c = _one_request(base, [base, base], P1)
    out = o.step(z, m, c, P1)
    assert out["pivots"]["n_commit"][0] == 1 and out["pivots"]["commit_pos"][0, 0] == 0
    assert out["pivots"]["commit_tok"][0, 0] == 2

    # everything confident -> M' empty -> DONE
    base = [_spike(V, 1, 10.0), _spike(V, 4, 9.0)]
    z, m, c = _one_request(base, [base, base], P1)
    out = o.step(z, m, c, P1)
    assert out["pivots"]["state"][0] == 1 and out["commit"]["winner"][0] == -3
    assert out["commit"]["mask_cnt"][0] == 0

    # no feasible row: tau_pivot above every mu -> skip
    prm = replace(P1, tau_pivot=0.99)
    base = [_spike(V, 1, 10.0), _uniform(V), _uniform(V)]
    z, m, c = _one_request(base, [base, base], prm)
    out = o.step(z, m, c, prm)
    assert out["pivots"]["state"][0] == 2 and out["commit"]["winner"][0] == -2
    assert list(out["commit"]["mask_pos"][0, :2]) == [1, 2]

    # single candidate (|C \ MASK| <= 1): the pivot has one dominant token -> skip
    base = [_spike(V, 1, 10.0), _spike(V, 0, 2.0), _spike(V, 3, 2.5)]
    z, m, c = _one_request(base, [base, base], P1)
    out = o.step(z, m, c, P1)
    assert out["pivots"]["state"][0] == 3 and out["commit"]["winner"][0] == -2

    # abstain: branches raise entropy -> [MASK] keeps the pivot masked
    base = [_spike(V, 1, 10.0), _uniform(V), _spike(V, 2, 3.0)]
    worse = [_uniform(V), _uniform(V), _uniform(V)]
    z, m, c = _one_request(base, [worse, worse], P1)
    out = o.step(z, m, c, P1)
    assert out["pivots"]["state"][0] == 0 and out["pivots"]["pivot_pos"][0, 0] == 1
    assert out["commit"]["winner"][0] == -1
    assert list(out["commit"]["mask_pos"][0, :out["commit"]["mask_cnt"][0]]) == [1, 2]

    # commit: branch 1 (token slot 1) collapses the downstream entropy
    better = [_uniform(V), _uniform(V), _spike(V, 2, 12.0)]
    z, m, c = _one_request(base, [worse, better], P1)
    out = o.step(z, m, c, P1)
    assert out["commit"]["winner"][0] == 1
    assert out["commit"]["commit_pos"][0] == 1 and out["commit"]["commit_tok"][0] == 1
    assert list(out["commit"]["mask_pos"][0, :out["commit"]["mask_cnt"][0]]) == [2]

    # exact ties: equal branch scores keep [MASK] (abstain)
    z, m, c = _one_request(base, [base, base], P1)
    out = o.step(z, m, c, P1)
    assert out["commit"]["winner"][0] == -1

    # n = 0: the pivot is the only row left -> mean entropy 0, [MASK] wins on plausibility
    prm = replace(P1, lam=0.5)
    base = [_spike(V, 1, 10.0), _uniform(V)]
    z, m, c = _one_request(base, [base, base], prm)
    out = o.step(z, m, c, prm)
    assert out["pivots"]["state"][0] == 0
    assert (out["scores"]["mean_H"][0, 0] == 0).all()
    assert out["commit"]["winner"][0] == -1


def pin_exact_thresholds(o):
    """Thresholds are inclusive: P^max >= tau, mu >= tau_pivot, p >= r P^max, N_tau uses >=."""
    # V = 2 uniform: P^max = 0.5 exactly -> both rows committed at tau = 0.5
    # (with a strict test neither passes and the fallback would commit one)
    prm = Params(k_max=2, r=1.0, tau_pivot=0.5, tau=0.5, lam=0.0, n_pivots=1, tokens_per_pivot=2)
    base = [_uniform(2), _uniform(2)]
    z, m, c = _one_request(base, [base, base], prm)
    out = o.step(z, m, c, prm)
    assert out["pivots"]["n_commit"][0] == 2 and out["pivots"]["state"][0] == 1

    # V = 4 uniform, k_max = 2: mu = 0.5 exactly -> feasible at tau_pivot = 0.5;
    # r = 1: p(v) = P^max for every token -> two candidates
    prm = Params(k_max=2, r=1.0, tau_pivot=0.5, tau=0.9, lam=0.0, n_pivots=1, tokens_per_pivot=2)
    base = [_spike(4, 0, 20.0), _uniform(4), _spike(4, 3, 30.0)]
    # downstream row (position 2) in each branch: V = 4 with P^max = 0.5 exactly
    half = np.full(4, -np.inf, np.float32)
    half[[0, 1]] = 0.0
    br = [_uniform(4), _uniform(4), half]
    z, m, c = _one_request(base, [br, br], prm)
    # base position 2: P^max = 0.72 < tau stays masked; its truncated entropy
    # (0.59) is below the uniform row's ln 2, so position 1 is the pivot
    z[0, 0, 2] = np.array([0.0, -1.0, -5.0, -5.0], np.float32)
    out = o.step(z, m, c, prm)
    piv = out["pivots"]
    assert piv["state"][0] == 0 and piv["pivot_pos"][0, 0] == 1, (piv["state"], piv["pivot_pos"])
    assert list(piv["cand_tok"][0, 0]) == [0, 1]
    # N_tau at tau = 0.5: position 2 of each branch has P^max = 0.5 exactly -> counted
    prm2 = replace(prm, tau=0.5)
    sc = o.score_branches(piv, out["branch"], out["base"], z[:, 0], prm2)
    assert sc["n_tau"][0, 0, 0] == 1 and sc["n_tau"][0, 0, 1] == 1


def _binary_entropy(t):
    return -t * math.log(t) - (1 - t) * math.log(1 - t)


def pin_propositions(o):
    """Prop. 1 (N_tau >= n - floor(n H-bar / h(tau))) and Prop. 2 (margin rule) on synthetic steps."""
    rng = np.random.default_rng(13)
    for trial in range(6):
        prm = Params(k_max=8, r=0.05, tau_pivot=0.0, tau=0.9, lam=float([0.1, 0.3, 0.5][trial % 3]),
                     n_pivots=2, tokens_per_pivot=2)
        z = _lookahead_case(rng, 1, 8, 16, prm, spread=0.7)
        mpos = np.arange(8, dtype=np.int32)[None]
        cnt = np.array([8], np.int32)
        out = o.step(z, mpos, cnt, prm)
        piv = out["pivots"]
        if piv["state"][0] != 0:
            continue
        n = int(piv["rem_cnt"][0]) - 1
        for tau in (0.5, 0.7, 0.9):
            sc = o.score_branches(piv, out["branch"], out["base"], z[:, 0], replace(prm, tau=tau))
            for j in range(prm.n_pivots):
                for cslot in range(prm.tokens_per_pivot + 1):
                    if sc["n_tau"][0, j, cslot] < 0:
                        continue
                    hb = sc["mean_H"][0, j, cslot]
                    bound = max(0, n - math.floor(n * hb / _binary_entropy(tau)))
                    assert sc["n_tau"][0, j, cslot] >= bound, (trial, tau, j, cslot)
        sc = out["scores"]
        lam = float(np.float32(prm.lam))
        for j in range(prm.n_pivots):
            s = sc["score"][0, j]
            valid = [cs for cs in range(prm.tokens_per_pivot + 1) if not np.isnan(s[cs])]
            if len(valid) < 2:
                continue
            hb, la = sc["mean_H"][0, j], sc["log_a"][0, j]
            best = out["commit"]["best_slot"][0, j]
            lagr = [hb[cs] - lam * la[cs] for cs in valid]
            assert min(lagr) == hb[best] - lam * la[best] or \
                abs(min(lagr) - (hb[best] - lam * la[best])) < 1e-12
            for c1 in valid:
                for d in valid:
                    lhs = s[c1] >= s[d]
                    rhs = hb[d] - hb[c1] >= lam * (la[d] - la[c1]) - 1e-12
                    if abs(s[c1] - s[d]) > 1e-9:
                        assert lhs == rhs, (trial, j, c1, d)
            # [MASK] plausibility is the anchor's top-1 probability: a_MASK >= a_c
            assert all(la[prm.tokens_per_pivot] >= la[cs] - 1e-12 for cs in valid)


# --------------------------------------------------------------------------
# LM head followed by the row statistics (the oracle of a fused contraction)
# --------------------------------------------------------------------------

def _bf16_bits(x) -> np.ndarray:
    """bf16 bits of values that bf16 holds exactly (checked)."""
    f = np.asarray(x, dtype=np.float32)
    bits = (f.view(np.uint32) >> 16).astype(np.uint16)
    assert ((bits.astype(np.uint32) << 16).view(np.float32) == f).all(), "value not exact in bf16"
    return bits


def pin_lmhead_worked_example(o):
    """d = 2, V = 3: h = (1, 2) and W = [[1, 0], [0, 1], [1, 1]] give z = (1, 2, 3)."""
    from oracle.lmhead import lmhead_row_stats
    st = lmhead_row_stats(o, _bf16_bits([[1, 2]]), _bf16_bits([[1, 0], [0, 1], [1, 1]]), 2)
    z = np.array([1.0, 2.0, 3.0])
    p = np.exp(z - z.max()) / np.exp(z - z.max()).sum()
    lse = math.log(np.exp(z).sum())
    close(st.zmax[0], 3.0, what="zmax")
    close(st.lse[0], lse, what="lse")
    close(st.H[0], -(p * np.log(p)).sum(), what="H")
    close(st.pmax[0], p[2], what="pmax")
    assert st.argmax[0] == 2
    assert list(st.topk_idx[0, :2]) == [2, 1]
    close(st.mu[0], p[2] + p[1], what="mu")
    close(st.htrunc[0], -(p[2] * math.log(p[2]) + p[1] * math.log(p[1])), what="htrunc")


def pin_lmhead_zero_hidden(o):
    """A zero hidden state makes every logit 0: the uniform row's closed forms."""
    from oracle.lmhead import lmhead_row_stats
    rng = np.random.default_rng(3)
    V, d, k = 300, 16, 10
    w = _bf16_bits(rng.integers(-8, 9, (V, d)).astype(np.float32))
    st = lmhead_row_stats(o, _bf16_bits(np.zeros((2, d))), w, k)
    close(st.H, math.log(V), what="H")
    close(st.pmax, 1.0 / V, what="pmax")
    close(st.mu, k / V, what="mu")
    assert (st.argmax == 0).all() and (st.topk_idx[:, :k] == np.arange(k)).all()


def pin_lmhead_token_shift(o):
    """Adding one vector u to every token's weights adds h.u to every logit of the
    row: the distribution, argmax and top-k stay, zmax and lse move by h.u."""
    from oracle.lmhead import lmhead_row_stats
    rng = np.random.default_rng(4)
    n, V, d, k = 4, 200, 8, 12
    h = rng.integers(-3, 4, (n, d)).astype(np.float32)
    w = rng.integers(-4, 5, (V, d)).astype(np.float32)
    u = rng.integers(-2, 3, d).astype(np.float32)
    a = lmhead_row_stats(o, _bf16_bits(h), _bf16_bits(w), k)
    b = lmhead_row_stats(o, _bf16_bits(h), _bf16_bits(w + u), k)
    shift = h.astype(np.float64) @ u.astype(np.float64)
    close(b.zmax, a.zmax + shift, what="zmax")
    close(b.lse, a.lse + shift, tol=1e-9, what="lse")
    for name in ("H", "pmax", "mu", "htrunc"):
        close(getattr(b, name), getattr(a, name), tol=1e-9, what=name)
    assert (a.argmax == b.argmax).all() and (a.topk_idx == b.topk_idx).all()


def pin_lmhead_token_permutation(o):
    """Token v of the permuted unembedding is token perm[v] of the original: the
    argmax and top-k tokens map back through perm (distinct logits)."""
    from oracle.lmhead import lmhead_row_stats
    rng = np.random.default_rng(5)
    V, d, k = 97, 3, 7
    w = np.zeros((V, d), np.float32)
    w[:, 0] = rng.permutation(V)           # z_v = w[v, 0] for h = (1, 0, 0): distinct
    w[:, 1:] = rng.integers(-5, 6, (V, d - 1))
    h = np.array([[1, 0, 0]], np.float32)
    perm = rng.permutation(V)
    a = lmhead_row_stats(o, _bf16_bits(h), _bf16_bits(w), k)
    b = lmhead_row_stats(o, _bf16_bits(h), _bf16_bits(w[perm]), k)
    assert a.argmax[0] == int(np.argmax(w[:, 0])) and perm[b.argmax[0]] == a.argmax[0]
    assert (perm[b.topk_idx[0, :k]] == a.topk_idx[0, :k]).all()
    close(b.H, a.H, tol=1e-12, what="H")


def _attn_case(seed, n_b, n_h, C, NB, G, D, spread=1.0):
    rng = np.random.default_rng(seed)
    n = C + NB * G
    return tuple(synth.bf16_round((rng.standard_normal((n_b, n_h, n, D)) * spread).astype(np.float32))
                 for _ in range(3))


def _bits_f64(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def pin_attention_dense_mask(o):
    """The packed attention equals masked softmax attention under the dense
    token-by-token mask written out from the isolation rule (a key is visible
    when it is a context token or lies in the query's own branch; context
    queries own branch 0), for every query at once."""
    from oracle.attention import packed_attention
    C, NB, G, D, scale = 5, 3, 4, 8, 0.37
    q, k, v = _attn_case(21, 2, 2, C, NB, G, D)
    out = packed_attention(q, k, v, C, NB, G, scale)
    seg = np.array([0] * C + [1 + j for j in range(NB) for _ in range(G)])
    own = np.where(seg == 0, 1, seg)
    visible = (seg[None, :] == 0) | (seg[None, :] == own[:, None])
    qf, kf, vf = _bits_f64(q), _bits_f64(k), _bits_f64(v)
    for b in range(2):
        for h in range(2):
            s = scale * qf[b, h] @ kf[b, h].T
            s = np.where(visible, s, -np.inf)
            p = np.exp(s - s.max(axis=1, keepdims=True))
            p /= p.sum(axis=1, keepdims=True)
            close(out[b, h], p @ vf[b, h], tol=1e-12, what="dense-mask attention")


def pin_attention_branch_is_plain_attention(o):
    """Each branch's queries get exactly plain (unmasked) attention over the
    sequence [context, that branch], and the context's queries plain attention
    over [context, branch 0]: a library routine (torch's scaled dot-product
    attention, fp64) on the unpacked sequence."""
    import torch
    from oracle.attention import packed_attention
    C, NB, G, D = 6, 4, 5, 16
    scale = 1.0 / math.sqrt(D)
    q, k, v = _attn_case(22, 1, 3, C, NB, G, D, spread=2.0)
    out = packed_attention(q, k, v, C, NB, G, scale)
    qf, kf, vf = (torch.from_numpy(_bits_f64(x)) for x in (q, k, v))
    for j in range(NB):
        idx = list(range(C)) + list(range(C + j * G, C + (j + 1) * G))
        ref = torch.nn.functional.scaled_dot_product_attention(qf[:, :, idx], kf[:, :, idx], vf[:, :, idx]).numpy()
        close(out[:, :, C + j * G:C + (j + 1) * G], ref[:, :, C:], tol=1e-12, what=f"branch {j}")
        if j == 0:
            close(out[:, :, :C], ref[:, :, :C], tol=1e-12, what="context")


def pin_attention_isolation(o):
    """Changing one branch's keys and values changes that branch's outputs
    only: the context and every other branch are bit-identical."""
    from oracle.attention import packed_attention
    C, NB, G, D = 4, 4, 3, 8
    q, k, v = _attn_case(23, 1, 2, C, NB, G, D)
    base = packed_attention(q, k, v, C, NB, G, 0.5)
    k2, v2 = k.copy(), v.copy()
    rows = slice(C + 2 * G, C + 3 * G)
    k2[:, :, rows] = synth.bf16_round(np.random.default_rng(24).standard_normal(k2[:, :, rows].shape).astype(np.float32))
    v2[:, :, rows] = synth.bf16_round(np.random.default_rng(25).standard_normal(v2[:, :, rows].shape).astype(np.float32))
    moved = packed_attention(q, k2, v2, C, NB, G, 0.5)
    keep = np.ones(C + NB * G, bool)
    keep[rows] = False
    assert np.array_equal(base[:, :, keep], moved[:, :, keep]), "another branch saw branch 2"
    assert not np.allclose(base[:, :, rows], moved[:, :, rows]), "branch 2 ignores its own keys"


def pin_attention_closed_forms(o):
    """Identical keys give uniform weights: the output is the mean of the
    visible values. A key whose score leads every other by 60 nats gives its
    own value."""
    from oracle.attention import packed_attention
    C, NB, G, D = 3, 3, 2, 4
    q, k, v = _attn_case(26, 1, 1, C, NB, G, D)
    k[:] = k[:, :, :1]
    out = packed_attention(q, k, v, C, NB, G, 0.8)
    vf = _bits_f64(v)[0, 0]
    for j in range(NB):
        vis = list(range(C)) + list(range(C + j * G, C + (j + 1) * G))
        close(out[0, 0, C + j * G:C + (j + 1) * G], np.broadcast_to(vf[vis].mean(axis=0), (G, D)), tol=1e-12,
              what=f"uniform weights, branch {j}")
    close(out[0, 0, :C], np.broadcast_to(vf[list(range(C + G))].mean(axis=0), (C, D)), tol=1e-12, what="context")
    # one dominant key in branch 1 (token C + G + 1): q . k = 60 / scale more than any other
    q2, k2, v2 = _attn_case(27, 1, 1, C, NB, G, D)
    qf = np.zeros((1, 1, C + NB * G, D))
    qf[..., 0] = 1.0
    kf = np.zeros_like(qf)
    kf[0, 0, C + G + 1, 0] = 60.0
    out = packed_attention(_bf16_bits(qf), _bf16_bits(kf), v2, C, NB, G, 1.0)
    close(out[0, 0, C + G:C + 2 * G], np.broadcast_to(_bits_f64(v2)[0, 0, C + G + 1], (G, D)), tol=1e-20,
          what="dominant key")


ALL_PINS = [
    pin_uniform_rows, pin_spike_rows, pin_two_level_rows, pin_rank_order, pin_library_crosscheck,
    pin_synth_rows_crosscheck, pin_invariants, pin_neg_inf_entries, pin_select_brute_force,
    pin_score_commit_brute_force, pin_score_closed_form, pin_control_flow, pin_exact_thresholds,
    pin_propositions, pin_lmhead_worked_example, pin_lmhead_zero_hidden, pin_lmhead_token_shift,
    pin_lmhead_token_permutation, pin_attention_dense_mask, pin_attention_branch_is_plain_attention,
    pin_attention_isolation, pin_attention_closed_forms,
]
