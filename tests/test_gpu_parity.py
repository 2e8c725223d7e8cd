"""GPU path vs the CPU oracle, through the C ABI (``-m gpu``).

* generator: the device twin writes the same bits as the host generator;
* row statistics: every output of ``rps_score_step`` in both modes, over
  dtypes, ragged vocabularies, row counts that split rows into many pieces,
  k from 1 to 32, and adversarial rows (ties, -inf, huge magnitudes);
* full steps on shrunken workloads: every stage against the oracle, over a
  hyper-parameter matrix that reaches every branch of Algorithm 1;
* full-size workloads: sampled rows against the oracle, and the decision
  stages re-run by the oracle on the GPU's own statistics;
* device-side error reporting on bad data.
"""
import numpy as np
import pytest
import torch

from gpu_harness import (GpuStep, assert_close, compare_stats, padded_tensor, piv_np, stats_np, to_device,
                         workload_inputs)
from oracle import default as oracle_default
from paper_2608_11742_gb300 import configs, synth
from paper_2608_11742_gb300.configs import Params

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rps():
    from paper_2608_11742_gb300.build import build
    build()
    from paper_2608_11742_gb300 import rps as r
    assert torch.cuda.is_available()
    return r


# ----------------------------------------------------------------------------- generator
def test_device_generator_matches_host(rps):
    for w, V, L in ((configs.TINY, None, None), (configs.SERVE.scaled(n_req=2, ragged=(3, 6)), 5000, 8)):
        w = w.scaled(**({} if V is None else dict(V=V, L=L)))
        valid = w.valid_rows()
        host = synth.make_logits(w.seed, w.n_req, w.n_branch, w.L, w.V, w.mixture, w.dtype, valid=valid)
        dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
        dev = torch.empty((w.n_req, 1 + w.n_branch, w.L, w.V), dtype=dt, device="cuda")
        synth.device_fill(dev, w.seed, w.mixture,
                          valid=None if valid is None else torch.from_numpy(valid).cuda())
        got = dev.view(torch.int16).cpu().numpy().view(np.uint16) if w.dtype == "bf16" else dev.cpu().numpy()
        assert (got.view(np.uint8) == host.view(np.uint8)).all(), w.name


def test_device_generator_full_size_rows(rps):
    w = configs.STEP
    dev = torch.empty((1, 1 + w.n_branch, w.L, w.V), dtype=torch.bfloat16, device="cuda")
    scale = torch.full((1, w.L), 1.0, device="cuda")
    scale[0, 5] = 1.25
    epoch = torch.zeros((1, w.L), dtype=torch.int32, device="cuda")
    epoch[0, 7] = 3
    synth.device_fill(dev, w.seed, w.mixture, step=2, scale=scale, epoch=epoch)
    rng = np.random.default_rng(0)
    for b, p in [(0, 5), (3, 5), (0, 7), (8, 7)] + [(int(rng.integers(0, 9)), int(rng.integers(0, 256)))
                                                  for _ in range(6)]:
        row = dev[0, b, p].view(torch.int16).cpu().numpy().view(np.uint16)
        want = synth.row_logits(w.seed, w.V, 0, b, p, w.mixture, "bf16", scale=float(scale[0, p]),
                                epoch=int(epoch[0, p]), step=2)
        assert (row == want).all(), (b, p)


# ----------------------------------------------------------------------------- row statistics
def _adversarial_rows(rng, n, V, bf16):
    z = rng.standard_normal((n, V)).astype(np.float32) * np.float32(2.0)
    for i in range(n):
        kind = i % 7
        if kind == 1:
            z[i] = 0.0                                  # all equal: ties everywhere
        elif kind == 2:
            z[i, rng.choice(V, V // 3, replace=False)] = -np.inf   # masked vocabulary
        elif kind == 3:
            z[i] *= np.float32(3e3)                     # large magnitudes
        elif kind == 4:
            z[i, rng.integers(0, V)] += np.float32(40.0)   # one dominant token
        elif kind == 5:
            z[i] = np.round(z[i])                       # heavy ties at small integers
        elif kind == 6:
            z[i, -1] = z[i].max() + 1                   # maximum in the ragged tail
    if bf16:
        return synth.bf16_round(z)
    return z


ROW_CASES = [
    # (dtype, V, n_rows, k)
    ("f32", 4096, 300, 10),
    ("bf16", 4096, 300, 10),
    ("bf16", 1003, 64, 32),      # V not a multiple of the 8-element unit
    ("f32", 1001, 64, 1),
    ("bf16", 126464, 3, 10),     # few long rows: each split over many warps
    ("bf16", 151936, 2, 16),
    ("f32", 126464, 3, 10),      # a sketch longer than one batch of loads per lane
    ("bf16", 40, 33, 32),        # rows shorter than one batch
    ("f32", 17, 5, 17),          # k == V
]


@pytest.mark.parametrize("dtype,V,n,k", ROW_CASES, ids=[f"{d}-V{V}-n{n}-k{k}" for d, V, n, k in ROW_CASES])
def test_row_stats_parity(rps, dtype, V, n, k):
    rng = np.random.default_rng(V + n + k)
    rows = _adversarial_rows(rng, n, V, dtype == "bf16")
    logits = rows.reshape(1, 1, n, V)
    t = padded_tensor(logits)
    o = oracle_default()
    ref = o.row_stats(rows, k)
    desc = torch.tensor([[0, 0, i] for i in range(n)], dtype=torch.int32, device="cuda")
    prm = Params(k_max=k)
    for topk in (True, False):
        buf = rps.RowStatsBuf.alloc(n, k if topk else 0, "cuda")
        ws = torch.zeros(rps.rps_workspace_bytes(n, V, k if topk else 0, t.dtype), dtype=torch.uint8, device="cuda")
        for rep in range(2):  # the second call checks the workspace is left ready
            rps.rps_score_step(t, desc, None, 1, n, prm, buf, ws)
            status, detail = rps.rps_poll_device_status()
            assert status == rps.RPS_OK, hex(detail)
            g = stats_np(buf)
            compare_stats(g, ref, np.arange(n), k if topk else 0, f"{dtype} V={V} topk={topk} rep={rep}")


def test_row_stats_mask_form_and_skips(rps):
    """Mask-form row lists, skipped entries (pos < 0) and NaN rows that must never be read."""
    rng = np.random.default_rng(3)
    n_req, L, V, k = 3, 10, 2048, 10
    z = rng.standard_normal((n_req, 2, L, V)).astype(np.float32)
    mask_pos = np.full((n_req, L), -1, np.int32)
    cnt = np.array([4, 0, 7], np.int32)
    for q in range(n_req):
        sel = np.sort(rng.choice(L, cnt[q], replace=False))
        mask_pos[q, :cnt[q]] = sel
        unmasked = np.setdiff1d(np.arange(L), sel)
        z[q, :, unmasked] = np.nan
    t = to_device(synth.bf16_round(z))
    zb = synth.bf16_round(z)
    buf = rps.RowStatsBuf.alloc(n_req * L, k, "cuda")
    ws = torch.zeros(rps.rps_workspace_bytes(n_req * L, V, k, t.dtype), dtype=torch.uint8, device="cuda")
    rps.rps_score_step(t, None, torch.from_numpy(cnt).cuda(), n_req, L, Params(k_max=k), buf, ws,
                       mask_pos=torch.from_numpy(mask_pos).cuda(), mask_branch=1)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_OK, hex(detail)
    g = stats_np(buf)
    o = oracle_default()
    ref = o.base_stats(zb, mask_pos, cnt, k, branch=1)
    slots = [q * L + i for q in range(n_req) for i in range(cnt[q])]
    compare_stats(g, ref, slots, k, "mask form")
    untouched = np.setdiff1d(np.arange(n_req * L), slots)
    assert np.isnan(g.H[untouched]).all(), "slots outside the mask were written"

    # explicit list with a skipped entry in the middle
    desc = torch.tensor([[0, 0, 1], [0, 0, -1], [2, 1, 3]], dtype=torch.int32, device="cuda")
    z2 = rng.standard_normal((3, 2, 4, V)).astype(np.float32)
    t2 = to_device(z2)
    buf2 = rps.RowStatsBuf.alloc(3, 0, "cuda")
    ws2 = torch.zeros(rps.rps_workspace_bytes(3, V, 0, t2.dtype), dtype=torch.uint8, device="cuda")
    rps.rps_score_step(t2, desc, None, 1, 3, Params(k_max=k), buf2, ws2)
    assert rps.rps_poll_device_status()[0] == rps.RPS_OK
    g2 = stats_np(buf2)
    assert np.isnan(g2.H[1])
    r2 = o.row_stats(np.stack([z2[0, 0, 1], z2[2, 1, 3]]), 0)
    assert_close(g2.H[[0, 2]], r2.H, "explicit list H")


def test_device_errors_are_reported(rps):
    V = 256
    z = np.random.default_rng(1).standard_normal((1, 1, 4, V)).astype(np.float32)
    z[0, 0, 2, 7] = np.nan
    t = to_device(z)
    buf = rps.RowStatsBuf.alloc(3, 0, "cuda")
    ws = torch.zeros(rps.rps_workspace_bytes(3, V, 0, t.dtype), dtype=torch.uint8, device="cuda")
    desc = torch.tensor([[0, 0, 0], [0, 0, 9], [0, 0, 2]], dtype=torch.int32, device="cuda")  # pos 9 out of range
    rps.rps_score_step(t, desc, None, 1, 3, Params(), buf, ws)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_ERR_DEVICE
    assert detail & rps.DEVERR_ROW_INDEX and detail & rps.DEVERR_NONFINITE
    g = stats_np(buf)
    assert np.isfinite(g.H[0]) and np.isnan(g.H[1]) and np.isnan(g.H[2]) and g.argmax[2] == -1
    assert rps.rps_poll_device_status()[0] == rps.RPS_OK, "the error word is cleared by polling"
    # a mask count above capacity is clamped and flagged
    cnt = torch.tensor([9], dtype=torch.int32, device="cuda")
    mpos = torch.arange(4, dtype=torch.int32, device="cuda").view(1, 4)
    buf4 = rps.RowStatsBuf.alloc(4, 0, "cuda")
    z[0, 0, 2, 7] = 0.0
    ws4 = torch.zeros(rps.rps_workspace_bytes(4, V, 0, torch.float32), dtype=torch.uint8, device="cuda")
    rps.rps_score_step(to_device(z), None, cnt, 1, 4, Params(), buf4, ws4, mask_pos=mpos)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_ERR_DEVICE and detail & rps.DEVERR_MASK


def test_topk_rows_with_few_finite_logits(rps):
    """Rows with fewer finite logits than k (the top-k bound is -inf, so every cell,
    the sketch's -inf padding included, is a candidate, and the list fills with -inf
    entries in token order) and with a few more, in top-k mode."""
    for dtype, V, k in (("bf16", 5003, 10), ("f32", 2049, 32)):
        rng = np.random.default_rng(V + k)
        counts = [1, 3, k - 1, k, k + 1, 40]
        rows = np.full((len(counts), V), -np.inf, np.float32)
        for i, c in enumerate(counts):
            rows[i, rng.choice(V, c, replace=False)] = rng.standard_normal(c).astype(np.float32) * np.float32(3.0)
        if dtype == "bf16":
            rows = synth.bf16_round(rows)
        n = len(counts)
        t = padded_tensor(rows.reshape(1, 1, n, V))
        ref = oracle_default().row_stats(rows, k)
        desc = torch.tensor([[0, 0, i] for i in range(n)], dtype=torch.int32, device="cuda")
        buf = rps.RowStatsBuf.alloc(n, k, "cuda")
        ws = torch.zeros(rps.rps_workspace_bytes(n, V, k, t.dtype), dtype=torch.uint8, device="cuda")
        rps.rps_score_step(t, desc, None, 1, n, Params(k_max=k), buf, ws)
        status, detail = rps.rps_poll_device_status()
        assert status == rps.RPS_OK, hex(detail)
        compare_stats(stats_np(buf), ref, np.arange(n), k, f"{dtype} V={V} few finite")


def test_topk_mode_device_errors(rps):
    """Top-k mode: a NaN row gives NaN statistics, an empty list and argmax -1; a bad
    descriptor leaves its slot untouched; a mask count above capacity is clamped."""
    V, k = 3001, 8
    rng = np.random.default_rng(11)
    z = rng.standard_normal((1, 1, 4, V)).astype(np.float32)
    z[0, 0, 2, 7] = np.nan
    t = padded_tensor(z)
    buf = rps.RowStatsBuf.alloc(3, k, "cuda")
    ws = torch.zeros(rps.rps_workspace_bytes(3, V, k, t.dtype), dtype=torch.uint8, device="cuda")
    desc = torch.tensor([[0, 0, 0], [0, 0, 9], [0, 0, 2]], dtype=torch.int32, device="cuda")  # pos 9 out of range
    rps.rps_score_step(t, desc, None, 1, 3, Params(k_max=k), buf, ws)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_ERR_DEVICE
    assert detail & rps.DEVERR_ROW_INDEX and detail & rps.DEVERR_NONFINITE
    g = stats_np(buf)
    compare_stats(g, oracle_default().row_stats(z[0, 0, :1], k), [0], k, "finite row")
    assert np.isnan(g.H[1]) and g.argmax[1] == -1 and (g.topk_idx[1] == -1).all(), "bad descriptor: untouched"
    assert np.isnan(g.H[2]) and g.argmax[2] == -1 and np.isnan(g.mu[2]) and np.isnan(g.htrunc[2])
    assert (g.topk_idx[2] == -1).all() and np.isnan(g.topk_logit[2]).all()
    # a mask count above capacity is clamped (all four rows scored) and flagged
    z[0, 0, 2, 7] = 0.0
    cnt = torch.tensor([9], dtype=torch.int32, device="cuda")
    mpos = torch.arange(4, dtype=torch.int32, device="cuda").view(1, 4)
    buf4 = rps.RowStatsBuf.alloc(4, k, "cuda")
    ws4 = torch.zeros(rps.rps_workspace_bytes(4, V, k, torch.float32), dtype=torch.uint8, device="cuda")
    rps.rps_score_step(padded_tensor(z), None, cnt, 1, 4, Params(k_max=k), buf4, ws4, mask_pos=mpos)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_ERR_DEVICE and detail & rps.DEVERR_MASK
    compare_stats(stats_np(buf4), oracle_default().row_stats(z[0, 0], k), np.arange(4), k, "clamped count")


# ----------------------------------------------------------------------------- full steps
PARAM_MATRIX = [
    Params(),                                                 # paper defaults (tau_pivot 0.9)
    configs.EXERCISE,                                         # every row feasible
    Params(tau_pivot=0.003, lam=0.3),
    Params(tau_pivot=0.03, tau=0.5, lam=0.5),
    Params(tau_pivot=0.0, tau=0.5, lam=0.0),
    Params(k_max=32, r=0.05, tau_pivot=0.0, n_pivots=1, tokens_per_pivot=32),   # adaptive C, one pivot
    Params(k_max=5, r=0.3, tau_pivot=0.0, lam=0.2, n_pivots=8, tokens_per_pivot=3),
    Params(tau=0.05, tau_pivot=0.0, lam=5.0),                 # plausibility dominates: abstain
    # the other commit rules of Eq. 2 and the ablation pivot strategies
    Params(tau_pivot=0.0, pivot_rule=1),                      # max-confidence pivots
    Params(tau_pivot=0.9, pivot_rule=2),                      # max-entropy pivots, no mass constraint
    Params(tau_pivot=0.0, commit_rule=1, commit_k=2),         # top-k confidence commits
    Params(tau_pivot=0.003, commit_rule=2, commit_k=3, pivot_rule=2),  # lowest-entropy commits
]

STEP_CASES = [
    ("tiny", configs.TINY, dict()),
    ("step-small", configs.STEP, dict(V=8192, L=64)),
    ("step-10-small", configs.STEP_10, dict(V=8192, L=64)),
    ("long-small", configs.LONG, dict(V=6000, L=96)),
    ("serve-small", configs.SERVE, dict(V=5003, L=40, n_req=4, ragged=(4, 40))),
    ("block-small", configs.BLOCK, dict(V=4096, n_req=12)),
]


@pytest.mark.parametrize("name,w,shrink", STEP_CASES, ids=[c[0] for c in STEP_CASES])
def test_step_parity(rps, name, w, shrink):
    w1, logits, mpos, mcnt = workload_inputs(w, **shrink)
    for prm in PARAM_MATRIX:
        if (prm.n_pivots, prm.tokens_per_pivot) == (4, 2):
            prm = w1.params(prm)
        if prm.n_branch == w1.n_branch:
            z = logits
        else:  # this parameter set packs a different number of lookahead branches
            z = synth.make_logits(w1.seed, w1.n_req, prm.n_branch, w1.L, w1.V, w1.mixture, w1.dtype,
                                  valid=w1.valid_rows())
        GpuStep(z, mpos, mcnt, prm).run_and_compare(f"{name} {prm}")


def test_step_parity_control_paths(rps):
    """Search, both skips, done, commit and abstain all occur, each matching the oracle."""
    states, winners = set(), set()
    w, logits, mpos, mcnt = workload_inputs(configs.TINY)
    flat = logits.copy()
    flat[:, 1:] = logits[:, :1] * np.float32(0.25)  # branches flatter than the anchor: [MASK] wins
    cases = [(logits, configs.EXERCISE), (logits, configs.PAPER), (logits, Params(tau=0.0, tau_pivot=0.0)),
             (flat, configs.EXERCISE), (logits, Params(tau=0.05, tau_pivot=0.0, lam=5.0))]
    for z, prm in cases:
        out = GpuStep(z, mpos, mcnt, w.params(prm)).run_and_compare(f"tiny {prm}")
        states.update(int(x) for x in out["piv"]["state"])
        winners.update(int(x) if x < 0 else 0 for x in out["commit"]["winner"])
    for name, w, shrink in (STEP_CASES[1], STEP_CASES[5]):
        w1, logits, mpos, mcnt = workload_inputs(w, **dict(shrink))
        out = GpuStep(logits, mpos, mcnt, w1.params(configs.EXERCISE)).run_and_compare(name)
        states.update(int(x) for x in out["piv"]["state"])
        winners.update(int(x) if x < 0 else 0 for x in out["commit"]["winner"])
    assert {0, 1}.issubset(states) and states & {2, 3}, states
    assert {0, -1, -2, -3}.issubset(winners), winners


# ----------------------------------------------------------------------------- full size
FULL = [("step", configs.STEP), ("step-10", configs.STEP_10), ("block", configs.BLOCK), ("serve", configs.SERVE),
        ("long", configs.LONG)]


@pytest.mark.parametrize("name,w", FULL, ids=[f[0] for f in FULL])
def test_full_size_sampled(rps, name, w):
    """Full-size step in the launch configuration the benchmark times: sampled rows
    against the oracle, decisions re-derived by the oracle from the GPU's statistics."""
    prm = w.params(configs.EXERCISE)
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    logits = torch.empty((w.n_req, 1 + w.n_branch, w.L, w.V), dtype=dt, device="cuda")
    valid = w.valid_rows()
    synth.device_fill(logits, w.seed, w.mixture, valid=None if valid is None else torch.from_numpy(valid).cuda())
    mpos, mcnt = w.mask()
    d_mpos, d_mcnt = torch.from_numpy(mpos).cuda(), torch.from_numpy(mcnt).cuda()
    step = rps.Step(w.n_req, w.L, w.V, prm, "cuda", dt)
    step.run(logits, d_mpos, d_mcnt)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_OK, hex(detail)
    o = oracle_default()
    base = stats_np(step.base)
    piv = piv_np(step.piv)
    rng = np.random.default_rng(0)

    # sampled base rows (top-k mode) against the oracle on host-generated rows
    slots = [(q, k) for q in range(w.n_req) for k in range(int(mcnt[q]))]
    pick = [slots[i] for i in rng.choice(len(slots), min(12, len(slots)), replace=False)]
    rows = np.stack([synth.row_logits(w.seed, w.V, q, 0, int(mpos[q, k]), w.mixture, w.dtype) for q, k in pick])
    ref = o.row_stats(rows, prm.k_max)
    sl = np.array([q * w.L + k for q, k in pick])
    for name_ in ("zmax", "lse", "H", "pmax", "mu", "htrunc"):
        assert_close(getattr(base, name_)[sl], getattr(ref, name_), f"{name} base {name_}")
    assert (base.argmax[sl] == ref.argmax).all()
    assert (base.topk_idx[sl] == ref.topk_idx).all()

    # sampled lookahead rows
    NB = prm.n_branch
    br = stats_np(step.branch)
    entries = [(q, i) for q in range(w.n_req) for i in range(int(piv["n_branch_rows"][q]))]
    if entries:
        pick = [entries[i] for i in rng.choice(len(entries), min(12, len(entries)), replace=False)]
        rows = []
        for q, i in pick:
            rq, rb, rp = (int(x) for x in piv["branch_rows"][q, i])
            rows.append(synth.row_logits(w.seed, w.V, rq, rb, rp, w.mixture, w.dtype))
        ref = o.row_stats(np.stack(rows), 0)
        sl = np.array([q * NB * w.L + i for q, i in pick])
        for name_ in ("zmax", "lse", "H", "pmax"):
            assert_close(getattr(br, name_)[sl], getattr(ref, name_), f"{name} branch {name_}")
        assert (br.argmax[sl] == ref.argmax).all()

    # decision stages: the oracle on the GPU's statistics gives the GPU's decisions
    from gpu_harness import MAX_EXCUSED, compare_commit, compare_scores, compare_select, scores_np, commit_np
    piv_o = o.select_pivots(mpos, mcnt, base, prm)
    compare_select(piv, piv_o, mcnt, w.L, prm.n_pivots, prm.tokens_per_pivot, {}, f"{name} select")
    anchor = logits[:, 0]
    if w.dtype == "bf16":
        anchor_np = anchor.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    else:
        anchor_np = anchor.contiguous().cpu().numpy()
    sc_o = o.score_branches(piv, br, base, anchor_np, prm)
    sc_g = scores_np(step.scores)
    compare_scores(sc_g, sc_o, prm, f"{name} scores")
    cm_o = o.commit(piv, sc_o, prm)
    assert len(compare_commit(commit_np(step.commit), cm_o, sc_g, sc_o, piv, prm, f"{name} commit")) <= MAX_EXCUSED
    assert (piv["state"] == 0).any(), "the exercise setting must reach the lookahead search"
