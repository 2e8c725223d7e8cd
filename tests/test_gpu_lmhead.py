"""LM head with the row statistics in its epilogue (rps_lmhead_row_stats).

The statistics of each row's logits z = h W^T are checked three ways:
1. the logits the epilogue folded (stored for the test) against the oracle's
   product, taken in fp64 and rounded once to fp32, within a bound of the
   accumulation error (1e-4 of sum |h_i w_i|), far below what a wrong operand
   descriptor or a dropped K slice gives;
2. the statistics against the streaming row-statistics kernel on those same
   fp32 logits: argmax and top-k identical, the rest within tolerance;
3. the statistics against the oracle (oracle/lmhead.py) within tolerance;
   argmax and top-k exact, except where the oracle's logits of the two tokens
   that trade places differ by less than twice the row's measured logit error.
"""
import numpy as np
import pytest
import torch

from gpu_harness import ATOL, RTOL, assert_close, compare_stats, stats_np
from oracle import default as oracle_default
from oracle.lmhead import bf16_to_f64, lmhead_logits
from paper_2608_11742_gb300 import rps, synth

pytestmark = pytest.mark.gpu


class Prm:
    def __init__(self, k):
        self.k_max, self.r, self.tau_pivot, self.tau, self.lam, self.n_pivots, self.tokens_per_pivot = \
            max(k, 1), 0.1, 0.0, 0.05, 0.1, 1, 1


def dev_bf16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def run_lmhead(h_bits, w_bits, k, logits=True):
    n, V = h_bits.shape[0], w_bits.shape[0]
    out = rps.RowStatsBuf.alloc(n, k, "cuda")
    ws = torch.empty(rps.rps_lmhead_workspace_bytes(n, V, k), dtype=torch.uint8, device="cuda")
    rps.rps_workspace_init(ws)
    lg = torch.full((n, V), float("nan"), device="cuda") if logits else None
    rps.rps_lmhead_row_stats(dev_bf16(h_bits), dev_bf16(w_bits), Prm(k) if k else None, out, ws, lg)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_OK, hex(detail)
    return out, lg, ws


def check(h_bits, w_bits, k, rows=None):
    n, V = h_bits.shape[0], w_bits.shape[0]
    out, lg, _ = run_lmhead(h_bits, w_bits, k)
    g = stats_np(out)
    lg = lg.cpu().numpy()
    rows = np.arange(n) if rows is None else np.asarray(rows)
    # 1. the folded logits against the oracle's product
    zo = lmhead_logits(h_bits[rows], w_bits)
    scale = np.abs(bf16_to_f64(h_bits[rows])) @ np.abs(bf16_to_f64(w_bits)).T
    err = np.abs(lg[rows].astype(np.float64) - zo)
    assert np.all(err <= 1e-4 * scale + 1e-6), f"logit error {err.max():.3e} against sum |h w| {scale.max():.3e}"
    # 2. the statistics against the streaming kernel on the same logits
    t = torch.from_numpy(lg).cuda().view(1, 1, n, V)
    ref_buf = rps.RowStatsBuf.alloc(n, k, "cuda")
    ws2 = torch.zeros(rps.rps_workspace_bytes(n, V, k, torch.float32), dtype=torch.uint8, device="cuda")
    rl = torch.tensor([[0, 0, r] for r in range(n)], dtype=torch.int32, device="cuda")
    rps.rps_score_step(t, rl, None, 1, n, Prm(k), ref_buf, ws2)
    assert rps.rps_poll_device_status() == (rps.RPS_OK, 0)
    compare_stats(g, stats_np(ref_buf), rows, k, "lmhead vs streaming kernel on its logits")
    # 3. the statistics against the oracle
    o = oracle_default().row_stats(zo.astype(np.float32), k)
    for name in ("zmax", "lse", "H", "pmax") + (("mu", "htrunc") if k else ()):
        assert_close(getattr(g, name)[rows], getattr(o, name), f"lmhead {name}")
    row_err = err.max(axis=1)
    for i, r in enumerate(rows):
        if g.argmax[r] != o.argmax[i]:
            assert abs(zo[i, g.argmax[r]] - zo[i, o.argmax[i]]) <= 2 * row_err[i], f"row {r} argmax"
        if k:
            for j in np.nonzero(g.topk_idx[r, :k] != o.topk_idx[i, :k])[0]:
                assert abs(zo[i, g.topk_idx[r, j]] - zo[i, o.topk_idx[i, j]]) <= 2 * row_err[i], f"row {r} rank {j}"
    return err.max()


@pytest.mark.parametrize("n,d,V,k", [
    (200, 128, 1000, 10),     # ragged rows and vocabulary, one tile per CTA
    (64, 64, 151936, 1),      # one K slice; the last vocabulary tile holds 128 tokens
    (130, 4096, 8192, 32),    # 64 K slices per tile, the longest list
    (1000, 512, 32768, 0),    # statistics only, eight row tiles, several tiles per CTA
])
def test_lmhead_parity(n, d, V, k):
    h, w = synth.lmhead_inputs(11, n, V, d)
    check(h, w, k)


@pytest.mark.parametrize("n", [300, 256])
def test_lmhead_full_vocabulary_sampled_rows(n):
    """n rows x vocabulary 126,464, twelve rows against the oracle: three row
    tiles (300 rows), or two (256 rows, the shape of a one-request step's base
    rows), with several vocabulary tiles per CTA through both accumulators."""
    d, V, k = 256, 126464, 10
    h, w = synth.lmhead_inputs(12, n, V, d)
    rows = np.random.default_rng(0).choice(n, 12, replace=False)
    check(h, w, k, rows)


def test_lmhead_wait_timeout_is_reported_and_the_workspace_recovers():
    """Every bounded wait gives up at once (testing hook): reported, nothing
    hangs, TMEM is released; the unhealthy workspace is refused; re-zeroed it works."""
    n, d, V, k = 130, 128, 2048, 10
    h, w = synth.lmhead_inputs(13, n, V, d)
    out = rps.RowStatsBuf.alloc(n, k, "cuda")
    ws = torch.empty(rps.rps_lmhead_workspace_bytes(n, V, k), dtype=torch.uint8, device="cuda")
    rps.rps_workspace_init(ws)
    hd, wd = dev_bf16(h), dev_bf16(w)
    rps.rps_debug_set_ring_wait_ns(0)
    try:
        rps.rps_lmhead_row_stats(hd, wd, Prm(k), out, ws)
        status, detail = rps.rps_poll_device_status()
    finally:
        rps.rps_debug_set_ring_wait_ns(2**64 - 1)
    assert status == rps.RPS_ERR_DEVICE and detail & rps.DEVERR_TIMEOUT, hex(detail)
    stale = rps.RowStatsBuf.alloc(n, k, "cuda")
    rps.rps_lmhead_row_stats(hd, wd, Prm(k), stale, ws)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_ERR_DEVICE and detail & rps.DEVERR_WORKSPACE and not detail & rps.DEVERR_TIMEOUT
    assert torch.isnan(stale.H).all()
    rps.rps_workspace_init(ws)
    good = rps.RowStatsBuf.alloc(n, k, "cuda")
    rps.rps_lmhead_row_stats(hd, wd, Prm(k), good, ws)
    assert rps.rps_poll_device_status() == (rps.RPS_OK, 0)
    o = oracle_default().row_stats(lmhead_logits(h, w), k)
    assert_close(stats_np(good).H, o.H, "H after re-zeroing")


@pytest.mark.parametrize("n,d,V,k", [(200, 128, 1000, 10), (300, 256, 126464, 16), (64, 64, 151936, 0)])
def test_lmhead_packed_unembedding_gives_the_same_bits(n, d, V, k):
    """The packed tile layout holds the same operands in the order the tensor
    cores read them: every statistic is bit-identical to the row-major path's."""
    h, w = synth.lmhead_inputs(14, n, V, d)
    hd, wd = dev_bf16(h), dev_bf16(w)
    packed = rps.rps_lmhead_pack_unembed(wd)
    outs = []
    for pk in (None, packed):
        out = rps.RowStatsBuf.alloc(n, k, "cuda")
        ws = torch.empty(rps.rps_lmhead_workspace_bytes(n, V, k), dtype=torch.uint8, device="cuda")
        rps.rps_workspace_init(ws)
        rps.rps_lmhead_row_stats(hd, wd, Prm(k) if k else None, out, ws, packed=pk)
        assert rps.rps_poll_device_status() == (rps.RPS_OK, 0)
        outs.append(out)
    from dataclasses import fields
    for f in fields(outs[0]):
        a, b = getattr(outs[0], f.name), getattr(outs[1], f.name)
        if a is None:
            continue
        assert torch.equal(a.nan_to_num(-7.0) if a.is_floating_point() else a,
                           b.nan_to_num(-7.0) if b.is_floating_point() else b), f.name
