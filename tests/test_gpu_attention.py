"""Branch-isolating packed-lookahead attention (rps_packed_attention_fwd)
against the oracle (oracle/attention.py).

Tolerance, from the arithmetic: the kernel rounds each probability to bf16
before it weights the values (relative error 2^-9) and rounds the output to
bf16 (2^-9), with fp32 scores and sums. So |out - ref| <= 2^-9 (sum_k p_k
|v_k|) + 2^-9 |ref| up to fp32 terms; the test allows 2^-8 of each. The first
term is the oracle's attention over |v| (the values with their sign bit
cleared). Isolation is also checked on the GPU bit for bit: changing one
branch's keys and values leaves every other output unchanged.
"""
import numpy as np
import pytest
import torch

from oracle.attention import packed_attention
from paper_2608_11742_gb300 import rps, synth

pytestmark = pytest.mark.gpu

D = 128


def inputs(seed, n_b, n_h, C, NB, G, key_growth=0.0):
    rng = np.random.default_rng(seed)
    n = C + NB * G
    q = rng.standard_normal((n_b, n_h, n, D)).astype(np.float32)
    k = rng.standard_normal((n_b, n_h, n, D)).astype(np.float32)
    v = rng.standard_normal((n_b, n_h, n, D)).astype(np.float32)
    if key_growth:  # scores that grow tile after tile: the running reference is raised, O rescaled
        k *= (1.0 + key_growth * (np.arange(n) // 128))[None, None, :, None].astype(np.float32)
    return synth.bf16_round(q), synth.bf16_round(k), synth.bf16_round(v)


def dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def run_gpu(q, k, v, C, NB, G, scale):
    out = torch.empty(q.shape, dtype=torch.bfloat16, device="cuda")
    vt = np.ascontiguousarray(np.swapaxes(v, 2, 3))
    rps.rps_packed_attention_fwd(dev(q), dev(k), dev(vt), out, C, NB, G, scale)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_OK, hex(detail)
    return out.float().cpu().numpy().astype(np.float64)


def check(q, k, v, C, NB, G, scale):
    g = run_gpu(q, k, v, C, NB, G, scale)
    ref = packed_attention(q, k, v, C, NB, G, scale)
    weighted_abs = packed_attention(q, k, v & np.uint16(0x7FFF), C, NB, G, scale)
    tol = 2.0 ** -8 * (weighted_abs + np.abs(ref)) + 1e-6
    bad = np.abs(g - ref) > tol
    assert not bad.any(), (f"{bad.sum()} outputs out of tolerance, worst {np.abs(g - ref)[bad].max():.3e} "
                           f"at {np.argwhere(bad)[:3].tolist()}")
    return g


@pytest.mark.parametrize("n_b,n_h,C,NB,G", [
    (1, 2, 128, 3, 128),   # whole tiles
    (2, 3, 200, 4, 40),    # ragged context and branches: the last key tile of each masks the rest
    (1, 2, 0, 3, 256),     # no context: each branch sees itself only
    (2, 4, 512, 9, 256),   # the lookahead shape: context 512, anchor + 8 branches of 256
    (3, 8, 0, 9, 96),      # one key tile per item, several items per CTA: every tile ends an item
    (4, 16, 64, 5, 64),    # two key tiles per item, two or three items per CTA
])
def test_packed_attention_parity(n_b, n_h, C, NB, G):
    q, k, v = inputs(31, n_b, n_h, C, NB, G)
    check(q, k, v, C, NB, G, 1.0 / np.sqrt(D))


def test_packed_attention_rescales_when_scores_grow():
    """Keys grow tile after tile, so each tile's maximum passes the running
    reference by more than the slack: O and the sum are rescaled in TMEM."""
    q, k, v = inputs(32, 1, 2, 256, 3, 256, key_growth=1.0)
    check(q, k, v, 256, 3, 256, 0.3)


def test_packed_attention_isolation_bit_for_bit():
    C, NB, G = 136, 4, 72
    q, k, v = inputs(33, 1, 2, C, NB, G)
    base = run_gpu(q, k, v, C, NB, G, 0.1)
    rows = slice(C + 2 * G, C + 3 * G)
    k2, v2 = k.copy(), v.copy()
    rng = np.random.default_rng(34)
    k2[:, :, rows] = synth.bf16_round(rng.standard_normal(k2[:, :, rows].shape).astype(np.float32))
    v2[:, :, rows] = synth.bf16_round(rng.standard_normal(v2[:, :, rows].shape).astype(np.float32))
    moved = run_gpu(q, k2, v2, C, NB, G, 0.1)
    keep = np.ones(C + NB * G, bool)
    keep[rows] = False
    assert np.array_equal(base[:, :, keep], moved[:, :, keep]), "another branch's output moved"
    assert not np.array_equal(base[:, :, rows], moved[:, :, rows])


def test_packed_attention_full_size_sampled():
    """The serving shape the bench times (8 requests x 32 heads, context 512,
    anchor + 8 branches of 256: 2,816 packed tokens), one launch over all of it;
    three (request, head) slices against the oracle."""
    n_b, n_h, C, NB, G = 8, 32, 512, 9, 256
    q, k, v = inputs(35, n_b, n_h, C, NB, G)
    g = run_gpu(q, k, v, C, NB, G, 1.0 / np.sqrt(D))
    for b, h in ((0, 0), (3, 17), (7, 31)):
        sl = (slice(b, b + 1), slice(h, h + 1))
        ref = packed_attention(q[sl], k[sl], v[sl], C, NB, G, 1.0 / np.sqrt(D))
        weighted_abs = packed_attention(q[sl], k[sl], v[sl] & np.uint16(0x7FFF), C, NB, G, 1.0 / np.sqrt(D))
        tol = 2.0 ** -8 * (weighted_abs + np.abs(ref)) + 1e-6
        err = np.abs(g[sl] - ref)
        assert not (err > tol).any(), f"slice ({b}, {h}): {(err > tol).sum()} outputs out of tolerance"


def test_packed_attention_wait_timeout_is_reported_and_the_next_launch_works():
    """Every bounded wait gives up at once (testing hook): the launch reports
    RPS_DEVERR_TIMEOUT and nothing hangs. Each role stops at its first wait, the
    two MMA issuers drain, and TMEM is released: the next, normal launch
    allocates it again and matches the oracle."""
    C, NB, G = 256, 3, 128
    q, k, v = inputs(36, 1, 2, C, NB, G)
    out = torch.empty(q.shape, dtype=torch.bfloat16, device="cuda")
    vt = np.ascontiguousarray(np.swapaxes(v, 2, 3))
    rps.rps_debug_set_ring_wait_ns(0)
    try:
        rps.rps_packed_attention_fwd(dev(q), dev(k), dev(vt), out, C, NB, G, 0.1)
        status, detail = rps.rps_poll_device_status()
    finally:
        rps.rps_debug_set_ring_wait_ns(2**64 - 1)
    assert status == rps.RPS_ERR_DEVICE and detail & rps.DEVERR_TIMEOUT, hex(detail)
    check(q, k, v, C, NB, G, 0.1)
