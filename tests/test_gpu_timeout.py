"""Bounded device waits that run out, seen on the host (failure detection
without a GPU fault).

The testing hook rps_debug_set_ring_wait_ns(0) makes every warp of the
row-statistics launch give up on its first ring-copy wait. Each warp still
waits (bounded) for the copies it issued before it stops, so nothing is left in
flight and the context stays usable. The call must report RPS_DEVERR_TIMEOUT;
a later call on the same, unhealthy workspace must write nothing and report
RPS_DEVERR_WORKSPACE; after rps_workspace_init the next call matches the oracle.
"""
import numpy as np
import pytest
import torch

from gpu_harness import compare_stats, padded_tensor, stats_np
from oracle import default as oracle_default
from paper_2608_11742_gb300 import rps, synth

pytestmark = pytest.mark.gpu

DEFAULT_WAIT = 2**64 - 1


@pytest.mark.parametrize("k", [0, 10])
def test_ring_wait_timeout_is_reported_and_the_workspace_recovers(k):
    V, n = 20011, 96
    z = synth.make_logits(5, 1, 0, n, V, (0.4, 0.3, 0.3), "bf16")  # [1][1][n][V]
    t = padded_tensor(z)
    prm = type("P", (), dict(k_max=10, r=0.1, tau_pivot=0.0, tau=0.05, lam=0.1, n_pivots=4, tokens_per_pivot=2))()
    ws = torch.empty(rps.rps_workspace_bytes(n, V, k, t.dtype), dtype=torch.uint8, device="cuda")
    rps.rps_workspace_init(ws)
    rows = torch.tensor([[0, 0, p] for p in range(n)], dtype=torch.int32, device="cuda")
    buf = rps.RowStatsBuf.alloc(n, k, "cuda")
    assert rps.rps_poll_device_status() == (rps.RPS_OK, 0)

    # 1. every ring wait gives up at once: reported, nothing hangs
    old = rps.rps_debug_set_ring_wait_ns(0)
    try:
        rps.rps_score_step(t, rows, None, 1, n, prm, buf, ws)
        status, detail = rps.rps_poll_device_status()
    finally:
        rps.rps_debug_set_ring_wait_ns(DEFAULT_WAIT)
    assert old == 200_000_000
    assert status == rps.RPS_ERR_DEVICE and detail & rps.DEVERR_TIMEOUT, (status, hex(detail))

    # 2. the same workspace without re-zeroing: refused on the device, nothing written
    stale = rps.RowStatsBuf.alloc(n, k, "cuda")
    rps.rps_score_step(t, rows, None, 1, n, prm, stale, ws)
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_ERR_DEVICE and detail & rps.DEVERR_WORKSPACE, (status, hex(detail))
    assert not detail & rps.DEVERR_TIMEOUT
    assert torch.isnan(stale.H).all() and (stale.argmax == -1).all(), "a refused call wrote statistics"

    # 3. re-zeroed: the next call is complete and matches the oracle, twice
    rps.rps_workspace_init(ws)
    ref = oracle_default().row_stats(z[0, 0], k)
    for rep in range(2):
        good = rps.RowStatsBuf.alloc(n, k, "cuda")
        rps.rps_score_step(t, rows, None, 1, n, prm, good, ws)
        assert rps.rps_poll_device_status() == (rps.RPS_OK, 0)
        compare_stats(stats_np(good), ref, np.arange(n), k, f"after re-zeroing, call {rep}")
