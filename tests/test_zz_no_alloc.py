"""rps_score_step_noalloc, the variant for callers that cannot allocate device memory.

Some callers cannot call cudaMalloc at all: plugins of a host runtime that owns
every device allocation, or bindings from languages without a CUDA allocator.
For them the library keeps a fixed scratch array on each device. This test calls
that entry point through the C ABI twice in a row and checks each result against
rps_score_step with a caller workspace, with the tolerances of the other parity
tests. The file name sorts last so that a stop-at-first-failure run has already
run every other test.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rps():
    from paper_2608_11742_gb300.build import build
    build()
    from paper_2608_11742_gb300 import rps as r
    assert torch.cuda.is_available()
    return r


def _rows(n, V, seed):
    from paper_2608_11742_gb300 import synth
    rng = np.random.default_rng(seed)
    z = rng.standard_normal((1, 1, n, V)).astype(np.float32) * np.float32(1.5)
    z[0, 0, :, rng.integers(0, V, n)] += np.float32(6.0)
    bits = synth.bf16_round(z)
    return torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)


@pytest.mark.parametrize("k", [0, 10])
def test_noalloc_matches_workspace_entry_point(rps, k):
    from gpu_harness import compare_stats, stats_np
    from paper_2608_11742_gb300.configs import Params
    n, V = 300, 6144
    prm = Params(k_max=max(k, 1))
    t = _rows(n, V, 7 + k)
    desc = torch.tensor([[0, 0, i] for i in range(n)], dtype=torch.int32, device="cuda")
    ref = rps.RowStatsBuf.alloc(n, k, "cuda")
    ws = torch.zeros(rps.rps_workspace_bytes(n, V, k, t.dtype), dtype=torch.uint8, device="cuda")
    rps.rps_score_step(t, desc, None, 1, n, prm, ref, ws)
    assert rps.rps_poll_device_status()[0] == rps.RPS_OK
    want = stats_np(ref)
    for call in range(2):
        got = rps.RowStatsBuf.alloc(n, k, "cuda")
        rps.rps_score_step_noalloc(t, desc, None, 1, n, prm, got)
        status, detail = rps.rps_poll_device_status()
        assert status == rps.RPS_OK, hex(detail)
        compare_stats(stats_np(got), want, np.arange(n), k, f"noalloc call {call}")


def test_noalloc_rejects_requests_beyond_the_scratch(rps):
    from paper_2608_11742_gb300.configs import Params
    V = 4096
    limit = 8 << 20
    n = 1
    while rps.rps_workspace_bytes(n, V, 10, torch.bfloat16) <= limit:
        n *= 2
    t = _rows(4, V, 1)
    desc = torch.zeros((n, 3), dtype=torch.int32, device="cuda")
    out = rps.RowStatsBuf.alloc(n, 10, "cuda")
    with pytest.raises(rps.RPSError) as e:
        rps.rps_score_step_noalloc(t, desc, None, 1, n, Params(), out)
    assert e.value.status == rps.RPS_ERR_UNSUPPORTED
    assert torch.isnan(out.H).all(), "a rejected call must not write its outputs"
