"""Edge cases of the scoring path on the GPU, element by element against the oracle:
the build's maximum sizes, a step with nothing masked, and degenerate
vocabularies (a single token, fewer tokens than one 16-byte unit)."""
import numpy as np
import pytest
import torch

from gpu_harness import GpuStep
from paper_2608_11742_gb300 import rps, synth
from paper_2608_11742_gb300.configs import Params

pytestmark = pytest.mark.gpu


def _logits(rng, n_req, nb, L, V, bf16=True, spread=1.5):
    """Random rows with one or a few spikes; the branches scale the base's spikes."""
    base = rng.standard_normal((n_req, 1, L, V)).astype(np.float32) * np.float32(spread)
    spikes = rng.integers(0, V, (n_req, L))
    amp = rng.uniform(0.0, 10.0, (n_req, L)).astype(np.float32)
    z = np.repeat(base, 1 + nb, axis=1)
    qi, li = np.arange(n_req)[:, None], np.arange(L)[None, :]
    for b in range(1 + nb):
        f = np.float32(1.0) if b == 0 else rng.uniform(0.8, 1.6, (n_req, L)).astype(np.float32)
        z[qi, b, li, spikes] += amp * f
    return synth.bf16_round(z) if bf16 else z


def _masks(rng, n_req, L, counts):
    pos = np.full((n_req, L), -1, np.int32)
    for q in range(n_req):
        pos[q, :counts[q]] = np.sort(rng.choice(L, counts[q], replace=False))
    return pos, np.asarray(counts, np.int32)


def test_largest_mask_and_pivot_counts():
    """L = RPS_MAX_POS positions, P = RPS_MAX_PIVOTS pivots of 4 tokens (64 branches),
    k_max = RPS_MAX_K, a top-k commit of RPS_MAX_COMMIT_K, and a ragged vocab."""
    rng = np.random.default_rng(11)
    P, K, L, V = 16, 4, 4096, 100
    z = _logits(rng, 1, P * K, L, V)
    pos, cnt = _masks(rng, 1, L, [L - 5])
    for prm in (Params(k_max=32, r=0.02, tau_pivot=0.0, tau=0.5, lam=0.2, n_pivots=P, tokens_per_pivot=K),
                Params(k_max=32, r=0.02, tau_pivot=0.0, tau=0.5, lam=0.2, n_pivots=P, tokens_per_pivot=K,
                       commit_rule=1, commit_k=16, pivot_rule=2)):
        out = GpuStep(z, pos, cnt, prm).run_and_compare(f"max sizes {prm}")
        assert out["piv"]["state"][0] == 0 and (out["piv"]["pivot_pos"][0] >= 0).sum() == P


def test_many_requests():
    """RPS_MAX_SEGMENTS requests of ragged mask counts in one call."""
    rng = np.random.default_rng(12)
    n_req, L, V, P, K = 1024, 8, 64, 2, 2
    z = _logits(rng, n_req, P * K, L, V)
    pos, cnt = _masks(rng, n_req, L, rng.integers(0, L + 1, n_req))
    prm = Params(k_max=8, r=0.05, tau_pivot=0.0, tau=0.5, lam=0.1, n_pivots=P, tokens_per_pivot=K)
    out = GpuStep(z, pos, cnt, prm).run_and_compare("1024 requests")
    states = set(out["piv"]["state"].tolist())
    assert 0 in states and 1 in states, states


def test_nothing_masked():
    """Every request already decoded: zero rows scored, state DONE, winner DONE."""
    rng = np.random.default_rng(13)
    n_req, L, V = 3, 6, 256
    z = _logits(rng, n_req, 8, L, V)
    pos = np.full((n_req, L), -1, np.int32)
    cnt = np.zeros(n_req, np.int32)
    out = GpuStep(z, pos, cnt, Params()).run_and_compare("nothing masked")
    assert (out["piv"]["state"] == rps.STATE_DONE).all() and (out["commit"]["winner"] == rps.WIN_DONE).all()
    assert (out["commit"]["mask_cnt"] == 0).all()


@pytest.mark.parametrize("V,bf16", [(1, False), (3, True), (7, True), (5, False)])
def test_tiny_vocabularies(V, bf16):
    """Vocabularies below one 16-byte unit (the ragged tail alone) and a single token
    (entropy 0, confidence 1, every row committed)."""
    rng = np.random.default_rng(14 + V)
    n_req, L = 2, 6
    K = max(1, min(2, V))
    z = _logits(rng, n_req, 2 * K, L, V, bf16=bf16)
    pos, cnt = _masks(rng, n_req, L, [L, 3])
    prm = Params(k_max=V, r=0.05, tau_pivot=0.0, tau=0.9 if V > 1 else 0.5, lam=0.1, n_pivots=2,
                 tokens_per_pivot=K)
    out = GpuStep(z, pos, cnt, prm).run_and_compare(f"V={V}")
    if V == 1:
        assert np.allclose(out["base"].H[[0, 1, 2]], 0.0, atol=1e-6) and np.allclose(out["base"].pmax[[0, 1, 2]], 1.0)
        assert (out["piv"]["state"] == 1).all(), "a single-token vocabulary commits everything"
