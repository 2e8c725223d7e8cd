"""The seeded generator: Philox known answers, bf16 rounding, value model."""
from pathlib import Path

import numpy as np
import pytest

from paper_2608_11742_gb300 import configs, synth

GOLDEN = Path(__file__).parent / "golden" / "philox4x32_10_kat.txt"


def test_philox_known_answers():
    rows = [l.split() for l in GOLDEN.read_text().splitlines() if l and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        c0, c1, c2, c3, k0, k1 = (int(x, 16) for x in r[:6])
        want = [int(x, 16) for x in r[6:]]
        got = [int(x) for x in synth.philox4x32_10(c0, c1, c2, c3, k0, k1)]
        assert got == want


def test_bf16_round_matches_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 10,
                        np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.0 - 2 ** -8, 3.3e38, -0.0, 0.0],
                                 np.float32)])
    ours = synth.bf16_round(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert (ours == ref).all()
    back = synth.bf16_to_f32(ours)
    assert (back == torch.from_numpy(ours.view(np.int16)).view(torch.bfloat16).float().numpy()).all()


def test_noise_moments():
    eps = np.concatenate([synth.noise_row(0, 50000, 0, p) for p in range(4)]).astype(np.float64)
    assert abs(eps.mean()) < 0.01
    assert abs(eps.var() - 1.0) < 0.01
    assert np.abs(eps).max() < 5.0


def test_regime_mixture_and_spikes():
    mix = (0.4, 0.3, 0.3)
    plans = [synth.row_plan(0, 126464, 0, p, mix) for p in range(3000)]
    freq = np.bincount([p.regime for p in plans], minlength=3) / len(plans)
    assert np.allclose(freq, mix, atol=0.03)
    for p in plans:
        if p.regime == synth.REGIME_LOW:
            assert len(p.spikes) == 1
        elif p.regime == synth.REGIME_MID:
            assert 2 <= len(p.spikes) <= 5 and len(set(p.spikes)) == len(p.spikes)
        else:
            assert p.spikes == ()


def test_branch_rows_scale_only_the_spike():
    mix = (0.4, 0.3, 0.3)
    for pos in range(12):
        plan = synth.row_plan(0, 4096, 0, pos, mix)
        base = synth.row_logits_f32(0, 4096, 0, 0, pos, mix)
        br = synth.row_logits_f32(0, 4096, 0, 3, pos, mix)
        f = synth.branch_factor(0, 0, 3, pos)
        assert 0.8 <= f < 1.6
        others = np.setdiff1d(np.arange(4096), np.array(plan.spikes, dtype=np.int64))
        assert (base[others] == br[others]).all()
        if plan.regime != synth.REGIME_HIGH:
            h = 12.0 if plan.regime == synth.REGIME_LOW else 4.0
            eps = synth.noise_row(0, 4096, 0, pos)
            s = list(plan.spikes)
            assert np.allclose(br[s] - eps[s], h * f, atol=1e-5)
            assert np.allclose(base[s] - eps[s], h, atol=1e-5)


def test_masks_and_counts():
    w = configs.STEP_10
    pos, cnt = w.mask()
    assert cnt[0] == 26  # 10 % of 256, rounded half up
    sel = pos[0, :26]
    assert (np.diff(sel) > 0).all() and sel.min() >= 0 and sel.max() < 256
    s = configs.SERVE
    pos, cnt = s.mask()
    assert ((cnt >= 16) & (cnt <= 256)).all() and len(set(cnt.tolist())) > 1
    valid = s.valid_rows()
    assert (valid.sum(1) == cnt).all()


def test_make_logits_pads_with_nan():
    w = configs.SERVE.scaled(V=64, L=8, n_req=2, ragged=(2, 6))
    valid = w.valid_rows()
    z = synth.make_logits(w.seed, w.n_req, w.n_branch, w.L, w.V, w.mixture, w.dtype, valid=valid)
    f = synth.bf16_to_f32(z)
    for q in range(w.n_req):
        for p in range(w.L):
            assert np.isnan(f[q, :, p]).all() == (not valid[q, p])
