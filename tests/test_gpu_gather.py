"""rps_gather_rows and Step.run_host: a step whose logits sit in page-locked host
memory copies only the rows it scores, and decides exactly what the same step
decides on the whole tensor in device memory."""
import ctypes as C

import numpy as np
import pytest
import torch

from gpu_harness import commit_np, piv_np, scores_np, stats_np
from paper_2608_11742_gb300 import configs, rps, synth

pytestmark = pytest.mark.gpu


def _pinned(z: np.ndarray, pad_to: int) -> torch.Tensor:
    """Page-locked host tensor of z, rows padded to a multiple of pad_to elements."""
    V = z.shape[-1]
    Vp = (V + pad_to - 1) // pad_to * pad_to
    if z.dtype == np.uint16:
        t = torch.empty(z.shape[:-1] + (Vp,), dtype=torch.bfloat16).pin_memory()
        t.view(torch.int16)[..., :V].copy_(torch.from_numpy(z.view(np.int16)))
    else:
        t = torch.empty(z.shape[:-1] + (Vp,), dtype=torch.float32).pin_memory()
        t[..., :V].copy_(torch.from_numpy(z))
    return t[..., :V]


def _device_like(h: torch.Tensor, fill_nan=True) -> torch.Tensor:
    Vp = h.stride(2)
    t = torch.empty(h.shape[:-1] + (Vp,), dtype=h.dtype, device="cuda")
    if fill_nan:
        t.fill_(float("nan"))
    return t[..., :h.shape[-1]]


def _outputs(step):
    return dict(base=stats_np(step.base), branch=stats_np(step.branch), piv=piv_np(step.piv),
                scores=scores_np(step.scores), commit=commit_np(step.commit))


def _assert_same(a, b, what):
    for part in ("base", "branch"):
        for name, x in vars(a[part]).items():
            y = getattr(b[part], name)
            if x is None:
                assert y is None
                continue
            assert np.array_equal(x, y, equal_nan=True), f"{what}: {part}.{name}"
    for part in ("piv", "scores", "commit"):
        for name, x in a[part].items():
            assert np.array_equal(x, b[part][name], equal_nan=True), f"{what}: {part}.{name}"


CASES = [
    # ragged masks, NaN padding outside them, a vocab with a ragged 16-byte tail
    (configs.SERVE, dict(n_req=3, L=48, V=3001, ragged=(4, 48), seed=5), configs.EXERCISE),
    (configs.TINY, dict(L=40, V=2050, seed=6), configs.Params(tau_pivot=0.003, lam=0.3)),
    (configs.BLOCK, dict(n_req=5, V=4096, seed=7), configs.EXERCISE),
]


@pytest.mark.parametrize("w,shrink,base_prm", CASES, ids=["serve-bf16", "tiny-f32", "block-bf16"])
def test_run_host_equals_device_run(w, shrink, base_prm):
    w = w.scaled(**shrink)
    prm = w.params(base_prm)
    z = synth.make_logits(w.seed, w.n_req, w.n_branch, w.L, w.V, w.mixture, w.dtype, valid=w.valid_rows())
    mask_pos, mask_cnt = w.mask()
    mp, mc = torch.from_numpy(mask_pos).cuda(), torch.from_numpy(mask_cnt).cuda()
    host = _pinned(z, 8)
    full = _device_like(host, fill_nan=False)
    full.copy_(host)
    ref_step = rps.Step(w.n_req, w.L, w.V, prm, "cuda", full.dtype)
    ref_step.run(full, mp, mc)
    torch.cuda.synchronize()
    ref = _outputs(ref_step)

    dev = _device_like(host)
    step = rps.Step(w.n_req, w.L, w.V, prm, "cuda", full.dtype)
    step.run_host(host, dev, mp, mc)
    torch.cuda.synchronize()
    assert rps.rps_poll_device_status()[0] == rps.RPS_OK
    _assert_same(_outputs(step), ref, w.name)

    # exactly the scored rows arrived; every other row still holds the NaN fill
    piv = ref["piv"]
    want = np.zeros(host.shape[:3], bool)
    for q in range(w.n_req):
        want[q, 0, mask_pos[q, :mask_cnt[q]]] = True
        for r in piv["branch_rows"].reshape(w.n_req, -1, 3)[q, :piv["n_branch_rows"][q]]:
            if r[2] >= 0:
                want[r[0], r[1], r[2]] = True
    got = dev.cpu()
    same = (got.view(torch.int16) == host.view(torch.int16)).all(-1).numpy() if got.dtype == torch.bfloat16 else \
        (got == host).all(-1).numpy()
    assert same[want].all(), "a gathered row differs from the host row"
    assert torch.isnan(got.float()).all(-1).numpy()[~want].all(), "a row outside the lists was written"
    assert want.sum() < want.size, "the case should leave rows behind"


def test_gather_device_to_device_strided_lists():
    """Explicit list with skipped entries and ragged counts; src and dst strides differ."""
    rng = np.random.default_rng(21)
    n_req, nb, L, V = 2, 3, 5, 1000
    src = torch.from_numpy(rng.standard_normal((n_req, nb, L, V)).astype(np.float32)).cuda()
    dst_store = torch.full((n_req, nb + 1, L, V + 24), float("nan"), device="cuda")
    dst = dst_store[:, 1:, :, :V]
    rows = torch.tensor([[0, 2, 4], [0, 0, -1], [1, 1, 3], [9, 9, 9],   # segment 0: 3 counted, 4th beyond count
                         [1, 0, 0], [1, 2, 2], [0, 0, 0], [0, 0, 0]],   # segment 1: 2 counted
                        dtype=torch.int32, device="cuda")
    cnt = torch.tensor([3, 2], dtype=torch.int32, device="cuda")
    rps.rps_gather_rows(src, rows, cnt, 2, 4, dst)
    torch.cuda.synchronize()
    assert rps.rps_poll_device_status()[0] == rps.RPS_OK
    got = dst.cpu()
    for r in ((0, 2, 4), (1, 1, 3), (1, 0, 0), (1, 2, 2)):
        assert torch.equal(got[r], src[r].cpu()), r
    written = {(0, 2, 4), (1, 1, 3), (1, 0, 0), (1, 2, 2)}
    for q in range(n_req):
        for b in range(nb):
            for p in range(L):
                if (q, b, p) not in written:
                    assert torch.isnan(got[q, b, p]).all(), (q, b, p)
    assert torch.isnan(dst_store[:, 0]).all() and torch.isnan(dst_store[..., V:]).all()


def test_gather_errors():
    V = 64
    src = torch.zeros((1, 1, 4, V), dtype=torch.bfloat16).pin_memory()
    dst = torch.full((1, 1, 4, V), float("nan"), dtype=torch.bfloat16, device="cuda")
    rows = torch.tensor([[0, 0, 1], [0, 0, 7]], dtype=torch.int32, device="cuda")  # pos 7 is out of range
    rps.rps_gather_rows(src, rows, None, 1, 2, dst)
    torch.cuda.synchronize()
    status, detail = rps.rps_poll_device_status()
    assert status == rps.RPS_ERR_DEVICE and detail & rps.DEVERR_ROW_INDEX
    got = dst.float().cpu()
    assert (got[0, 0, 1] == 0).all() and torch.isnan(got[0, 0, [0, 2, 3]]).all()

    pageable = torch.zeros((1, 1, 4, V), dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        rps.rps_gather_rows(pageable, rows[:1], None, 1, 1, dst)
    # the library refuses a pageable source and a destination outside device memory
    s, d = rps.logits_desc(pageable), rps.logits_desc(dst)
    rl = rps.RpsRowList(rows.data_ptr(), None, 1, 1, None, 0)
    st = rps._lib.rps_gather_rows(C.byref(s), C.byref(rl), C.byref(d), None)
    assert st == rps.RPS_ERR_INVALID_ARG
    s2, d2 = rps.logits_desc(dst), rps.logits_desc(src)
    assert rps._lib.rps_gather_rows(C.byref(s2), C.byref(rl), C.byref(d2), None) == rps.RPS_ERR_INVALID_ARG
    mis = torch.zeros((1, 1, 4, V + 1), dtype=torch.bfloat16, device="cuda")[..., 1:]
    with pytest.raises(rps.RPSError):
        rps.rps_gather_rows(mis, rows[:1], None, 1, 1, dst)
    assert rps.rps_poll_device_status()[0] == rps.RPS_OK
