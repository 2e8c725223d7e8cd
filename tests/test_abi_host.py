"""C-ABI checks that need no GPU: exports, host-side validation, workspace sizing.

Only calls that return before any CUDA call are made here (argument errors,
size queries, status strings); no compute entry point runs without a GPU.
"""
import ctypes as C
import re
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]
INCLUDE = ROOT / "include"
PKG = ROOT / "paper_2608_11742_gb300"


@pytest.fixture(scope="module")
def libs():
    from paper_2608_11742_gb300.build import build
    built = build()
    return {name: C.CDLL(str(path)) for name, path in built.items()}


def declared_functions(header: Path):
    text = re.sub(r"/\*.*?\*/", "", header.read_text(), flags=re.S)
    text = re.sub(r"//.*", "", text)
    return sorted(set(re.findall(r"\b(rps_\w+)\s*\(", text)) - {"rps_stream_t"})


def test_every_declared_symbol_is_exported(libs):
    owners = {"rps.h": "librps.so", "rps_synth.h": "librps_synth.so"}
    for header in sorted(INCLUDE.glob("*.h")):
        lib = libs[owners[header.name]]
        names = declared_functions(header)
        assert names, header
        for name in names:
            assert hasattr(lib, name), f"{name} declared in {header.name} is not exported"


def test_status_strings_and_version(libs):
    lib = libs["librps.so"]
    lib.rps_status_string.restype = C.c_char_p
    for code in range(6):
        assert lib.rps_status_string(code).startswith(b"RPS_")
    assert lib.rps_status_string(99) == b"unknown rps_status"
    lib.rps_version.restype = C.c_int32
    assert lib.rps_version() >= 100


def test_workspace_bytes(libs):
    lib = libs["librps.so"]
    lib.rps_workspace_bytes.restype = C.c_size_t
    lib.rps_workspace_bytes.argtypes = [C.c_int64, C.c_int64, C.c_int32, C.c_int32]
    bf16, f32 = 1, 0
    a = lib.rps_workspace_bytes(256, 126464, bf16, 10)
    b = lib.rps_workspace_bytes(256, 126464, bf16, 0)
    assert a > b > 0
    assert lib.rps_workspace_bytes(256, 126464, f32, 10) > a  # the top-k sketch is element-sized
    assert lib.rps_workspace_bytes(256, 126464, f32, 0) == b
    assert lib.rps_workspace_bytes(512, 126464, bf16, 10) > a
    assert lib.rps_workspace_bytes(0, 126464, bf16, 10) == 0
    assert lib.rps_workspace_bytes(16, 0, bf16, 10) == 0
    assert lib.rps_workspace_bytes(16, 100, bf16, 33) == 0
    assert lib.rps_workspace_bytes(16, 100, 7, 10) == 0


def _binding_types():
    # the ctypes structures of the binding, without loading torch CUDA state
    import paper_2608_11742_gb300.rps as r
    return r


def test_host_rejects_bad_arguments(libs):
    r = _binding_types()
    lib = r._lib
    fake = 1 << 20  # never dereferenced: every case fails validation first
    good_logits = r.RpsLogits(fake, r.RPS_BF16, 1, 9, 32, 4096, 9 * 32 * 4096, 32 * 4096, 4096)
    rows = r.RpsRowList(fake, None, 1, 32, None, 0)
    prm = r.RpsParams(10, 0.1, 0.9, 0.9, 0.1, 4, 2)
    out = r.RpsRowStats(fake, fake, fake, fake, fake, fake, fake, fake, fake)
    ws = lib.rps_workspace_bytes(32, 4096, r.RPS_BF16, 10)

    def score(logits=good_logits, rows=rows, prm=prm, out=out, ws_ptr=fake, ws_bytes=ws):
        return lib.rps_score_step(C.byref(logits), C.byref(rows), C.byref(prm), C.byref(out), ws_ptr, ws_bytes, None)

    bad = r.RpsLogits(*[getattr(good_logits, f) for f, _ in r.RpsLogits._fields_])
    bad.data = fake + 2  # not 16-byte aligned
    assert score(logits=bad) == r.RPS_ERR_INVALID_ARG
    bad.data = fake
    bad.pos_stride = 4095  # rows not 16-byte aligned
    assert score(logits=bad) == r.RPS_ERR_INVALID_ARG
    bad.pos_stride = 4096
    bad.dtype = 7
    assert score(logits=bad) == r.RPS_ERR_INVALID_ARG
    assert score(ws_bytes=ws - 1) == r.RPS_ERR_INVALID_ARG
    assert score(ws_ptr=None) == r.RPS_ERR_INVALID_ARG
    big_k = r.RpsParams(33, 0.1, 0.9, 0.9, 0.1, 4, 2)
    assert score(prm=big_k) == r.RPS_ERR_UNSUPPORTED
    no_rows = r.RpsRowList(None, None, 1, 32, None, 0)
    assert score(rows=no_rows) == r.RPS_ERR_INVALID_ARG
    many = r.RpsRowList(fake, None, 2000, 4, None, 0)
    assert score(rows=many) == r.RPS_ERR_UNSUPPORTED
    missing = r.RpsRowStats(fake, None, fake, fake, fake, fake, fake, fake, fake)
    assert score(out=missing) == r.RPS_ERR_INVALID_ARG
    no_mu = r.RpsRowStats(fake, fake, fake, fake, fake, None, fake, fake, fake)
    assert score(out=no_mu) == r.RPS_ERR_INVALID_ARG

    piv = r.RpsPivots(*([fake] * len(r._PIVOT_FIELDS)))

    def select(prm=prm, n_req=1, L=32, piv=piv):
        return lib.rps_select_pivots(C.byref(out), n_req, L, fake, fake, C.byref(prm), C.byref(piv), None)

    assert select(n_req=0) == r.RPS_ERR_INVALID_ARG
    assert select(L=5000) == r.RPS_ERR_UNSUPPORTED
    assert select(prm=r.RpsParams(10, 0.0, 0.9, 0.9, 0.1, 4, 2)) == r.RPS_ERR_INVALID_ARG   # r = 0
    assert select(prm=r.RpsParams(10, 1.5, 0.9, 0.9, 0.1, 4, 2)) == r.RPS_ERR_INVALID_ARG   # r > 1
    assert select(prm=r.RpsParams(10, 0.1, 0.9, 0.9, -0.1, 4, 2)) == r.RPS_ERR_INVALID_ARG  # lambda < 0
    assert select(prm=r.RpsParams(10, 0.1, 0.9, 0.9, 0.1, 4, 11)) == r.RPS_ERR_INVALID_ARG  # K > k_max
    assert select(prm=r.RpsParams(10, 0.1, 0.9, 0.9, 0.1, 17, 2)) == r.RPS_ERR_UNSUPPORTED  # P > 16
    nan = float("nan")
    assert select(prm=r.RpsParams(10, 0.1, nan, 0.9, 0.1, 4, 2)) == r.RPS_ERR_INVALID_ARG
    assert select(prm=r.RpsParams(10, 0.1, 0.9, 0.9, 0.1, 4, 2, 3, 0, 0)) == r.RPS_ERR_INVALID_ARG  # pivot rule
    assert select(prm=r.RpsParams(10, 0.1, 0.9, 0.9, 0.1, 4, 2, 0, 3, 1)) == r.RPS_ERR_INVALID_ARG  # commit rule
    assert select(prm=r.RpsParams(10, 0.1, 0.9, 0.9, 0.1, 4, 2, 0, 1, 0)) == r.RPS_ERR_INVALID_ARG  # top-k, k = 0
    assert select(prm=r.RpsParams(10, 0.1, 0.9, 0.9, 0.1, 4, 2, 0, 2, 17)) == r.RPS_ERR_UNSUPPORTED  # k > 16
    holes = r.RpsPivots(*([fake] * (len(r._PIVOT_FIELDS) - 1) + [None]))
    assert select(piv=holes) == r.RPS_ERR_INVALID_ARG

    sc = r.RpsBranchScores(fake, fake, fake, fake)
    assert lib.rps_score_branches(C.byref(good_logits), 9, C.byref(out), C.byref(out), 1, 32, C.byref(piv),
                                  C.byref(prm), C.byref(sc), None) == r.RPS_ERR_INVALID_ARG  # anchor branch
    assert lib.rps_score_branches(C.byref(good_logits), 0, C.byref(out), C.byref(out), 2, 32, C.byref(piv),
                                  C.byref(prm), C.byref(sc), None) == r.RPS_ERR_INVALID_ARG  # n_req > tensor
    cm = r.RpsCommitOut(fake, fake, fake, fake, fake, fake, fake, fake)
    alias = r.RpsCommitOut(fake, fake, fake, fake, fake, fake, piv.rem_pos, fake)
    assert lib.rps_commit(C.byref(sc), 1, 32, C.byref(piv), C.byref(prm), C.byref(alias), None) \
        == r.RPS_ERR_INVALID_ARG
    assert lib.rps_commit(C.byref(sc), 0, 32, C.byref(piv), C.byref(prm), C.byref(cm), None) \
        == r.RPS_ERR_INVALID_ARG

    synth = libs["librps_synth.so"]
    synth.rps_synth_fill.restype = C.c_int32
    synth.rps_synth_fill.argtypes = [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int64,
                                     C.c_int64, C.c_int64, C.c_int64, C.c_uint32, C.c_uint64, C.c_uint64,
                                     C.c_uint32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
    assert synth.rps_synth_fill(fake + 4, 1, 1, 8, 32, 4096, 0, 0, 4096, 0, 1, 2, 0, None, None, None, None) == 1
    assert synth.rps_synth_fill(fake, 1, 1, 8, 32, 4096, 0, 0, 4096, 0, 3, 2, 0, None, None, None, None) == 1
