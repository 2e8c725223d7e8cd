"""ctypes binding of ``librps.so`` (declared in ``include/rps.h``).

Argument marshalling only: each function takes torch CUDA tensors, passes their
device pointers and the current stream to the C ABI function of the same name,
and raises ``RPSError`` on a non-OK status. Every step of the scoring path runs
in the library's CUDA kernels; there is no fallback. Importing this module
raises ImportError when the library has not been built.

Buffers (``RowStatsBuf``, ``PivotsBuf``, ``ScoresBuf``, ``CommitBuf``) are
allocated once by the caller and reused; ``Step`` strings the five calls of
one decoding step together on preallocated buffers.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass, fields
from pathlib import Path
from typing import Optional

import torch

import os

# RPS_LIBRARY selects another build of the library (for example a tuning variant).
LIB_PATH = Path(os.environ.get("RPS_LIBRARY", Path(__file__).resolve().parent / "librps.so"))
if not LIB_PATH.exists():
    raise ImportError(f"{LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
_lib = C.CDLL(str(LIB_PATH))

RPS_OK, RPS_ERR_INVALID_ARG, RPS_ERR_UNSUPPORTED, RPS_ERR_CUDA, RPS_ERR_DEVICE, RPS_ERR_TIMEOUT = range(6)
RPS_F32, RPS_BF16 = 0, 1
STATE_SEARCH, STATE_DONE, STATE_NO_FEASIBLE, STATE_NO_CANDIDATES = 0, 1, 2, 3
WIN_ANCHOR, WIN_SKIP, WIN_DONE = -1, -2, -3
DEVERR_ROW_INDEX, DEVERR_NONFINITE, DEVERR_MASK, DEVERR_TOKEN = 0x1, 0x2, 0x4, 0x8
DEVERR_TIMEOUT, DEVERR_WORKSPACE = 0x10, 0x20

_p = C.c_void_p


class RpsParams(C.Structure):
    _fields_ = [("k_max", C.c_int32), ("r", C.c_float), ("tau_pivot", C.c_float), ("tau", C.c_float),
                ("lambda_", C.c_float), ("n_pivots", C.c_int32), ("tokens_per_pivot", C.c_int32),
                ("pivot_rule", C.c_int32), ("commit_rule", C.c_int32), ("commit_k", C.c_int32)]


class RpsLogits(C.Structure):
    _fields_ = [("data", _p), ("dtype", C.c_int32), ("n_req", C.c_int32), ("n_branch", C.c_int32),
                ("n_pos", C.c_int32), ("vocab", C.c_int64), ("req_stride", C.c_int64),
                ("branch_stride", C.c_int64), ("pos_stride", C.c_int64)]


class RpsRowList(C.Structure):
    _fields_ = [("rows", _p), ("seg_cnt", _p), ("n_seg", C.c_int32), ("cap", C.c_int32),
                ("mask_pos", _p), ("mask_branch", C.c_int32)]


class RpsRowStats(C.Structure):
    _fields_ = [(n, _p) for n in ("zmax", "lse", "H", "pmax", "argmax", "mu", "htrunc", "topk_idx", "topk_logit")]


_PIVOT_FIELDS = ("n_commit", "commit_pos", "commit_tok", "rem_cnt", "rem_k", "rem_pos", "state", "pivot_k",
                 "pivot_pos", "n_cand", "cand_tok", "branch_valid", "branch_off", "branch_cnt", "n_branch_rows",
                 "branch_rows")


class RpsPivots(C.Structure):
    _fields_ = [(n, _p) for n in _PIVOT_FIELDS]


class RpsBranchScores(C.Structure):
    _fields_ = [(n, _p) for n in ("mean_H", "n_tau", "log_a", "score")]


class RpsCommitOut(C.Structure):
    _fields_ = [(n, _p) for n in ("best_slot", "gain", "winner", "commit_pos", "commit_tok", "margin", "mask_pos",
                                  "mask_cnt")]


_lib.rps_workspace_bytes.restype = C.c_size_t
_lib.rps_workspace_bytes.argtypes = [C.c_int64, C.c_int64, C.c_int32, C.c_int32]
_lib.rps_workspace_init.restype = C.c_int
_lib.rps_workspace_init.argtypes = [_p, C.c_size_t, _p]
_lib.rps_score_step.restype = C.c_int
_lib.rps_score_step.argtypes = [C.POINTER(RpsLogits), C.POINTER(RpsRowList), C.POINTER(RpsParams),
                                C.POINTER(RpsRowStats), _p, C.c_size_t, _p]
_lib.rps_score_step_noalloc.restype = C.c_int
_lib.rps_score_step_noalloc.argtypes = [C.POINTER(RpsLogits), C.POINTER(RpsRowList), C.POINTER(RpsParams),
                                        C.POINTER(RpsRowStats), _p]
_lib.rps_select_pivots.restype = C.c_int
_lib.rps_select_pivots.argtypes = [C.POINTER(RpsRowStats), C.c_int32, C.c_int32, _p, _p, C.POINTER(RpsParams),
                                   C.POINTER(RpsPivots), _p]
_lib.rps_score_branches.restype = C.c_int
_lib.rps_score_branches.argtypes = [C.POINTER(RpsLogits), C.c_int32, C.POINTER(RpsRowStats),
                                    C.POINTER(RpsRowStats), C.c_int32, C.c_int32, C.POINTER(RpsPivots),
                                    C.POINTER(RpsParams), C.POINTER(RpsBranchScores), _p]
_lib.rps_commit.restype = C.c_int
_lib.rps_commit.argtypes = [C.POINTER(RpsBranchScores), C.c_int32, C.c_int32, C.POINTER(RpsPivots),
                            C.POINTER(RpsParams), C.POINTER(RpsCommitOut), _p]
_lib.rps_score_and_commit.restype = C.c_int
_lib.rps_score_and_commit.argtypes = [C.POINTER(RpsLogits), C.c_int32, C.POINTER(RpsRowStats),
                                      C.POINTER(RpsRowStats), C.c_int32, C.c_int32, C.POINTER(RpsPivots),
                                      C.POINTER(RpsParams), C.POINTER(RpsBranchScores), C.POINTER(RpsCommitOut), _p]
_lib.rps_run_step.restype = C.c_int
_lib.rps_run_step.argtypes = [C.POINTER(RpsLogits), C.c_int32, C.c_int32, _p, _p, C.POINTER(RpsParams),
                              C.POINTER(RpsRowStats), C.POINTER(RpsPivots), C.POINTER(RpsRowStats),
                              C.POINTER(RpsBranchScores), C.POINTER(RpsCommitOut), _p, C.c_size_t, _p, C.c_size_t, _p]
_lib.rps_decode_advance.restype = C.c_int
_lib.rps_decode_advance.argtypes = [C.POINTER(RpsPivots), C.POINTER(RpsCommitOut), C.c_int32, C.c_int32, C.c_int32,
                                    _p, _p, _p, _p, _p, _p, _p]
_lib.rps_gather_rows.restype = C.c_int
_lib.rps_gather_rows.argtypes = [C.POINTER(RpsLogits), C.POINTER(RpsRowList), C.POINTER(RpsLogits), _p]
_lib.rps_poll_device_status.restype = C.c_int
_lib.rps_poll_device_status.argtypes = [_p, C.POINTER(C.c_uint32)]
_lib.rps_status_string.restype = C.c_char_p
_lib.rps_status_string.argtypes = [C.c_int]
_lib.rps_version.restype = C.c_int32
_lib.rps_version.argtypes = []
class RpsLmhead(C.Structure):
    _fields_ = [("hidden", _p), ("unembed", _p), ("n_rows", C.c_int32), ("d", C.c_int32), ("vocab", C.c_int64),
                ("hidden_stride", C.c_int64), ("unembed_stride", C.c_int64), ("unembed_packed", C.c_int32)]


_lib.rps_lmhead_packed_bytes.restype = C.c_size_t
_lib.rps_lmhead_packed_bytes.argtypes = [C.c_int64, C.c_int32]
_lib.rps_lmhead_pack_unembed.restype = C.c_int
_lib.rps_lmhead_pack_unembed.argtypes = [_p, C.c_int64, C.c_int32, C.c_int64, _p, C.c_size_t, _p]
_lib.rps_lmhead_workspace_bytes.restype = C.c_size_t
_lib.rps_lmhead_workspace_bytes.argtypes = [C.c_int32, C.c_int64, C.c_int32]
_lib.rps_lmhead_row_stats.restype = C.c_int
_lib.rps_lmhead_row_stats.argtypes = [C.POINTER(RpsLmhead), C.POINTER(RpsParams), C.POINTER(RpsRowStats), _p, _p,
                                      C.c_size_t, _p]
class RpsPackedAttention(C.Structure):
    _fields_ = [("q", _p), ("k", _p), ("vt", _p), ("out", _p), ("n_batch", C.c_int32), ("n_heads", C.c_int32),
                ("head_dim", C.c_int32), ("n_context", C.c_int32), ("n_branch", C.c_int32),
                ("branch_len", C.c_int32), ("scale", C.c_float)]


_lib.rps_packed_attention_fwd.restype = C.c_int
_lib.rps_packed_attention_fwd.argtypes = [C.POINTER(RpsPackedAttention), _p]
_lib.rps_debug_set_ring_wait_ns.restype = C.c_uint64
_lib.rps_debug_set_ring_wait_ns.argtypes = [C.c_uint64]


class RPSError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {_lib.rps_status_string(status).decode()}")


def _check(status: int, where: str) -> None:
    if status != RPS_OK:
        raise RPSError(status, where)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def params(p) -> RpsParams:
    """C struct from any object with the ``configs.Params`` fields."""
    return RpsParams(p.k_max, p.r, p.tau_pivot, p.tau, p.lam, p.n_pivots, p.tokens_per_pivot,
                     getattr(p, "pivot_rule", 0), getattr(p, "commit_rule", 0), getattr(p, "commit_k", 0))


def logits_desc(t: torch.Tensor) -> RpsLogits:
    """Descriptor of a ``[n_req][n_branch][n_pos][vocab]`` bf16 / fp32 CUDA tensor."""
    if t.dim() != 4 or t.stride(3) != 1:
        raise ValueError("logits must be 4-D with a contiguous vocab dimension")
    if t.dtype == torch.bfloat16:
        dt = RPS_BF16
    elif t.dtype == torch.float32:
        dt = RPS_F32
    else:
        raise TypeError(f"logits must be bf16 or fp32, got {t.dtype}")
    n_req, nb, L, V = t.shape
    return RpsLogits(t.data_ptr(), dt, n_req, nb, L, V, t.stride(0), t.stride(1), t.stride(2))


# --------------------------------------------------------------------------- buffers
@dataclass
class RowStatsBuf:
    zmax: torch.Tensor
    lse: torch.Tensor
    H: torch.Tensor
    pmax: torch.Tensor
    argmax: torch.Tensor
    mu: Optional[torch.Tensor] = None
    htrunc: Optional[torch.Tensor] = None
    topk_idx: Optional[torch.Tensor] = None
    topk_logit: Optional[torch.Tensor] = None

    @staticmethod
    def alloc(n: int, k: int, device) -> "RowStatsBuf":
        f = lambda *s: torch.full(s, float("nan"), dtype=torch.float32, device=device)
        i = lambda *s: torch.full(s, -1, dtype=torch.int32, device=device)
        if k > 0:
            return RowStatsBuf(f(n), f(n), f(n), f(n), i(n), f(n), f(n), i(n, k), f(n, k))
        return RowStatsBuf(f(n), f(n), f(n), f(n), i(n))

    def c(self) -> RpsRowStats:
        return RpsRowStats(*(_ptr(getattr(self, f.name)) for f in fields(self)))


@dataclass
class PivotsBuf:
    n_commit: torch.Tensor
    commit_pos: torch.Tensor
    commit_tok: torch.Tensor
    rem_cnt: torch.Tensor
    rem_k: torch.Tensor
    rem_pos: torch.Tensor
    state: torch.Tensor
    pivot_k: torch.Tensor
    pivot_pos: torch.Tensor
    n_cand: torch.Tensor
    cand_tok: torch.Tensor
    branch_valid: torch.Tensor
    branch_off: torch.Tensor
    branch_cnt: torch.Tensor
    n_branch_rows: torch.Tensor
    branch_rows: torch.Tensor

    @staticmethod
    def alloc(n_req: int, L: int, P: int, K: int, device) -> "PivotsBuf":
        i = lambda *s: torch.full(s, -1, dtype=torch.int32, device=device)
        NB = P * K
        return PivotsBuf(i(n_req), i(n_req, L), i(n_req, L), i(n_req), i(n_req, L), i(n_req, L), i(n_req),
                         i(n_req, P), i(n_req, P), i(n_req, P), i(n_req, P, K),
                         torch.zeros(n_req, NB, dtype=torch.uint8, device=device), i(n_req, NB), i(n_req, NB),
                         i(n_req), i(n_req, NB * L, 3))

    def c(self) -> RpsPivots:
        return RpsPivots(*(_ptr(getattr(self, n)) for n in _PIVOT_FIELDS))


@dataclass
class ScoresBuf:
    mean_H: torch.Tensor
    n_tau: torch.Tensor
    log_a: torch.Tensor
    score: torch.Tensor

    @staticmethod
    def alloc(n_req: int, P: int, K: int, device) -> "ScoresBuf":
        f = lambda: torch.full((n_req, P, K + 1), float("nan"), dtype=torch.float32, device=device)
        return ScoresBuf(f(), torch.full((n_req, P, K + 1), -1, dtype=torch.int32, device=device), f(), f())

    def c(self) -> RpsBranchScores:
        return RpsBranchScores(*(_ptr(getattr(self, f.name)) for f in fields(self)))


@dataclass
class CommitBuf:
    best_slot: torch.Tensor
    gain: torch.Tensor
    winner: torch.Tensor
    commit_pos: torch.Tensor
    commit_tok: torch.Tensor
    margin: torch.Tensor
    mask_pos: torch.Tensor
    mask_cnt: torch.Tensor

    @staticmethod
    def alloc(n_req: int, L: int, P: int, device) -> "CommitBuf":
        i = lambda *s: torch.full(s, -1, dtype=torch.int32, device=device)
        f = lambda *s: torch.full(s, float("nan"), dtype=torch.float32, device=device)
        return CommitBuf(i(n_req, P), f(n_req, P), i(n_req), i(n_req), i(n_req), f(n_req), i(n_req, L), i(n_req))

    def c(self) -> RpsCommitOut:
        return RpsCommitOut(*(_ptr(getattr(self, f.name)) for f in fields(self)))


# --------------------------------------------------------------------------- ABI calls
def rps_version() -> int:
    return _lib.rps_version()


def rps_debug_set_ring_wait_ns(ns: int) -> int:
    """Testing hook: the row-statistics kernels' limit on each ring-copy wait
    (0 gives up at once; ``2**64 - 1`` restores the default). Returns the previous limit."""
    return _lib.rps_debug_set_ring_wait_ns(ns)


def rps_status_string(status: int) -> str:
    return _lib.rps_status_string(status).decode()


def rps_workspace_bytes(max_rows: int, vocab: int, k_max: int, dtype=RPS_BF16) -> int:
    """Workspace bytes; dtype is an RPS_* code or a torch dtype of the logits."""
    if not isinstance(dtype, int):
        dtype = RPS_BF16 if dtype == torch.bfloat16 else RPS_F32
    n = _lib.rps_workspace_bytes(max_rows, vocab, dtype, k_max)
    if n == 0:
        raise RPSError(RPS_ERR_INVALID_ARG, "rps_workspace_bytes")
    return n


def rps_workspace_init(ws: torch.Tensor, stream=None) -> None:
    _check(_lib.rps_workspace_init(ws.data_ptr(), ws.numel() * ws.element_size(), _stream(stream)),
           "rps_workspace_init")


def rps_score_step(logits: torch.Tensor, rows: Optional[torch.Tensor], seg_cnt: Optional[torch.Tensor], n_seg: int,
                   cap: int, prm, out: RowStatsBuf, ws: torch.Tensor, stream=None,
                   mask_pos: Optional[torch.Tensor] = None, mask_branch: int = 0) -> None:
    desc = logits_desc(logits)
    rl = RpsRowList(_ptr(rows), _ptr(seg_cnt), n_seg, cap, _ptr(mask_pos), mask_branch)
    p = params(prm)
    st = out.c()
    _check(_lib.rps_score_step(C.byref(desc), C.byref(rl), C.byref(p), C.byref(st), ws.data_ptr(),
                               ws.numel() * ws.element_size(), _stream(stream)), "rps_score_step")


def rps_score_step_noalloc(logits: torch.Tensor, rows: Optional[torch.Tensor], seg_cnt: Optional[torch.Tensor],
                           n_seg: int, cap: int, prm, out: RowStatsBuf, stream=None,
                           mask_pos: Optional[torch.Tensor] = None, mask_branch: int = 0) -> None:
    """rps_score_step with the library's fixed scratch instead of a caller workspace,
    for callers that cannot allocate device memory (see include/rps.h)."""
    desc = logits_desc(logits)
    rl = RpsRowList(_ptr(rows), _ptr(seg_cnt), n_seg, cap, _ptr(mask_pos), mask_branch)
    p = params(prm)
    st = out.c()
    _check(_lib.rps_score_step_noalloc(C.byref(desc), C.byref(rl), C.byref(p), C.byref(st), _stream(stream)),
           "rps_score_step_noalloc")


def rps_gather_rows(src: torch.Tensor, rows: Optional[torch.Tensor], seg_cnt: Optional[torch.Tensor], n_seg: int,
                    cap: int, dst: torch.Tensor, stream=None, mask_pos: Optional[torch.Tensor] = None,
                    mask_branch: int = 0) -> None:
    """Copy the listed rows of ``src`` (a CUDA tensor, or a page-locked CPU tensor the
    GPU reads over the host link) into the same places of the CUDA tensor ``dst``."""
    if src.shape != dst.shape or src.dtype != dst.dtype:
        raise ValueError("src and dst must have the same shape and dtype")
    if not src.is_cuda and not src.is_pinned():
        raise ValueError("a host src must be page-locked (pin_memory)")
    s, d = logits_desc(src), logits_desc(dst)
    rl = RpsRowList(_ptr(rows), _ptr(seg_cnt), n_seg, cap, _ptr(mask_pos), mask_branch)
    _check(_lib.rps_gather_rows(C.byref(s), C.byref(rl), C.byref(d), _stream(stream)), "rps_gather_rows")


def rps_select_pivots(base: RowStatsBuf, n_req: int, L: int, mask_pos: torch.Tensor, mask_cnt: torch.Tensor, prm,
                      out: PivotsBuf, stream=None) -> None:
    b, p, o = base.c(), params(prm), out.c()
    _check(_lib.rps_select_pivots(C.byref(b), n_req, L, mask_pos.data_ptr(), mask_cnt.data_ptr(), C.byref(p),
                                  C.byref(o), _stream(stream)), "rps_select_pivots")


def rps_score_branches(anchor_logits: torch.Tensor, anchor_branch: int, anchor: RowStatsBuf, branch: RowStatsBuf,
                       n_req: int, L: int, piv: PivotsBuf, prm, out: ScoresBuf, stream=None) -> None:
    d, a, b, pv, p, o = logits_desc(anchor_logits), anchor.c(), branch.c(), piv.c(), params(prm), out.c()
    _check(_lib.rps_score_branches(C.byref(d), anchor_branch, C.byref(a), C.byref(b), n_req, L, C.byref(pv),
                                   C.byref(p), C.byref(o), _stream(stream)), "rps_score_branches")


def rps_commit(scores: ScoresBuf, n_req: int, L: int, piv: PivotsBuf, prm, out: CommitBuf, stream=None) -> None:
    s, pv, p, o = scores.c(), piv.c(), params(prm), out.c()
    _check(_lib.rps_commit(C.byref(s), n_req, L, C.byref(pv), C.byref(p), C.byref(o), _stream(stream)),
           "rps_commit")


def rps_score_and_commit(anchor_logits: torch.Tensor, anchor_branch: int, anchor: RowStatsBuf, branch: RowStatsBuf,
                         n_req: int, L: int, piv: PivotsBuf, prm, scores: ScoresBuf, out: CommitBuf,
                         stream=None) -> None:
    d, a, b, pv, p = logits_desc(anchor_logits), anchor.c(), branch.c(), piv.c(), params(prm)
    s, o = scores.c(), out.c()
    _check(_lib.rps_score_and_commit(C.byref(d), anchor_branch, C.byref(a), C.byref(b), n_req, L, C.byref(pv),
                                     C.byref(p), C.byref(s), C.byref(o), _stream(stream)), "rps_score_and_commit")


def rps_run_step(logits: torch.Tensor, n_req: int, L: int, mask_pos: torch.Tensor, mask_cnt: torch.Tensor, prm,
                 base: RowStatsBuf, piv: PivotsBuf, branch: RowStatsBuf, scores: ScoresBuf, out: CommitBuf,
                 ws_base: torch.Tensor, ws_branch: torch.Tensor, stream=None) -> None:
    d, p = logits_desc(logits), params(prm)
    b, pv, br, sc, o = base.c(), piv.c(), branch.c(), scores.c(), out.c()
    _check(_lib.rps_run_step(C.byref(d), n_req, L, mask_pos.data_ptr(), mask_cnt.data_ptr(), C.byref(p), C.byref(b),
                             C.byref(pv), C.byref(br), C.byref(sc), C.byref(o), ws_base.data_ptr(),
                             ws_base.numel() * ws_base.element_size(), ws_branch.data_ptr(),
                             ws_branch.numel() * ws_branch.element_size(), _stream(stream)), "rps_run_step")


def rps_decode_advance(piv: PivotsBuf, commit: CommitBuf, n_req: int, B: int, L_total: int, tokens, block, mask_pos,
                       mask_cnt, done, steps=None, stream=None) -> None:
    pv, cm = piv.c(), commit.c()
    _check(_lib.rps_decode_advance(C.byref(pv), C.byref(cm), n_req, B, L_total, tokens.data_ptr(), block.data_ptr(),
                                   mask_pos.data_ptr(), mask_cnt.data_ptr(), done.data_ptr(),
                                   None if steps is None else steps.data_ptr(), _stream(stream)),
           "rps_decode_advance")


def rps_poll_device_status(stream=None):
    """Synchronise and return (status, detail bits); clears the device error word."""
    detail = C.c_uint32(0)
    st = _lib.rps_poll_device_status(_stream(stream), C.byref(detail))
    return st, detail.value


def rps_lmhead_workspace_bytes(n_rows: int, vocab: int, k_max: int) -> int:
    n = _lib.rps_lmhead_workspace_bytes(n_rows, vocab, k_max)
    if n == 0:
        raise RPSError(RPS_ERR_INVALID_ARG, "rps_lmhead_workspace_bytes")
    return n


def rps_lmhead_pack_unembed(unembed: torch.Tensor, stream=None) -> torch.Tensor:
    """The unembedding ``[V][d]`` (bf16 CUDA tensor) in the LM head's packed tile
    layout, as a new uint8 CUDA tensor (a one-time re-layout of the weight)."""
    if unembed.dtype != torch.bfloat16 or unembed.dim() != 2 or unembed.stride(1) != 1:
        raise ValueError("unembed must be a bf16 [V][d] tensor with d contiguous")
    V, d = unembed.shape
    n = _lib.rps_lmhead_packed_bytes(V, d)
    if n == 0:
        raise RPSError(RPS_ERR_INVALID_ARG, "rps_lmhead_packed_bytes")
    packed = torch.empty(n, dtype=torch.uint8, device=unembed.device)
    _check(_lib.rps_lmhead_pack_unembed(unembed.data_ptr(), V, d, unembed.stride(0), packed.data_ptr(), n,
                                        _stream(stream)), "rps_lmhead_pack_unembed")
    return packed


def rps_lmhead_row_stats(hidden: torch.Tensor, unembed: torch.Tensor, prm, out: RowStatsBuf, ws: torch.Tensor,
                         logits_out: Optional[torch.Tensor] = None, stream=None,
                         packed: Optional[torch.Tensor] = None) -> None:
    """Row statistics of ``hidden @ unembed.T`` (bf16 CUDA tensors ``[n][d]`` and
    ``[V][d]``) into ``out``; ``logits_out`` (fp32 ``[n][V]``, testing) also
    receives the logits. With ``packed`` (from rps_lmhead_pack_unembed of the
    same unembedding) the kernel reads the packed copy instead."""
    if hidden.dtype != torch.bfloat16 or unembed.dtype != torch.bfloat16:
        raise TypeError("hidden and unembed must be bf16")
    if hidden.dim() != 2 or unembed.dim() != 2 or hidden.stride(1) != 1 or unembed.stride(1) != 1:
        raise ValueError("hidden [n][d] and unembed [V][d] with d contiguous")
    src = unembed.data_ptr() if packed is None else packed.data_ptr()
    lm = RpsLmhead(hidden.data_ptr(), src, hidden.shape[0], hidden.shape[1], unembed.shape[0],
                   hidden.stride(0), unembed.stride(0), 0 if packed is None else 1)
    p = params(prm) if prm is not None else None
    st = out.c()
    _check(_lib.rps_lmhead_row_stats(C.byref(lm), None if p is None else C.byref(p), C.byref(st), _ptr(logits_out),
                                     ws.data_ptr(), ws.numel() * ws.element_size(), _stream(stream)),
           "rps_lmhead_row_stats")


def rps_packed_attention_fwd(q: torch.Tensor, k: torch.Tensor, vt: torch.Tensor, out: torch.Tensor, n_context: int,
                             n_branch: int, branch_len: int, scale: float, stream=None) -> None:
    """Branch-isolating attention of a packed lookahead sequence: q, k, out
    ``[batch][heads][tokens][128]`` and vt ``[batch][heads][128][tokens]``, bf16 CUDA tensors."""
    for t in (q, k, vt, out):
        if t.dtype != torch.bfloat16 or not t.is_contiguous() or t.dim() != 4:
            raise ValueError("q, k, vt and out must be contiguous 4-D bf16 tensors")
    n_b, n_h, n_tok, d = q.shape
    if k.shape != q.shape or out.shape != q.shape or vt.shape != (n_b, n_h, d, n_tok):
        raise ValueError("shapes: q, k, out [b][h][tokens][d] and vt [b][h][d][tokens]")
    if n_tok != n_context + n_branch * branch_len:
        raise ValueError("tokens must be n_context + n_branch * branch_len")
    a = RpsPackedAttention(q.data_ptr(), k.data_ptr(), vt.data_ptr(), out.data_ptr(), n_b, n_h, d, n_context,
                           n_branch, branch_len, scale)
    _check(_lib.rps_packed_attention_fwd(C.byref(a), _stream(stream)), "rps_packed_attention_fwd")


# --------------------------------------------------------------------------- one step
class Step:
    """Preallocated buffers and the ABI calls of one RPS decoding step.

    The base branch (0) of ``logits`` is the anchor, as in the workloads here.
    Kernels launched per ``run`` (one rps_run_step call): row statistics of the
    masked base rows and their top-k lists (top-k mode: two launches), pivot
    selection, row statistics of the lookahead rows, and branch scores with the
    commit decision in one launch. ``run_calls`` makes the same five launches
    through the separate calls.
    """
    LAUNCHES = 5

    def __init__(self, n_req: int, L: int, V: int, prm, device, dtype=torch.bfloat16):
        self.n_req, self.L, self.V, self.prm = n_req, L, V, prm
        P, K, k = prm.n_pivots, prm.tokens_per_pivot, prm.k_max
        self.NB = P * K
        self.base = RowStatsBuf.alloc(n_req * L, k, device)
        self.branch = RowStatsBuf.alloc(n_req * self.NB * L, 0, device)
        self.piv = PivotsBuf.alloc(n_req, L, P, K, device)
        self.scores = ScoresBuf.alloc(n_req, P, K, device)
        self.commit = CommitBuf.alloc(n_req, L, P, device)
        base_ws = rps_workspace_bytes(n_req * L, V, k, dtype)
        br_ws = rps_workspace_bytes(n_req * self.NB * L, V, 0, dtype)
        self.ws_base = torch.empty(base_ws, dtype=torch.uint8, device=device)
        self.ws_branch = torch.empty(br_ws, dtype=torch.uint8, device=device)
        rps_workspace_init(self.ws_base)
        rps_workspace_init(self.ws_branch)

    def score_base(self, logits, mask_pos, mask_cnt, stream=None):
        rps_score_step(logits, None, mask_cnt, self.n_req, self.L, self.prm, self.base, self.ws_base, stream,
                       mask_pos=mask_pos, mask_branch=0)

    def select(self, mask_pos, mask_cnt, stream=None):
        rps_select_pivots(self.base, self.n_req, self.L, mask_pos, mask_cnt, self.prm, self.piv, stream)

    def score_branch_rows(self, logits, stream=None):
        rps_score_step(logits, self.piv.branch_rows, self.piv.n_branch_rows, self.n_req, self.NB * self.L, self.prm,
                       self.branch, self.ws_branch, stream)

    def score(self, logits, stream=None):
        rps_score_branches(logits, 0, self.base, self.branch, self.n_req, self.L, self.piv, self.prm, self.scores,
                           stream)

    def decide(self, stream=None):
        rps_commit(self.scores, self.n_req, self.L, self.piv, self.prm, self.commit, stream)

    def score_and_decide(self, logits, stream=None):
        rps_score_and_commit(logits, 0, self.base, self.branch, self.n_req, self.L, self.piv, self.prm, self.scores,
                             self.commit, stream)

    def run(self, logits, mask_pos, mask_cnt, stream=None):
        rps_run_step(logits, self.n_req, self.L, mask_pos, mask_cnt, self.prm, self.base, self.piv, self.branch,
                     self.scores, self.commit, self.ws_base, self.ws_branch, stream)

    def run_calls(self, logits, mask_pos, mask_cnt, stream=None):
        self.score_base(logits, mask_pos, mask_cnt, stream)
        self.select(mask_pos, mask_cnt, stream)
        self.score_branch_rows(logits, stream)
        self.score_and_decide(logits, stream)

    def run_host(self, host_logits, dev_logits, mask_pos, mask_cnt, stream=None):
        """``run`` on logits that sit in page-locked host memory: only the rows the
        step reads (the masked base rows, then the listed lookahead rows) are
        gathered into ``dev_logits`` before they are scored; the lookahead list
        stays on the device, so there is no host synchronisation in the step."""
        n_req, L = self.n_req, self.L
        rps_gather_rows(host_logits, None, mask_cnt, n_req, L, dev_logits, stream, mask_pos=mask_pos, mask_branch=0)
        self.score_base(dev_logits, mask_pos, mask_cnt, stream)
        self.select(mask_pos, mask_cnt, stream)
        rps_gather_rows(host_logits, self.piv.branch_rows, self.piv.n_branch_rows, n_req, self.NB * L, dev_logits,
                        stream)
        self.score_branch_rows(dev_logits, stream)
        self.score_and_decide(dev_logits, stream)
