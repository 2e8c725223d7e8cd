"""ctypes front end of the CPU oracle (``rps_oracle.c``).

TEST INFRASTRUCTURE. Only the test-suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg use this module; the library never imports it.

Logits are numpy arrays: ``uint16`` holds bf16 bit patterns, ``float32`` holds
fp32 logits. Statistics come back in fp64.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass
from pathlib import Path
from typing import Optional

import numpy as np

from .build import LIBRARY, build_oracle, oracle_up_to_date

STATE_SEARCH, STATE_DONE, STATE_NO_FEASIBLE, STATE_NO_CANDIDATES = 0, 1, 2, 3
WIN_ANCHOR, WIN_SKIP, WIN_DONE = -1, -2, -3

_i32p = np.ctypeslib.ndpointer(dtype=np.int32, flags="C_CONTIGUOUS")
_i64p = np.ctypeslib.ndpointer(dtype=np.int64, flags="C_CONTIGUOUS")
_f64p = np.ctypeslib.ndpointer(dtype=np.float64, flags="C_CONTIGUOUS")
_u8p = np.ctypeslib.ndpointer(dtype=np.uint8, flags="C_CONTIGUOUS")


def dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.uint16:
        return 1
    if a.dtype == np.float32:
        return 0
    raise TypeError(f"logits must be uint16 (bf16 bits) or float32, got {a.dtype}")


@dataclass
class RowStats:
    zmax: np.ndarray
    lse: np.ndarray
    H: np.ndarray
    pmax: np.ndarray
    mu: Optional[np.ndarray]
    htrunc: Optional[np.ndarray]
    argmax: np.ndarray
    topk_idx: Optional[np.ndarray]    # [n][k]
    topk_logit: Optional[np.ndarray]  # [n][k]

    @staticmethod
    def empty(n: int, k: int) -> "RowStats":
        nan = lambda: np.full(n, np.nan)
        return RowStats(nan(), nan(), nan(), nan(), nan(), nan(), np.full(n, -1, np.int32),
                        np.full((n, max(k, 1)), -1, np.int32), np.full((n, max(k, 1)), np.nan))

    def scatter(self, dst: "RowStats", where: np.ndarray) -> None:
        for name in ("zmax", "lse", "H", "pmax", "mu", "htrunc", "argmax"):
            src = getattr(self, name)
            if src is not None:
                getattr(dst, name)[where] = src
        if self.topk_idx is not None and dst.topk_idx is not None:
            k = self.topk_idx.shape[1]
            dst.topk_idx[where, :k] = self.topk_idx
            dst.topk_logit[where, :k] = self.topk_logit


class Oracle:
    def __init__(self, path: Path = LIBRARY):
        path = Path(path)
        if path == LIBRARY and not oracle_up_to_date():
            build_oracle()
        self.lib = C.CDLL(str(path))
        L = self.lib
        L.rps_oracle_row_stats.restype = C.c_int64
        L.rps_oracle_row_stats.argtypes = [C.c_void_p, C.c_int32, C.c_int64, _i64p, C.c_int64, C.c_int32,
                                           _f64p, _f64p, _f64p, _f64p, C.c_void_p, C.c_void_p, _i32p,
                                           C.c_void_p, C.c_void_p]
        L.rps_oracle_select_pivots.restype = None
        L.rps_oracle_select_pivots.argtypes = (
            [C.c_int32, C.c_int32, _i32p, _i32p, _f64p, _f64p, _i32p, _f64p, _f64p, _f64p, _i32p, _f64p,
             C.c_int32, C.c_double, C.c_double, C.c_double, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int32]
            + [_i32p] * 11 + [_u8p, _i32p, _i32p, _i32p, _i32p])
        L.rps_oracle_score_branches.restype = None
        L.rps_oracle_score_branches.argtypes = (
            [C.c_int32] * 4 + [_i32p] * 7 + [_u8p, _i32p, _i32p] + [_f64p] * 6
            + [C.c_void_p, C.c_int32, C.c_int64, C.c_int64, C.c_double, C.c_double,
               _f64p, _i32p, _f64p, _f64p])
        L.rps_oracle_commit.restype = None
        L.rps_oracle_commit.argtypes = (
            [C.c_int32] * 4 + [_i32p] * 4 + [_u8p, _f64p, _i32p, _i32p, _i32p, _f64p]
            + [_i32p] * 3 + [_f64p, _i32p, _i32p])

    # ------------------------------------------------------------------ rows
    def row_stats_at(self, tensor: np.ndarray, row_off: np.ndarray, k: int) -> RowStats:
        """Statistics of the rows starting at element offsets ``row_off`` of ``tensor``."""
        t = np.ascontiguousarray(tensor)
        V = t.shape[-1]
        off = np.ascontiguousarray(row_off, dtype=np.int64)
        n = off.shape[0]
        if n and (off.min() < 0 or off.max() + V > t.size):
            raise IndexError("row offset outside the tensor")
        st = RowStats.empty(n, k)
        if k == 0:
            st.mu = st.htrunc = st.topk_idx = st.topk_logit = None
        mu_p = st.mu.ctypes.data if k else None
        ht_p = st.htrunc.ctypes.data if k else None
        ti_p = st.topk_idx.ctypes.data if k else None
        tl_p = st.topk_logit.ctypes.data if k else None
        self.lib.rps_oracle_row_stats(t.ctypes.data, dtype_code(t), V, off, n, k, st.zmax, st.lse, st.H,
                                      st.pmax, mu_p, ht_p, st.argmax, ti_p, tl_p)
        return st

    def row_stats(self, rows: np.ndarray, k: int) -> RowStats:
        """Statistics of each row of a 2-D ``[n][V]`` array."""
        rows = np.ascontiguousarray(rows)
        if rows.ndim == 1:
            rows = rows[None]
        off = np.arange(rows.shape[0], dtype=np.int64) * rows.shape[1]
        return self.row_stats_at(rows, off, k)

    # ------------------------------------------------------------ decisions
    def select_pivots(self, mask_pos, mask_cnt, base: RowStats, params) -> dict:
        n_req, L = mask_pos.shape
        P, K, k_max = params.n_pivots, params.tokens_per_pivot, params.k_max
        NB = P * K
        z = lambda *s, v=0: np.full(s, v, dtype=np.int32)
        out = dict(n_commit=z(n_req), commit_pos=z(n_req, L, v=-1), commit_tok=z(n_req, L, v=-1),
                   rem_cnt=z(n_req), rem_k=z(n_req, L, v=-1), rem_pos=z(n_req, L, v=-1), state=z(n_req),
                   pivot_k=z(n_req, P), pivot_pos=z(n_req, P), n_cand=z(n_req, P), cand_tok=z(n_req, P, K),
                   branch_valid=np.zeros((n_req, NB), np.uint8), branch_off=z(n_req, NB),
                   branch_cnt=z(n_req, NB), n_branch_rows=z(n_req),
                   branch_rows=z(n_req, NB * L, 3, v=-1))
        ti = np.ascontiguousarray(base.topk_idx[:, :k_max], dtype=np.int32)
        tl = np.ascontiguousarray(base.topk_logit[:, :k_max], dtype=np.float64)
        self.lib.rps_oracle_select_pivots(
            n_req, L, np.ascontiguousarray(mask_pos, np.int32), np.ascontiguousarray(mask_cnt, np.int32),
            base.zmax, base.pmax, base.argmax, base.mu, base.htrunc, base.H, ti, tl, k_max,
            float(np.float32(params.r)), float(np.float32(params.tau_pivot)), float(np.float32(params.tau)),
            P, K, getattr(params, "commit_rule", 0), getattr(params, "commit_k", 0), getattr(params, "pivot_rule", 0),
            out["n_commit"], out["commit_pos"], out["commit_tok"], out["rem_cnt"], out["rem_k"],
            out["rem_pos"], out["state"], out["pivot_k"], out["pivot_pos"], out["n_cand"], out["cand_tok"],
            out["branch_valid"], out["branch_off"], out["branch_cnt"], out["n_branch_rows"],
            out["branch_rows"])
        return out

    def score_branches(self, piv: dict, branch: RowStats, anchor: RowStats, anchor_logits: np.ndarray,
                       params) -> dict:
        """``anchor_logits`` is the anchor branch, shaped ``[n_req][L][V]`` (any strides)."""
        n_req, L = piv["rem_k"].shape
        P, K = params.n_pivots, params.tokens_per_pivot
        shape = (n_req, P, K + 1)
        out = dict(mean_H=np.full(shape, np.nan), n_tau=np.full(shape, -1, np.int32),
                   log_a=np.full(shape, np.nan), score=np.full(shape, np.nan))
        a = anchor_logits
        esz = a.dtype.itemsize
        if a.strides[-1] != esz:
            raise ValueError("anchor rows must be contiguous")
        self.lib.rps_oracle_score_branches(
            n_req, L, P, K, piv["state"], piv["rem_cnt"], piv["rem_k"], piv["pivot_k"], piv["pivot_pos"],
            piv["n_cand"], piv["cand_tok"], piv["branch_valid"], piv["branch_off"], piv["branch_cnt"],
            np.ascontiguousarray(branch.H), np.ascontiguousarray(branch.pmax),
            np.ascontiguousarray(anchor.H), np.ascontiguousarray(anchor.pmax),
            np.ascontiguousarray(anchor.lse), np.ascontiguousarray(anchor.zmax),
            a.ctypes.data, dtype_code(a), a.strides[0] // esz, a.strides[1] // esz,
            float(np.float32(params.lam)), float(np.float32(params.tau)),
            out["mean_H"], out["n_tau"], out["log_a"], out["score"])
        return out

    def commit(self, piv: dict, scores: dict, params) -> dict:
        n_req, L = piv["rem_k"].shape
        P, K = params.n_pivots, params.tokens_per_pivot
        out = dict(best_slot=np.full((n_req, P), -1, np.int32), gain=np.full((n_req, P), np.nan),
                   winner=np.zeros(n_req, np.int32), commit_pos=np.zeros(n_req, np.int32),
                   commit_tok=np.zeros(n_req, np.int32), margin=np.zeros(n_req),
                   mask_cnt=np.zeros(n_req, np.int32), mask_pos=np.full((n_req, L), -1, np.int32))
        self.lib.rps_oracle_commit(
            n_req, L, P, K, piv["state"], piv["pivot_pos"], piv["n_cand"], piv["cand_tok"],
            piv["branch_valid"], np.ascontiguousarray(scores["score"]), piv["rem_cnt"], piv["rem_pos"],
            out["best_slot"], out["gain"], out["winner"], out["commit_pos"], out["commit_tok"],
            out["margin"], out["mask_cnt"], out["mask_pos"])
        return out

    # ------------------------------------------------------------ full step
    def base_stats(self, logits: np.ndarray, mask_pos, mask_cnt, k_max: int, branch: int = 0) -> RowStats:
        """Statistics of the masked rows of one branch, in ``[req * L + k]`` layout."""
        n_req, nb1, L, V = logits.shape
        st = RowStats.empty(n_req * L, k_max)
        where, off = [], []
        for q in range(n_req):
            for k in range(int(mask_cnt[q])):
                where.append(q * L + k)
                off.append(((q * nb1 + branch) * L + int(mask_pos[q, k])) * V)
        if where:
            self.row_stats_at(logits, np.array(off, np.int64), k_max).scatter(st, np.array(where))
        return st

    def branch_stats(self, logits: np.ndarray, piv: dict, n_branch: int) -> RowStats:
        """Statistics of the listed lookahead rows, compact layout ``[req * NB * L + i]``."""
        n_req, nb1, L, V = logits.shape
        st = RowStats.empty(n_req * n_branch * L, 0)
        where, off = [], []
        for q in range(n_req):
            rows = piv["branch_rows"][q]
            for i in range(int(piv["n_branch_rows"][q])):
                rq, rb, rp = (int(x) for x in rows[i])
                where.append(q * n_branch * L + i)
                off.append(((rq * nb1 + rb) * L + rp) * V)
        if where:
            self.row_stats_at(logits, np.array(off, np.int64), 0).scatter(st, np.array(where))
        return st

    def step(self, logits: np.ndarray, mask_pos, mask_cnt, params) -> dict:
        """One decoding step of the scoring path with the base branch as anchor."""
        n_req, nb1, L, V = logits.shape
        if nb1 != 1 + params.n_branch:
            raise ValueError("branch count does not match the parameters")
        base = self.base_stats(logits, mask_pos, mask_cnt, params.k_max)
        piv = self.select_pivots(mask_pos, mask_cnt, base, params)
        br = self.branch_stats(logits, piv, params.n_branch)
        sc = self.score_branches(piv, br, base, logits[:, 0], params)
        cm = self.commit(piv, sc, params)
        return dict(base=base, pivots=piv, branch=br, scores=sc, commit=cm)


_DEFAULT: Optional[Oracle] = None


def default() -> Oracle:
    global _DEFAULT
    if _DEFAULT is None:
        _DEFAULT = Oracle()
    return _DEFAULT
