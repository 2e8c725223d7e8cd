"""Seeded synthetic logits for the RPS scoring path (host twin of ``csrc/synth.cu``).

This module is input generation only: it holds none of the scoring arithmetic
(no softmax, entropy, top-k or decision rule). It serves both the CPU oracle and
the CUDA path, which is why it lives on its own.

Workload shape (Sec. 3 "Decoding" and Algorithm 1 of the paper): one denoising
step produces, for every request, a base prediction plus one lookahead branch per
(pivot slot, candidate token) pair, each a ``[positions x vocab]`` block of logits.
The tensor layout is ``[n_req][1 + n_branch][L][V]``, branch 0 being the base
(which also serves as the anchor branch of Eq. 4).

Value model, per (request, position):

* a regime is drawn once: low entropy (one token raised by +12), mid entropy
  (2-5 distinct tokens raised by +4 each) or high entropy (no spike, logits / 0.5);
* every entry carries noise ``eps`` with unit variance;
* lookahead branch ``b`` repeats the base logits with the spike amplitude scaled
  by a factor ``f`` drawn uniformly from [0.8, 1.6);
* the result is rounded to bf16 (round to nearest even) or kept in fp32.

Exact reproducibility between this numpy code and the CUDA generator is the
design goal, so every step is integer arithmetic or a single IEEE-754 fp32
operation with round-to-nearest:

* counters are hashed with Philox4x32-10 (Salmon, Moraes, Dror, Shaw,
  "Parallel random numbers: as easy as 1, 2, 3", SC'11), written here from
  that published definition;
* ``eps`` is a scaled Irwin-Hall sum of eight 16-bit uniforms (variance 1,
  support about +-4.9 sigma), which needs no transcendental function and so has
  the same bits on both sides. It stands in for N(0, 1).
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Optional, Sequence

import numpy as np

# Philox4x32 multipliers and Weyl key increments (Salmon et al., SC'11).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85

# Stream tags, placed in the low byte of counter word 3.
TAG_NOISE = 1
TAG_REGIME = 2
TAG_SPIKES = 3
TAG_BRANCH = 4
TAG_MASK = 5
TAG_COUNT = 6

# Second key word: constant so that a seed alone selects the stream family.
KEY1 = 0x52505331

REGIME_LOW, REGIME_MID, REGIME_HIGH = 0, 1, 2
SPIKE_LOW = np.float32(12.0)
SPIKE_MID = np.float32(4.0)
HIGH_GAIN = np.float32(2.0)  # logits / 0.5
# eps = (2*S - 8*65535) * sqrt(1.5) / 131072 with S the sum of eight 16-bit uniforms.
EPS_SCALE = np.float32(math.sqrt(1.5) / 131072.0)
EPS_OFFSET = 8 * 65535
BRANCH_F_LO = np.float32(0.8)
BRANCH_F_SPAN = np.float32(0.8)
TWO_M24 = np.float32(2.0 ** -24)
MAX_SPIKE_DRAWS = 16  # Philox calls per row when drawing mid-regime tokens

_M32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Philox4x32 with 10 rounds over broadcastable uint32 arrays.

    Returns four uint32 arrays. Round i maps the counter (c0, c1, c2, c3) with key
    (k0, k1) to (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2), hi(M0*c0) ^ c3 ^ k1, lo(M0*c0)),
    and the key is advanced by the Weyl constants between rounds.
    """
    c0, c1, c2, c3 = (np.asarray(x, dtype=np.uint64) & _M32 for x in (c0, c1, c2, c3))
    k0 = np.uint64(int(k0) & 0xFFFFFFFF)
    k1 = np.uint64(int(k1) & 0xFFFFFFFF)
    m0 = np.uint64(PHILOX_M0)
    m1 = np.uint64(PHILOX_M1)
    for rnd in range(10):
        if rnd:
            k0 = np.uint64((int(k0) + PHILOX_W0) & 0xFFFFFFFF)
            k1 = np.uint64((int(k1) + PHILOX_W1) & 0xFFFFFFFF)
        p0 = m0 * c0
        p1 = m1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _M32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _M32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return tuple(x.astype(np.uint32) for x in (c0, c1, c2, c3))


def _tag(tag: int, epoch: int = 0) -> int:
    return (tag & 0xFF) | ((epoch & 0xFFFFFF) << 8)


def regime_thresholds(mixture: Sequence[float]):
    """Integer thresholds (t_low, t_mid) on a uint32 draw for a (low, mid, high) mixture."""
    p_low, p_mid, p_high = (float(p) for p in mixture)
    if min(p_low, p_mid, p_high) < 0 or abs(p_low + p_mid + p_high - 1.0) > 1e-9:
        raise ValueError(f"bad regime mixture {mixture}")
    t_low = min(int(round(p_low * 2 ** 32)), 2 ** 32)
    t_mid = min(int(round((p_low + p_mid) * 2 ** 32)), 2 ** 32)
    return t_low, t_mid


def bf16_round(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bits (uint16), round to nearest even. NaN stays NaN."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = ((b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16))
    out = rounded.astype(np.uint16)
    nan = np.isnan(np.asarray(x, dtype=np.float32))
    if nan.any():
        out = np.where(nan, np.uint16(0x7FC0), out)
    return out


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bits (uint16) -> fp32 values (exact)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclass(frozen=True)
class RowPlan:
    """The per-(request, position) draws that shape a row."""
    regime: int
    spikes: tuple  # token ids raised by the spike (empty for the high regime)


def row_plan(seed: int, V: int, req: int, pos: int, mixture) -> RowPlan:
    """Regime and spike tokens of position ``pos`` of request ``req``."""
    t_low, t_mid = regime_thresholds(mixture)
    x0, x1, x2, _ = philox4x32_10(0, pos, req, _tag(TAG_REGIME), seed, KEY1)
    x0, x1, x2 = int(x0), int(x1), int(x2)
    if x0 < t_low:
        return RowPlan(REGIME_LOW, (x1 % V,))
    if x0 < t_mid:
        want = min(2 + x2 % 4, V)
        toks: list = []
        for q in range(MAX_SPIKE_DRAWS):
            words = philox4x32_10(q, pos, req, _tag(TAG_SPIKES), seed, KEY1)
            for w in words:
                t = int(w) % V
                if len(toks) < want and t not in toks:
                    toks.append(t)
            if len(toks) >= want:
                break
        return RowPlan(REGIME_MID, tuple(toks))
    return RowPlan(REGIME_HIGH, ())


def noise_row(seed: int, V: int, req: int, pos: int, epoch: int = 0) -> np.ndarray:
    """fp32 noise for one (request, position), shared by the base and all its branches."""
    v = np.arange(V, dtype=np.uint64)
    x = philox4x32_10(v, pos, req, _tag(TAG_NOISE, epoch), seed, KEY1)
    s = np.zeros(V, dtype=np.int64)
    for w in x:
        w = w.astype(np.int64)
        s += (w & 0xFFFF) + (w >> 16)
    centred = (2 * s - EPS_OFFSET).astype(np.float32)  # exact: |value| < 2**20
    return centred * EPS_SCALE


def branch_factor(seed: int, req: int, branch: int, pos: int, step: int = 0) -> np.float32:
    """Spike scale factor in [0.8, 1.6) of lookahead branch ``branch`` (>= 1) at ``pos``."""
    x0, _, _, _ = philox4x32_10(branch, pos, req, _tag(TAG_BRANCH, step), seed, KEY1)
    u = np.float32(int(x0) >> 8) * TWO_M24
    return np.float32(BRANCH_F_LO + np.float32(BRANCH_F_SPAN * u))


def row_logits_f32(seed: int, V: int, req: int, branch: int, pos: int, mixture,
                   scale: float = 1.0, epoch: int = 0, step: int = 0) -> np.ndarray:
    """fp32 logits of row (req, branch, pos) before any bf16 rounding."""
    plan = row_plan(seed, V, req, pos, mixture)
    eps = noise_row(seed, V, req, pos, epoch)
    if plan.regime == REGIME_HIGH:
        return eps * HIGH_GAIN
    h = SPIKE_LOW if plan.regime == REGIME_LOW else SPIKE_MID
    f = np.float32(1.0) if branch == 0 else branch_factor(seed, req, branch, pos, step)
    amp = np.float32(np.float32(h * np.float32(scale)) * f)
    z = eps.copy()
    idx = np.array(plan.spikes, dtype=np.int64)
    z[idx] = eps[idx] + amp
    return z


def row_logits(seed: int, V: int, req: int, branch: int, pos: int, mixture, dtype: str,
               scale: float = 1.0, epoch: int = 0, step: int = 0) -> np.ndarray:
    """One row as stored: uint16 bf16 bits for ``dtype == 'bf16'``, float32 otherwise."""
    z = row_logits_f32(seed, V, req, branch, pos, mixture, scale, epoch, step)
    return bf16_round(z) if dtype == "bf16" else z


def make_logits(seed: int, n_req: int, n_branch: int, L: int, V: int, mixture, dtype: str,
                valid: Optional[np.ndarray] = None, scale: Optional[np.ndarray] = None,
                epoch: Optional[np.ndarray] = None, step: int = 0) -> np.ndarray:
    """Full ``[n_req][1 + n_branch][L][V]`` tensor (host; small shapes only).

    ``valid[req, pos] == 0`` fills that position's rows with NaN in every branch
    (padding that a correct scorer never reads). ``scale`` and ``epoch`` are the
    per-(request, position) spike scale and noise epoch used by multi-step replay.
    """
    np_dtype = np.uint16 if dtype == "bf16" else np.float32
    out = np.empty((n_req, 1 + n_branch, L, V), dtype=np_dtype)
    nan = np.uint16(0x7FC0) if dtype == "bf16" else np.float32(np.nan)
    for req in range(n_req):
        for pos in range(L):
            if valid is not None and not valid[req, pos]:
                out[req, :, pos, :] = nan
                continue
            sc = 1.0 if scale is None else float(scale[req, pos])
            ep = 0 if epoch is None else int(epoch[req, pos])
            for b in range(1 + n_branch):
                out[req, b, pos] = row_logits(seed, V, req, b, pos, mixture, dtype, sc, ep, step)
    return out


def masked_positions(seed: int, req: int, L: int, count: int) -> np.ndarray:
    """A seeded random subset of ``count`` positions out of ``L``, in increasing order."""
    if not 0 <= count <= L:
        raise ValueError("count out of range")
    pos = np.arange(L, dtype=np.uint64)
    key = philox4x32_10(pos, 0, req, _tag(TAG_MASK), seed, KEY1)[0].astype(np.int64)
    order = np.lexsort((np.arange(L), key))
    return np.sort(order[:count]).astype(np.int32)


def ragged_count(seed: int, req: int, lo: int, hi: int) -> int:
    """Masked count of request ``req`` drawn uniformly from [lo, hi]."""
    x0 = int(philox4x32_10(req, 0, 0, _tag(TAG_COUNT), seed, KEY1)[0])
    return lo + x0 % (hi - lo + 1)


# ---------------------------------------------------------------------------
# Device twin (librps_synth.so): the same bits, written straight into HBM.
# ---------------------------------------------------------------------------
_SYNTH_LIB = None


def _synth_lib():
    global _SYNTH_LIB
    if _SYNTH_LIB is None:
        import ctypes as C
        from pathlib import Path
        path = Path(__file__).resolve().parent / "librps_synth.so"
        if not path.exists():
            raise ImportError(f"{path} is missing: build the CUDA libraries first")
        lib = C.CDLL(str(path))
        lib.rps_synth_fill.restype = C.c_int32
        lib.rps_synth_fill.argtypes = [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int64,
                                       C.c_int64, C.c_int64, C.c_int64, C.c_uint32, C.c_uint64, C.c_uint64,
                                       C.c_uint32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
        lib.rps_synth_fill_blocks.restype = C.c_int32
        lib.rps_synth_fill_blocks.argtypes = [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_int64,
                                              C.c_int64, C.c_int64, C.c_int64, C.c_uint32, C.c_uint64, C.c_uint64,
                                              C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p]
        lib.rps_synth_advance.restype = C.c_int32
        lib.rps_synth_advance.argtypes = [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p,
                                          C.c_void_p, C.c_void_p, C.c_uint32, C.c_void_p]
        _SYNTH_LIB = lib
    return _SYNTH_LIB


def device_fill(out, seed: int, mixture, step: int = 0, scale=None, epoch=None, valid=None, stream=None) -> None:
    """Fill a CUDA tensor ``[n_req][1 + n_branch][L][V]`` (bf16 or fp32) on the device.

    ``scale`` (float32), ``epoch`` (int32) and ``valid`` (uint8) are optional
    ``[n_req][L]`` CUDA tensors with the meaning of ``make_logits``.
    """
    import torch
    if out.dim() != 4 or out.stride(3) != 1:
        raise ValueError("out must be 4-D with a contiguous last dimension")
    dtype = {torch.bfloat16: 1, torch.float32: 0}[out.dtype]
    n_req, nb1, L, V = out.shape
    t_low, t_mid = regime_thresholds(mixture)
    if stream is None:
        stream = torch.cuda.current_stream()
    ptr = lambda t: None if t is None else t.data_ptr()
    rc = _synth_lib().rps_synth_fill(out.data_ptr(), dtype, n_req, nb1 - 1, L, V, out.stride(0), out.stride(1),
                                     out.stride(2), seed, t_low, t_mid, step, ptr(scale), ptr(epoch), ptr(valid),
                                     stream.cuda_stream)
    if rc != 0:
        raise RuntimeError(f"rps_synth_fill failed with code {rc}")


def device_fill_blocks(out, seed: int, mixture, d_step, d_block, L_total: int, scale, epoch, stream=None) -> None:
    """Decode mode of ``device_fill``: ``out`` is ``[n_req][1 + n_branch][B][V]``, the
    current block of every request (row p is response position ``d_block[q] * B + p``;
    rows past ``L_total`` are NaN). ``d_step`` (int32 [1]), ``d_block`` (int32 [n_req]),
    ``scale`` (float32) and ``epoch`` (int32) ``[n_req][L_total]`` are CUDA tensors."""
    import torch
    dtype = {torch.bfloat16: 1, torch.float32: 0}[out.dtype]
    n_req, nb1, B, V = out.shape
    t_low, t_mid = regime_thresholds(mixture)
    if stream is None:
        stream = torch.cuda.current_stream()
    rc = _synth_lib().rps_synth_fill_blocks(out.data_ptr(), dtype, n_req, nb1 - 1, B, V, out.stride(0), out.stride(1),
                                            out.stride(2), seed, t_low, t_mid, d_step.data_ptr(), d_block.data_ptr(),
                                            L_total, scale.data_ptr(), epoch.data_ptr(), stream.cuda_stream)
    if rc != 0:
        raise RuntimeError(f"rps_synth_fill_blocks failed with code {rc}")


def device_advance(winner, B: int, L_total: int, d_block, d_step, scale, epoch, seed: int, stream=None) -> None:
    """Apply one step's winner codes to the generator state of each current block,
    then advance the step counter (all CUDA tensors; see ``rps_synth_advance``)."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    rc = _synth_lib().rps_synth_advance(winner.data_ptr(), winner.shape[0], B, L_total, d_block.data_ptr(),
                                        d_step.data_ptr(), scale.data_ptr(), epoch.data_ptr(), seed,
                                        stream.cuda_stream)
    if rc != 0:
        raise RuntimeError(f"rps_synth_advance failed with code {rc}")


def lmhead_inputs(seed: int, n_rows: int, V: int, d: int, logit_scale: float = 3.0):
    """Seeded LM-head operands as bf16 bits (uint16): hidden [n_rows][d] with
    unit-variance entries, and an unembedding [V][d] whose entries have standard
    deviation logit_scale / sqrt(d), so that the logits h W^T spread over about
    logit_scale nats per standard deviation. numpy's PCG64 normal generator."""
    rng = np.random.default_rng(seed)
    h = rng.standard_normal((n_rows, d), dtype=np.float32)
    w = rng.standard_normal((V, d), dtype=np.float32)
    w *= np.float32(logit_scale / np.sqrt(d))
    return bf16_round(h), bf16_round(w)
