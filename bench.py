#!/usr/bin/env python
"""Benchmark of the RPS scoring path (rps_score_step / rps_select_pivots /
rps_score_branches / rps_commit) on GB300.

A step is one pass of the whole path over one decoding step's synthetic logits:
row statistics of the masked base rows (top-k mode), standard commit and pivot
selection, row statistics of the lookahead rows, benefit scores and the commit
decision. The headline workload is the largest one that fits one GPU, the
batched serving step: 8 requests x 256 positions, vocab 151,936, bf16 logits,
1 base + 16 lookahead branches (8 pivots x top-2), ragged masked counts
U{16..256} with NaN-padded unmasked rows. Every other workload (the generation
step at 100 / 50 / 10 % masked, the long generation's first step and its whole
64-step replay, the KV-cache block step and the tiny fp32 step) gets a record of
its own under `per_workload`, each with the roofline of its lookahead
row-statistics launch and its whole-step fraction of the HBM peak.

Timing: the launches of a step are captured in one CUDA graph; each timed
replay is preceded by an L2 flush (a 256 MB buffer is written, then read back,
so that L2 holds none of the step's data and no dirty lines whose write-back
would land inside the timed region) and bracketed by CUDA events on the
launching stream. Event nodes between kernels would break the programmatic
dependent launch that overlaps each kernel's start with its predecessor's end,
so the step graph has none; a second timed loop replays the same step captured
with an event node around each kernel, on the same stream, for the per-kernel
times and the roofline of the lookahead row-statistics kernel (the dominant
kernel). SM clocks and throttle reasons are sampled with nvidia-smi during both.
The roofline's `traffic` (DRAM bytes of one launch, from ncu) is reported only
while the kernel sources hash to the value recorded beside it.

`value` is scored logit rows per second over the whole job (N replicas, one per
GPU, no collective in the data path: weak scaling). `e2e` is the same metric
through the C ABI with the step's logits in pinned host memory: the gather of
the rows the step scores, the copy of the mask, the step, and the read-back of
the decisions are all inside the timed region. `--impl reference` times the CPU oracle (the only other implementation
of this path) on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time
from pathlib import Path

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

METRIC = "lookahead-scoring logit rows/s and achieved HBM GB/s (fraction of GB300 peak)"
HEADLINE = "serve"
OTHERS = ("step", "step-50", "step-10", "long", "block", "tiny")
REPLAY_STEPS = 64
FLUSH_BYTES = 256 << 20
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
LMHEAD_D = 4096  # hidden size of the 126,464-token model
KERNEL_SOURCES = ("paper_2608_11742_gb300/csrc/rowstats.cu", "paper_2608_11742_gb300/csrc/rps_internal.cuh")


class L2Flush:
    """Write a buffer larger than L2, then read it back: the read evicts the
    written lines (their write-back happens here, outside the timed region) and
    leaves only clean lines of the flush buffer in L2."""

    def __init__(self, device):
        import torch
        self.buf = torch.zeros(FLUSH_BYTES // 4, dtype=torch.float32, device=device)
        self.sink = torch.zeros((), dtype=torch.float32, device=device)

    def __call__(self):
        import torch
        self.buf.add_(1)
        torch.sum(self.buf, dim=0, out=self.sink)


def kernel_source_hash() -> str:
    import hashlib
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        h.update((ROOT / rel).read_bytes())
    return h.hexdigest()


def recorded_traffic(workload: str):
    """DRAM bytes per launch of the lookahead kernel, if recorded for the current sources."""
    tf = ROOT / "profiles" / "traffic.json"
    if not tf.exists():
        return None
    d = json.loads(tf.read_text())
    if d.get("source_sha256") != kernel_source_hash():
        return None
    return d.get("workloads", {}).get(workload)


def describe(w) -> str:
    return (f"{w.name}: {w.n_req} request(s) x {w.L} positions, vocab {w.V}, {w.dtype} logits, "
            f"1 base + {w.n_branch} lookahead branches ({w.n_pivots} pivots x top-{w.tokens_per_pivot}), "
            f"mixture {w.mixture}, masked {'ragged ' + str(w.ragged) if w.ragged else w.masked_frac}")


def peaks():
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        d = json.loads(p.read_text())
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def tensor_peak():
    """Dense bf16 tensor-core peak (TFLOP/s) for a kernel timed alone: the measured burst figure."""
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        return float(json.loads(p.read_text())["bf16_tflops"]), "measured"
    return FALLBACK_BF16_TFLOPS, "fallback"


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def max_over_ranks(x: float) -> float:
    """Largest value of x over the ranks (the slowest replica sets the job's step time)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: int, world: int, ms_per_step: float) -> float:
    """Units per second of the whole job: every replica scores its own step in ms_per_step."""
    return world * units_per_rank / (ms_per_step / 1e3)


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = [l.split(",") for l in open(self.path).read().splitlines() if l.strip()]
        os.unlink(self.path)
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
                for n, v in zip(names, r[5:9]):
                    if v.strip().lower() == "active":
                        reasons.add(n)
            except (ValueError, IndexError):
                continue
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------- GPU arm
class Workload:
    """Device-resident inputs, buffers and the captured step of one workload."""

    def __init__(self, w, prm, device):
        import torch
        from paper_2608_11742_gb300 import rps, synth
        self.w, self.prm, self.device = w, prm, device
        dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
        self.logits = torch.empty((w.n_req, 1 + w.n_branch, w.L, w.V), dtype=dt, device=device)
        valid = w.valid_rows()
        synth.device_fill(self.logits, w.seed, w.mixture,
                          valid=None if valid is None else torch.from_numpy(valid).to(device))
        mpos, mcnt = w.mask()
        self.mpos = torch.from_numpy(mpos).to(device)
        self.mcnt = torch.from_numpy(mcnt).to(device)
        self.step = rps.Step(w.n_req, w.L, w.V, prm, device, dt)
        self.stream = torch.cuda.Stream(device)
        self.ev = None
        with torch.cuda.stream(self.stream):
            self.step.run(self.logits, self.mpos, self.mcnt)
        self.stream.synchronize()
        status, detail = rps.rps_poll_device_status()
        if status != rps.RPS_OK:
            raise RuntimeError(f"device error bits {detail:#x}")
        self.base_rows = int(mcnt.sum())
        self.branch_rows = int(self.step.piv.n_branch_rows.sum())
        self.graph = self._capture()

    KERNELS = ("base_rows_topk", "select", "lookahead_rows", "score_commit")

    def _capture(self):
        import torch
        calls = (lambda: self.step.score_base(self.logits, self.mpos, self.mcnt),
                 lambda: self.step.select(self.mpos, self.mcnt),
                 lambda: self.step.score_branch_rows(self.logits),
                 lambda: self.step.score_and_decide(self.logits))
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=self.stream):
            self.step.run(self.logits, self.mpos, self.mcnt)  # the five launches of rps_run_step
        # the same step with an event node before and after every kernel
        self.graph_ev = torch.cuda.CUDAGraph()
        try:
            ev = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(5)]
        except TypeError:  # torch without external events: one graph per kernel
            ev = None
        if ev:
            with torch.cuda.graph(self.graph_ev, stream=self.stream):
                for i, call in enumerate(calls):
                    ev[i].record()
                    call()
                ev[4].record()
        else:
            self.kernel_graphs = []
            for call in calls:
                kg = torch.cuda.CUDAGraph()
                with torch.cuda.graph(kg, stream=self.stream):
                    call()
                self.kernel_graphs.append(kg)
        self.ev = ev
        return g

    def rows(self):
        return self.base_rows + self.branch_rows

    def bytes(self):
        return self.rows() * self.w.V * self.w.elem_bytes

    def branch_bytes(self):
        return self.branch_rows * self.w.V * self.w.elem_bytes

    def time(self, steps, warmup, flush):
        """Step times (event-free graph), then per-kernel times (graph with event nodes)."""
        import torch
        s = self.stream
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        step_ms = []
        for i in range(warmup + steps):
            with torch.cuda.stream(s):
                flush()
                e0.record(s)
                self.graph.replay()
                e1.record(s)
            s.synchronize()
            if i >= warmup:
                step_ms.append(e0.elapsed_time(e1))
        self.kernel_ms = {k: [] for k in self.KERNELS}
        for i in range(warmup + steps):
            if self.ev:
                with torch.cuda.stream(s):
                    flush()
                    self.graph_ev.replay()
                s.synchronize()
                if i >= warmup:
                    for j, name in enumerate(self.KERNELS):
                        self.kernel_ms[name].append(self.ev[j].elapsed_time(self.ev[j + 1]))
            else:
                with torch.cuda.stream(s):
                    flush()
                for j, name in enumerate(self.KERNELS):
                    with torch.cuda.stream(s):
                        e0.record(s)
                        self.kernel_graphs[j].replay()
                        e1.record(s)
                    s.synchronize()
                    if i >= warmup:
                        self.kernel_ms[name].append(e0.elapsed_time(e1))
        return step_ms, self.kernel_ms["lookahead_rows"]

    def e2e(self, steps, warmup):
        """Same step through the C ABI from pinned host buffers, copies included.

        The logits stay in page-locked host memory: the step gathers the rows it
        scores (masked base rows, then the listed lookahead rows) over the host
        link, with no host synchronisation inside the step. The mask is copied
        in and the decisions read back every step. The whole-tensor copy is
        timed too, for context."""
        import torch
        host = torch.empty(self.logits.shape, dtype=self.logits.dtype, pin_memory=True)
        host.copy_(self.logits)
        hpos = self.mpos.cpu().pin_memory()
        hcnt = self.mcnt.cpu().pin_memory()
        c = self.step.commit
        outs = [c.winner, c.commit_pos, c.commit_tok, c.mask_cnt, c.mask_pos, self.step.piv.n_commit,
                self.step.piv.commit_pos, self.step.piv.commit_tok]
        hout = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in outs]
        dlog, dpos, dcnt = torch.empty_like(self.logits), torch.empty_like(self.mpos), torch.empty_like(self.mcnt)
        s = self.stream
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

        def timed(body):
            ms = []
            for i in range(warmup + steps):
                with torch.cuda.stream(s):
                    e0.record(s)
                    dpos.copy_(hpos, non_blocking=True)
                    dcnt.copy_(hcnt, non_blocking=True)
                    body()
                    for h, d in zip(hout, outs):
                        h.copy_(d, non_blocking=True)
                    e1.record(s)
                s.synchronize()
                if i >= warmup:
                    ms.append(e0.elapsed_time(e1))
            return ms

        ms = timed(lambda: self.step.run_host(host, dlog, dpos, dcnt))
        decisions = [h.clone() for h in hout]

        def full():
            dlog.copy_(host, non_blocking=True)
            self.step.run(dlog, dpos, dcnt)
        ms_full = timed(full)
        if not all(torch.equal(a, b) for a, b in zip(decisions, hout)):
            raise RuntimeError("the gathered step decided differently from the whole-tensor step")
        mask_bytes = hpos.numel() * 4 + hcnt.numel() * 4
        h2d = self.bytes() + mask_bytes
        h2d_full = host.numel() * host.element_size() + mask_bytes
        d2h = sum(h.numel() * h.element_size() for h in hout)
        del dlog
        return ms, h2d, d2h, ms_full, h2d_full


def workload_record(x, step_ms, peak: float, peak_kind: str) -> dict:
    """Step time, whole-step HBM fraction and the roofline of the dominant
    (lookahead row-statistics) launch of one timed workload."""
    ts = statistics.mean(step_ms)
    kernel_us = {k: statistics.mean(v) * 1e3 for k, v in x.kernel_ms.items() if v}
    la_ms = kernel_us["lookahead_rows"] / 1e3
    base_ms = kernel_us["base_rows_topk"] / 1e3
    la_gbs = x.branch_bytes() / (la_ms / 1e3) / 1e9
    base_bytes = x.base_rows * x.w.V * x.w.elem_bytes
    return {"workload": describe(x.w), "rows_per_step": x.rows(), "base_rows": x.base_rows,
            "lookahead_rows": x.branch_rows, "bytes_per_step": x.bytes(),
            "step_us": ts * 1e3, "p50_step_us": statistics.median(step_ms) * 1e3,
            "p90_step_us": sorted(step_ms)[int(0.9 * (len(step_ms) - 1))] * 1e3,
            "rows_per_s": x.rows() / (ts / 1e3), "gbs": x.bytes() / (ts / 1e3) / 1e9,
            "frac": x.bytes() / (ts / 1e3) / 1e9 / peak,
            "kernel_us": kernel_us,
            "roofline": {"bound": "hbm", "kernel": "row statistics of the lookahead rows (statistics-only mode)",
                         "algorithmic_bytes_per_launch": x.branch_bytes(), "launch_ms": la_ms, "achieved": la_gbs,
                         "peak": peak, "peak_kind": peak_kind, "unit": "GB/s", "frac": la_gbs / peak},
            "base_launches": {"kernel": "row statistics of the masked base rows with the top-k sketch, then the "
                                        "top-k search (two launches)",
                              "algorithmic_bytes_per_launch": base_bytes, "launch_ms": base_ms,
                              "achieved": base_bytes / (base_ms / 1e3) / 1e9,
                              "frac": base_bytes / (base_ms / 1e3) / 1e9 / peak}}


def long_replay(configs, device, flush, peak: float) -> dict:
    """The long workload's whole 64-step replay (1 request x 512 positions, vocab
    126,464, 1 base + 16 branches): each step's logits are written by the seeded
    generator and L2 is flushed outside the timed region; the step then scores
    them, and the decision moves the generator (a committed branch becomes the
    next base, a skip draws fresh noise) and the mask (committed positions leave
    it) for the next step, all on the device."""
    import torch
    from paper_2608_11742_gb300.decode import DecodeLoop
    w = configs.LONG
    prm = w.params(configs.EXERCISE)
    loop = DecodeLoop(w.n_req, w.L, w.L, w.V, prm, w.seed, w.mixture, device)
    stream = torch.cuda.Stream(device)
    base_n, branch_n = [], []

    def between():
        flush()
        base_n.append(loop.mask_cnt.sum())

    def after():
        branch_n.append(loop.step.piv.n_branch_rows.sum())

    steps, score_ms, _ = loop.run_split(stream, max_steps=REPLAY_STEPS, between=between, after=after)
    base = [int(v) for v in torch.stack(base_n[:steps]).cpu()]
    branch = [int(v) for v in torch.stack(branch_n[:steps]).cpu()]
    rows = sum(base) + sum(branch)
    t = sum(score_ms) / 1e3
    gbs = rows * w.V * w.elem_bytes / t / 1e9
    del loop
    return {"workload": describe(w) + f", replayed for {steps} decode steps on the device",
            "steps": steps, "rows": rows, "base_rows_first_last": [base[0], base[-1]],
            "lookahead_rows_first_last": [branch[0], branch[-1]],
            "rows_per_s": rows / t, "gbs": gbs, "frac": gbs / peak,
            "mean_step_us": statistics.mean(score_ms) * 1e3, "p50_step_us": statistics.median(score_ms) * 1e3,
            "timing": "CUDA events around each step's scoring graph (the five launches of the step); the "
                      "generator's write of the step's 2.2 GB of logits, an L2 flush and the decision's "
                      "advance of the generator and the mask run outside the timed region"}


def lmhead_run(configs, device, flush, steps: int, warmup: int) -> dict:
    """The LM head with the statistics in its epilogue (rps_lmhead_row_stats) on
    the step workload's scored rows: 256 base rows in top-k mode (k 10) and
    1,152 lookahead rows statistics-only, hidden size 4,096, vocabulary 126,464.
    Random bf16 operands (seeded); each launch is timed alone with CUDA events
    after an L2 flush. cuBLAS (torch.matmul to bf16 logits) on the same shapes is
    timed beside it for context: it writes the logits the fused kernel never does."""
    import torch
    from paper_2608_11742_gb300 import rps
    w = configs.STEP
    prm = w.params(configs.EXERCISE)
    peak_tf, peak_kind = tensor_peak()
    hbm, _ = peaks()
    V, d = w.V, LMHEAD_D
    g = torch.Generator(device=device)
    g.manual_seed(7)
    W = (torch.randn((V, d), generator=g, device=device) * (3.0 / d ** 0.5)).to(torch.bfloat16)
    Wp = rps.rps_lmhead_pack_unembed(W)  # the one-time packed tile layout (outside every timed region)
    parts = {"base rows (top-k)": (256, prm.k_max), "lookahead rows (statistics)": (1152, 0)}
    out = {"workload": f"{sum(n for n, _ in parts.values())} scored rows of the step workload, hidden size {d}, "
                       f"vocabulary {V}, bf16 operands (seeded random), fp32 accumulation",
           "peak_tflops": peak_tf, "peak_kind": peak_kind, "launches": {}}
    stream = torch.cuda.Stream(device)
    total_ms = total_flop = 0.0
    for name, (n, k) in parts.items():
        h = torch.randn((n, d), generator=g, device=device).to(torch.bfloat16)
        buf = rps.RowStatsBuf.alloc(n, k, device)
        ws = torch.empty(rps.rps_lmhead_workspace_bytes(n, V, k), dtype=torch.uint8, device=device)
        rps.rps_workspace_init(ws)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

        def timed(fn):
            ms = []
            for i in range(warmup + steps):
                with torch.cuda.stream(stream):
                    flush()
                    e0.record(stream)
                    fn()
                    e1.record(stream)
                stream.synchronize()
                if i >= warmup:
                    ms.append(e0.elapsed_time(e1))
            return statistics.mean(ms)

        t = timed(lambda: rps.rps_lmhead_row_stats(h, W, prm if k else None, buf, ws, packed=Wp))
        t_rm = timed(lambda: rps.rps_lmhead_row_stats(h, W, prm if k else None, buf, ws))
        st, detail = rps.rps_poll_device_status(stream)
        if st != rps.RPS_OK:
            raise RuntimeError(f"lmhead device error {detail:#x}")
        t_cublas = timed(lambda: torch.matmul(h, W.t()))
        flop = 2.0 * n * d * V
        tf = flop / (t / 1e3) / 1e12
        out["launches"][name] = {
            "rows": n, "k": k, "ms": t, "tflops": tf, "frac_of_tensor_peak": tf / peak_tf,
            "unembedding_gbs": V * d * 2 / (t / 1e3) / 1e9, "unembedding_frac_of_hbm": V * d * 2 / (t / 1e3) / 1e9 / hbm,
            "row_major_unembedding_ms": t_rm,
            "cublas_matmul_ms": t_cublas, "cublas_tflops": flop / (t_cublas / 1e3) / 1e12,
            "logit_bytes_not_written": n * V * 2}
        total_ms += t
        total_flop += flop
        del h, buf, ws
    out["step_ms"] = total_ms
    out["tflops"] = total_flop / (total_ms / 1e3) / 1e12
    out["frac_of_tensor_peak"] = out["tflops"] / peak_tf
    out["roofline"] = {"bound": "tensor", "kernel": "lmhead_kernel (tcgen05) + merge, both launches",
                       "achieved": out["tflops"], "peak": peak_tf, "unit": "TFLOP/s", "frac": out["frac_of_tensor_peak"],
                       "algorithmic_flop_per_step": total_flop}
    out["unembedding_layout"] = "packed tiles (rps_lmhead_pack_unembed, once); row_major_unembedding_ms times [V][d]"
    del W, Wp
    return out


def attention_run(device, flush, steps: int, warmup: int) -> dict:
    """The branch-isolating attention of the packed lookahead forward pass
    (rps_packed_attention_fwd) at the serving shape: 8 requests x 32 heads x
    head dim 128, a 512-token context and the anchor plus 8 branches of the
    256-token generation region (2,816 packed tokens). Random bf16 inputs
    (seeded); CUDA events after an L2 flush. torch's scaled-dot-product
    attention with the same mask written out densely is timed for context."""
    import torch
    from paper_2608_11742_gb300 import rps
    B, H, D, C, NB, G = 8, 32, 128, 512, 9, 256
    n = C + NB * G
    g = torch.Generator(device=device)
    g.manual_seed(9)
    q, k, v = (torch.randn((B, H, n, D), generator=g, device=device).to(torch.bfloat16) for _ in range(3))
    vt = v.transpose(2, 3).contiguous()
    out = torch.empty_like(q)
    scale = D ** -0.5
    stream = torch.cuda.Stream(device)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn):
        ms = []
        for i in range(warmup + steps):
            with torch.cuda.stream(stream):
                flush()
                e0.record(stream)
                fn()
                e1.record(stream)
            stream.synchronize()
            if i >= warmup:
                ms.append(e0.elapsed_time(e1))
        return statistics.mean(ms)

    t = timed(lambda: rps.rps_packed_attention_fwd(q, k, vt, out, C, NB, G, scale))
    st, detail = rps.rps_poll_device_status(stream)
    if st != rps.RPS_OK:
        raise RuntimeError(f"attention device error {detail:#x}")
    pairs = C * (C + G) + NB * G * (C + G)  # visible (query, key) pairs per head
    flop = 4.0 * D * B * H * pairs
    peak_tf, peak_kind = tensor_peak()
    tf = flop / (t / 1e3) / 1e12
    rec = {"workload": f"{B} requests x {H} heads x head dim {D}: context {C} + {NB} branches (anchor and "
                       f"{NB - 1} candidates) x {G} tokens = {n} packed tokens, bf16",
           "ms": t, "tflops": tf, "frac_of_tensor_peak": tf / peak_tf, "peak_tflops": peak_tf, "peak_kind": peak_kind,
           "algorithmic_flop": flop, "visible_fraction_of_dense": pairs / (n * n),
           "roofline": {"bound": "tensor", "kernel": "packed_attention_kernel (tcgen05)", "achieved": tf,
                        "peak": peak_tf, "unit": "TFLOP/s", "frac": tf / peak_tf}}
    seg = torch.cat([torch.zeros(C, dtype=torch.int64)] + [torch.full((G,), 1 + j) for j in range(NB)]).to(device)
    own = torch.where(seg == 0, torch.ones_like(seg), seg)
    mask = (seg[None, :] == 0) | (seg[None, :] == own[:, None])
    try:
        t_sdpa = timed(lambda: torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=mask))
        rec["torch_sdpa_dense_mask_ms"] = t_sdpa
    except RuntimeError as exc:  # no kernel for this mask / size
        rec["torch_sdpa_dense_mask_ms"] = f"unavailable: {exc}"[:200]
    del q, k, v, vt, out, mask
    return rec


def decode_run(configs, device):
    """A whole response decoded on the device (Algorithm 1): the block workload's
    64 requests x 32-position blocks extended to 256 positions. The denoiser
    forward pass is the seeded generator (a stub); its time is reported apart."""
    import torch
    from paper_2608_11742_gb300.decode import DecodeLoop
    w = configs.BLOCK
    prm = w.params(configs.EXERCISE)
    L_total = 256
    loop = DecodeLoop(w.n_req, w.L, L_total, w.V, prm, w.seed, w.mixture, device)
    stream = torch.cuda.Stream(device)
    steps, score_ms, total_ms = loop.run_split(stream)
    rows = int(loop.steps.sum().item())  # request-steps
    tokens = w.n_req * L_total
    mean_ms = statistics.mean(score_ms)
    return {"workload": f"{w.n_req} requests x {L_total} positions in blocks of {w.L}, vocab {w.V}, bf16, "
                        f"1 base + {w.n_branch} lookahead branches, mixture {w.mixture}",
            "decoded": bool(loop.done.all().item()) and bool((loop.tokens >= 0).all().item()),
            "steps": steps, "request_steps": rows, "tokens": tokens,
            "scoring_ms_per_step": mean_ms, "scoring_p50_ms": statistics.median(score_ms),
            "tokens_per_s_scoring": tokens / (sum(score_ms) / 1e3),
            "total_ms_with_stub": total_ms,
            "launches_per_step": DecodeLoop.LAUNCHES,
            "timing": "CUDA events around the graph of the scoring step (row statistics, selection, lookahead "
                      "rows, scores and commit), replayed after the stub's graph wrote the step's 4.66 GB of "
                      "logits (larger than L2); the generator's and the decode state's advance (three launches) "
                      "replay after it, outside the timed region"}


def cpu_sample(w, n_take: int = 64):
    """A bounded sample of one step's rows, in the step's proportions: base rows
    (scored in top-k mode) and lookahead rows (statistics only)."""
    import numpy as np
    from paper_2608_11742_gb300 import synth
    mpos, mcnt = w.mask()
    rng = np.random.default_rng(0)
    n_base = max(1, int(round(n_take / (1 + w.n_branch))))
    base, branch = [], []
    for i in range(n_take):
        q = int(rng.integers(0, w.n_req))
        pos = int(mpos[q, int(rng.integers(0, max(int(mcnt[q]), 1)))])
        b = 0 if i < n_base else int(rng.integers(1, 1 + w.n_branch))
        (base if b == 0 else branch).append(synth.row_logits(w.seed, w.V, q, b, pos, w.mixture, w.dtype))
    return np.stack(base), np.stack(branch)


def time_oracle(sample, k_max: int, budget_s: float):
    """Rows per second of the oracle as it stands (single thread) over the sample, repeated for budget_s."""
    from oracle import default as oracle_default
    o = oracle_default()
    rb, rr = sample
    done, t0, elapsed = 0, time.perf_counter(), 0.0
    while elapsed < budget_s:
        o.row_stats(rb, k_max)
        o.row_stats(rr, 0)
        done += len(rb) + len(rr)
        elapsed = time.perf_counter() - t0
    return done / elapsed, done, elapsed


def all_cores_entry(w, sample, k_max: int, budget_s: float) -> dict:
    """The same oracle in one process per logical CPU at once (summed rates)."""
    from oracle.parallel import rows_per_second_all_cores
    rows_s, done, procs = rows_per_second_all_cores(sample, k_max, budget_s)
    return {"value": rows_s, "unit": "rows/s", "cores": procs,
            "sample": f"{procs} processes, each the single-threaded oracle over the same sample for about "
                      f"{budget_s:.0f} s ({done} rows in all; {rows_s * w.V * w.elem_bytes / 1e9:.3f} GB/s)"}


def host_cpu() -> dict:
    """The host's logical CPU count and model (lscpu where present, else the platform)."""
    import os, platform, subprocess
    model = platform.processor() or platform.machine()
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name:"):
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    return {"nproc": os.cpu_count(), "model": model, "machine": platform.machine()}


def cpu_baseline(w, prm, budget_s: float):
    sample = cpu_sample(w)
    rows_s, done, elapsed = time_oracle(sample, prm.k_max, budget_s)
    return {"value": rows_s, "unit": "rows/s", "cores": 1, "kind": "oracle", "host": host_cpu(),
            "sample": f"{done} rows of the {w.name} workload ({len(sample[0])} base rows in top-k mode and "
                      f"{len(sample[1])} lookahead rows, repeated) scored by the single-threaded fp64 oracle in "
                      f"{elapsed:.1f} s ({rows_s * w.V * w.elem_bytes / 1e9:.3f} GB/s)",
            "all_cores": all_cores_entry(w, sample, prm.k_max, min(4.0, budget_s))}


def run_gpu(args):
    import torch
    from paper_2608_11742_gb300 import configs, rps
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    flush = L2Flush(device)
    peak, peak_kind = peaks()

    w = configs.ALL[args.workload]
    prm = w.params(configs.EXERCISE)
    wl = Workload(w, prm, device)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        step_ms, _ = wl.time(args.steps, args.warmup, flush)
    clocks = clk.summary()
    t_step = max_over_ranks(statistics.mean(step_ms))
    rows = wl.rows()
    value = whole_job_rate(rows, world, t_step)
    traffic = recorded_traffic(args.workload)

    rec = workload_record(wl, step_ms, peak, peak_kind)
    out = {
        "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": describe(w), "input_dtype": w.dtype,
                   "params": {"k_max": prm.k_max, "r": prm.r, "tau_pivot": prm.tau_pivot, "tau": prm.tau,
                              "lambda": prm.lam, "n_pivots": prm.n_pivots, "tokens_per_pivot": prm.tokens_per_pivot},
                   "rows_per_step": rows, "base_rows": wl.base_rows, "lookahead_rows": wl.branch_rows,
                   "bytes_per_step": wl.bytes(), "l2": "flushed before every timed step (256 MB buffer written, then read back)",
                   "timing": "step: CUDA events around an event-free graph of the step; per-kernel and roofline: a "
                             "second timed loop of the same step graph with an event node around each kernel",
                   "parallelism": f"{world} independent replica(s), no collective"},
        "achieved_gbs": wl.bytes() / (t_step / 1e3) / 1e9,
        "frac_of_hbm_peak": wl.bytes() / (t_step / 1e3) / 1e9 / peak,
        "roofline": dict(rec["roofline"], traffic=traffic),
        "clocks": clocks,
        "gpu_launches": rps.Step.LAUNCHES * args.steps,
        "kernel_us": rec["kernel_us"],
        "p50_step_us": rec["p50_step_us"],
        "base_launches": rec["base_launches"],
    }
    del wl
    torch.cuda.empty_cache()

    if not args.skip_others:
        per = {}
        for name in OTHERS:
            wo = configs.ALL[name]
            x = Workload(wo, wo.params(configs.EXERCISE), device)
            sm, _ = x.time(max(5, args.steps // 2), 3, flush)
            per[name] = workload_record(x, sm, peak, peak_kind)
            del x
            torch.cuda.empty_cache()
        per["long-replay"] = long_replay(configs, device, flush, peak)
        torch.cuda.empty_cache()
        out["per_workload"] = per

    if not args.skip_decode:
        out["decode"] = decode_run(configs, device)
        torch.cuda.empty_cache()

    if not args.skip_lmhead:
        out["lmhead"] = lmhead_run(configs, device, flush, max(5, args.steps // 2), 3)
        torch.cuda.empty_cache()
        out["attention"] = attention_run(device, flush, max(5, args.steps // 2), 3)
        torch.cuda.empty_cache()

    if not args.skip_e2e:
        wl = Workload(w, prm, device)
        ms, h2d, d2h, ms_full, h2d_full = wl.e2e(max(3, args.steps // 4), 3)
        te = max_over_ranks(statistics.mean(ms))
        tf = max_over_ranks(statistics.mean(ms_full))
        out["e2e"] = {"value": whole_job_rate(rows, world, te), "unit": "rows/s", "h2d_bytes_per_step": h2d,
                      "d2h_bytes_per_step": d2h, "ms_per_step": te,
                      "path": "Step.run_host: scored rows gathered from pinned host memory",
                      "whole_tensor_copy": {"value": whole_job_rate(rows, world, tf), "ms_per_step": tf,
                                            "h2d_bytes_per_step": h2d_full}}
        del wl
        torch.cuda.empty_cache()

    if rank == 0 and world == 1 and not args.skip_cpu:
        out["cpu_baseline"] = cpu_baseline(w, prm, args.cpu_seconds)
        out["cpu_baseline"].pop("seconds", None)

    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    if rank == 0:
        print(json.dumps(out))


def run_reference(args):
    """The CPU oracle as the reference arm, on the host cores, same metric and workload."""
    from paper_2608_11742_gb300 import configs
    rank, world, _ = dist_env()
    if rank != 0:
        return
    w = configs.ALL[args.workload]
    prm = w.params(configs.EXERCISE)
    per_step = max(0.5, args.cpu_seconds / max(1, args.steps + args.warmup))
    sample = cpu_sample(w)
    vals = []
    for i in range(args.warmup + args.steps):
        rows_s, _, _ = time_oracle(sample, prm.k_max, per_step)
        if i >= args.warmup:
            vals.append(rows_s)
    value = statistics.mean(vals)
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": None, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": describe(w), "input_dtype": w.dtype},
           "cpu_baseline": {"value": value, "unit": "rows/s", "cores": 1, "kind": "oracle", "host": host_cpu(),
                            "sample": f"each step: about {per_step:.1f} s of the single-threaded fp64 oracle on a "
                                      f"64-row sample of the workload ({len(sample[0])} base rows in top-k mode, "
                                      f"{len(sample[1])} lookahead rows)",
                            "all_cores": all_cores_entry(w, sample, prm.k_max, 4.0)},
           "e2e": {"value": value, "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out))


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", default=HEADLINE)
    ap.add_argument("--skip-others", action="store_true")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--skip-decode", action="store_true")
    ap.add_argument("--skip-lmhead", action="store_true")
    ap.add_argument("--only-lmhead", action="store_true",
                    help="time the tensor-core extensions alone (LM head with the statistics epilogue, packed "
                         "lookahead attention) and print their records")
    ap.add_argument("--skip-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    elif args.only_lmhead:
        import torch
        from paper_2608_11742_gb300 import configs
        device = torch.device("cuda", dist_env()[2])
        torch.cuda.set_device(device)
        flush = L2Flush(device)
        print(json.dumps({"lmhead": lmhead_run(configs, device, flush, args.steps, args.warmup),
                          "attention": attention_run(device, flush, args.steps, args.warmup)}))
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
