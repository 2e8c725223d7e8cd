// abi.cu -- host side of the C ABI declared in include/rps.h: argument checks,
// launch configuration, workspace layout and the device error word.
#include <cmath>
#include <algorithm>
#include <cstring>
#include <atomic>
#include <mutex>

#include "rps_internal.cuh"

namespace rps {
namespace {

// Sticky error word of each device (one copy per device context).
__device__ uint32_t g_device_error;

constexpr int kMaxDevices = 64;
constexpr size_t kAlign = 256;

struct DeviceInfo {
    bool ready = false;
    int sm_count = 0;
    int blocks[2] = {0, 0};  // resident row-statistics blocks per SM, by dtype
    uint32_t *err = nullptr;
};

std::mutex g_mutex;
DeviceInfo g_devices[kMaxDevices];

// Limit of the row-statistics kernels' wait for each ring chunk (see
// rps_debug_set_ring_wait_ns).
constexpr uint64_t kRingWaitNs = 200ull * 1000 * 1000;
std::atomic<uint64_t> g_ring_wait_ns{kRingWaitNs};

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

rps_status device_info(DeviceInfo *out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RPS_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mutex);
    DeviceInfo &d = g_devices[dev];
    if (!d.ready) {
        if (cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return RPS_ERR_CUDA;
        for (int dt = 0; dt < 2; ++dt)
            if (row_stats_occupancy(dt, &d.blocks[dt]) != cudaSuccess || d.blocks[dt] < 1) return RPS_ERR_CUDA;
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_device_error) != cudaSuccess) return RPS_ERR_CUDA;
        d.err = static_cast<uint32_t *>(p);
        d.ready = true;
    }
    *out = d;
    return RPS_OK;
}

bool finite(float x) { return std::isfinite(x); }

// Checks the parameters a call uses; `need_search` adds r, tau_pivot, P and K.
rps_status check_params(const rps_params *p, bool need_search) {
    if (!p) return RPS_ERR_INVALID_ARG;
    if (p->k_max < 1) return RPS_ERR_INVALID_ARG;
    if (p->k_max > RPS_MAX_K) return RPS_ERR_UNSUPPORTED;
    if (!need_search) return RPS_OK;
    if (!finite(p->r) || !(p->r > 0.f) || p->r > 1.f) return RPS_ERR_INVALID_ARG;
    if (!finite(p->tau) || !finite(p->tau_pivot)) return RPS_ERR_INVALID_ARG;
    if (!finite(p->lambda) || p->lambda < 0.f) return RPS_ERR_INVALID_ARG;
    if (p->n_pivots < 1 || p->tokens_per_pivot < 1 || p->tokens_per_pivot > p->k_max) return RPS_ERR_INVALID_ARG;
    if (p->n_pivots > RPS_MAX_PIVOTS) return RPS_ERR_UNSUPPORTED;
    if (p->pivot_rule < RPS_PIVOT_TRUNCATED_ENTROPY || p->pivot_rule > RPS_PIVOT_MAX_ENTROPY) return RPS_ERR_INVALID_ARG;
    if (p->commit_rule < RPS_COMMIT_THRESHOLD || p->commit_rule > RPS_COMMIT_TOPK_LOW_ENTROPY) return RPS_ERR_INVALID_ARG;
    if (p->commit_rule != RPS_COMMIT_THRESHOLD) {
        if (p->commit_k < 1) return RPS_ERR_INVALID_ARG;
        if (p->commit_k > RPS_MAX_COMMIT_K) return RPS_ERR_UNSUPPORTED;
    }
    return RPS_OK;
}

rps_status check_logits(const rps_logits *l) {
    if (!l || !l->data) return RPS_ERR_INVALID_ARG;
    if (l->dtype != RPS_F32 && l->dtype != RPS_BF16) return RPS_ERR_INVALID_ARG;
    if (l->vocab < 1 || l->vocab > INT32_MAX || l->n_req < 1 || l->n_branch < 1 || l->n_pos < 1)
        return RPS_ERR_INVALID_ARG;
    if (l->req_stride < 0 || l->branch_stride < 0 || l->pos_stride < 0) return RPS_ERR_INVALID_ARG;
    const int64_t esize = l->dtype == RPS_BF16 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(l->data) % 16 != 0) return RPS_ERR_INVALID_ARG;
    if ((l->req_stride * esize) % 16 || (l->branch_stride * esize) % 16 || (l->pos_stride * esize) % 16)
        return RPS_ERR_INVALID_ARG;
    return RPS_OK;
}

struct WorkspaceLayout {
    size_t health, ticket, part, sketch, norm, piece, total;
};

// The health word (its own 256-byte line), tickets, partial records, and in
// top-k mode the sketch (one element-sized entry per cell: one lane's units of
// one 2 KB ring chunk), each row's B, ln S, 1 / S and first piece length, and
// the launch's piece length.
WorkspaceLayout layout(int64_t max_rows, int64_t vocab, int32_t dtype, int32_t k) {
    WorkspaceLayout w;
    const size_t rows = static_cast<size_t>(max_rows);
    const size_t esize = dtype == RPS_BF16 ? 2 : 4;
    const size_t units = (static_cast<size_t>(vocab) * esize + 15) / 16;
    w.health = 0;
    w.ticket = kAlign;
    w.part = w.ticket + align_up(rows * sizeof(uint32_t));
    w.sketch = w.part + align_up(rows * kMaxPartials * sizeof(Partial));
    w.norm = w.sketch + (k > 0 ? align_up(rows * static_cast<size_t>(sketch_entries(units)) * esize) : 0);
    w.piece = w.norm + (k > 0 ? align_up(rows * sizeof(float4)) : 0);
    w.total = w.piece + (k > 0 ? align_up(sizeof(int32_t)) : 0);
    return w;
}

rps_status from_cuda(cudaError_t e) { return e == cudaSuccess ? RPS_OK : RPS_ERR_CUDA; }

}  // namespace

uint32_t *device_error_word() {
    DeviceInfo dev;
    return device_info(&dev) == RPS_OK ? dev.err : nullptr;
}

uint64_t ring_wait_limit_ns() { return g_ring_wait_ns.load(std::memory_order_relaxed); }

}  // namespace rps

using namespace rps;

extern "C" {

size_t rps_workspace_bytes(int64_t max_rows, int64_t vocab, int32_t dtype, int32_t k_max) {
    if (max_rows < 1 || vocab < 1 || k_max < 0 || k_max > RPS_MAX_K) return 0;
    if (dtype != RPS_F32 && dtype != RPS_BF16) return 0;
    return layout(max_rows, vocab, dtype, k_max).total;
}

rps_status rps_workspace_init(void *d_ws, size_t ws_bytes, rps_stream_t stream) {
    if (!d_ws || ws_bytes == 0) return RPS_ERR_INVALID_ARG;
    return from_cuda(cudaMemsetAsync(d_ws, 0, ws_bytes, reinterpret_cast<cudaStream_t>(stream)));
}

}  // extern "C"

namespace rps {
namespace {

}  // namespace

rps_status check_row_stats_args(const rps_logits *logits, const rps_row_list *rows, const rps_params *prm,
                                const rps_row_stats *out, int32_t *k_out) {
    rps_status st = check_logits(logits);
    if (st != RPS_OK) return st;
    if (!rows || (!rows->rows && !rows->mask_pos) || rows->n_seg < 1 || rows->cap < 1) return RPS_ERR_INVALID_ARG;
    if (rows->n_seg > RPS_MAX_SEGMENTS) return RPS_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(rows->n_seg) * rows->cap > INT32_MAX / 3) return RPS_ERR_INVALID_ARG;
    if (!out || !out->zmax || !out->lse || !out->H || !out->pmax || !out->argmax) return RPS_ERR_INVALID_ARG;
    int32_t k = 0;
    if (out->topk_idx) {
        if ((st = check_params(prm, false)) != RPS_OK) return st;
        if (!out->topk_logit || !out->mu || !out->htrunc) return RPS_ERR_INVALID_ARG;
        if (prm->k_max > logits->vocab) return RPS_ERR_INVALID_ARG;
        k = prm->k_max;
    }
    *k_out = k;
    return RPS_OK;
}

namespace {

// Checks the arguments of a row-statistics launch and fills its kernel
// arguments and grid.
rps_status prepare_row_stats(const rps_logits *logits, const rps_row_list *rows, const rps_params *prm,
                             const rps_row_stats *out, void *d_ws, size_t ws_bytes, RowStatsArgs *ap,
                             int *grid_out, int *topk_grid_out) {
    int32_t k = 0;
    rps_status st = check_row_stats_args(logits, rows, prm, out, &k);
    if (st != RPS_OK) return st;
    const int64_t max_rows = static_cast<int64_t>(rows->n_seg) * rows->cap;
    const WorkspaceLayout w = layout(max_rows, logits->vocab, logits->dtype, k);
    if (!d_ws || ws_bytes < w.total || reinterpret_cast<uintptr_t>(d_ws) % 16 != 0) return RPS_ERR_INVALID_ARG;

    DeviceInfo dev;
    if ((st = device_info(&dev)) != RPS_OK) return st;
    const int esize = logits->dtype == RPS_BF16 ? 2 : 4;
    const int per_unit = 16 / esize;

    RowStatsArgs &a = *ap;
    std::memset(&a, 0, sizeof a);
    a.data = logits->data;
    a.vocab = logits->vocab;
    a.req_stride = logits->req_stride;
    a.branch_stride = logits->branch_stride;
    a.pos_stride = logits->pos_stride;
    a.n_req = logits->n_req;
    a.n_branch = logits->n_branch;
    a.n_pos = logits->n_pos;
    a.rows = rows->rows;
    a.seg_cnt = rows->seg_cnt;
    a.n_seg = rows->n_seg;
    a.cap = rows->cap;
    a.mask_pos = rows->mask_pos;
    a.mask_branch = rows->mask_branch;
    a.k = k;
    a.zmax = out->zmax;
    a.lse = out->lse;
    a.H = out->H;
    a.pmax = out->pmax;
    a.argmax = out->argmax;
    a.mu = out->mu;
    a.htrunc = out->htrunc;
    a.topk_idx = out->topk_idx;
    a.topk_logit = out->topk_logit;
    char *ws = static_cast<char *>(d_ws);
    a.ticket = reinterpret_cast<uint32_t *>(ws + w.ticket);
    a.health = reinterpret_cast<uint32_t *>(ws + w.health);
    a.ring_wait_ns = g_ring_wait_ns.load(std::memory_order_relaxed);
    a.part = reinterpret_cast<Partial *>(ws + w.part);
    a.sketch = k > 0 ? static_cast<void *>(ws + w.sketch) : nullptr;
    a.norm = k > 0 ? reinterpret_cast<float4 *>(ws + w.norm) : nullptr;
    a.sketch_piece = k > 0 ? reinterpret_cast<int32_t *>(ws + w.piece) : nullptr;
    a.units_per_row = (logits->vocab + per_unit - 1) / per_unit;
    a.sketch_stride = sketch_entries(a.units_per_row);
    const int grid = dev.sm_count * dev.blocks[logits->dtype];
    a.warps = grid * (kStatThreads / 32);
    *topk_grid_out = static_cast<int>(std::min<int64_t>((max_rows + kTopkWarps - 1) / kTopkWarps,
                                                         static_cast<int64_t>(dev.sm_count) * 16));
    a.min_piece = (a.units_per_row + (kMaxPartials - 2) - 1) / (kMaxPartials - 2);
    a.err = dev.err;
    *grid_out = grid;
    return RPS_OK;
}

}  // namespace
}  // namespace rps

extern "C" {

rps_status rps_score_step(const rps_logits *logits, const rps_row_list *rows, const rps_params *prm,
                          const rps_row_stats *out, void *d_ws, size_t ws_bytes, rps_stream_t stream) {
    RowStatsArgs a;
    int grid = 0, topk_grid = 0;
    const rps_status st = prepare_row_stats(logits, rows, prm, out, d_ws, ws_bytes, &a, &grid, &topk_grid);
    if (st != RPS_OK) return st;
    return from_cuda(launch_row_stats(a, logits->dtype, grid, topk_grid, reinterpret_cast<cudaStream_t>(stream)));
}


}  // extern "C"

namespace rps {
namespace {

rps_status make_select_args(const rps_row_stats *base, int32_t n_req, int32_t L, const int32_t *d_mask_pos,
                            const int32_t *d_mask_cnt, const rps_params *prm, const rps_pivots *out,
                            SelectArgs *ap) {
    rps_status st = check_params(prm, true);
    if (st != RPS_OK) return st;
    if (!base || !base->zmax || !base->pmax || !base->argmax || !base->mu || !base->htrunc || !base->H ||
        !base->topk_idx || !base->topk_logit)
        return RPS_ERR_INVALID_ARG;
    if (n_req < 1 || L < 1 || !d_mask_pos || !d_mask_cnt) return RPS_ERR_INVALID_ARG;
    if (L > RPS_MAX_POS) return RPS_ERR_UNSUPPORTED;
    if (!out || !out->n_commit || !out->commit_pos || !out->commit_tok || !out->rem_cnt || !out->rem_k ||
        !out->rem_pos || !out->state || !out->pivot_k || !out->pivot_pos || !out->n_cand || !out->cand_tok ||
        !out->branch_valid || !out->branch_off || !out->branch_cnt || !out->n_branch_rows || !out->branch_rows)
        return RPS_ERR_INVALID_ARG;
    DeviceInfo dev;
    if ((st = device_info(&dev)) != RPS_OK) return st;
    SelectArgs &a = *ap;
    a.zmax = base->zmax;
    a.pmax = base->pmax;
    a.mu = base->mu;
    a.htrunc = base->htrunc;
    a.H = base->H;
    a.topk_logit = base->topk_logit;
    a.argmax = base->argmax;
    a.topk_idx = base->topk_idx;
    a.k_max = prm->k_max;
    a.mask_pos = d_mask_pos;
    a.mask_cnt = d_mask_cnt;
    a.n_req = n_req;
    a.L = L;
    a.P = prm->n_pivots;
    a.K = prm->tokens_per_pivot;
    a.tau = prm->tau;
    a.tau_pivot = prm->tau_pivot;
    a.log_r = std::log(static_cast<double>(prm->r));
    a.pivot_rule = prm->pivot_rule;
    a.commit_rule = prm->commit_rule;
    a.commit_k = prm->commit_k;
    a.out = *out;
    a.err = dev.err;
    a.early = 0;
    return RPS_OK;
}

}  // namespace
}  // namespace rps

extern "C" {

rps_status rps_select_pivots(const rps_row_stats *base, int32_t n_req, int32_t L, const int32_t *d_mask_pos,
                             const int32_t *d_mask_cnt, const rps_params *prm, const rps_pivots *out,
                             rps_stream_t stream) {
    SelectArgs a;
    const rps_status st = make_select_args(base, n_req, L, d_mask_pos, d_mask_cnt, prm, out, &a);
    if (st != RPS_OK) return st;
    return from_cuda(launch_select(a, reinterpret_cast<cudaStream_t>(stream)));
}


}  // extern "C"

namespace rps {
namespace {

rps_status make_score_args(const rps_logits *anchor_logits, int32_t anchor_branch, const rps_row_stats *anchor,
                           const rps_row_stats *branch, int32_t n_req, int32_t L, const rps_pivots *piv,
                           const rps_params *prm, const rps_branch_scores *out, ScoreArgs *a) {
    rps_status st = check_params(prm, true);
    if (st != RPS_OK) return st;
    if ((st = check_logits(anchor_logits)) != RPS_OK) return st;
    if (anchor_branch < 0 || anchor_branch >= anchor_logits->n_branch) return RPS_ERR_INVALID_ARG;
    if (n_req < 1 || L < 1 || n_req > anchor_logits->n_req) return RPS_ERR_INVALID_ARG;
    if (L > RPS_MAX_POS) return RPS_ERR_UNSUPPORTED;
    if (!anchor || !anchor->zmax || !anchor->lse || !anchor->H || !anchor->pmax) return RPS_ERR_INVALID_ARG;
    if (!branch || !branch->H || !branch->pmax) return RPS_ERR_INVALID_ARG;
    if (!piv || !piv->state || !piv->rem_cnt || !piv->rem_k || !piv->pivot_k || !piv->pivot_pos || !piv->n_cand ||
        !piv->cand_tok || !piv->branch_valid || !piv->branch_off || !piv->branch_cnt)
        return RPS_ERR_INVALID_ARG;
    if (!out || !out->mean_H || !out->n_tau || !out->log_a || !out->score) return RPS_ERR_INVALID_ARG;
    a->anchor_data = anchor_logits->data;
    a->dtype = anchor_logits->dtype;
    a->vocab = anchor_logits->vocab;
    a->req_stride = anchor_logits->req_stride;
    a->pos_stride = anchor_logits->pos_stride;
    a->branch_offset = static_cast<int64_t>(anchor_branch) * anchor_logits->branch_stride;
    a->n_pos = anchor_logits->n_pos;
    a->a_H = anchor->H;
    a->a_pmax = anchor->pmax;
    a->a_lse = anchor->lse;
    a->a_zmax = anchor->zmax;
    a->b_H = branch->H;
    a->b_pmax = branch->pmax;
    a->piv = *piv;
    a->n_req = n_req;
    a->L = L;
    a->P = prm->n_pivots;
    a->K = prm->tokens_per_pivot;
    a->lambda = prm->lambda;
    a->tau = prm->tau;
    a->out = *out;
    a->err = nullptr;
    a->early = 0;
    return RPS_OK;
}

rps_status make_commit_args(const rps_branch_scores *scores, int32_t n_req, int32_t L, const rps_pivots *piv,
                            const rps_params *prm, const rps_commit_out *out, CommitArgs *a) {
    rps_status st = check_params(prm, true);
    if (st != RPS_OK) return st;
    if (!scores || !scores->score || n_req < 1 || L < 1) return RPS_ERR_INVALID_ARG;
    if (L > RPS_MAX_POS) return RPS_ERR_UNSUPPORTED;
    if (!piv || !piv->state || !piv->pivot_pos || !piv->n_cand || !piv->cand_tok || !piv->branch_valid ||
        !piv->rem_cnt || !piv->rem_pos)
        return RPS_ERR_INVALID_ARG;
    if (!out || !out->best_slot || !out->gain || !out->winner || !out->commit_pos || !out->commit_tok ||
        !out->margin || !out->mask_pos || !out->mask_cnt)
        return RPS_ERR_INVALID_ARG;
    if (out->mask_pos == piv->rem_pos) return RPS_ERR_INVALID_ARG;
    a->score = scores->score;
    a->piv = *piv;
    a->n_req = n_req;
    a->L = L;
    a->P = prm->n_pivots;
    a->K = prm->tokens_per_pivot;
    a->out = *out;
    return RPS_OK;
}

}  // namespace
}  // namespace rps

extern "C" {

rps_status rps_score_branches(const rps_logits *anchor_logits, int32_t anchor_branch,
                              const rps_row_stats *anchor, const rps_row_stats *branch, int32_t n_req,
                              int32_t L, const rps_pivots *piv, const rps_params *prm,
                              const rps_branch_scores *out, rps_stream_t stream) {
    ScoreArgs a;
    rps_status st = make_score_args(anchor_logits, anchor_branch, anchor, branch, n_req, L, piv, prm, out, &a);
    if (st != RPS_OK) return st;
    DeviceInfo dev;
    if ((st = device_info(&dev)) != RPS_OK) return st;
    a.err = dev.err;
    return from_cuda(launch_score(a, reinterpret_cast<cudaStream_t>(stream)));
}

rps_status rps_commit(const rps_branch_scores *scores, int32_t n_req, int32_t L, const rps_pivots *piv,
                      const rps_params *prm, const rps_commit_out *out, rps_stream_t stream) {
    CommitArgs a;
    rps_status st = make_commit_args(scores, n_req, L, piv, prm, out, &a);
    if (st != RPS_OK) return st;
    DeviceInfo dev;
    if ((st = device_info(&dev)) != RPS_OK) return st;
    return from_cuda(launch_commit(a, reinterpret_cast<cudaStream_t>(stream)));
}

rps_status rps_score_and_commit(const rps_logits *anchor_logits, int32_t anchor_branch,
                                const rps_row_stats *anchor, const rps_row_stats *branch, int32_t n_req, int32_t L,
                                const rps_pivots *piv, const rps_params *prm, const rps_branch_scores *scores,
                                const rps_commit_out *out, rps_stream_t stream) {
    ScoreArgs s;
    CommitArgs c;
    rps_status st = make_score_args(anchor_logits, anchor_branch, anchor, branch, n_req, L, piv, prm, scores, &s);
    if (st != RPS_OK) return st;
    if ((st = make_commit_args(scores, n_req, L, piv, prm, out, &c)) != RPS_OK) return st;
    DeviceInfo dev;
    if ((st = device_info(&dev)) != RPS_OK) return st;
    s.err = dev.err;
    return from_cuda(launch_score_commit(s, c, reinterpret_cast<cudaStream_t>(stream)));
}

rps_status rps_run_step(const rps_logits *logits, int32_t n_req, int32_t L, const int32_t *d_mask_pos,
                        const int32_t *d_mask_cnt, const rps_params *prm, const rps_row_stats *base,
                        const rps_pivots *piv, const rps_row_stats *branch, const rps_branch_scores *scores,
                        const rps_commit_out *out, void *d_ws_base, size_t ws_base_bytes, void *d_ws_branch,
                        size_t ws_branch_bytes, rps_stream_t stream) {
    // every argument is checked before anything is enqueued
    if (!piv || !piv->branch_rows || !piv->n_branch_rows || !prm || !base || !base->topk_idx || !branch ||
        branch->topk_idx)
        return RPS_ERR_INVALID_ARG;
    if (prm->n_pivots < 1 || prm->tokens_per_pivot < 1 || L < 1) return RPS_ERR_INVALID_ARG;
    if (static_cast<int64_t>(prm->n_pivots) * prm->tokens_per_pivot * L > INT32_MAX / 3) return RPS_ERR_INVALID_ARG;
    rps_row_list rows_base;
    rows_base.rows = nullptr;
    rows_base.seg_cnt = d_mask_cnt;
    rows_base.n_seg = n_req;
    rows_base.cap = L;
    rows_base.mask_pos = d_mask_pos;
    rows_base.mask_branch = 0;
    rps_row_list rows_la;
    rows_la.rows = piv->branch_rows;
    rows_la.seg_cnt = piv->n_branch_rows;
    rows_la.n_seg = n_req;
    rows_la.cap = prm->n_pivots * prm->tokens_per_pivot * L;
    rows_la.mask_pos = nullptr;
    rows_la.mask_branch = 0;
    RowStatsArgs a_base, a_la;
    SelectArgs sel;
    ScoreArgs sc;
    CommitArgs cm;
    int grid_base = 0, grid_la = 0, topk_grid_base = 0, topk_grid_la = 0;
    rps_status st;
    if ((st = prepare_row_stats(logits, &rows_base, prm, base, d_ws_base, ws_base_bytes, &a_base, &grid_base,
                                &topk_grid_base)) != RPS_OK)
        return st;
    if ((st = make_select_args(base, n_req, L, d_mask_pos, d_mask_cnt, prm, piv, &sel)) != RPS_OK) return st;
    if ((st = prepare_row_stats(logits, &rows_la, prm, branch, d_ws_branch, ws_branch_bytes, &a_la, &grid_la,
                                &topk_grid_la)) != RPS_OK)
        return st;
    if ((st = make_score_args(logits, 0, base, branch, n_req, L, piv, prm, scores, &sc)) != RPS_OK) return st;
    if ((st = make_commit_args(scores, n_req, L, piv, prm, out, &cm)) != RPS_OK) return st;
    if (d_ws_base == d_ws_branch) return RPS_ERR_INVALID_ARG;
    sc.err = a_la.err;
    // inside one step the select launch follows the base statistics only, and
    // score and commit follow the lookahead statistics only
    sel.early = 1;
    sc.early = 1;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = launch_row_stats(a_base, logits->dtype, grid_base, topk_grid_base, s);
    if (e == cudaSuccess) e = launch_select(sel, s);
    if (e == cudaSuccess) e = launch_row_stats(a_la, logits->dtype, grid_la, topk_grid_la, s);
    if (e == cudaSuccess) e = launch_score_commit(sc, cm, s);
    return from_cuda(e);
}

rps_status rps_poll_device_status(rps_stream_t stream, uint32_t *detail) {
    if (detail) *detail = 0;
    if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) return RPS_ERR_CUDA;
    DeviceInfo dev;
    rps_status st = device_info(&dev);
    if (st != RPS_OK) return st;
    uint32_t v = 0;
    if (cudaMemcpy(&v, dev.err, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return RPS_ERR_CUDA;
    if (v == 0) return RPS_OK;
    const uint32_t zero = 0;
    if (cudaMemcpy(dev.err, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess) return RPS_ERR_CUDA;
    if (detail) *detail = v;
    return RPS_ERR_DEVICE;
}

const char *rps_status_string(rps_status status) {
    switch (status) {
    case RPS_OK: return "RPS_OK";
    case RPS_ERR_INVALID_ARG: return "RPS_ERR_INVALID_ARG: argument rejected on the host";
    case RPS_ERR_UNSUPPORTED: return "RPS_ERR_UNSUPPORTED: outside this build's limits";
    case RPS_ERR_CUDA: return "RPS_ERR_CUDA: a CUDA runtime call failed";
    case RPS_ERR_DEVICE: return "RPS_ERR_DEVICE: a kernel flagged bad data";
    case RPS_ERR_TIMEOUT: return "RPS_ERR_TIMEOUT: a bounded device wait gave up";
    }
    return "unknown rps_status";
}

int32_t rps_version(void) { return 300; }

uint64_t rps_debug_set_ring_wait_ns(uint64_t ns) {
    return g_ring_wait_ns.exchange(ns == UINT64_MAX ? kRingWaitNs : ns);
}

}  // extern "C"
