// rps_internal.cuh -- declarations shared by the library's translation units.
#pragma once

#include <cstdint>
#include <utility>

#include <cuda_runtime.h>

#include "rps.h"

namespace rps {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kMaxPartials = 32;   // partial records per row (one merging warp)
#ifndef RPS_STAT_THREADS
#define RPS_STAT_THREADS 1024
#endif
constexpr int kStatThreads = RPS_STAT_THREADS;  // threads per block of the row-statistics kernel (one block per SM: no launch-slot skew)
#ifndef RPS_STAT_BLOCKS_PER_SM
#define RPS_STAT_BLOCKS_PER_SM 1
#endif
constexpr int kStatBlocksPerSm = RPS_STAT_BLOCKS_PER_SM;
#ifndef RPS_TOPK_WARPS
#define RPS_TOPK_WARPS 4
#endif
#ifndef RPS_TOPK_MIN_BLOCKS
#define RPS_TOPK_MIN_BLOCKS 4
#endif
constexpr int kTopkWarps = RPS_TOPK_WARPS;            // warps (rows in flight) per block of the top-k launch
constexpr int kTopkMinBlocks = RPS_TOPK_MIN_BLOCKS;   // resident blocks per SM it is compiled for
// Sketch entries per row slot: 32 per ring chunk of the row under the cut of
// its statistics launch, at most units / 4 + 32 * kMaxPartials (at most
// kMaxPartials pieces hold a part of a row, each may end in a partial chunk).
__host__ __device__ constexpr int64_t sketch_entries(int64_t units) {
    return ((units + 3) / 4 + 32 * kMaxPartials + 7) / 8 * 8;
}
// Shape of each warp's shared-memory ring (overridable at build time for tuning).
#ifndef RPS_RING_UNITS_PER_LANE
#define RPS_RING_UNITS_PER_LANE 4
#endif
#ifndef RPS_RING_STAGES
#define RPS_RING_STAGES 2
#endif
constexpr int kBatch = RPS_RING_UNITS_PER_LANE;  // 16-byte units a lane takes from each ring buffer
constexpr int kStages = RPS_RING_STAGES;         // ring buffers (bulk copies in flight) per warp

// Partial statistics of one row segment, base-2 online softmax:
// s = sum 2^u, t = sum u 2^u with u = (z - mref) * log2(e); mx = max z and
// amax its lowest token index.
struct __align__(16) Partial {
    float mref;
    float s;
    float t;
    float mx;
    int32_t amax;
    int32_t pad[3];
};

struct RowStatsArgs {
    const void *data;
    int64_t vocab;
    int64_t req_stride, branch_stride, pos_stride;
    int32_t n_req, n_branch, n_pos;
    const int32_t *rows;
    const int32_t *seg_cnt;
    int32_t n_seg, cap;
    const int32_t *mask_pos;  // mask form of the row list when rows == nullptr
    int32_t mask_branch;
    int32_t k;  // top-k size, 0 = statistics only
    // outputs
    float *zmax, *lse, *H, *pmax, *mu, *htrunc, *topk_logit;
    int32_t *argmax, *topk_idx;
    // workspace
    Partial *part;        // [slots][kMaxPartials]
    void *sketch;         // [slots][sketch_stride] per-(chunk, lane) maxima (top-k mode)
    int64_t sketch_stride;  // sketch entries per slot (a multiple of 8)
    float4 *norm;         // [slots] B, ln S, 1 / S of each row's base-2 softmax and its sketch's len0 (top-k mode)
    int32_t *sketch_piece;  // [1] units per piece of the sketch layout (top-k mode)
    uint32_t *ticket;     // [slots]
    uint32_t *health;     // workspace health word: 0, or non-zero once a launch on this workspace gave up
    uint64_t ring_wait_ns;  // limit of a warp's wait for its next ring chunk (0: give up at once)
    // decomposition: the rows' 16-byte units are split evenly over `warps` warps
    int64_t units_per_row;
    int32_t warps;
    int64_t min_piece;    // at least ceil(units_per_row / (kMaxPartials - 1))
    uint32_t *err;
};

// Top-k mode (a.k > 0) takes two launches: the statistics launch, which also
// leaves the sketch and B, ln S, 1 / S, then the top-k launch of topk_grid blocks.
cudaError_t launch_row_stats(const RowStatsArgs &a, int dtype, int grid, int topk_grid, cudaStream_t stream);
cudaError_t row_stats_occupancy(int dtype, int *blocks_per_sm);

struct SelectArgs {
    // base statistics [q * L + k]
    const float *zmax, *pmax, *mu, *htrunc, *H, *topk_logit;
    const int32_t *argmax, *topk_idx;
    int32_t k_max;
    const int32_t *mask_pos, *mask_cnt;
    int32_t n_req, L, P, K;
    float tau, tau_pivot;
    double log_r;
    int32_t pivot_rule, commit_rule, commit_k;
    rps_pivots out;
    uint32_t *err;
    int32_t early;  // the mask predates the previous launch (see select_kernel)
};

struct ScoreArgs {
    const void *anchor_data;
    int32_t dtype;
    int64_t vocab, req_stride, pos_stride, branch_offset;
    int32_t n_pos;
    const float *a_H, *a_pmax, *a_lse, *a_zmax;  // anchor statistics [q * L + k]
    const float *b_H, *b_pmax;                   // branch statistics, compact [q * NB * L + i]
    rps_pivots piv;
    int32_t n_req, L, P, K;
    float lambda, tau;
    rps_branch_scores out;
    uint32_t *err;
    int32_t early;  // the pivots and anchor statistics predate the previous launch (see score_commit_kernel)
};

struct CommitArgs {
    const float *score;
    rps_pivots piv;
    int32_t n_req, L, P, K;
    rps_commit_out out;
};

cudaError_t launch_select(const SelectArgs &a, cudaStream_t stream);
cudaError_t launch_score(const ScoreArgs &a, cudaStream_t stream);
cudaError_t launch_commit(const CommitArgs &a, cudaStream_t stream);
cudaError_t launch_score_commit(const ScoreArgs &s, const CommitArgs &c, cudaStream_t stream);

// The calling device's sticky error word (nullptr if the device cannot be queried).
uint32_t *device_error_word();

// The current limit of a kernel's wait for an asynchronous copy (rps_debug_set_ring_wait_ns).
uint64_t ring_wait_limit_ns();

// The host-side argument rules of rps_score_step (everything but the
// workspace), checked before anything is enqueued; *k_out is the top-k size
// (0 in statistics-only mode). Shared by every row-statistics entry point.
rps_status check_row_stats_args(const rps_logits *logits, const rps_row_list *rows, const rps_params *prm,
                                const rps_row_stats *out, int32_t *k_out);

// ---------------------------------------------------------------- launches
// Every kernel of the library is launched with programmatic stream
// serialization: it may start while the previous kernel on the stream finishes,
// and waits (pdl_wait) for that kernel's completion and memory before reading
// anything. When the previous kernel is not one of ours this is the ordinary
// stream order.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Waits until the previous kernel on the stream has completed and its writes are visible.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Lets the next kernel on the stream begin launching (it still waits in pdl_wait).
__device__ __forceinline__ void pdl_launch_next() { asm volatile("griddepcontrol.launch_dependents;" :::); }

// ---------------------------------------------------------------- device
__device__ __forceinline__ void flag_error(uint32_t *err, uint32_t bits) {
    if (err) atomicOr(err, bits);
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFull, v, o));
    return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

__device__ __forceinline__ int warp_sum_int(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

__device__ __forceinline__ int warp_min_int(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(kFull, v, o));
    return v;
}

}  // namespace rps
