// decide.cu -- per-request decision kernels of one RPS step, one block per
// request, over the block-level steps of decide_device.cuh:
//
//   select_kernel        select_request                   -> rps_select_pivots
//   score_kernel         score_request                    -> rps_score_branches
//   commit_kernel        commit_request                   -> rps_commit
//   score_commit_kernel  score_commit_request             -> rps_score_and_commit
#include "decide_device.cuh"

namespace rps {
namespace {

// a.early: the mask predates the previous launch (the base rows' statistics),
// so it is staged before waiting for that launch. The next launch (the
// lookahead rows' statistics) is released only at the end: its blocks would
// otherwise sit, waiting, on this block's SM while it works.
__global__ void __launch_bounds__(kSelectThreads) select_kernel(const SelectArgs a) {
    if (!a.early) pdl_wait();
    extern __shared__ __align__(16) unsigned char sel_smem[];
    select_request(a, blockIdx.x, sel_smem, a.early != 0);
    pdl_launch_next();
}

__global__ void __launch_bounds__(kScoreThreads) score_kernel(const ScoreArgs a) {
    pdl_wait();
    pdl_launch_next();
    __shared__ PivotView v;
    __shared__ SlotPre pre[kMaxSlots];
    extern __shared__ __align__(16) int32_t view_smem[];
    stage_view(a.piv, blockIdx.x, a.L, a.P, a.K, v, view_smem, view_smem + a.L);
    __syncthreads();
    score_prepare(a, blockIdx.x, v, view_smem, pre);
    __syncthreads();
    score_finish(a, blockIdx.x, v, pre, nullptr);
}

__global__ void __launch_bounds__(kScoreThreads) commit_kernel(const CommitArgs a) {
    pdl_wait();
    pdl_launch_next();
    __shared__ PivotView v;
    __shared__ float sc[kMaxSlots];
    extern __shared__ __align__(16) int32_t view_smem[];
    const int q = blockIdx.x;
    stage_view(a.piv, q, a.L, a.P, a.K, v, view_smem, view_smem + a.L);
    for (int i = threadIdx.x; i < a.P * (a.K + 1); i += blockDim.x)
        sc[i] = a.score[static_cast<int64_t>(q) * a.P * (a.K + 1) + i];
    __syncthreads();
    if (threadIdx.x < 32) commit_request(a, q, v, view_smem + a.L, sc);
}

// s.early: the pivots and the anchor's statistics come from launches before the
// previous one (the lookahead rows' statistics), so the first half of the
// scores runs before waiting for that launch.
__global__ void __launch_bounds__(kScoreThreads) score_commit_kernel(const ScoreArgs s, const CommitArgs c) {
    if (!s.early) pdl_wait();
    pdl_launch_next();
    extern __shared__ __align__(16) unsigned char sc_smem[];
    score_commit_request(s, c, blockIdx.x, sc_smem, s.early != 0);
}

}  // namespace

cudaError_t launch_select(const SelectArgs &a, cudaStream_t stream) {
    const size_t smem = select_smem_bytes(a.L);
    if (smem > 48 * 1024) {
        const cudaError_t e =
            cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    return launch_pdl(select_kernel, dim3(a.n_req), dim3(kSelectThreads), smem, stream, a);
}

cudaError_t launch_score(const ScoreArgs &a, cudaStream_t stream) {
    return launch_pdl(score_kernel, dim3(a.n_req), dim3(kScoreThreads), view_smem_bytes(a.L), stream, a);
}

cudaError_t launch_commit(const CommitArgs &a, cudaStream_t stream) {
    return launch_pdl(commit_kernel, dim3(a.n_req), dim3(kScoreThreads), view_smem_bytes(a.L), stream, a);
}

cudaError_t launch_score_commit(const ScoreArgs &s, const CommitArgs &c, cudaStream_t stream) {
    const size_t smem = score_commit_smem_bytes(s.L);
    if (smem > 48 * 1024) {
        const cudaError_t e = cudaFuncSetAttribute(score_commit_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    return launch_pdl(score_commit_kernel, dim3(s.n_req), dim3(kScoreThreads), smem, stream, s, c);
}

}  // namespace rps
