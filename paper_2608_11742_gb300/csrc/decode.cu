// decode.cu -- the outer loop of Algorithm 1 over semi-autoregressive blocks
// (rps_decode_advance): record a step's committed tokens in the response and
// move a request whose block is fully decoded on to its next block.
#include "rps_internal.cuh"

namespace rps {
namespace {

struct AdvanceArgs {
    rps_pivots piv;
    rps_commit_out commit;
    int32_t B, L_total;
    int32_t *tokens, *block, *mask_pos, *mask_cnt, *done, *steps;
    uint32_t *err;
};

// One block per request. Positions of the commit lists are block-local.
__global__ void __launch_bounds__(256) advance_kernel(const AdvanceArgs a) {
    pdl_wait();
    pdl_launch_next();
    const int q = blockIdx.x, tid = threadIdx.x;
    const int B = a.B;
    const int64_t mq = static_cast<int64_t>(q) * B;
    if (a.done[q]) {
        if (tid == 0) a.mask_cnt[q] = 0;
        return;
    }
    if (tid == 0 && a.steps) a.steps[q] += 1;
    const int blk = a.block[q];
    const int first = blk * B;
    const int n_here = min(B, a.L_total - first);  // positions of this block
    int32_t *x = a.tokens + static_cast<int64_t>(q) * a.L_total + first;
    // the standard commit S (Eq. 2) and the committed pivot
    int n_s = a.piv.n_commit[q];
    if (n_s < 0 || n_s > B) {
        if (tid == 0) flag_error(a.err, RPS_DEVERR_MASK);
        n_s = 0;
    }
    for (int i = tid; i < n_s; i += blockDim.x) {
        const int p = a.piv.commit_pos[mq + i];
        if (p >= 0 && p < n_here) x[p] = a.piv.commit_tok[mq + i];
        else flag_error(a.err, RPS_DEVERR_MASK);
    }
    if (tid == 0) {
        const int p = a.commit.commit_pos[q];
        if (p >= 0 && p < n_here) x[p] = a.commit.commit_tok[q];
    }
    // the mask of the next step
    int cnt = a.commit.mask_cnt[q];
    if (cnt < 0 || cnt > B) {
        if (tid == 0) flag_error(a.err, RPS_DEVERR_MASK);
        cnt = 0;
    }
    if (cnt > 0) {
        if (a.commit.mask_pos != a.mask_pos)
            for (int i = tid; i < cnt; i += blockDim.x) a.mask_pos[mq + i] = a.commit.mask_pos[mq + i];
        if (tid == 0) a.mask_cnt[q] = cnt;
        return;
    }
    // block decoded: the next one, all masked, or the end of the response
    const int next = first + B;
    if (next < a.L_total) {
        const int n_next = min(B, a.L_total - next);
        for (int i = tid; i < n_next; i += blockDim.x) a.mask_pos[mq + i] = i;
        if (tid == 0) {
            a.block[q] = blk + 1;
            a.mask_cnt[q] = n_next;
        }
    } else if (tid == 0) {
        a.done[q] = 1;
        a.mask_cnt[q] = 0;
    }
}

}  // namespace

cudaError_t launch_advance(const AdvanceArgs &a, int n_req, cudaStream_t stream) {
    return launch_pdl(advance_kernel, dim3(n_req), dim3(256), 0, stream, a);
}

}  // namespace rps

using namespace rps;

extern "C" rps_status rps_decode_advance(const rps_pivots *piv, const rps_commit_out *commit, int32_t n_req,
                                         int32_t B, int32_t L_total, int32_t *d_tokens, int32_t *d_block,
                                         int32_t *d_mask_pos, int32_t *d_mask_cnt, int32_t *d_done,
                                         int32_t *d_steps, rps_stream_t stream) {
    if (!piv || !commit || n_req < 1 || B < 1 || L_total < 1 || !d_tokens || !d_block || !d_mask_pos ||
        !d_mask_cnt || !d_done)
        return RPS_ERR_INVALID_ARG;
    if (!piv->n_commit || !piv->commit_pos || !piv->commit_tok || !commit->commit_pos || !commit->commit_tok ||
        !commit->mask_pos || !commit->mask_cnt)
        return RPS_ERR_INVALID_ARG;
    if (B > RPS_MAX_POS) return RPS_ERR_UNSUPPORTED;
    AdvanceArgs a;
    a.piv = *piv;
    a.commit = *commit;
    a.B = B;
    a.L_total = L_total;
    a.tokens = d_tokens;
    a.block = d_block;
    a.mask_pos = d_mask_pos;
    a.mask_cnt = d_mask_cnt;
    a.done = d_done;
    a.steps = d_steps;
    a.err = device_error_word();
    if (!a.err) return RPS_ERR_CUDA;
    return launch_advance(a, n_req, reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess ? RPS_OK : RPS_ERR_CUDA;
}
