// gather.cu -- rps_gather_rows: copy the rows of a row list from one logit tensor
// to another (a caller's page-locked host memory, read by the GPU over the
// host link, into device memory), so that a step moves only the rows it scores.
#include <cstring>

#include "rps_internal.cuh"

namespace rps {
namespace {

struct GatherArgs {
    const char *src;
    char *dst;
    int32_t esize;
    int64_t vocab;
    int64_t s_req, s_branch, s_pos;  // element strides of src
    int64_t d_req, d_branch, d_pos;  // element strides of dst
    int32_t n_req, n_branch, n_pos;
    const int32_t *rows, *seg_cnt, *mask_pos;
    int32_t n_seg, cap, mask_branch;
    uint32_t *err;
};

constexpr int kGatherThreads = 256;
constexpr int kInFlight = 8;  // 16-byte loads a thread keeps in flight

// One block per row slot of the list: whole 16-byte units, then the ragged tail.
__global__ void __launch_bounds__(kGatherThreads) gather_kernel(const GatherArgs a) {
    pdl_wait();
    pdl_launch_next();
    const int64_t slot = blockIdx.x;
    const int seg = static_cast<int>(slot / a.cap), i = static_cast<int>(slot % a.cap);
    if (a.seg_cnt) {
        int c = a.seg_cnt[seg];
        c = c < 0 ? 0 : (c > a.cap ? a.cap : c);
        if (i >= c) return;
    }
    int32_t req, br, pos;
    if (a.rows) {
        req = a.rows[slot * 3 + 0];
        br = a.rows[slot * 3 + 1];
        pos = a.rows[slot * 3 + 2];
    } else {
        req = seg;
        br = a.mask_branch;
        pos = a.mask_pos[slot];
    }
    if (pos < 0) return;
    if (req < 0 || req >= a.n_req || br < 0 || br >= a.n_branch || pos >= a.n_pos) {
        if (threadIdx.x == 0) flag_error(a.err, RPS_DEVERR_ROW_INDEX);
        return;
    }
    const char *s = a.src + (req * a.s_req + br * a.s_branch + static_cast<int64_t>(pos) * a.s_pos) * a.esize;
    char *d = a.dst + (req * a.d_req + br * a.d_branch + static_cast<int64_t>(pos) * a.d_pos) * a.esize;
    const int64_t bytes = a.vocab * a.esize;
    const int64_t units = bytes / 16;
    const uint4 *su = reinterpret_cast<const uint4 *>(s);
    uint4 *du = reinterpret_cast<uint4 *>(d);
    for (int64_t u0 = threadIdx.x; u0 < units; u0 += static_cast<int64_t>(kInFlight) * blockDim.x) {
        uint4 v[kInFlight];
#pragma unroll
        for (int j = 0; j < kInFlight; ++j) {
            const int64_t u = u0 + static_cast<int64_t>(j) * blockDim.x;
            if (u < units) v[j] = __ldcs(su + u);
        }
#pragma unroll
        for (int j = 0; j < kInFlight; ++j) {
            const int64_t u = u0 + static_cast<int64_t>(j) * blockDim.x;
            if (u < units) du[u] = v[j];
        }
    }
    for (int64_t b = units * 16 + threadIdx.x; b < bytes; b += blockDim.x) d[b] = s[b];
}

}  // namespace
}  // namespace rps

using namespace rps;

extern "C" rps_status rps_gather_rows(const rps_logits *src, const rps_row_list *rows, const rps_logits *dst,
                                      rps_stream_t stream) {
    if (!src || !dst || !src->data || !dst->data || !rows) return RPS_ERR_INVALID_ARG;
    if (src->dtype != dst->dtype || (src->dtype != RPS_F32 && src->dtype != RPS_BF16)) return RPS_ERR_INVALID_ARG;
    if (src->vocab != dst->vocab || src->vocab < 1 || src->n_req != dst->n_req || src->n_branch != dst->n_branch ||
        src->n_pos != dst->n_pos || src->n_req < 1 || src->n_branch < 1 || src->n_pos < 1)
        return RPS_ERR_INVALID_ARG;
    if ((!rows->rows && !rows->mask_pos) || rows->n_seg < 1 || rows->cap < 1) return RPS_ERR_INVALID_ARG;
    if (static_cast<int64_t>(rows->n_seg) * rows->cap > INT32_MAX / 3) return RPS_ERR_INVALID_ARG;
    const int64_t esize = src->dtype == RPS_BF16 ? 2 : 4;
    for (const rps_logits *l : {src, dst}) {
        if (reinterpret_cast<uintptr_t>(l->data) % 16 || (l->req_stride * esize) % 16 ||
            (l->branch_stride * esize) % 16 || (l->pos_stride * esize) % 16)
            return RPS_ERR_INVALID_ARG;
    }
    // src: device memory, or page-locked host memory the device reads through its alias
    const void *s_dev = src->data;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, src->data) != cudaSuccess) {
        cudaGetLastError();
        return RPS_ERR_INVALID_ARG;
    }
    if (at.type == cudaMemoryTypeHost) {
        void *p = nullptr;
        if (cudaHostGetDevicePointer(&p, const_cast<void *>(src->data), 0) != cudaSuccess || !p) {
            cudaGetLastError();
            return RPS_ERR_INVALID_ARG;
        }
        s_dev = p;
    } else if (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged) {
        return RPS_ERR_INVALID_ARG;  // pageable host memory: the device cannot read it safely
    }
    if (cudaPointerGetAttributes(&at, dst->data) != cudaSuccess) {
        cudaGetLastError();
        return RPS_ERR_INVALID_ARG;
    }
    if (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged) return RPS_ERR_INVALID_ARG;
    GatherArgs a;
    a.src = static_cast<const char *>(s_dev);
    a.dst = const_cast<char *>(static_cast<const char *>(dst->data));  // dst is the written tensor
    a.esize = static_cast<int32_t>(esize);
    a.vocab = src->vocab;
    a.s_req = src->req_stride;
    a.s_branch = src->branch_stride;
    a.s_pos = src->pos_stride;
    a.d_req = dst->req_stride;
    a.d_branch = dst->branch_stride;
    a.d_pos = dst->pos_stride;
    a.n_req = src->n_req;
    a.n_branch = src->n_branch;
    a.n_pos = src->n_pos;
    a.rows = rows->rows;
    a.seg_cnt = rows->seg_cnt;
    a.mask_pos = rows->mask_pos;
    a.n_seg = rows->n_seg;
    a.cap = rows->cap;
    a.mask_branch = rows->mask_branch;
    a.err = device_error_word();
    if (!a.err) return RPS_ERR_CUDA;
    const int slots = rows->n_seg * rows->cap;
    return launch_pdl(gather_kernel, dim3(slots), dim3(kGatherThreads), 0, reinterpret_cast<cudaStream_t>(stream),
                      a) == cudaSuccess
               ? RPS_OK
               : RPS_ERR_CUDA;
}
