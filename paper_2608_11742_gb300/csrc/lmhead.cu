// lmhead.cu -- row statistics straight from the LM head (rps_lmhead_row_stats).
//
// Each scored row's logits are z = h W^T: its hidden state h (d bf16) against
// the unembedding W (one row of d bf16 weights per token). The paper's p_i is
// the softmax of that row (Sec. 2 notation), and the statistics of Eq. 1 and
// Eq. 3 follow from it. Here the contraction runs on the tensor cores and the
// statistics are folded in its epilogue, so the logits never reach HBM.
//
// Contraction. A CTA owns one tile of 128 hidden rows and one contiguous range
// of 256-token vocabulary tiles (a "split"); the CTAs of every row tile take
// the same splits, so they stream the same unembedding tiles at the same pace
// and each tile comes from HBM once, the other row tiles finding it in L2.
//   warp 0      TMA producer: per 64-wide slice of d, the hidden tile (128 x
//               64) and the unembedding tile (256 x 64), 128-byte swizzle,
//               into a ring of kStages shared-memory stages (mbarrier
//               completion, bounded waits);
//   warp 1      MMA issuer: tcgen05.mma kind::f16 (bf16 x bf16 -> f32), M = 128,
//               N = 256, K = 16, four per stage, into one of two TMEM
//               accumulators (128 lanes x 256 columns each), so that the
//               epilogue of one tile overlaps the contraction of the next;
//               it also allocates and frees the 512 TMEM columns;
//   warps 2-5   epilogue: thread = row (TMEM lane). tcgen05.ld brings its 256
//               logits; pass 1 finds the tile maximum, pass 2 folds the
//               logits into the row's base-2 online softmax record (B, S, T
//               with S = sum 2^u, T = sum u 2^u, u = z log2(e) - B), the
//               running maximum and argmax, and, in top-k mode, a sorted
//               register list of the KMAX largest logits.
// At the end of its range each epilogue thread leaves its row's record and
// list in the workspace; a second launch (one warp per row) merges the splits
// and writes the statistics, with the same formulas as the streaming kernel.
//
// Every mbarrier wait is bounded (%globaltimer). A role whose wait runs out
// flags RPS_DEVERR_TIMEOUT, marks the workspace unhealthy and raises a CTA
// abort flag that ends the other roles' waits; the producer then waits,
// bounded, for the copies it issued, the MMA issuer for the MMAs it issued,
// and TMEM is freed before the CTA exits.
#include <cuda.h>  // CUtensorMap and the tensor-map encoder's signature (no link against the driver)
#include <cudaTypedefs.h>

#include <algorithm>
#include <cfloat>
#include <climits>
#include <cstring>
#include <mutex>

#include "rps_internal.cuh"
#include "umma_desc.h"

namespace rps {
namespace {

constexpr int kTileM = 128;                 // hidden rows per tile (TMEM lanes)
constexpr int kTileN = 256;                 // tokens per tile (accumulator columns)
constexpr int kTileK = 64;                  // d per stage: one 128-byte swizzle row of bf16
constexpr int kMmaK = 16;                   // K of one tcgen05.mma kind::f16
constexpr int kStages = 4;
constexpr int kABytes = kTileM * kTileK * 2;  // 16 KB
constexpr int kBBytes = kTileN * kTileK * 2;  // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kThreads = 192;               // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr int kEpiWarps = 4;
constexpr uint32_t kTmemCols = 2 * kTileN;  // two accumulators
constexpr int kMaxSplits = 256;
constexpr int kSmemBytes = kStages * kStageBytes + 1024;  // + slack to align the ring to 1024 bytes
constexpr int kMergeThreads = 256;
constexpr uint64_t kDrainNs = 200ull * 1000 * 1000;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// One split's record of a row.
struct __align__(16) LmPartial {
    float B;   // base-2 reference
    float s;   // sum 2^u
    float t;   // sum u 2^u
    float mx;  // largest logit
    int32_t amax;
    int32_t pad[3];
};

struct LmArgs {
    int32_t n_rows, d, n_vt, splits, kmax, k;
    const uint8_t *w_packed;  // unembedding in the packed tile layout, or nullptr (tensor map)
    int64_t vocab;
    LmPartial *part;   // [n_rows][splits]
    float2 *lists;     // [n_rows][splits][kmax]: (logit, token id as int bits)
    float *logits_out; // optional [n_rows][vocab]
    uint32_t *health;
    uint32_t *err;
    uint64_t wait_ns;
    float *zmax, *lse, *H, *pmax, *mu, *htrunc, *topk_logit;
    int32_t *argmax, *topk_idx;
};

// ---------------------------------------------------------------- PTX
__device__ __forceinline__ uint32_t saddr(const void *p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(saddr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(saddr(bar)) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(saddr(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(saddr(bar)), "r"(parity)
        : "memory");
    return done != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int c0, int c1, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            saddr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(saddr(bar))
        : "memory");
}
// Plain bulk copy of `bytes` contiguous bytes into shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     saddr(dst)),
                 "l"(src), "r"(bytes), "r"(saddr(bar))
                 : "memory");
}
__device__ __forceinline__ void prefetch_map(const CUtensorMap *map) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t *slot, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(slot)), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] x B[smem]^T, bf16 inputs, f32 accumulator; accumulate != 0 adds to D.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrives on `bar` once every tcgen05 operation this thread issued before has completed.
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(saddr(bar))
                 : "memory");
}

// 32 consecutive f32 columns of this thread's TMEM lane (the warp's 32 lanes at once).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// ---------------------------------------------------------------- bounded waits
struct Ctl {
    uint64_t full[kStages], empty[kStages], acc_full[2], acc_empty[2], mma_done;
    uint32_t tmem_base;
    int abort_flag;
    int skip;
};

// Waits for phase `parity` of `bar`. False when the CTA aborts: this wait ran
// out (then it flags the timeout, marks the workspace and raises the abort
// flag) or another role already aborted.
__device__ bool wait_or_abort(uint64_t *bar, uint32_t parity, Ctl &c, const LmArgs &a) {
    if (a.wait_ns != 0 && mbar_try_wait(bar, parity)) return true;
    const uint64_t start = global_ns();
    while (a.wait_ns != 0) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*reinterpret_cast<volatile int *>(&c.abort_flag)) return false;
        if (global_ns() - start > a.wait_ns) break;
    }
    flag_error(a.err, RPS_DEVERR_TIMEOUT);
    atomicExch(a.health, 1u);
    *reinterpret_cast<volatile int *>(&c.abort_flag) = 1;
    return false;
}

// A wait that only ends early when the phase completes (drains before exit).
// wait_or_abort for every lane of a warp that goes on to warp-wide tcgen05
// instructions: the warp leaves together, on the same answer.
template <typename Ctl_, typename Args_>
__device__ __forceinline__ bool warp_wait_or_abort(uint64_t *bar, uint32_t parity, Ctl_ &c, const Args_ &a) {
    return __all_sync(kFull, wait_or_abort(bar, parity, c, a));
}

__device__ void wait_drain(uint64_t *bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return;
    const uint64_t start = global_ns();
    while (global_ns() - start < kDrainNs)
        if (mbar_try_wait(bar, parity)) return;
}

// ---------------------------------------------------------------- epilogue state
template <int KMAX>
struct RowState {
    float B, s, t, mx;
    int amx;
    float lv[KMAX > 0 ? KMAX : 1];
    int li[KMAX > 0 ? KMAX : 1];
};

// Inserts (z, id) into the sorted list (logit desc; ids arrive in increasing
// order, so equal logits keep the lower id first). Called for z > lv[KMAX-1].
template <int KMAX>
__device__ __forceinline__ void list_insert(RowState<KMAX> &st, float z, int id) {
    float cv = z;
    int ci = id;
#pragma unroll
    for (int i = 0; i < KMAX; ++i) {
        const bool sw = cv > st.lv[i];
        const float tv = st.lv[i];
        const int ti = st.li[i];
        st.lv[i] = sw ? cv : tv;
        st.li[i] = sw ? ci : ti;
        cv = sw ? tv : cv;
        ci = sw ? ti : ci;
    }
}

template <int KMAX>
__global__ void __launch_bounds__(kThreads, 1)
    lmhead_kernel(const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_w, const LmArgs a) {
    extern __shared__ uint8_t dyn_smem[];
    __shared__ Ctl c;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rt = blockIdx.x / a.splits, split = blockIdx.x - rt * a.splits;
    const int vt0 = static_cast<int>(static_cast<int64_t>(split) * a.n_vt / a.splits);
    const int vt1 = static_cast<int>(static_cast<int64_t>(split + 1) * a.n_vt / a.splits);
    const int n_tiles = vt1 - vt0;
    const int kblocks = a.d / kTileK;
    // the ring starts on a 1024-byte boundary (the 128-byte swizzle's period)
    uint8_t *ring = dyn_smem + ((1024u - (saddr(dyn_smem) & 1023u)) & 1023u);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&c.full[s], 1);
            mbar_init(&c.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&c.acc_full[b], 1);
            mbar_init(&c.acc_empty[b], kEpiWarps);
        }
        mbar_init(&c.mma_done, 1);
        c.abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0 && lane == 0) {
        prefetch_map(&tm_h);
        prefetch_map(&tm_w);
    }
    if (warp == 1) {
        tmem_alloc(&c.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    // the hidden rows may come from the previous kernel on the stream
    pdl_wait();
    pdl_launch_next();
    if (threadIdx.x == 0) c.skip = __ldcg(a.health) != 0;
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = c.tmem_base;
    if (c.skip) {  // a workspace an earlier launch gave up on: write nothing
        if (threadIdx.x == 0) flag_error(a.err, RPS_DEVERR_WORKSPACE);
    } else if (warp == 0) {
        if (lane == 0) {  // ---------------------------------------- TMA producer
            uint32_t it = 0;
            bool ok = true;
            for (int t = 0; t < n_tiles && ok; ++t) {
                const int vt = vt0 + t;
                for (int kb = 0; kb < kblocks; ++kb) {
                    const int s = it % kStages;
                    const uint32_t ph = (it / kStages) & 1;
                    if (!wait_or_abort(&c.empty[s], ph ^ 1, c, a)) {
                        ok = false;
                        break;
                    }
                    uint8_t *sa = ring + s * kStageBytes;
                    mbar_expect_tx(&c.full[s], kStageBytes);
                    tma_load_2d(sa, &tm_h, kb * kTileK, rt * kTileM, &c.full[s]);
                    if (a.w_packed)  // one contiguous 32 KB block, already in the swizzled image
                        bulk_load(sa + kABytes, a.w_packed + (static_cast<int64_t>(vt) * kblocks + kb) * kBBytes,
                                  kBBytes, &c.full[s]);
                    else
                        tma_load_2d(sa + kABytes, &tm_w, kb * kTileK, vt * kTileN, &c.full[s]);
                    ++it;
                }
            }
            // every copy issued lands before the CTA leaves, whichever role
            // aborted (in a normal run these phases have long completed)
            for (uint32_t j = it > kStages ? it - kStages : 0; j < it; ++j)
                wait_drain(&c.full[j % kStages], (j / kStages) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ---------------------------------------- MMA issuer
            constexpr uint32_t idesc = umma::instr_desc_bf16(kTileM, kTileN);
            uint32_t it = 0;
            bool ok = true;
            for (int t = 0; t < n_tiles && ok; ++t) {
                const int buf = t & 1;
                const uint32_t use = static_cast<uint32_t>(t >> 1);
                if (!wait_or_abort(&c.acc_empty[buf], (use & 1) ^ 1, c, a)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + static_cast<uint32_t>(buf * kTileN);
                for (int kb = 0; kb < kblocks; ++kb) {
                    const int s = it % kStages;
                    const uint32_t ph = (it / kStages) & 1;
                    if (!wait_or_abort(&c.full[s], ph, c, a)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = saddr(ring + s * kStageBytes);
                    const uint64_t ad = umma::smem_desc_kmajor_sw128(sa);
                    const uint64_t bd = umma::smem_desc_kmajor_sw128(sa + kABytes);
#pragma unroll
                    for (int k = 0; k < kTileK / kMmaK; ++k)
                        mma_bf16(d_tmem, umma::advance_k16(ad, k), umma::advance_k16(bd, k), idesc,
                                 (kb | k) != 0 ? 1u : 0u);
                    mma_commit(&c.empty[s]);  // the stage is free once these MMAs have read it
                    ++it;
                }
                if (ok) mma_commit(&c.acc_full[buf]);
            }
            // every MMA issued has completed before TMEM is freed
            mma_commit(&c.mma_done);
            wait_drain(&c.mma_done, 0);
        }
        __syncwarp();
    } else {  // ---------------------------------------------------- epilogue
        const int q = warp & 3;  // this warp's quarter of the TMEM lanes
        const int row = rt * kTileM + q * 32 + lane;
        const bool live = row < a.n_rows;
        RowState<KMAX> st;
        st.B = -INFINITY;
        st.s = 0.f;
        st.t = 0.f;
        st.mx = -INFINITY;
        st.amx = INT_MAX;
#pragma unroll
        for (int i = 0; i < (KMAX > 0 ? KMAX : 1); ++i) {
            st.lv[i] = -INFINITY;
            st.li[i] = INT_MAX;
        }
        bool ok = true;
        for (int t = 0; t < n_tiles; ++t) {
            const int buf = t & 1;
            const uint32_t use = static_cast<uint32_t>(t >> 1);
            if (!warp_wait_or_abort(&c.acc_full[buf], use & 1, c, a)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t tbase = tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(buf * kTileN);
            const int col0 = (vt0 + t) * kTileN;
            const int ncol = static_cast<int>(min(static_cast<int64_t>(kTileN), a.vocab - col0));
            // pass 1: the tile's maximum and its lowest column
            float tm = -INFINITY;
            int ta = INT_MAX;
            for (int ch = 0; ch < kTileN / 32; ++ch) {
                float v[32];
                tmem_ld32(tbase + ch * 32, v);
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const int cc = ch * 32 + i;
                    if (cc < ncol && v[i] > tm) {
                        tm = v[i];
                        ta = col0 + cc;
                    }
                }
            }
            if (tm > st.mx) {
                st.mx = tm;
                st.amx = ta;
            }
            // the base-2 reference follows the running maximum
            const float nb = fmaxf(st.B, tm * kLog2e);
            if (nb > st.B) {
                if (st.s > 0.f) {
                    const float dl = st.B - nb;
                    const float f = ex2(dl);
                    st.t = f * fmaf(dl, st.s, st.t);
                    st.s *= f;
                }
                st.B = nb;
            }
            // pass 2: the sums, the top-k list, and (testing only) the logits
            for (int ch = 0; ch < kTileN / 32; ++ch) {
                float v[32];
                tmem_ld32(tbase + ch * 32, v);
                const int nv = min(32, ncol - ch * 32);  // valid columns of this chunk (32 but in the last tile)
                if (nv < 32) {
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (i >= nv) v[i] = -INFINITY;  // contributes 2^-inf = 0 and never enters the list
                }
                float ps[2] = {0.f, 0.f}, pt[2] = {0.f, 0.f};
                uint32_t cand = 0;  // columns that pass the list's last entry
                const float thr = KMAX > 0 ? st.lv[KMAX > 0 ? KMAX - 1 : 0] : INFINITY;
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const float u = fmaf(v[i], kLog2e, -st.B);
                    const float e = ex2(u);
                    ps[i & 1] += e;
                    pt[i & 1] = fmaf(e > 0.f ? u : 0.f, e, pt[i & 1]);
                    if (KMAX > 0 && v[i] > thr) cand |= 1u << i;
                }
                st.s += ps[0] + ps[1];
                st.t += pt[0] + pt[1];
                // the few candidates, one copy of the insertion (the list only
                // grows stricter, so each is checked again against it)
#pragma unroll 1
                while (KMAX > 0 && cand) {
                    const int i = __ffs(cand) - 1;
                    cand &= cand - 1;
                    float x = v[0];
#pragma unroll
                    for (int j = 1; j < 32; ++j) x = j == i ? v[j] : x;
                    if (x > st.lv[KMAX > 0 ? KMAX - 1 : 0]) list_insert<KMAX>(st, x, col0 + ch * 32 + i);
                }
                if (a.logits_out && live) {
                    float *dst = a.logits_out + static_cast<int64_t>(row) * a.vocab + col0 + ch * 32;
                    for (int i = 0; i < 32; ++i)
                        if (ch * 32 + i < ncol) dst[i] = v[i];
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.acc_empty[buf]);
        }
        if (ok && live) {
            const int64_t slot = static_cast<int64_t>(row) * a.splits + split;
            LmPartial p;
            p.B = st.B;
            p.s = st.s;
            p.t = st.t;
            p.mx = st.mx;
            p.amax = st.amx;
            p.pad[0] = p.pad[1] = p.pad[2] = 0;
            a.part[slot] = p;
            if (KMAX > 0) {
                float2 *l = a.lists + slot * KMAX;
#pragma unroll
                for (int i = 0; i < (KMAX > 0 ? KMAX : 1); ++i) l[i] = make_float2(st.lv[i], __int_as_float(st.li[i]));
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ---------------------------------------------------------------- merge
__device__ __forceinline__ bool better(float v, int i, float w, int j) { return v > w || (v == w && i < j); }

// One warp per row: the splits' records give zmax, lse, H, P^max and argmax;
// in top-k mode a k-way merge of the splits' sorted lists gives T_i, mu and
// the truncated entropy (Eq. 3). Lane l owns splits l, l + 32, ...
template <int KMAX>
__global__ void __launch_bounds__(kMergeThreads) lmhead_merge_kernel(const LmArgs a) {
    constexpr int kPerLane = kMaxSplits / 32;
    __shared__ int head_all[kMergeThreads / 32][kMaxSplits];
    pdl_wait();
    pdl_launch_next();
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    if (__ldcg(a.health) != 0) {
        if (blockIdx.x == 0 && threadIdx.x == 0) flag_error(a.err, RPS_DEVERR_WORKSPACE);
        return;
    }
    int *head = head_all[wib];
    const int warps = gridDim.x * (kMergeThreads / 32);
    for (int row = blockIdx.x * (kMergeThreads / 32) + wib; row < a.n_rows; row += warps) {
        const LmPartial *pr = a.part + static_cast<int64_t>(row) * a.splits;
        // the largest reference of the row's live records
        float M = -INFINITY, mx = -INFINITY;
        int am = INT_MAX;
        bool nan = false;
        for (int j = lane; j < a.splits; j += 32) {
            const LmPartial p = pr[j];
            if (p.s > 0.f) M = fmaxf(M, p.B);
            if (p.s != p.s) nan = true;
            if (p.mx > mx || (p.mx == mx && p.amax < am)) {
                mx = p.mx;
                am = p.amax;
            }
        }
        M = warp_max(M);
        float S = 0.f, T = 0.f;
        for (int j = lane; j < a.splits; j += 32) {
            const LmPartial p = pr[j];
            if (p.s > 0.f) {
                const float dl = p.B - M;
                const float f = ex2(dl);
                S = fmaf(f, p.s, S);
                T = fmaf(f, fmaf(dl, p.s, p.t), T);
            }
        }
        S = warp_sum(S);
        T = warp_sum(T);
        nan = __any_sync(kFull, nan);
        const float rmx = warp_max(mx);
        const int ram = warp_min_int(mx == rmx ? am : INT_MAX);
        const bool ok = !nan && rmx > -INFINITY && S > 0.f && !(T != T) && ram != INT_MAX;
        float lse = NAN, H = NAN, pmax = NAN, lnS = NAN, invS = NAN;
        if (ok) {
            lnS = logf(S);
            invS = 1.f / S;
            lse = fmaf(M, kLn2, lnS);
            H = fmaxf(lnS - kLn2 * T * invS, 0.f);
            pmax = ex2(fmaf(rmx, kLog2e, -M)) * invS;
        }
        if (lane == 0) {
            a.zmax[row] = ok ? rmx : NAN;
            a.lse[row] = lse;
            a.H[row] = H;
            a.pmax[row] = pmax;
            a.argmax[row] = ok ? ram : -1;
            if (!ok) flag_error(a.err, RPS_DEVERR_NONFINITE);
        }
        if constexpr (KMAX > 0) {  // (the statistics-only form has no lists)
            if (a.k == 0) continue;
            // k-way merge: rank r goes to lane r
            for (int j = lane; j < a.splits; j += 32) head[j] = 0;
            __syncwarp();
            const float2 *ls = a.lists + static_cast<int64_t>(row) * a.splits * KMAX;
            float tv = -INFINITY;
            int ti = INT_MAX;
            for (int r = 0; r < a.k; ++r) {
                float bv = -INFINITY;
                int bi = INT_MAX, bj = -1;
    #pragma unroll
                for (int m = 0; m < kPerLane; ++m) {
                    const int j = lane + 32 * m;
                    if (j < a.splits && head[j] < KMAX) {
                        const float2 e = ls[j * KMAX + head[j]];
                        const int id = __float_as_int(e.y);
                        if (bj < 0 || better(e.x, id, bv, bi)) {
                            bv = e.x;
                            bi = id;
                            bj = j;
                        }
                    }
                }
                // warp-wide best (logit desc, token asc)
                float wv = bv;
                int wi = bi, wl = bj < 0 ? INT_MAX : lane;
    #pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    const float ov = __shfl_xor_sync(kFull, wv, o);
                    const int oi = __shfl_xor_sync(kFull, wi, o);
                    const int ol = __shfl_xor_sync(kFull, wl, o);
                    if (ol != INT_MAX && (wl == INT_MAX || better(ov, oi, wv, wi))) {
                        wv = ov;
                        wi = oi;
                        wl = ol;
                    }
                }
                if (lane == wl) ++head[bj];
                if (lane == r) {
                    tv = wl == INT_MAX ? -INFINITY : wv;
                    ti = wl == INT_MAX ? INT_MAX : wi;
                }
                __syncwarp();
            }
            // mu and the truncated entropy against the row's reference, as the streaming kernel forms them
            float p = 0.f, h = 0.f;
            if (ok && lane < a.k && ti != INT_MAX) {
                const float u = fmaf(tv, kLog2e, -M);
                p = ex2(u) * invS;
                if (p > 0.f) h = -p * (u * kLn2 - lnS);
            }
            const float mu = warp_sum(p), ht = warp_sum(h);
            if (lane == 0) {
                a.mu[row] = ok ? mu : NAN;
                a.htrunc[row] = ok ? ht : NAN;
            }
            if (lane < a.k) {
                a.topk_idx[static_cast<int64_t>(row) * a.k + lane] = ti == INT_MAX ? -1 : ti;
                a.topk_logit[static_cast<int64_t>(row) * a.k + lane] = ti == INT_MAX ? NAN : tv;
            }
        }
    }
}

// ---------------------------------------------------------------- packed unembedding
// The packed layout holds, for vocabulary tile vt and d slice kb, the 256 x 64
// block W[256 vt + n][64 kb + k] as the 32 KB image a TMA load with 128-byte
// swizzle would leave in shared memory: row n at byte 128 n, its 16-byte
// chunk c at chunk position c ^ (n % 8). Rows past the vocabulary are zero.
// One thread per 16-byte chunk of the packed tensor.
__global__ void pack_unembed_kernel(const uint4 *w, int64_t vocab, int32_t d, int64_t stride_elems, uint4 *out,
                                    int64_t n_chunks) {
    const int kblocks = d / kTileK;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n_chunks;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t blk = i / (kBBytes / 16);
        const int in = static_cast<int>(i - blk * (kBBytes / 16));  // chunk within the block image
        const int n = in >> 3, pos = in & 7, c = pos ^ (n & 7);     // row, stored position, source chunk
        const int64_t vt = blk / kblocks;
        const int kb = static_cast<int>(blk - vt * kblocks);
        const int64_t row = vt * kTileN + n;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (row < vocab) v = w[(row * stride_elems + static_cast<int64_t>(kb) * kTileK) / 8 + c];
        out[i] = v;
    }
}

// ---------------------------------------------------------------- host
struct LmDevice {
    bool ready = false;
    int sm_count = 0;
};
constexpr int kMaxDevices = 64;
std::mutex g_lm_mutex;
LmDevice g_lm_devices[kMaxDevices];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

rps_status lm_device(LmDevice *out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RPS_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_lm_mutex);
    if (!g_encode) {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !fn)
            return RPS_ERR_CUDA;
        g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    LmDevice &d = g_lm_devices[dev];
    if (!d.ready) {
        if (cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return RPS_ERR_CUDA;
        const int kmaxes[3] = {0, 16, 32};
        for (int i = 0; i < 3; ++i) {
            cudaError_t e = kmaxes[i] == 0   ? cudaFuncSetAttribute(lmhead_kernel<0>,
                                                                    cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes)
                            : kmaxes[i] == 16 ? cudaFuncSetAttribute(lmhead_kernel<16>,
                                                                     cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes)
                                              : cudaFuncSetAttribute(lmhead_kernel<32>,
                                                                     cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
            if (e != cudaSuccess) return RPS_ERR_CUDA;
        }
        d.ready = true;
    }
    *out = d;
    return RPS_OK;
}

// 2-D bf16 tensor map over rows x d (d contiguous), box of 64 x box_rows, 128-byte swizzle.
rps_status make_map(CUtensorMap *m, const void *base, int64_t rows, int32_t d, int64_t stride_elems, int box_rows) {
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(stride_elems) * 2};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(kTileK), static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t es[2] = {1, 1};
    const CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
                                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? RPS_OK : RPS_ERR_CUDA;
}

int list_len(int32_t k) { return k == 0 ? 0 : (k <= 16 ? 16 : 32); }

struct LmLayout {
    size_t health, part, lists, total;
};

LmLayout lm_layout(int32_t n_rows, int64_t vocab, int32_t k) {
    const int64_t n_vt = (vocab + kTileN - 1) / kTileN;
    const size_t cap = static_cast<size_t>(n_rows) * static_cast<size_t>(std::min<int64_t>(n_vt, kMaxSplits));
    auto up = [](size_t x) { return (x + 255) / 256 * 256; };
    LmLayout l;
    l.health = 0;
    l.part = 256;
    l.lists = l.part + up(cap * sizeof(LmPartial));
    l.total = l.lists + up(cap * static_cast<size_t>(list_len(k)) * sizeof(float2));
    return l;
}

}  // namespace
}  // namespace rps

using namespace rps;

extern "C" {

size_t rps_lmhead_packed_bytes(int64_t vocab, int32_t d) {
    if (vocab < 1 || vocab > INT32_MAX || d < kTileK || d % kTileK) return 0;
    return static_cast<size_t>((vocab + kTileN - 1) / kTileN) * (d / kTileK) * kBBytes;
}

rps_status rps_lmhead_pack_unembed(const void *unembed, int64_t vocab, int32_t d, int64_t stride, void *packed,
                                   size_t packed_bytes, rps_stream_t stream) {
    if (!unembed || !packed || reinterpret_cast<uintptr_t>(unembed) % 16 || reinterpret_cast<uintptr_t>(packed) % 16)
        return RPS_ERR_INVALID_ARG;
    const size_t need = rps_lmhead_packed_bytes(vocab, d);
    if (need == 0 || stride < d || stride % 8 || packed_bytes < need) return RPS_ERR_INVALID_ARG;
    const int64_t n_chunks = static_cast<int64_t>(need / 16);
    const int grid = static_cast<int>(std::min<int64_t>((n_chunks + 255) / 256, 152 * 16));
    pack_unembed_kernel<<<grid, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint4 *>(unembed), vocab, d, stride, static_cast<uint4 *>(packed), n_chunks);
    return cudaGetLastError() == cudaSuccess ? RPS_OK : RPS_ERR_CUDA;
}

size_t rps_lmhead_workspace_bytes(int32_t n_rows, int64_t vocab, int32_t k_max) {
    if (n_rows < 1 || vocab < 1 || vocab > INT32_MAX || k_max < 0 || k_max > RPS_MAX_K) return 0;
    return lm_layout(n_rows, vocab, k_max).total;
}

rps_status rps_lmhead_row_stats(const rps_lmhead *lm, const rps_params *prm, const rps_row_stats *out,
                                float *d_logits_out, void *d_ws, size_t ws_bytes, rps_stream_t stream) {
    if (!lm || !lm->hidden || !lm->unembed || !out) return RPS_ERR_INVALID_ARG;
    if (lm->n_rows < 1 || lm->vocab < 1 || lm->vocab > INT32_MAX || lm->d < kTileK || lm->d % kTileK != 0)
        return RPS_ERR_INVALID_ARG;
    if (lm->hidden_stride < lm->d || lm->hidden_stride % 8) return RPS_ERR_INVALID_ARG;
    if (!lm->unembed_packed && (lm->unembed_stride < lm->d || lm->unembed_stride % 8)) return RPS_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(lm->hidden) % 16 || reinterpret_cast<uintptr_t>(lm->unembed) % 16)
        return RPS_ERR_INVALID_ARG;
    if (!out->zmax || !out->lse || !out->H || !out->pmax || !out->argmax) return RPS_ERR_INVALID_ARG;
    int32_t k = 0;
    if (out->topk_idx) {
        if (!prm || prm->k_max < 1) return RPS_ERR_INVALID_ARG;
        if (prm->k_max > RPS_MAX_K) return RPS_ERR_UNSUPPORTED;
        if (prm->k_max > lm->vocab || !out->topk_logit || !out->mu || !out->htrunc) return RPS_ERR_INVALID_ARG;
        k = prm->k_max;
    }
    const LmLayout w = lm_layout(lm->n_rows, lm->vocab, k);
    if (!d_ws || ws_bytes < w.total || reinterpret_cast<uintptr_t>(d_ws) % 16) return RPS_ERR_INVALID_ARG;
    LmDevice dev;
    rps_status st = lm_device(&dev);
    if (st != RPS_OK) return st;
    uint32_t *err = device_error_word();
    if (!err) return RPS_ERR_CUDA;

    const int n_rt = (lm->n_rows + kTileM - 1) / kTileM;
    const int n_vt = static_cast<int>((lm->vocab + kTileN - 1) / kTileN);
    const int splits = std::max(1, std::min({dev.sm_count / n_rt, n_vt, kMaxSplits}));
    CUtensorMap tm_h, tm_w;
    if ((st = make_map(&tm_h, lm->hidden, lm->n_rows, lm->d, lm->hidden_stride, kTileM)) != RPS_OK) return st;
    if (lm->unembed_packed) {  // the tensor map is not read; the hidden map stands in its slot
        tm_w = tm_h;
    } else if ((st = make_map(&tm_w, lm->unembed, lm->vocab, lm->d, lm->unembed_stride, kTileN)) != RPS_OK) {
        return st;
    }

    LmArgs a;
    std::memset(&a, 0, sizeof a);
    a.n_rows = lm->n_rows;
    a.d = lm->d;
    a.n_vt = n_vt;
    a.splits = splits;
    a.kmax = list_len(k);
    a.k = k;
    a.vocab = lm->vocab;
    char *ws = static_cast<char *>(d_ws);
    a.health = reinterpret_cast<uint32_t *>(ws + w.health);
    a.part = reinterpret_cast<LmPartial *>(ws + w.part);
    a.lists = reinterpret_cast<float2 *>(ws + w.lists);
    a.logits_out = d_logits_out;
    a.w_packed = lm->unembed_packed ? static_cast<const uint8_t *>(lm->unembed) : nullptr;
    a.err = err;
    a.wait_ns = ring_wait_limit_ns();
    a.zmax = out->zmax;
    a.lse = out->lse;
    a.H = out->H;
    a.pmax = out->pmax;
    a.argmax = out->argmax;
    a.mu = out->mu;
    a.htrunc = out->htrunc;
    a.topk_idx = out->topk_idx;
    a.topk_logit = out->topk_logit;

    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const dim3 grid(n_rt * splits), block(kThreads);
    cudaError_t e;
    if (a.kmax == 0) e = launch_pdl(lmhead_kernel<0>, grid, block, kSmemBytes, s, tm_h, tm_w, a);
    else if (a.kmax == 16) e = launch_pdl(lmhead_kernel<16>, grid, block, kSmemBytes, s, tm_h, tm_w, a);
    else e = launch_pdl(lmhead_kernel<32>, grid, block, kSmemBytes, s, tm_h, tm_w, a);
    if (e != cudaSuccess) return RPS_ERR_CUDA;
    const dim3 mgrid(std::min((lm->n_rows + kMergeThreads / 32 - 1) / (kMergeThreads / 32), dev.sm_count * 8));
    if (a.kmax == 0) e = launch_pdl(lmhead_merge_kernel<0>, mgrid, dim3(kMergeThreads), 0, s, a);
    else if (a.kmax == 16) e = launch_pdl(lmhead_merge_kernel<16>, mgrid, dim3(kMergeThreads), 0, s, a);
    else e = launch_pdl(lmhead_merge_kernel<32>, mgrid, dim3(kMergeThreads), 0, s, a);
    return e == cudaSuccess ? RPS_OK : RPS_ERR_CUDA;
}

}  // extern "C"
