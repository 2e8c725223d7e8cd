// attention.cu -- branch-isolating attention of the packed lookahead forward
// pass (rps_packed_attention_fwd; Sec. 3.1 "Lookahead scoring", Fig. 2 right).
//
// The lookahead pass scores every candidate branch of a step in one forward
// pass over a packed sequence [context | branch 0 | branch 1 | ... ] (branch 0
// is the anchor: the normal sequence's own generation region). A branch's
// queries attend to the context and to their own branch, the context's
// queries to the normal sequence (context and branch 0). The mask is
// block-structured, so no mask is ever formed: a query tile walks exactly the
// key tiles of its two visible segments, and the last tile of a segment masks
// the keys past its end.
//
// One persistent CTA per SM takes work items (batch, head, 128-query tile):
//   warp 0      TMA producer: the Q tile (128 x 128, two 64-wide swizzle
//               atoms), then per key tile K (128 keys x 128) and V^T (128 dims
//               x 128 keys; V is stored transposed so that both MMA operands
//               are K-major), 128-byte swizzle, two stages;
//   warp 1      MMA issuer: S = Q K^T (M 128, N 128, K 128) into one of two
//               TMEM buffers, then O += P V^T into the TMEM accumulator once
//               the softmax has written P; it also allocates and frees TMEM;
//   warps 2-5   softmax: thread = query row. Pass 1 over its S row (tcgen05.ld)
//               finds the tile maximum; the base-2 reference m is raised only
//               when a score passes it by more than 8 (then O and the running
//               sum are rescaled in TMEM); pass 2 writes P = 2^(s c - m) as bf16
//               into shared memory in the swizzled layout the MMA reads. At the
//               end of an item O / l is written to global memory as bf16.
// Every wait is bounded; a role whose wait runs out flags RPS_DEVERR_TIMEOUT
// and raises the CTA's abort flag, copies and MMAs in flight are drained and
// TMEM is freed before the CTA exits.
#include <cuda.h>  // CUtensorMap and the tensor-map encoder's signature (no link against the driver)
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include "rps_internal.cuh"
#include "umma_desc.h"

namespace rps {
namespace {

constexpr int kD = 128;                      // head dimension
constexpr int kBQ = 128;                     // queries per tile (TMEM lanes)
constexpr int kBK = 128;                     // keys per tile
constexpr int kAtom = 64 * 128 * 2;          // one 128-row x 64-column bf16 swizzle atom: 16 KB
constexpr int kQBytes = 2 * kAtom;           // Q tile: two atoms along d
constexpr int kKBytes = 2 * kAtom;           // K tile: two atoms along d
constexpr int kVBytes = 2 * kAtom;           // V^T tile: two atoms along the keys
constexpr int kPBytes = 2 * kAtom;           // P tile: two atoms along the keys
constexpr int kKvStages = 2;
constexpr int kKvBytes = kKBytes + kVBytes;
constexpr int kSmemBytes = kQBytes + kKvStages * kKvBytes + kPBytes + 1024;
constexpr int kThreads = 192;
constexpr int kSoftWarps = 4;
constexpr uint32_t kTmemCols = 512;          // S buffers at columns 0 and 128, O at 256
constexpr uint32_t kOCol = 256;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescale = 8.0f;             // base-2 units a score may pass the reference by
constexpr uint64_t kDrainNs = 200ull * 1000 * 1000;

struct AttnArgs {
    int32_t n_bh, n_heads, n_tokens, n_context, n_branch, branch_len;
    int32_t q_tiles_ctx, q_tiles_branch, items;  // query tiles of the context, of one branch; work items
    float c;                                     // scale * log2(e)
    __nv_bfloat16 *out;
    uint32_t *err;
    uint64_t wait_ns;
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
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(saddr(bar))
                 : "memory");
}
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
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
        "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
        "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
        "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
        "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
        "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
        "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
        "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
        "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
        "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// ---------------------------------------------------------------- work items
// Item w = (bh, query tile); query tiles: the context's, then each branch's.
// Its key tiles: the context's, then those of the one visible branch.
struct Item {
    int bh, q_start, q_len;     // queries [q_start, q_start + q_len) of the packed sequence (q_len <= 128)
    int seg_b;                  // visible branch (0 for the context's queries)
    int n_ctx_tiles, n_tiles;   // key tiles: context tiles first
};

__device__ __forceinline__ Item item_of(const AttnArgs &a, int w) {
    Item it;
    const int per_bh = a.q_tiles_ctx + a.n_branch * a.q_tiles_branch;
    it.bh = w / per_bh;
    int t = w - it.bh * per_bh;
    if (t < a.q_tiles_ctx) {
        it.seg_b = 0;
        it.q_start = t * kBQ;
        it.q_len = min(kBQ, a.n_context - it.q_start);
    } else {
        t -= a.q_tiles_ctx;
        const int b = t / a.q_tiles_branch;
        const int qt = t - b * a.q_tiles_branch;
        it.seg_b = b;
        it.q_start = a.n_context + b * a.branch_len + qt * kBQ;
        it.q_len = min(kBQ, a.branch_len - qt * kBQ);
    }
    it.n_ctx_tiles = a.q_tiles_ctx;
    it.n_tiles = a.q_tiles_ctx + a.q_tiles_branch;
    return it;
}

// First key and number of valid keys of key tile j of an item.
__device__ __forceinline__ void key_tile(const AttnArgs &a, const Item &it, int j, int &k0, int &valid) {
    if (j < it.n_ctx_tiles) {
        k0 = j * kBK;
        valid = min(kBK, a.n_context - k0);
    } else {
        const int jj = j - it.n_ctx_tiles;
        k0 = a.n_context + it.seg_b * a.branch_len + jj * kBK;
        valid = min(kBK, a.branch_len - jj * kBK);
    }
}

struct Ctl {
    uint64_t q_full, q_empty, kv_full[kKvStages], kv_empty[kKvStages], s_full[2], p_full, pv_done, o_free, mma_done;
    uint32_t tmem_base;
    int abort_flag;
};

__device__ bool wait_or_abort(uint64_t *bar, uint32_t parity, Ctl &c, const AttnArgs &a) {
    if (a.wait_ns != 0 && mbar_try_wait(bar, parity)) return true;
    const uint64_t start = global_ns();
    while (a.wait_ns != 0) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*reinterpret_cast<volatile int *>(&c.abort_flag)) return false;
        if (global_ns() - start > a.wait_ns) break;
    }
    flag_error(a.err, RPS_DEVERR_TIMEOUT);
    *reinterpret_cast<volatile int *>(&c.abort_flag) = 1;
    return false;
}

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

__global__ void __launch_bounds__(kThreads, 1)
    packed_attention_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                            const __grid_constant__ CUtensorMap tm_vt, const AttnArgs a) {
    extern __shared__ uint8_t dyn_smem[];
    __shared__ Ctl c;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t *base = dyn_smem + ((1024u - (saddr(dyn_smem) & 1023u)) & 1023u);
    uint8_t *sq = base;
    uint8_t *skv = base + kQBytes;
    uint8_t *sp = skv + kKvStages * kKvBytes;

    if (threadIdx.x == 0) {
        mbar_init(&c.q_full, 1);
        mbar_init(&c.q_empty, 1);
        for (int s = 0; s < kKvStages; ++s) {
            mbar_init(&c.kv_full[s], 1);
            mbar_init(&c.kv_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) mbar_init(&c.s_full[b], 1);
        mbar_init(&c.p_full, kSoftWarps);
        mbar_init(&c.pv_done, 1);
        mbar_init(&c.o_free, kSoftWarps);
        mbar_init(&c.mma_done, 1);
        c.abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        tmem_alloc(&c.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    pdl_wait();
    pdl_launch_next();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = c.tmem_base;
    constexpr uint32_t idesc = umma::instr_desc_bf16(kBQ, kBK);

    if (warp == 0) {
        if (lane == 0) {  // -------------------------------------------- TMA producer
            uint32_t g = 0;  // key tiles issued (all items)
            int n_items = 0;
            bool ok = true;
            for (int w = blockIdx.x; w < a.items && ok; w += gridDim.x, ++n_items) {
                const Item it = item_of(a, w);
                if (!wait_or_abort(&c.q_empty, (n_items & 1) ^ 1, c, a)) break;
                mbar_expect_tx(&c.q_full, kQBytes);
                const int qrow = it.bh * a.n_tokens + it.q_start;
                tma_load_2d(sq, &tm_q, 0, qrow, &c.q_full);
                tma_load_2d(sq + kAtom, &tm_q, 64, qrow, &c.q_full);
                for (int j = 0; j < it.n_tiles; ++j, ++g) {
                    const int s = g % kKvStages;
                    if (!wait_or_abort(&c.kv_empty[s], ((g / kKvStages) & 1) ^ 1, c, a)) {
                        ok = false;
                        break;
                    }
                    int k0, valid;
                    key_tile(a, it, j, k0, valid);
                    uint8_t *sk = skv + s * kKvBytes, *sv = sk + kKBytes;
                    mbar_expect_tx(&c.kv_full[s], kKvBytes);
                    const int krow = it.bh * a.n_tokens + k0;
                    tma_load_2d(sk, &tm_k, 0, krow, &c.kv_full[s]);
                    tma_load_2d(sk + kAtom, &tm_k, 64, krow, &c.kv_full[s]);
                    tma_load_2d(sv, &tm_vt, k0, it.bh * kD, &c.kv_full[s]);
                    tma_load_2d(sv + kAtom, &tm_vt, k0 + 64, it.bh * kD, &c.kv_full[s]);
                }
            }
            // every copy issued lands before the CTA leaves
            for (uint32_t j = g > kKvStages ? g - kKvStages : 0; j < g; ++j)
                wait_drain(&c.kv_full[j % kKvStages], (j / kKvStages) & 1);
            if (n_items > 0) wait_drain(&c.q_full, (n_items - 1) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {  // -------------------------------------------- MMA issuer
            uint32_t g = 0;  // key tiles consumed (all items)
            int n_items = 0;
            bool ok = true;
            for (int w = blockIdx.x; w < a.items && ok; w += gridDim.x, ++n_items) {
                const Item it = item_of(a, w);
                if (!wait_or_abort(&c.q_full, n_items & 1, c, a)) break;
                tc_fence_after();
                const uint64_t qd = umma::smem_desc_kmajor_sw128(saddr(sq));
                const uint64_t qd1 = umma::smem_desc_kmajor_sw128(saddr(sq + kAtom));
                const uint64_t pd = umma::smem_desc_kmajor_sw128(saddr(sp));
                const uint64_t pd1 = umma::smem_desc_kmajor_sw128(saddr(sp + kAtom));
                for (int j = 0; j <= it.n_tiles && ok; ++j) {
                    if (j < it.n_tiles) {  // S_j = Q K_j^T
                        const uint32_t gj = g + j;
                        const int s = gj % kKvStages;
                        if (!wait_or_abort(&c.kv_full[s], (gj / kKvStages) & 1, c, a)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint8_t *sk = skv + s * kKvBytes;
                        const uint64_t kd = umma::smem_desc_kmajor_sw128(saddr(sk));
                        const uint64_t kd1 = umma::smem_desc_kmajor_sw128(saddr(sk + kAtom));
                        const uint32_t sbuf = tmem + (gj & 1) * kBK;
#pragma unroll
                        for (int k = 0; k < 8; ++k)
                            mma_bf16(sbuf, umma::advance_k16(k < 4 ? qd : qd1, k & 3),
                                     umma::advance_k16(k < 4 ? kd : kd1, k & 3), idesc, k != 0);
                        mma_commit(&c.s_full[gj & 1]);
                        if (j == it.n_tiles - 1) mma_commit(&c.q_empty);  // Q is no longer read
                    }
                    if (j >= 1) {  // O += P_{j-1} V_{j-1}
                        const uint32_t gp = g + j - 1;
                        if (j == 1 && !wait_or_abort(&c.o_free, (n_items & 1) ^ 1, c, a)) {
                            ok = false;
                            break;
                        }
                        if (!wait_or_abort(&c.p_full, gp & 1, c, a)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint8_t *sv = skv + (gp % kKvStages) * kKvBytes + kKBytes;
                        const uint64_t vd = umma::smem_desc_kmajor_sw128(saddr(sv));
                        const uint64_t vd1 = umma::smem_desc_kmajor_sw128(saddr(sv + kAtom));
#pragma unroll
                        for (int k = 0; k < 8; ++k)
                            mma_bf16(tmem + kOCol, umma::advance_k16(k < 4 ? pd : pd1, k & 3),
                                     umma::advance_k16(k < 4 ? vd : vd1, k & 3), idesc, (j > 1 || k != 0) ? 1u : 0u);
                        mma_commit(&c.kv_empty[gp % kKvStages]);
                        mma_commit(&c.pv_done);
                    }
                }
                g += it.n_tiles;
            }
            mma_commit(&c.mma_done);
            wait_drain(&c.mma_done, 0);
        }
        __syncwarp();
    } else {  // ---------------------------------------------------- softmax
        const int q = warp & 3;
        const int r = q * 32 + lane;  // query row in the tile (TMEM lane)
        const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
        uint32_t g = 0;
        int n_items = 0;
        for (int w = blockIdx.x; w < a.items; w += gridDim.x, ++n_items) {
            const Item it = item_of(a, w);
            float m = -INFINITY, l = 0.f;
            bool ok = true;
            for (int j = 0; j < it.n_tiles; ++j) {
                const uint32_t gj = g + j;
                if (!warp_wait_or_abort(&c.s_full[gj & 1], (gj >> 1) & 1, c, a)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                int k0, valid;
                key_tile(a, it, j, k0, valid);
                const uint32_t sbuf = tmem + lane_off + (gj & 1) * kBK;
                // pass 1: the tile's largest visible score
                float tmx = -INFINITY;
                for (int ch = 0; ch < kBK / 32; ++ch) {
                    float v[32];
                    tmem_ld32(sbuf + ch * 32, v);
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (ch * 32 + i < valid) tmx = fmaxf(tmx, v[i]);
                }
                const float tm = tmx * a.c;
                float f = 1.f;
                bool rescale = false;
                if (m == -INFINITY) {
                    m = tm;
                } else if (tm > m + kRescale) {
                    f = ex2(m - tm);
                    m = tm;
                    rescale = true;
                }
                // P and O of the previous tile are free once its PV has completed
                if (j >= 1) {
                    if (!warp_wait_or_abort(&c.pv_done, (gj - 1) & 1, c, a)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    // tcgen05.ld / st are warp-wide (.sync.aligned): the warp
                    // rescales together when any of its rows needs it, the
                    // other rows by f = 1
                    if (__any_sync(kFull, rescale)) {
                        for (int ch = 0; ch < kD / 32; ++ch) {
                            float o[32];
                            tmem_ld32(tmem + lane_off + kOCol + ch * 32, o);
#pragma unroll
                            for (int i = 0; i < 32; ++i) o[i] *= f;
                            tmem_st32(tmem + lane_off + kOCol + ch * 32, o);
                        }
                    }
                }
                l *= f;
                // pass 2: P = 2^(s c - m) into the swizzled P tile (row r)
                for (int ch = 0; ch < kBK / 32; ++ch) {
                    float v[32];
                    tmem_ld32(sbuf + ch * 32, v);
                    uint32_t pk[16];
#pragma unroll
                    for (int i = 0; i < 32; i += 2) {
                        const float p0 = ch * 32 + i < valid ? ex2(fmaf(v[i], a.c, -m)) : 0.f;
                        const float p1 = ch * 32 + i + 1 < valid ? ex2(fmaf(v[i + 1], a.c, -m)) : 0.f;
                        l += p0 + p1;
                        pk[i / 2] = pack_bf16(p0, p1);
                    }
                    // 32 keys = four 16-byte chunks of one atom row
                    const int atom = ch >> 1;
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int chunk = (ch & 1) * 4 + u;
                        uint4 *dst = reinterpret_cast<uint4 *>(sp + atom * kAtom + r * 128 + ((chunk ^ (r & 7)) << 4));
                        *dst = make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
                    }
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // P visible to the MMA
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&c.p_full);
            }
            if (!ok) break;
            const uint32_t glast = g + it.n_tiles - 1;
            if (!warp_wait_or_abort(&c.pv_done, glast & 1, c, a)) break;
            tc_fence_after();
            // O / l of this row, bf16, to global memory
            const bool live = r < it.q_len;
            const float inv = 1.f / l;
            __nv_bfloat16 *dst = a.out + (static_cast<int64_t>(it.bh) * a.n_tokens + it.q_start + r) * kD;
            for (int ch = 0; ch < kD / 32; ++ch) {
                float o[32];
                tmem_ld32(tmem + lane_off + kOCol + ch * 32, o);
                if (live) {
                    uint4 *d4 = reinterpret_cast<uint4 *>(dst + ch * 32);
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        d4[u] = make_uint4(pack_bf16(o[8 * u] * inv, o[8 * u + 1] * inv),
                                           pack_bf16(o[8 * u + 2] * inv, o[8 * u + 3] * inv),
                                           pack_bf16(o[8 * u + 4] * inv, o[8 * u + 5] * inv),
                                           pack_bf16(o[8 * u + 6] * inv, o[8 * u + 7] * inv));
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.o_free);  // O may be overwritten by the next item
            g += it.n_tiles;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ---------------------------------------------------------------- host
std::mutex g_attn_mutex;
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
bool g_attr_set[64] = {};
int g_sm_count[64] = {};

rps_status attn_setup(int *sm_count) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return RPS_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_attn_mutex);
    if (!g_encode) {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !fn)
            return RPS_ERR_CUDA;
        g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    if (!g_attr_set[dev]) {
        if (cudaDeviceGetAttribute(&g_sm_count[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            return RPS_ERR_CUDA;
        if (cudaFuncSetAttribute(packed_attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) !=
            cudaSuccess)
            return RPS_ERR_CUDA;
        g_attr_set[dev] = true;
    }
    *sm_count = g_sm_count[dev];
    return RPS_OK;
}

rps_status map_2d(CUtensorMap *m, const void *base, int64_t rows, int64_t cols) {
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
    const cuuint32_t box[2] = {64, 128};
    const cuuint32_t es[2] = {1, 1};
    const CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
                                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? RPS_OK : RPS_ERR_CUDA;
}

}  // namespace
}  // namespace rps

using namespace rps;

extern "C" rps_status rps_packed_attention_fwd(const rps_packed_attention *p, rps_stream_t stream) {
    if (!p || !p->q || !p->k || !p->vt || !p->out) return RPS_ERR_INVALID_ARG;
    if (p->head_dim != kD) return RPS_ERR_UNSUPPORTED;
    if (p->n_batch < 1 || p->n_heads < 1 || p->n_context < 0 || p->n_branch < 1 || p->branch_len < 1)
        return RPS_ERR_INVALID_ARG;
    if (p->n_context % 8 || p->branch_len % 8) return RPS_ERR_INVALID_ARG;
    if (!(p->scale > 0.f) || !std::isfinite(p->scale)) return RPS_ERR_INVALID_ARG;
    for (const void *x : {p->q, p->k, p->vt, static_cast<const void *>(p->out)})
        if (reinterpret_cast<uintptr_t>(x) % 16) return RPS_ERR_INVALID_ARG;
    const int64_t n_tokens = static_cast<int64_t>(p->n_context) + static_cast<int64_t>(p->n_branch) * p->branch_len;
    const int64_t n_bh = static_cast<int64_t>(p->n_batch) * p->n_heads;
    if (n_tokens > INT32_MAX / 2 || n_bh * n_tokens > INT32_MAX || n_bh * kD > INT32_MAX) return RPS_ERR_UNSUPPORTED;
    int sm_count = 0;
    rps_status st = attn_setup(&sm_count);
    if (st != RPS_OK) return st;
    uint32_t *err = device_error_word();
    if (!err) return RPS_ERR_CUDA;
    CUtensorMap tq, tk, tv;
    if ((st = map_2d(&tq, p->q, n_bh * n_tokens, kD)) != RPS_OK) return st;
    if ((st = map_2d(&tk, p->k, n_bh * n_tokens, kD)) != RPS_OK) return st;
    if ((st = map_2d(&tv, p->vt, n_bh * kD, n_tokens)) != RPS_OK) return st;
    AttnArgs a;
    std::memset(&a, 0, sizeof a);
    a.n_bh = static_cast<int32_t>(n_bh);
    a.n_heads = p->n_heads;
    a.n_tokens = static_cast<int32_t>(n_tokens);
    a.n_context = p->n_context;
    a.n_branch = p->n_branch;
    a.branch_len = p->branch_len;
    a.q_tiles_ctx = (p->n_context + kBQ - 1) / kBQ;
    a.q_tiles_branch = (p->branch_len + kBQ - 1) / kBQ;
    const int64_t items = n_bh * (a.q_tiles_ctx + static_cast<int64_t>(p->n_branch) * a.q_tiles_branch);
    if (items > INT32_MAX) return RPS_ERR_UNSUPPORTED;
    a.items = static_cast<int32_t>(items);
    a.c = p->scale * kLog2e;
    a.out = static_cast<__nv_bfloat16 *>(p->out);
    a.err = err;
    a.wait_ns = ring_wait_limit_ns();
    const int grid = static_cast<int>(std::min<int64_t>(items, sm_count));
    const cudaError_t e = launch_pdl(packed_attention_kernel, dim3(grid), dim3(kThreads), kSmemBytes,
                                     reinterpret_cast<cudaStream_t>(stream), tq, tk, tv, a);
    return e == cudaSuccess ? RPS_OK : RPS_ERR_CUDA;
}
