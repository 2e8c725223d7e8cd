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
//   warp 0      TMA producer of Q (128 x 128, two 64-wide swizzle atoms) and,
//               per key tile, K (128 keys x 128), 128-byte swizzle, two stages;
//   warp 6      TMA producer of V^T (128 dims x 128 keys: V is stored
//               transposed so that both MMA operands are K-major), two stages
//               of their own, so that K runs ahead of V (K is free once S is
//               computed, V only once P V is);
//   warp 1      MMA issuer: S = Q K^T (M 128, N 128, K 128) into one of two
//               TMEM buffers, then O += P V^T into the TMEM accumulator once
//               the softmax has written P; it also allocates and frees TMEM;
//   warps 2-5   softmax: thread = query row. Pass 1 over its S row (tcgen05.ld)
//               finds the tile maximum; the base-2 reference m is raised only
//               when a score passes it by more than 8 (then O and the running
//               sum are rescaled in TMEM); pass 2 writes P = 2^(s c - m) as bf16
//               into one of two shared-memory buffers, in the swizzled layout
//               the MMA reads, while the MMA still reads the other. At the end
//               of an item O / l is written to global memory as bf16.
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
constexpr int kKvStages = 2;
constexpr int kQBufs = 2;                    // the next item's Q loads while this item runs
constexpr int kSBufs = 3;                    // S (and P, in place) of key tile g in TMEM buffer g % 3
constexpr int kStageBytes = 32 * 64;           // per softmax warp: 32 rows x 32 bf16 of O on their way out
constexpr int kSmemBytes = kQBufs * kQBytes + kKvStages * (kKBytes + kVBytes) + 8 * kStageBytes + 1024;
constexpr int kThreads = 384;                // warps 0 and 10 TMA, 1 and 11 MMA, 2-9 softmax
constexpr int kSoftWarps = 8;                // two per TMEM lane quarter: one per half of the keys
constexpr int kVWarp = 10;
constexpr int kPvWarp = 11;
constexpr uint32_t kTmemCols = 512;          // S buffers at columns 0, 128 and 256, O at 384
constexpr uint32_t kOCol = kSBufs * kBK;
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
// D[tmem] (+)= A[tmem] x B[smem]^T: the A operand (128 rows x 16 bf16, two per
// 32-bit column, lane = row) read from tensor memory.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void tmem_st32_u(uint32_t taddr, const uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
        "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]),
        "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]),
        "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint4 v) {
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr)
                 : "memory");
    return v;
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
// 32 columns without waiting: the registers are valid only after tmem_wait_dep on them.
__device__ __forceinline__ void tmem_ld32_async(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
}
// Waits for this thread's outstanding tcgen05.ld; naming the registers as
// operands keeps every later use of them after the wait.
__device__ __forceinline__ void tmem_wait_dep(uint32_t (&r)[32]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                   "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                   "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                   "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                   "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
                 :
                 : "memory");
}

// Packed fp32 pairs (one instruction for two lanes of work).
typedef unsigned long long f2;
__device__ __forceinline__ f2 pack2(float lo, float hi) {
    f2 r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void unpack2(f2 v, float &lo, float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ f2 fma2(f2 a, f2 b, f2 c) {
    f2 r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ f2 add2(f2 a, f2 b) {
    f2 r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
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

// The CTA's items w = blockIdx.x + n * gridDim.x, walked in order: (bh, index
// within bh) moves on by the grid's quotient and remainder, so the walk needs
// no division per item (one at the start).
struct ItemWalk {
    int per_bh, step_bh, step_t;  // items per (batch, head); gridDim.x = step_bh * per_bh + step_t
    int bh, t;                    // the current item
    float inv_qtb;                // 1 / query tiles per branch
};

__device__ __forceinline__ ItemWalk item_walk(const AttnArgs &a) {
    ItemWalk wk;
    wk.per_bh = a.q_tiles_ctx + a.n_branch * a.q_tiles_branch;
    wk.bh = static_cast<int>(blockIdx.x) / wk.per_bh;
    wk.t = static_cast<int>(blockIdx.x) - wk.bh * wk.per_bh;
    wk.step_bh = static_cast<int>(gridDim.x) / wk.per_bh;
    wk.step_t = static_cast<int>(gridDim.x) - wk.step_bh * wk.per_bh;
    wk.inv_qtb = 1.f / static_cast<float>(a.q_tiles_branch);
    return wk;
}

__device__ __forceinline__ void item_next(ItemWalk &wk) {
    wk.t += wk.step_t;
    wk.bh += wk.step_bh;
    if (wk.t >= wk.per_bh) {
        wk.t -= wk.per_bh;
        ++wk.bh;
    }
}

// item_of for the walk's current item; the branch index is the float quotient
// moved to the exact floor (it is off by at most one for these sizes; the
// loops make the result exact regardless)
__device__ __forceinline__ Item item_at(const AttnArgs &a, const ItemWalk &wk) {
    Item it;
    it.bh = wk.bh;
    int t = wk.t;
    if (t < a.q_tiles_ctx) {
        it.seg_b = 0;
        it.q_start = t * kBQ;
        it.q_len = min(kBQ, a.n_context - it.q_start);
    } else {
        t -= a.q_tiles_ctx;
        int b = __float2int_rz(static_cast<float>(t) * wk.inv_qtb);
        while (b > 0 && b * a.q_tiles_branch > t) --b;
        while ((b + 1) * a.q_tiles_branch <= t) ++b;
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

// Moves (item n, key tile j) of the CTA's key-tile sequence one tile on:
// the loops walk the sequence in order, with no division per tile.
__device__ __forceinline__ void next_tile(int &n, int &j, int T) {
    if (++j == T) {
        j = 0;
        ++n;
    }
}

struct Ctl {
    uint64_t q_full[kQBufs], q_empty[kQBufs], k_full[kKvStages], k_empty[kKvStages], v_full[kKvStages],
        v_empty[kKvStages];
    // s_full and p_full per S / P buffer: the softmax may arrive on P up to three
    // tiles ahead of the MMA's wait (P of tile u needs S of tile u, issued after
    // the MMA saw P of tile u - 3), one phase ahead on each of three barriers
    uint64_t s_full[kSBufs], p_full[kSBufs], pv_done[kSBufs], o_ready, o_free, mma_done;
    // the two halves of a row trade their tile maxima and, at the end of an
    // item, their sums: (stamp << 32 | value bits), double-buffered by parity
    uint64_t xmax[2][2][kBQ], xsum[2][2][kBQ];  // [parity][half][row]
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

// Waits (warp-wide) until the P V product of global key tile x has completed.
// Product x completes phase x / 3 of pv_done[x % 3] (one phase per product
// that reads P from S buffer x % 3). The softmax waits for it at tile x + 1,
// before a rescale of O: S of tile x + 1 was issued only after product x - 2
// had completed, and product x + 3 needs P that this softmax has not made, so
// the barrier is at phase x / 3 (pending) or x / 3 + 1 (done), which its
// parity tells apart.
__device__ __forceinline__ bool wait_pv(uint32_t x, Ctl &c, const AttnArgs &a) {
    return warp_wait_or_abort(&c.pv_done[x % kSBufs], (x / kSBufs) & 1, c, a);
}

// Publishes this half-row's value for the partner half (stamp != 0).
__device__ __forceinline__ void xput(uint64_t *slot, uint32_t stamp, float v) {
    const uint64_t x = (static_cast<uint64_t>(stamp) << 32) | __float_as_uint(v);
    asm volatile("st.volatile.shared.u64 [%0], %1;" ::"r"(saddr(slot)), "l"(x) : "memory");
}

// The partner half's value with `stamp`, bounded like every other wait; the
// warp leaves together (false: the CTA aborts).
__device__ bool xget(uint64_t *slot, uint32_t stamp, float &v, Ctl &c, const AttnArgs &a) {
    uint64_t x = 0;
    bool ok = false;
    const uint64_t start = global_ns();
    for (uint32_t n = 0;; ++n) {
        asm volatile("ld.volatile.shared.u64 %0, [%1];" : "=l"(x) : "r"(saddr(slot)) : "memory");
        if (static_cast<uint32_t>(x >> 32) == stamp) {
            ok = true;
            break;
        }
        if (*reinterpret_cast<volatile int *>(&c.abort_flag)) break;
        if ((n & 63) == 63 && (a.wait_ns == 0 || global_ns() - start > a.wait_ns)) {
            flag_error(a.err, RPS_DEVERR_TIMEOUT);
            *reinterpret_cast<volatile int *>(&c.abort_flag) = 1;
            break;
        }
    }
    v = __uint_as_float(static_cast<uint32_t>(x));
    return __all_sync(kFull, ok);
}

// O / l of this thread's half-row of item n (64 of the 128 columns), bf16, to
// global memory, once the item's last product is done (o_ready, one phase per
// item); then O is released to the MMA (o_free). The row sum is the two
// halves' sums added in a fixed order.
__device__ bool read_out(const Item &it, int n, float l_half, uint32_t tmem, uint32_t lane_off, int r, int h, int lane,
                         uint32_t stage, Ctl &c, const AttnArgs &a) {
    if (!warp_wait_or_abort(&c.o_ready, n & 1, c, a)) return false;
    tc_fence_after();
    const uint32_t stamp = static_cast<uint32_t>(n) + 1u;
    xput(&c.xsum[n & 1][h][r], stamp, l_half);
    float other;
    if (!xget(&c.xsum[n & 1][h ^ 1][r], stamp, other, c, a)) return false;
    const float l = h == 0 ? l_half + other : other + l_half;
    const float inv = 1.f / l;
    uint32_t o[2][32];
#pragma unroll
    for (int ch = 0; ch < 2; ++ch) tmem_ld32_async(tmem + lane_off + kOCol + h * 64 + ch * 32, o[ch]);
#pragma unroll
    for (int ch = 0; ch < 2; ++ch) tmem_wait_dep(o[ch]);
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&c.o_free);  // O may take the next item
    // The warp's 32 rows go out through its shared-memory stage, 32 columns at
    // a time: written a row per thread, read back so that each store
    // instruction covers 64 contiguous bytes of 8 rows (a row per thread would
    // touch 32 lines per instruction). The 16-byte chunk index is XORed with
    // bits 1-2 of the row, so that neither the writes nor the reads put two
    // threads of a quarter-warp in one bank group.
    const int row0 = r - lane;  // first row of the warp's lane quarter
    __nv_bfloat16 *dst = a.out + (static_cast<int64_t>(it.bh) * a.n_tokens + it.q_start + row0) * kD + h * 64;
#pragma unroll
    for (int ch = 0; ch < 2; ++ch) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const uint32_t *x = o[ch] + 8 * u;
            st_shared_v4(stage + lane * 64 + ((u ^ ((lane >> 1) & 3)) << 4),
                         make_uint4(pack_bf16(__uint_as_float(x[0]) * inv, __uint_as_float(x[1]) * inv),
                                    pack_bf16(__uint_as_float(x[2]) * inv, __uint_as_float(x[3]) * inv),
                                    pack_bf16(__uint_as_float(x[4]) * inv, __uint_as_float(x[5]) * inv),
                                    pack_bf16(__uint_as_float(x[6]) * inv, __uint_as_float(x[7]) * inv)));
        }
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int rr = i * 8 + (lane >> 2), cc = lane & 3;
            const uint4 v = ld_shared_v4(stage + rr * 64 + ((cc ^ ((rr >> 1) & 3)) << 4));
            if (row0 + rr < it.q_len)
                *reinterpret_cast<uint4 *>(dst + static_cast<int64_t>(rr) * kD + ch * 32 + cc * 8) = v;
        }
        __syncwarp();  // the stage is rewritten next
    }
    return true;
}

__global__ void __launch_bounds__(kThreads, 1)
    packed_attention_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                            const __grid_constant__ CUtensorMap tm_vt, const AttnArgs a) {
    extern __shared__ uint8_t dyn_smem[];
    __shared__ Ctl c;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t *base = dyn_smem + ((1024u - (saddr(dyn_smem) & 1023u)) & 1023u);
    uint8_t *sq = base;                          // Q buffers
    uint8_t *sk = sq + kQBufs * kQBytes;         // K stages
    uint8_t *sv = sk + kKvStages * kKBytes;      // V^T stages
    uint8_t *so = sv + kKvStages * kVBytes;      // output stages of the softmax warps
    // Every item has the same number of key tiles (the context's and one
    // branch's), so the CTA's key tiles are numbered globally: tile t is tile
    // t % T of the CTA's item t / T.
    const int T = a.q_tiles_ctx + a.q_tiles_branch;
    const int my_items = blockIdx.x < static_cast<unsigned>(a.items)
                             ? (a.items - 1 - static_cast<int>(blockIdx.x)) / static_cast<int>(gridDim.x) + 1
                             : 0;
    const uint32_t tiles = static_cast<uint32_t>(my_items) * T;

    if (threadIdx.x == 0) {
        for (int b = 0; b < kQBufs; ++b) {
            mbar_init(&c.q_full[b], 1);
            mbar_init(&c.q_empty[b], 1);
        }
        for (int s = 0; s < kKvStages; ++s) {
            mbar_init(&c.k_full[s], 1);
            mbar_init(&c.k_empty[s], 1);
            mbar_init(&c.v_full[s], 1);
            mbar_init(&c.v_empty[s], 1);
        }
        for (int b = 0; b < kSBufs; ++b) {
            mbar_init(&c.s_full[b], 1);
            mbar_init(&c.p_full[b], kSoftWarps);
        }
        for (int b = 0; b < kSBufs; ++b) mbar_init(&c.pv_done[b], 1);
        mbar_init(&c.o_ready, 1);
        mbar_init(&c.o_free, kSoftWarps);
        mbar_init(&c.mma_done, 2);  // one commit from each MMA issuer
        c.abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    for (int i = threadIdx.x; i < 2 * 2 * kBQ; i += kThreads) {  // stamp 0: nothing published
        (&c.xmax[0][0][0])[i] = 0;
        (&c.xsum[0][0][0])[i] = 0;
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
        if (lane == 0) {  // -------------------------------------------- Q and K producer
            uint32_t t = 0;  // key tiles issued
            int n_q = 0;     // Q tiles issued
            bool ok = true;
            Item it{};
            ItemWalk wk = item_walk(a);
            for (int n = 0, j = 0; t < tiles && ok; ++t, next_tile(n, j, T)) {
                if (j == 0) {  // this item's Q, into buffer n % 2 once item n - 2 has left it
                    if (n > 0) item_next(wk);
                    it = item_at(a, wk);
                    const int b = n & 1;
                    if (!wait_or_abort(&c.q_empty[b], ((n >> 1) & 1) ^ 1, c, a)) break;
                    mbar_expect_tx(&c.q_full[b], kQBytes);
                    const int qrow = it.bh * a.n_tokens + it.q_start;
                    tma_load_2d(sq + b * kQBytes, &tm_q, 0, qrow, &c.q_full[b]);
                    tma_load_2d(sq + b * kQBytes + kAtom, &tm_q, 64, qrow, &c.q_full[b]);
                    ++n_q;
                }
                const int s = t % kKvStages;
                if (!wait_or_abort(&c.k_empty[s], ((t / kKvStages) & 1) ^ 1, c, a)) {
                    ok = false;
                    break;
                }
                int k0, valid;
                key_tile(a, it, j, k0, valid);
                uint8_t *dst = sk + s * kKBytes;
                mbar_expect_tx(&c.k_full[s], kKBytes);
                const int krow = it.bh * a.n_tokens + k0;
                tma_load_2d(dst, &tm_k, 0, krow, &c.k_full[s]);
                tma_load_2d(dst + kAtom, &tm_k, 64, krow, &c.k_full[s]);
            }
            // every copy issued lands before the CTA leaves
            for (uint32_t x = t > kKvStages ? t - kKvStages : 0; x < t; ++x)
                wait_drain(&c.k_full[x % kKvStages], (x / kKvStages) & 1);
            for (int n = n_q > kQBufs ? n_q - kQBufs : 0; n < n_q; ++n) wait_drain(&c.q_full[n & 1], (n >> 1) & 1);
        }
    } else if (warp == kVWarp) {
        if (lane == 0) {  // -------------------------------------------- V producer
            uint32_t t = 0;
            Item it{};
            ItemWalk wk = item_walk(a);
            for (int n = 0, j = 0; t < tiles; ++t, next_tile(n, j, T)) {
                if (j == 0) {
                    if (n > 0) item_next(wk);
                    it = item_at(a, wk);
                }
                const int s = t % kKvStages;
                if (!wait_or_abort(&c.v_empty[s], ((t / kKvStages) & 1) ^ 1, c, a)) break;
                int k0, valid;
                key_tile(a, it, j, k0, valid);
                uint8_t *dst = sv + s * kVBytes;
                mbar_expect_tx(&c.v_full[s], kVBytes);
                tma_load_2d(dst, &tm_vt, k0, it.bh * kD, &c.v_full[s]);
                tma_load_2d(dst + kAtom, &tm_vt, k0 + 64, it.bh * kD, &c.v_full[s]);
            }
            for (uint32_t x = t > kKvStages ? t - kKvStages : 0; x < t; ++x)
                wait_drain(&c.v_full[x % kKvStages], (x / kKvStages) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {  // -------------------------------------------- S issuer
            bool ok = true;
            int n = 0, j = 0;
            for (uint32_t t = 0; t < tiles && ok; ++t, next_tile(n, j, T)) {  // S_t = Q K_t^T into buffer t % 3
                const int qb = n & 1, s = t % kKvStages;
                // the buffer holds P of tile t - 3 until that product has completed
                // (it comes from the other issuer: issue order does not protect it)
                if ((j == 0 && !wait_or_abort(&c.q_full[qb], (n >> 1) & 1, c, a)) ||
                    (t >= kSBufs && !wait_or_abort(&c.pv_done[t % kSBufs], ((t - kSBufs) / kSBufs) & 1, c, a)) ||
                    !wait_or_abort(&c.k_full[s], (t / kKvStages) & 1, c, a)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint64_t qd = umma::smem_desc_kmajor_sw128(saddr(sq + qb * kQBytes));
                const uint64_t qd1 = umma::smem_desc_kmajor_sw128(saddr(sq + qb * kQBytes + kAtom));
                const uint64_t kd = umma::smem_desc_kmajor_sw128(saddr(sk + s * kKBytes));
                const uint64_t kd1 = umma::smem_desc_kmajor_sw128(saddr(sk + s * kKBytes + kAtom));
                const uint32_t sbuf = tmem + (t % kSBufs) * kBK;
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16(sbuf, umma::advance_k16(k < 4 ? qd : qd1, k & 3), umma::advance_k16(k < 4 ? kd : kd1, k & 3),
                             idesc, k != 0);
                mma_commit(&c.k_empty[s]);  // K stage free once S is computed
                mma_commit(&c.s_full[t % kSBufs]);
                if (j == T - 1) mma_commit(&c.q_empty[qb]);  // this Q is no longer read
            }
            mma_commit(&c.mma_done);
            wait_drain(&c.mma_done, 0);
        }
        __syncwarp();
    } else if (warp == kPvWarp) {
        if (lane == 0) {  // -------------------------------------------- P V issuer
            bool ok = true;
            int n = 0, j = 0;
            for (uint32_t t = 0; t < tiles && ok; ++t, next_tile(n, j, T)) {  // O += P_t V_t
                // the first product of an item overwrites O: the previous item's read-out must be done
                if ((j == 0 && !wait_or_abort(&c.o_free, (n & 1) ^ 1, c, a)) ||
                    !wait_or_abort(&c.p_full[t % kSBufs], (t / kSBufs) & 1, c, a) ||
                    !wait_or_abort(&c.v_full[t % kKvStages], (t / kKvStages) & 1, c, a)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint8_t *vb = sv + (t % kKvStages) * kVBytes;
                const uint64_t vd = umma::smem_desc_kmajor_sw128(saddr(vb));
                const uint64_t vd1 = umma::smem_desc_kmajor_sw128(saddr(vb + kAtom));
                // P of keys 16k..16k+15: columns (k / 4) * 64 + (k % 4) * 8 of S buffer t % 3
                // (each half-row wrote its 64 keys, two per column, over its own first 32 columns)
                const uint32_t pcol = tmem + (t % kSBufs) * kBK;
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16_ts(tmem + kOCol, pcol + (k >> 2) * 64 + (k & 3) * 8,
                                umma::advance_k16(k < 4 ? vd : vd1, k & 3), idesc, (j > 0 || k != 0) ? 1u : 0u);
                mma_commit(&c.v_empty[t % kKvStages]);
                mma_commit(&c.pv_done[t % kSBufs]);
                if (j == T - 1) mma_commit(&c.o_ready);  // the item's O is complete
            }
            mma_commit(&c.mma_done);
            wait_drain(&c.mma_done, 0);
        }
        __syncwarp();
    } else {  // ---------------------------------------------------- softmax (warps 2-9)
        // warp w reads TMEM lane quarter w % 4 (rows 32 q .. 32 q + 31) and half
        // h of each S row (keys 64 h .. 64 h + 63); the two halves of a row
        // agree on its maximum through the exchange slots
        const int q = warp & 3, h = (warp - 2) >> 2;
        const int r = q * 32 + lane;  // query row in the tile (TMEM lane)
        const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
        const uint32_t stage = saddr(so + (warp - 2) * kStageBytes);
        float m = -INFINITY, l = 0.f;
        // The read-out of item n waits until the first P of item n + 1 is out:
        // by then its last product has had the softmax of a whole tile to finish.
        Item pend_it{};
        int pend_n = -1;
        float pend_l = 0.f;
        bool ok = true;
        Item it{};
        ItemWalk wk = item_walk(a);
        int n = 0, j = 0;
        for (uint32_t t = 0; t < tiles && ok; ++t, next_tile(n, j, T)) {
            if (j == 0) {
                if (n > 0) item_next(wk);
                it = item_at(a, wk);
                m = -INFINITY;
                l = 0.f;
            }
            const int sb = t % kSBufs;
            if (!warp_wait_or_abort(&c.s_full[sb], (t / kSBufs) & 1, c, a)) {
                ok = false;
                break;
            }
            tc_fence_after();
            int k0, valid;
            key_tile(a, it, j, k0, valid);
            const uint32_t sbuf = tmem + lane_off + sb * kBK + h * 64;
            // this half-row's 64 scores in one round of loads
            uint32_t sr[2][32];
#pragma unroll
            for (int ch = 0; ch < 2; ++ch) tmem_ld32_async(sbuf + ch * 32, sr[ch]);
#pragma unroll
            for (int ch = 0; ch < 2; ++ch) tmem_wait_dep(sr[ch]);
            if (valid < kBK) {  // keys past the segment's end take no weight
#pragma unroll
                for (int ch = 0; ch < 2; ++ch)
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (h * 64 + ch * 32 + i >= valid) sr[ch][i] = __float_as_uint(-INFINITY);
            }
            // the half's largest score (eight independent chains), then the row's
            float mx8[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) mx8[i] = -INFINITY;
#pragma unroll
            for (int ch = 0; ch < 2; ++ch)
#pragma unroll
                for (int i = 0; i < 32; ++i) mx8[i & 7] = fmaxf(mx8[i & 7], __uint_as_float(sr[ch][i]));
            const float hmx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                                    fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
            xput(&c.xmax[t & 1][h][r], t + 1, hmx);
            float omx;
            if (!xget(&c.xmax[t & 1][h ^ 1][r], t + 1, omx, c, a)) {
                ok = false;
                break;
            }
            const float tm = fmaxf(hmx, omx) * a.c;  // the same in both halves
            float f = 1.f;
            bool rescale = false;
            if (m == -INFINITY) {
                m = tm;
            } else if (tm > m + kRescale) {
                f = ex2(m - tm);
                m = tm;
                rescale = true;
            }
            // tcgen05.ld / st are warp-wide (.sync.aligned): the warp rescales
            // its half of O together when any of its rows needs it, the other
            // rows by f = 1, once the product of the previous tile is done
            if (__any_sync(kFull, rescale)) {
                if (!wait_pv(t - 1, c, a)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int ch = 0; ch < 2; ++ch) {
                    float o[32];
                    tmem_ld32(tmem + lane_off + kOCol + h * 64 + ch * 32, o);
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[i] *= f;
                    tmem_st32(tmem + lane_off + kOCol + h * 64 + ch * 32, o);
                }
            }
            l *= f;
            // P = 2^(s c - m) (a masked key gives 2^-inf = 0), bf16 pairs, over
            // the first 32 columns of this half's S (already in registers)
            const f2 cc = pack2(a.c, a.c), mm = pack2(-m, -m);
            f2 lsum[4] = {pack2(0.f, 0.f), pack2(0.f, 0.f), pack2(0.f, 0.f), pack2(0.f, 0.f)};
            uint32_t pk[32];
#pragma unroll
            for (int ch = 0; ch < 2; ++ch)
#pragma unroll
                for (int i = 0; i < 32; i += 2) {
                    const f2 u = fma2(pack2(__uint_as_float(sr[ch][i]), __uint_as_float(sr[ch][i + 1])), cc, mm);
                    float u0, u1;
                    unpack2(u, u0, u1);
                    const float p0 = ex2(u0), p1 = ex2(u1);
                    lsum[(i >> 1) & 3] = add2(lsum[(i >> 1) & 3], pack2(p0, p1));
                    pk[ch * 16 + i / 2] = pack_bf16(p0, p1);
                }
            tmem_st32_u(sbuf, pk);
            {
                float l0, l1;
                unpack2(add2(add2(lsum[0], lsum[1]), add2(lsum[2], lsum[3])), l0, l1);
                l += l0 + l1;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&c.p_full[sb]);
            if (j == 0 && pend_n >= 0) {
                if (!read_out(pend_it, pend_n, pend_l, tmem, lane_off, r, h, lane, stage, c, a)) {
                    ok = false;
                    break;
                }
                pend_n = -1;
            }
            if (j == T - 1) {
                pend_it = it;
                pend_n = n;
                pend_l = l;
            }
        }
        if (ok && pend_n >= 0) read_out(pend_it, pend_n, pend_l, tmem, lane_off, r, h, lane, stage, c, a);
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
