// rowstats.cu -- fused single-pass row statistics of logit rows (rps_score_step).
//
// For every listed row z (V logits) one pass over HBM yields
//   zmax, argmax (Eq. 1), lse, H = -sum p log p, P^max (Sec. 2 notation) and,
//   in top-k mode, T_i, mu_i and the truncated entropy of Eq. 3.
//
// Work split. One block of kStatThreads per SM; each warp streams one piece. With
// at least as many warps as rows, each row is cut into equal pieces, so that no
// piece crosses a row boundary; otherwise the rows' 16-byte units are laid end
// to end and cut into equal contiguous pieces (a piece covers the tail of one
// row, whole rows and the head of another). Either way every warp streams about
// the same number of bytes. Each (warp, row) pair leaves a partial record in the
// workspace and the last warp to finish a row (atomic ticket, no waiting) merges
// the at most kMaxPartials records and writes the row.
//
// Data movement. Each warp owns a ring of shared-memory buffers of 2 KB.
// Lane 0 keeps every free buffer filled by a bulk asynchronous copy (cp.async.bulk, completion
// counted on an mbarrier per buffer) in flight ahead of the warp, across row
// boundaries; the lanes read their four 16-byte units of each buffer from shared
// memory. Bytes in flight therefore cost no registers. Every mbarrier wait is
// bounded: on expiry the warp flags RPS_DEVERR_TIMEOUT, waits (bounded) for its
// own copies and stops.
//
// Per lane, a row segment is reduced as a base-2 online softmax against an
// exponent reference B (in base-2 units) that is raised only when a value exceeds
// it by more than kSlack nats (rare):
//   u = fma(z, log2(e), -B)  (the product is exact inside the fma),
//   s = sum 2^u, t = sum u 2^u,
//   H = ln S - ln2 * T / S,  lse = ln2 * B + ln S   (after merging lanes / pieces)
// and P^max, mu and the truncated entropy take their exponents the same way, so
// a rounding of B is a common factor of numerator and denominator.
// The exact maximum is tracked per unit; its token index is resolved once per
// segment by re-reading the unit that holds it (in top-k mode it is rank 0 of
// the top-k list instead).
//
// Top-k mode (k <= 32) is two launches. This one also records, per row, the
// maximum of every cell -- one lane's four units of one ring chunk, 64 bytes of
// logits 512 bytes apart -- densely in the workspace (the sketch), and the row's
// B, ln S and 1 / S. topk_rows_kernel then takes one warp per row slot: the k-th
// largest of its lanes' largest sketch entries bounds the row's k-th largest
// logit from below (k lanes each saw a different cell holding an element at
// least that large), so only the few cells that reach it are read again and
// their elements at or above it merged into a warp-distributed sorted list.
//
// -inf logits or NaN make the first pass's sums NaN; the segment is then rescanned
// from global memory with clamped exponents (SAFE), which scores -inf as
// probability 0 and flags NaN input as RPS_DEVERR_NONFINITE.
#include <cfloat>
#include <climits>

#include "rps_internal.cuh"

namespace rps {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kSlack = 8.0f;          // nats the reference may trail the maximum
constexpr int kChunkUnits = 32 * kBatch;  // 16-byte units per ring buffer (2 KB)
constexpr int kCandBatch = 32;  // top-k candidates merged at a time
constexpr uint64_t kWaitLimitNs = 200ull * 1000 * 1000;  // a bulk copy normally lands within microseconds
constexpr uint32_t kUnhealthy = 1u;  // health word of a workspace a launch gave up on

// ---------------------------------------------------------------- PTX helpers
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Packed fp32 pairs (sm_100+ f32x2 arithmetic): one instruction per two lanes of work.
typedef unsigned long long f2;

__device__ __forceinline__ f2 pack2(float lo, float hi) {
    f2 r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void unpack2(f2 v, float &lo, float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ f2 mul2(f2 a, f2 b) {
    f2 r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ f2 add2(f2 a, f2 b) {
    f2 r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ f2 fma2(f2 a, f2 b, f2 c) {
    f2 r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}

// Streaming 16-byte load: read once, do not keep in L1.
__device__ __forceinline__ uint4 ld_stream(const void *p) {
    uint4 v;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
        : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
        : "l"(p));
    return v;
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Shared-memory 16-byte load the compiler may not merge with an earlier one (a
// second read of a ring unit costs less than keeping the first in registers).
__device__ __forceinline__ uint4 lds_again(const uint4 *p) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(smem_u32(p)));
    return v;
}

// 16-byte asynchronous global -> shared copy (L2 only), and the wait for all of
// this thread's outstanding ones.
__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }

// Orders this thread's earlier shared-memory accesses before later async-proxy writes.
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Arm `bar` for `bytes` and start a bulk copy of them from global memory into `dst`.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Waits for phase `parity` of `bar`, giving up after limit_ns (at once when 0).
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity, uint64_t limit_ns = kWaitLimitNs) {
    if (limit_ns == 0) return false;
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t start = global_ns();
    while (global_ns() - start < limit_ns)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}

__device__ __forceinline__ uint32_t bf16x2_max(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// ---------------------------------------------------------------- element types
template <int DT>
struct Elem;

template <>
struct Elem<RPS_BF16> {
    static constexpr int N = 8;
    static constexpr int kBytes = 2;
    __device__ static __forceinline__ void unpack(const uint4 &w, float (&y)[8]) {
        y[0] = __uint_as_float(w.x << 16);
        y[1] = __uint_as_float(w.x & 0xffff0000u);
        y[2] = __uint_as_float(w.y << 16);
        y[3] = __uint_as_float(w.y & 0xffff0000u);
        y[4] = __uint_as_float(w.z << 16);
        y[5] = __uint_as_float(w.z & 0xffff0000u);
        y[6] = __uint_as_float(w.w << 16);
        y[7] = __uint_as_float(w.w & 0xffff0000u);
    }
    __device__ static __forceinline__ float unit_max(const uint4 &w) {
        const uint32_t m = bf16x2_max(bf16x2_max(w.x, w.y), bf16x2_max(w.z, w.w));
        return fmaxf(__uint_as_float(m << 16), __uint_as_float(m & 0xffff0000u));
    }
    // per-(chunk, lane) maximum kept for the top-k second pass: the bf16 bits
    typedef uint16_t Sketch;
    static constexpr uint32_t kNegInf2 = 0xff80ff80u;  // a 32-bit word of -inf sketch entries
    __device__ static __forceinline__ Sketch to_sketch(float v) { return static_cast<uint16_t>(__float_as_uint(v) >> 16); }
    // running maximum of whole units, kept as a packed bf16 pair
    typedef uint32_t Acc;
    __device__ static __forceinline__ Acc acc_init() { return 0xff80ff80u; }  // (-inf, -inf)
    __device__ static __forceinline__ Acc acc_add(Acc m, const uint4 &w) {
        return bf16x2_max(bf16x2_max(m, w.x), bf16x2_max(bf16x2_max(w.y, w.z), w.w));
    }
    __device__ static __forceinline__ float acc_value(Acc m) {
        return fmaxf(__uint_as_float(m << 16), __uint_as_float(m & 0xffff0000u));
    }
    __device__ static __forceinline__ float load1(const char *row, int64_t e) {
        return __uint_as_float(static_cast<uint32_t>(reinterpret_cast<const uint16_t *>(row)[e]) << 16);
    }
    // element i of a staged unit held as four 32-bit words
    __device__ static __forceinline__ float pick(const uint32_t *words, int i) {
        uint32_t w = words[i >> 1];
        return __uint_as_float((i & 1) ? (w & 0xffff0000u) : (w << 16));
    }
};

template <>
struct Elem<RPS_F32> {
    static constexpr int N = 4;
    static constexpr int kBytes = 4;
    __device__ static __forceinline__ void unpack(const uint4 &w, float (&y)[4]) {
        y[0] = __uint_as_float(w.x);
        y[1] = __uint_as_float(w.y);
        y[2] = __uint_as_float(w.z);
        y[3] = __uint_as_float(w.w);
    }
    __device__ static __forceinline__ float unit_max(const uint4 &w) {
        return fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)), fmaxf(__uint_as_float(w.z), __uint_as_float(w.w)));
    }
    typedef float Sketch;
    static constexpr uint32_t kNegInf2 = 0xff800000u;
    __device__ static __forceinline__ Sketch to_sketch(float v) { return v; }
    typedef float Acc;
    __device__ static __forceinline__ Acc acc_init() { return -INFINITY; }
    __device__ static __forceinline__ Acc acc_add(Acc m, const uint4 &w) { return fmaxf(m, unit_max(w)); }
    __device__ static __forceinline__ float acc_value(Acc m) { return m; }
    __device__ static __forceinline__ float load1(const char *row, int64_t e) {
        return reinterpret_cast<const float *>(row)[e];
    }
    __device__ static __forceinline__ float pick(const uint32_t *words, int i) { return __uint_as_float(words[i]); }
};

// True when this lane holds at least one unit of a chunk of n_units units.
__device__ __forceinline__ bool j0_valid(int n_units, int lane) { return lane < n_units; }

// ---------------------------------------------------------------- online softmax
struct LaneState {
    float mref;       // exponent reference B (base-2 units), -inf until the first finite value
    f2 s, t;          // pairwise partial sums of 2^u and u 2^u, u = fma(z, log2(e), -B)
    float mx;         // exact running maximum
    int best;         // unit (or first unit of the ring chunk) where mx was first reached, -1 if none
    bool best_chunk;  // best names a ring chunk: this lane's units best + 32 j, j < kBatch
    bool bad;         // NaN input seen (SAFE scan only)
};

__device__ __forceinline__ void lane_init(LaneState &L) {
    L.mref = -INFINITY;
    L.s = pack2(0.f, 0.f);
    L.t = pack2(0.f, 0.f);
    L.mx = -INFINITY;
    L.best = -1;
    L.best_chunk = false;
    L.bad = false;
}

// Raise the exponent reference to m log2(e) (rare: only when m exceeds it by kSlack nats).
__device__ __forceinline__ void raise_reference(LaneState &L, float m) {
    const float mb = m * kLog2e;
    if (mb > L.mref + kSlack * kLog2e) {
        float slo, shi;
        unpack2(L.s, slo, shi);
        if (slo + shi > 0.f) {
            const float d = L.mref - mb;
            const float a = ex2(d);
            const f2 a2 = pack2(a, a);
            L.t = mul2(a2, fma2(pack2(d, d), L.s, L.t));
            L.s = mul2(a2, L.s);
        }
        L.mref = mb;
    }
}

// Sums of n values (n even or the last value alone). The exponent is one fma,
// z log2(e) - B, rounded once: large logits lose no absolute precision.
template <int N, bool SAFE>
__device__ __forceinline__ void accumulate(LaneState &L, const float (&y)[N], int n) {
    const f2 m2 = pack2(-L.mref, -L.mref);
    const f2 l2 = pack2(kLog2e, kLog2e);
#pragma unroll
    for (int i = 0; i < N; i += 2) {
        const bool v0 = i < n, v1 = i + 1 < n;
        if (!v0) break;
        const f2 u2 = fma2(pack2(y[i], v1 ? y[i + 1] : y[i]), l2, m2);
        float u0, u1;
        unpack2(u2, u0, u1);
        if (SAFE) {
            L.bad |= (y[i] != y[i]) || (v1 && y[i + 1] != y[i + 1]);
            u0 = fmaxf(u0, -1000.f);
            u1 = fmaxf(u1, -1000.f);
        }
        const float e0v = ex2(u0);
        const float e1v = v1 ? ex2(u1) : 0.f;
        const f2 e2 = pack2(e0v, e1v);
        const f2 uu = SAFE ? pack2(u0, u1) : u2;
        L.s = add2(L.s, e2);
        L.t = fma2(uu, e2, L.t);
    }
}

// Fold one unit of n valid values (n == N except for a ragged row tail).
template <int N, bool SAFE>
__device__ __forceinline__ void fold_unit(LaneState &L, const float (&y)[N], int n, int unit) {
    float vmax = -INFINITY;
#pragma unroll
    for (int i = 0; i < N; ++i)
        if (i < n) vmax = fmaxf(vmax, y[i]);
    if (vmax > L.mx) {
        L.mx = vmax;
        L.best = unit;
        L.best_chunk = false;
    }
    raise_reference(L, vmax);
    accumulate<N, SAFE>(L, y, n);
}

// Fold this lane's units of one ring chunk (the fast path). The chunk's maximum
// comes from packed compares; the exact argmax is resolved once per segment.
// SKETCH: every lane records its maximum (-inf without units) at key + lane.
template <int DT, bool SKETCH>
__device__ __forceinline__ float fold_chunk(LaneState &L, typename Elem<DT>::Sketch *sketch, const uint4 *buf,
                                            int n_units, int cu, int key, int lane) {
    using E = Elem<DT>;
    constexpr int N = E::N;
    typename E::Acc acc = E::acc_init();
#pragma unroll
    for (int j = 0; j < kBatch; ++j)
        if (j * 32 + lane < n_units) acc = E::acc_add(acc, buf[j * 32 + lane]);
    const float cmax = j0_valid(n_units, lane) ? E::acc_value(acc) : -INFINITY;
    if (cmax > L.mx) {
        L.mx = cmax;
        L.best = cu;
        L.best_chunk = true;
    }
    raise_reference(L, cmax);
    if (SKETCH) sketch[key + lane] = E::to_sketch(cmax);
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
        if (j * 32 + lane < n_units) {
            float y[N];
            E::unpack(lds_again(buf + j * 32 + lane), y);
            accumulate<N, false>(L, y, N);
        }
    }
    return cmax;
}

// The ragged last unit of a row (fewer than N values), folded by lane 0.
template <int DT, bool SAFE>
__device__ __forceinline__ void fold_tail(LaneState &L, const char *row, int V, int lane) {
    using E = Elem<DT>;
    constexpr int N = E::N;
    const int e0 = (V / N) * N;
    const int n = V - e0;
    if (lane != 0 || n == 0) return;
    float y[N];
#pragma unroll
    for (int i = 0; i < N; ++i) y[i] = i < n ? E::load1(row, e0 + i) : -INFINITY;
    fold_unit<N, SAFE>(L, y, n, V / N);
}

// Rescan of a segment straight from global memory with clamped exponents; used
// when the fast pass saw -inf or NaN.
template <int DT>
__device__ void rescan_safe(LaneState &L, const char *row, int V, int u0, int u1, int lane) {
    using E = Elem<DT>;
    constexpr int N = E::N;
    lane_init(L);
    const int full_end = min(u1, V / N);
    for (int u = u0 + lane; u < full_end; u += 32) {
        float y[N];
        E::unpack(ld_stream(row + static_cast<size_t>(u) * 16), y);
        fold_unit<N, true>(L, y, N, u);
    }
    if (u1 > V / N) fold_tail<DT, true>(L, row, V, lane);
}

// ---------------------------------------------------------------- top-k
// True when (av, ai) ranks before (bv, bi): larger logit, then lower token id.
__device__ __forceinline__ bool ranks_before(float av, int ai, float bv, int bi) {
    return av > bv || (av == bv && ai < bi);
}

// Insert a warp-uniform candidate into the warp's sorted list (lane j = rank j).
__device__ __forceinline__ void topk_insert(float &tv, int &ti, float cv, int ci, int k, int lane) {
    const unsigned keep = (k >= 32) ? kFull : ((1u << k) - 1u);
    const int pos = __popc(__ballot_sync(kFull, ranks_before(tv, ti, cv, ci)) & keep);
    if (pos >= k) return;
    const float uv = __shfl_up_sync(kFull, tv, 1);
    const int ui = __shfl_up_sync(kFull, ti, 1);
    if (lane == pos) {
        tv = cv;
        ti = ci;
    } else if (lane > pos) {
        tv = uv;
        ti = ui;
    }
}

// k-th largest of the 32 lane values (bitonic sort, descending), 1 <= k <= 32.
__device__ __forceinline__ float warp_kth_largest(float x, int k, int lane) {
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const float o = __shfl_xor_sync(kFull, x, stride);
            const bool keep_max = ((lane & size) == 0) == ((lane & stride) == 0);
            x = keep_max ? fmaxf(x, o) : fminf(x, o);
        }
    }
    return __shfl_sync(kFull, x, k - 1);
}

// Merges one candidate per lane (sentinel -inf / INT_MAX for none) into the
// warp-distributed sorted list: bitonic sort of the 32 candidates in rank order,
// then the element-wise better of the list and the reversed candidates (the 32
// best of both, as a bitonic sequence), then a bitonic merge. Fixed cost,
// independent of how many candidates are real.
__device__ __forceinline__ void pair_step(float &v, int &i, int stride, bool keep_better) {
    const float ov = __shfl_xor_sync(kFull, v, stride);
    const int oi = __shfl_xor_sync(kFull, i, stride);
    if (keep_better == ranks_before(ov, oi, v, i)) {
        v = ov;
        i = oi;
    }
}

// The list holds nothing yet: each real candidate's rank among the 32 is the
// count of candidates before it (candidates are distinct, so ranks are); ranks
// below k go to buf[rank] (kCandBatch entries), then lane j takes rank j.
// Independent shuffles instead of a sorting network's dependent stages.
__device__ __forceinline__ void warp_rank_into_list(float &tv, int &ti, float cv, int ci, int k, int lane,
                                                    float2 *buf) {
    const bool real = ci != INT_MAX;
    int rank = 0;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        const float ov = __shfl_sync(kFull, cv, j);
        const int oi = __shfl_sync(kFull, ci, j);
        rank += ranks_before(ov, oi, cv, ci);
    }
    const int n = __popc(__ballot_sync(kFull, real));
    __syncwarp();
    if (real && rank < k) buf[rank] = make_float2(cv, __int_as_float(ci));
    __syncwarp();
    const float2 e = lane < k && lane < n ? buf[lane] : make_float2(-INFINITY, __int_as_float(INT_MAX));
    tv = e.x;
    ti = __float_as_int(e.y);
    __syncwarp();
}

__device__ __forceinline__ void warp_merge_batch(float &tv, int &ti, float cv, int ci, int k, int lane) {
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1)
            pair_step(cv, ci, stride, ((lane & size) == 0) == ((lane & stride) == 0));
    }
    const float rv = __shfl_sync(kFull, cv, 31 - lane);
    const int ri = __shfl_sync(kFull, ci, 31 - lane);
    if (ranks_before(rv, ri, tv, ti)) {
        tv = rv;
        ti = ri;
    }
#pragma unroll
    for (int stride = 16; stride > 0; stride >>= 1) pair_step(tv, ti, stride, (lane & stride) == 0);
    if (lane >= k) {
        tv = -INFINITY;
        ti = INT_MAX;
    }
}

// Candidates of a row's ragged last unit (top-k mode).
template <int DT>
__device__ __forceinline__ void topk_tail(const char *row, int V, int k, int lane, float &tv, int &ti) {
    using E = Elem<DT>;
    constexpr int N = E::N;
    const int e0 = (V / N) * N;
    const int n = V - e0;
#pragma unroll
    for (int i = 0; i < N; ++i) {
        const float cv = i < n ? E::load1(row, e0 + i) : -INFINITY;
        const float th = __shfl_sync(kFull, tv, k - 1);
        if (i < n && cv >= th) topk_insert(tv, ti, cv, e0 + i, k, lane);
    }
}

// ---------------------------------------------------------------- row records
// Lowest token index holding value MX among the units this lane recorded as best
// (INT_MAX if none).
template <int DT>
__device__ __forceinline__ int resolve_argmax(const char *row, int V, const LaneState &L, float MX, int lane) {
    using E = Elem<DT>;
    constexpr int N = E::N;
    if (L.best < 0 || !(L.mx == MX)) return INT_MAX;
    const int full_units = V / N;
    const int n_units = L.best_chunk ? kBatch : 1;
    for (int j = 0; j < n_units; ++j) {
        const int u = L.best_chunk ? L.best + j * 32 + lane : L.best;
        const int e0 = u * N;
        const int n = u < full_units ? N : V - e0;
        if (n <= 0) break;
        float y[N];
        if (n == N) {
            E::unpack(ld_stream(row + static_cast<size_t>(e0) * E::kBytes), y);
        } else {
#pragma unroll
            for (int i = 0; i < N; ++i) y[i] = i < n ? E::load1(row, e0 + i) : -INFINITY;
        }
#pragma unroll
        for (int i = 0; i < N; ++i)
            if (i < n && y[i] == MX) return e0 + i;
    }
    return INT_MAX;
}

struct RowTotals {
    float M, S, T, MX;
    int AM;
};

// Combine per-lane (or per-piece) records into one: max reference, rescaled sums.
__device__ __forceinline__ RowTotals combine(float mref, float s, float t, float mx, int am) {
    RowTotals r;
    const bool live = s > 0.f;
    r.M = warp_max(live ? mref : -INFINITY);
    float a = 0.f, d = 0.f;
    if (live) {
        d = mref - r.M;
        a = ex2(d);
    }
    // a NaN s (bad input) must survive the merge
    r.S = warp_sum(live ? a * s : (s != s ? s : 0.f));
    r.T = warp_sum(live ? a * fmaf(d, s, t) : 0.f);
    r.MX = warp_max(mx);
    r.AM = warp_min_int(mx == r.MX ? am : INT_MAX);
    return r;
}

// mu (Eq. 3) and the truncated entropy of the warp's list (lane j = rank j)
// against the row's reference B and sum S: p_v = 2^fma(z_v, log2(e), -B) / S.
__device__ __forceinline__ void topk_mass(float tv, float M, float lnS, float invS, int k, int lane, float &mu,
                                          float &ht) {
    float p = 0.f, h = 0.f;
    if (lane < k) {
        const float u = fmaf(tv, kLog2e, -M);
        p = ex2(u) * invS;
        if (p > 0.f) h = -p * (u * kLn2 - lnS);
    }
    mu = warp_sum(p);
    ht = warp_sum(h);
}

// SKETCH: the row's B, ln S, 1 / S and sketch segment 0 (len0) are kept for
// the top-k launch.
template <bool SKETCH>
__device__ __forceinline__ void write_row(const RowStatsArgs &a, int64_t slot, const RowTotals &r, int lane,
                                          int len0) {
    const bool ok = (r.MX > -INFINITY) && (r.S > 0.f) && !(r.S != r.S) && !(r.T != r.T) && (r.AM != INT_MAX);
    // Probabilities are formed against the reference B like the sums, p_v =
    // 2^fma(z_v, log2(e), -B) / S, never as exp(z_v - lse): with large logits
    // lse carries an absolute rounding error of ulp(lse) that the exponential
    // would amplify.
    float lse = NAN, H = NAN, pmax = NAN, lnS = NAN, invS = NAN;
    if (ok) {
        lnS = logf(r.S);
        invS = 1.f / r.S;
        lse = fmaf(r.M, kLn2, lnS);
        H = fmaxf(lnS - kLn2 * r.T * invS, 0.f);
        pmax = ex2(fmaf(r.MX, kLog2e, -r.M)) * invS;
    }
    if (lane == 0) {
        a.zmax[slot] = ok ? r.MX : NAN;
        a.lse[slot] = lse;
        a.H[slot] = H;
        a.pmax[slot] = pmax;
        if (!SKETCH) a.argmax[slot] = ok ? r.AM : -1;
        if (!ok) flag_error(a.err, RPS_DEVERR_NONFINITE);
        if (SKETCH) a.norm[slot] = make_float4(r.M, lnS, invS, __int_as_float(len0));
    }
}

// ---------------------------------------------------------------- segments
// Rows of the list: the exclusive prefix of the segment counts (clamped to
// capacity) into seg_start, RPS_MAX_SEGMENTS / THREADS segments per thread and
// a block-wide scan; returns the total. Every thread of the block must call it.
template <int THREADS>
__device__ __forceinline__ int64_t count_rows(const RowStatsArgs &a, int32_t *seg_start, int32_t *warp_total, int lane,
                                              int wib) {
    if (!a.seg_cnt) return static_cast<int64_t>(a.n_seg) * a.cap;
    if (a.n_seg == 1) {  // one request: no scan (locate reads seg_start[0] only)
        int32_t v = a.seg_cnt[0];
        if (v < 0 || v > a.cap) {
            if (blockIdx.x == 0 && threadIdx.x == 0) flag_error(a.err, RPS_DEVERR_MASK);
            v = v < 0 ? 0 : a.cap;
        }
        if (threadIdx.x == 0) {
            seg_start[0] = 0;
            seg_start[1] = v;
        }
        __syncthreads();
        return v;
    }
    constexpr int kPer = RPS_MAX_SEGMENTS / THREADS;
    static_assert(RPS_MAX_SEGMENTS % THREADS == 0, "segments split evenly over the threads");
    int32_t c[kPer];
    int32_t local = 0;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        const int sg = threadIdx.x * kPer + i;
        int32_t v = sg < a.n_seg ? a.seg_cnt[sg] : 0;
        if (v < 0 || v > a.cap) {
            if (blockIdx.x == 0) flag_error(a.err, RPS_DEVERR_MASK);
            v = v < 0 ? 0 : a.cap;
        }
        c[i] = v;
        local += v;
    }
    int32_t incl = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t n = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += n;
    }
    if (lane == 31) warp_total[wib] = incl;
    __syncthreads();
    // exclusive prefix of the warps' totals: a shuffle scan in every warp
    static_assert(THREADS <= 32 * 32, "one warp scans the warps' totals");
    const int32_t wt = lane < THREADS / 32 ? warp_total[lane] : 0;
    int32_t wincl = wt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t n = __shfl_up_sync(kFull, wincl, o);
        if (lane >= o) wincl += n;
    }
    int32_t run = __shfl_sync(kFull, wincl - wt, wib) + incl - local;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
        seg_start[threadIdx.x * kPer + i] = run;
        run += c[i];
    }
    if (threadIdx.x == THREADS - 1) seg_start[RPS_MAX_SEGMENTS] = run;
    __syncthreads();
    return seg_start[a.n_seg];
}

struct Segment {
    int64_t slot;
    const char *row;
    int u0, u1;   // row-local unit range of this piece
    bool valid;   // false: skipped entry or bad descriptor
    bool bad;     // bad descriptor (to flag)
};

// The row of list entry s.slot of segment seg: validity and row pointer. CG:
// loads through L2.
template <int DT, bool CG = false>
__device__ __forceinline__ void describe(const RowStatsArgs &a, int seg, Segment &s) {
    int32_t req, br, pos;
    if (a.rows) {
        const int32_t *e = a.rows + s.slot * 3;
        req = CG ? __ldcg(e) : e[0];
        br = CG ? __ldcg(e + 1) : e[1];
        pos = CG ? __ldcg(e + 2) : e[2];
    } else {
        req = seg;
        br = a.mask_branch;
        pos = CG ? __ldcg(a.mask_pos + s.slot) : a.mask_pos[s.slot];
    }
    s.bad = pos >= 0 && (req < 0 || req >= a.n_req || br < 0 || br >= a.n_branch || pos >= a.n_pos);
    s.valid = pos >= 0 && !s.bad;
    s.row = s.valid ? static_cast<const char *>(a.data) +
                          (req * a.req_stride + br * a.branch_stride + static_cast<int64_t>(pos) * a.pos_stride) *
                              Elem<DT>::kBytes
                    : nullptr;
}

// Row r of the concatenated list -> (segment, entry) -> output slot and row pointer.
template <int DT>
__device__ __forceinline__ void locate(const RowStatsArgs &a, const int32_t *seg_start, int64_t r, Segment &s) {
    int seg;
    if (a.seg_cnt) {
        int lo = 0, hi = a.n_seg;  // s with seg_start[s] <= r < seg_start[s + 1]
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (seg_start[mid] <= r) lo = mid;
            else hi = mid;
        }
        seg = lo;
        s.slot = static_cast<int64_t>(lo) * a.cap + (r - seg_start[lo]);
    } else {
        seg = static_cast<int>(r / a.cap);
        s.slot = r;
    }
    describe<DT>(a, seg, s);
}

// The cut of the rows' units into pieces, one per warp. Aligned: each row is
// cut into equal pieces (at most ceil(nv / min_piece) per row), so that no
// piece crosses a row boundary, where a warp's stream stops for the row's
// record; taken when it leaves at most an eighth of the warps idle. Otherwise
// all units are cut evenly (pieces of at least min_piece units). Returns the
// units per piece.
__device__ __forceinline__ int64_t piece_units(const RowStatsArgs &a, int64_t total_rows, int64_t nv,
                                               bool &aligned) {
    aligned = false;
    if (total_rows <= a.warps) {  // 32-bit arithmetic: rows, warps and units of a row fit
        const int rows = static_cast<int>(total_rows), n = static_cast<int>(nv), mp = static_cast<int>(a.min_piece);
        const int ppr = min(a.warps / rows, (n + mp - 1) / mp);
        const int piece = (n + ppr - 1) / ppr;
        const int cpr = (n + piece - 1) / piece;
        if (8 * static_cast<int64_t>(rows) * cpr >= 7 * static_cast<int64_t>(a.warps)) {
            aligned = true;
            return piece;
        }
    }
    return max((total_rows * nv + a.warps - 1) / a.warps, a.min_piece);
}

// Sketch layout of one row under the cut of piece_units (top-k mode). The
// pieces that hold a part of the row are its segments: segment 0 = [0, len0),
// then pieces of `piece` units (the last one shorter). Each segment's ring
// chunks start at the segment start; the sketch holds 32 entries per chunk,
// segments in row order: ch0 chunks for segment 0, then cps per piece, then
// -inf to the end of the slot's stride. The statistics launch passes len0 per
// row and piece per launch to the top-k launch.
struct SketchRow {
    int len0;   // units of segment 0
    int ch0;    // its chunks of whole units
    int piece;  // units per further segment (the row length when there is none)
    int cps;    // chunks per further segment
};

__device__ __forceinline__ SketchRow sketch_row(int len0, int piece, int full_units) {
    SketchRow q;
    q.len0 = len0;
    q.ch0 = (min(len0, full_units) + kChunkUnits - 1) / kChunkUnits;
    q.piece = piece;
    q.cps = (piece + kChunkUnits - 1) / kChunkUnits;
    return q;
}

// Segment 0 of row r under a cut of `piece` units per warp.
__device__ __forceinline__ int sketch_len0(int64_t r, int64_t nv, int64_t piece, bool aligned) {
    const int64_t off = aligned ? 0 : (r * nv) % piece;  // units of the first piece spent on earlier rows
    return static_cast<int>(min(piece - off, nv));
}

// Sketch entry of the first chunk of the segment starting at unit u0.
__device__ __forceinline__ int sketch_key(const SketchRow &q, int u0) {
    return u0 == 0 ? 0 : 32 * (q.ch0 + (u0 - q.len0) / q.piece * q.cps);
}

// The units of sketch entry e of the row: first unit and count (units first +
// 32 t, t < count, of one lane of one ring chunk).
__device__ __forceinline__ void sketch_cell(const SketchRow &q, int full_units, int e, int &first, int &count) {
    const int chunk = e >> 5, l = e & 31;
    int cu, end;
    if (chunk < q.ch0) {
        cu = chunk * kChunkUnits;
        end = q.len0;
    } else {
        const int j = (chunk - q.ch0) / q.cps;
        const int s0 = q.len0 + j * q.piece;
        cu = s0 + (chunk - q.ch0 - j * q.cps) * kChunkUnits;
        end = s0 + q.piece;
    }
    end = min(min(end, cu + kChunkUnits), full_units);
    first = cu + l;
    count = first < end ? min((end - first + 31) / 32, kBatch) : 0;
}

// A warp's unit range: `left` units from unit u of row r on.
struct Walk {
    int64_t r;
    int u;
    int64_t left;
};

// Walks the row segments of a warp's range.
template <int DT>
__device__ __forceinline__ bool next_segment(const RowStatsArgs &a, const int32_t *seg_start, int64_t nv, Walk &w,
                                             int64_t &r, Segment &s) {
    if (w.left <= 0) return false;
    r = w.r;
    s.u0 = w.u;
    s.u1 = static_cast<int>(min(nv, static_cast<int64_t>(w.u) + w.left));
    w.left -= s.u1 - s.u0;
    ++w.r;
    w.u = 0;
    locate<DT>(a, seg_start, r, s);
    return true;
}

// Lane 0's copy engine: the next run of at most kChunkUnits whole units of the
// piece, in the order the warp consumes them (valid segments only).
template <int DT>
struct Producer {
    Walk w;
    Segment s;
    int cu;      // next unit to copy in the current segment
    int cu_end;  // end of its whole units
    bool have;

    __device__ __forceinline__ void init(const Walk &w0) {
        w = w0;
        have = false;
        cu = cu_end = 0;
    }

    __device__ __forceinline__ bool next(const RowStatsArgs &a, const int32_t *seg_start, int64_t nv, int full_units,
                                         const char *&src, uint32_t &bytes) {
        while (!have || cu >= cu_end) {
            int64_t r;
            if (!next_segment<DT>(a, seg_start, nv, w, r, s)) return false;
            have = s.valid;
            cu = s.u0;
            cu_end = min(s.u1, full_units);
        }
        const int n = min(kChunkUnits, cu_end - cu);
        src = s.row + static_cast<size_t>(cu) * 16;
        bytes = static_cast<uint32_t>(n) * 16u;
        cu += n;
        return true;
    }
};

// SKETCH (first launch of top-k mode): also the sketch (layout of sketch_row)
// and each row's B, ln S and 1 / S for the top-k launch.
template <int DT, bool SKETCH>
__global__ void __launch_bounds__(kStatThreads, kStatBlocksPerSm) row_stats_kernel(const RowStatsArgs a) {
    constexpr int kWarps = kStatThreads / 32;
    using E = Elem<DT>;
    constexpr int N = E::N;
    extern __shared__ __align__(128) uint4 dyn[];
    __shared__ int32_t seg_start[RPS_MAX_SEGMENTS + 1];
    __shared__ int32_t warp_total[kWarps];
    constexpr int kRing = kStages;
    __shared__ __align__(8) uint64_t bars[kWarps][kRing];

    pdl_wait();
    pdl_launch_next();
    const int lane = threadIdx.x & 31;
    const int wib = threadIdx.x >> 5;
    const int warp = blockIdx.x * kWarps + wib;
    uint4 *ring = dyn + wib * (kRing * kChunkUnits);
    uint64_t *bar = bars[wib];

    // (loaded here, tested after the row count, so that the two loads overlap)
    const uint32_t health = __ldcg(a.health);
    const int64_t total_rows = count_rows<kStatThreads>(a, seg_start, warp_total, lane, wib);
    // A workspace an earlier launch gave up on holds tickets of rows it never
    // finished: merging on them would write wrong rows, so nothing is written.
    if (health != 0) {
        if (threadIdx.x == 0) flag_error(a.err, RPS_DEVERR_WORKSPACE);
        return;
    }

    const int64_t nv = a.units_per_row;
    const int64_t total = total_rows * nv;
    if (total == 0) return;
    // With at least as many warps as rows, each row is cut into equal pieces
    // (aligned: no piece crosses a row boundary, where a warp's stream would
    // stop for the row's record); otherwise the units are cut evenly.
    __shared__ int64_t cut_cpr[kWarps];  // pieces per row of an aligned cut, 0 for the even cut
    if (lane == 0) cut_cpr[wib] = 0;
    bool aligned = false;
    const int64_t piece = piece_units(a, total_rows, nv, aligned);
    if (SKETCH && blockIdx.x == 0 && threadIdx.x == 0) *a.sketch_piece = static_cast<int>(min(piece, nv));
    Walk w0;
    if (aligned) {  // (32-bit: piece and the pieces per row are below the row length)
        const int cpr = (static_cast<int>(nv) + static_cast<int>(piece) - 1) / static_cast<int>(piece);
        const int row0 = warp / cpr, part = warp - row0 * cpr;
        if (row0 >= total_rows) return;
        w0.r = row0;
        w0.u = part * static_cast<int>(piece);
        w0.left = min(piece, nv - w0.u);
        if (lane == 0) cut_cpr[wib] = cpr;
    } else {
        const int64_t g_begin = static_cast<int64_t>(warp) * piece;
        if (g_begin >= total) return;
        w0.r = g_begin / nv;
        w0.u = static_cast<int>(g_begin - w0.r * nv);
        w0.left = min(piece, total - g_begin);
    }
    const int V = static_cast<int>(a.vocab);
    const int full_units = V / N;

    // Ring set-up: one mbarrier per buffer, then up to kRing copies in flight.
    if (lane == 0) {
        for (int i = 0; i < kRing; ++i) mbar_init(bar + i, 1);
        fence_mbar_init();
    }
    __syncwarp();
    Producer<DT> prod;
    prod.init(w0);
    int issued = 0;
    if (lane == 0) {
        const char *src;
        uint32_t bytes;
        while (issued < kRing && prod.next(a, seg_start, nv, full_units, src, bytes)) {
            bulk_load(ring + issued * kChunkUnits, src, bytes, bar + issued);
            ++issued;
        }
    }
    issued = __shfl_sync(kFull, issued, 0);
    int acquired = 0, released = 0;

    // Waits for the next ring chunk; false when it does not land within the
    // limit. The warp then flags the error, marks the workspace unhealthy (its
    // rows' tickets stay incomplete), waits -- bounded -- for every copy it
    // issued, the one that timed out included, so that none still writes into
    // its ring, and must stop.
    auto acquire = [&](int &st) -> bool {
        st = acquired % kRing;
        if (mbar_wait_bounded(bar + st, (acquired / kRing) & 1, a.ring_wait_ns)) {
            ++acquired;
            return true;
        }
        if (lane == 0) {
            flag_error(a.err, RPS_DEVERR_TIMEOUT);
            atomicExch(a.health, kUnhealthy);
            for (int c = acquired; c < issued; ++c) mbar_wait_bounded(bar + (c % kRing), (c / kRing) & 1);
        }
        __syncwarp();
        return false;
    };
    // Hands the oldest held buffer back to the copy engine, which refills it.
    auto release = [&]() {
        const int st = released % kRing;
        fence_proxy_async();
        __syncwarp();
        ++released;
        if (lane == 0) {
            const char *src;
            uint32_t bytes;
            if (prod.next(a, seg_start, nv, full_units, src, bytes)) {
                bulk_load(ring + st * kChunkUnits, src, bytes, bar + st);
                ++issued;
            }
        }
        issued = __shfl_sync(kFull, issued, 0);
    };

    Walk walk = w0;
    int64_t r;
    Segment s;
    while (next_segment<DT>(a, seg_start, nv, walk, r, s)) {
        if (!s.valid) {
            if (s.bad && lane == 0) flag_error(a.err, RPS_DEVERR_ROW_INDEX);
            continue;
        }
        LaneState L;
        lane_init(L);
        typename E::Sketch *sketch =
            SKETCH ? static_cast<typename E::Sketch *>(a.sketch) + s.slot * a.sketch_stride : nullptr;
        const int cend = min(s.u1, full_units);
        int key = SKETCH ? sketch_key(sketch_row(sketch_len0(r, nv, piece, aligned), static_cast<int>(min(piece, nv)),
                                                 full_units),
                                      s.u0)
                         : 0;
        for (int cu = s.u0; cu < cend; cu += kChunkUnits) {
            int st;
            if (!acquire(st)) return;
            fold_chunk<DT, SKETCH>(L, sketch, ring + st * kChunkUnits, min(kChunkUnits, cend - cu), cu, key,
                                         lane);
            key += 32;
            release();
        }
        if (SKETCH && s.u1 == nv) {  // the rest of the slot's sketch reads as -inf
            constexpr int kPerVec = 16 / static_cast<int>(sizeof(typename E::Sketch));
            uint4 *p = reinterpret_cast<uint4 *>(sketch);
            const uint4 ninf = make_uint4(E::kNegInf2, E::kNegInf2, E::kNegInf2, E::kNegInf2);
            for (int v = key / kPerVec + lane; v < a.sketch_stride / kPerVec; v += 32) p[v] = ninf;
        }
        if (s.u1 > full_units) fold_tail<DT, false>(L, s.row, V, lane);
        {
            float a0, a1, b0, b1;
            unpack2(L.s, a0, a1);
            unpack2(L.t, b0, b1);
            const float chk = a0 + a1 + b0 + b1;
            if (__any_sync(kFull, chk != chk)) {
                rescan_safe<DT>(L, s.row, V, s.u0, s.u1, lane);
                if (L.bad) L.s = pack2(NAN, NAN);
            }
        }
        // (sketch mode: the top-k launch takes the argmax from its list)
        const int am = SKETCH ? 0 : resolve_argmax<DT>(s.row, V, L, warp_max(L.mx), lane);
        float s_lo, s_hi, t_lo, t_hi;
        unpack2(L.s, s_lo, s_hi);
        unpack2(L.t, t_lo, t_hi);
        RowTotals rt = combine(L.mref, s_lo + s_hi, t_lo + t_hi, L.mx, am);

        // the pieces (warps) that hold a part of row r
        int64_t w_first;
        int count;
        // (read back from shared memory so that it is not kept live through the stream)
        const int64_t cpr = *reinterpret_cast<volatile int64_t *>(&cut_cpr[wib]);
        if (cpr > 0) {
            w_first = r * cpr;
            count = static_cast<int>(cpr);
        } else {
            w_first = (r * nv) / piece;
            count = static_cast<int>(((r + 1) * nv - 1) / piece - w_first + 1);
        }
        const int64_t slot = s.slot;
        if (count == 1) {
            write_row<SKETCH>(a, slot, rt, lane, SKETCH ? sketch_len0(r, nv, piece, aligned) : 0);
            continue;
        }
        const int my = static_cast<int>(warp - w_first);
        Partial *part = a.part + slot * kMaxPartials;
        if (lane == 0) {
            Partial p;
            p.mref = rt.M;
            p.s = rt.S;
            p.t = rt.T;
            p.mx = rt.MX;
            p.amax = rt.AM;
            p.pad[0] = p.pad[1] = p.pad[2] = 0;
            part[my] = p;
        }
        __threadfence();
        __syncwarp();
        unsigned prior = 0;
        if (lane == 0) {
            prior = atomicAdd(a.ticket + slot, 1u);
            // a ticket at or past the piece count was left by an unfinished
            // launch or was never zeroed
            if (prior >= static_cast<unsigned>(count)) flag_error(a.err, RPS_DEVERR_WORKSPACE);
        }
        prior = __shfl_sync(kFull, prior, 0);
        if (prior != static_cast<unsigned>(count - 1)) continue;

        // Last piece of this row to finish: merge every record.
        __threadfence();
        if (lane == 0) a.ticket[slot] = 0;  // ready for the next call
        Partial p;
        p.mref = -INFINITY;
        p.s = 0.f;
        p.t = 0.f;
        p.mx = -INFINITY;
        p.amax = INT_MAX;
        if (lane < count) {
            const float4 q = __ldcg(reinterpret_cast<const float4 *>(part + lane));
            p.mref = q.x;
            p.s = q.y;
            p.t = q.z;
            p.mx = q.w;
            p.amax = __ldcg(&part[lane].amax);
        }
        rt = combine(p.mref, p.s, p.t, p.mx, p.amax);
        write_row<SKETCH>(a, slot, rt, lane, SKETCH ? sketch_len0(r, nv, piece, aligned) : 0);
    }
}

// ---------------------------------------------------------------- top-k launch
// Second launch of top-k mode (k <= 32), one warp per slot of the row list. Its statistics
// launch left the row's sketch -- the maximum of every cell, a cell being one
// lane's units of one ring chunk -- and B, ln S, 1 / S. The k-th largest of the 32
// lanes' largest sketch entries bounds the row's k-th largest logit from below
// (k lanes each saw a different cell holding an element at least that large),
// so only the cells whose maximum reaches the bound -- about k of them -- are
// read again, and their elements at or above it enter the warp-distributed
// sorted list (lane j = rank j, logit desc then token asc).
constexpr int kCellCap = 256;  // candidate cells a warp buffers before reloading them
constexpr int kSketchVecs = 24;  // 16-byte sketch loads a lane keeps in flight (up to 768 vectors a slot in one round)
static_assert(kSketchVecs <= 32, "one hit bit per vector");

// Merges the elements at or above max(theta, current k-th entry) of the staged
// cells (lane j: units first + 32 t at stage[t * 32 + j], t < count).
template <int DT>
__device__ __forceinline__ void merge_staged_cells(const uint4 *stage, int first, int count, int k, int lane,
                                                   float theta, float &tv, int &ti, float2 *cand, bool &empty) {
    using E = Elem<DT>;
    constexpr int N = E::N;
    static_assert(kBatch * N <= 32, "a cell's elements fit one mask word");
    const float th = empty ? theta : fmaxf(__shfl_sync(kFull, tv, k - 1), theta);
    uint32_t cm = 0;
#pragma unroll
    for (int t = 0; t < kBatch; ++t) {
        if (t < count) {
            const uint4 w = stage[t * 32 + lane];
            if (E::unit_max(w) >= th) {
                float y[N];
                E::unpack(w, y);
#pragma unroll
                for (int i = 0; i < N; ++i)
                    if (y[i] >= th) cm |= 1u << (t * N + i);
            }
        }
    }
    const int c = __popc(cm);
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += n;
    }
    const int total = __shfl_sync(kFull, incl, 31);
    const uint32_t *words = reinterpret_cast<const uint32_t *>(stage);
    for (int done = 0; done < total; done += kCandBatch) {
        int slot = incl - c;
        uint32_t bits = cm;
        while (bits) {
            const int bit = __ffs(bits) - 1;
            bits &= bits - 1;
            if (slot >= done && slot < done + kCandBatch) {
                const int t = bit / N, i = bit % N;
                cand[slot - done] = make_float2(E::pick(words + (t * 32 + lane) * 4, i),
                                                __int_as_float((first + 32 * t) * N + i));
            }
            ++slot;
        }
        __syncwarp();
        const float2 e = done + lane < total ? cand[lane] : make_float2(-INFINITY, __int_as_float(INT_MAX));
        __syncwarp();
        if (empty) warp_rank_into_list(tv, ti, e.x, __float_as_int(e.y), k, lane, cand);
        else warp_merge_batch(tv, ti, e.x, __float_as_int(e.y), k, lane);
        empty = false;
        __syncwarp();
    }
}

// Reloads the buffered cells cells[0, n) (sketch entries), 32 at a time, and
// merges their elements.
template <int DT>
__device__ void merge_sketch_cells(const char *row, const int32_t *cells, int n, const SketchRow &cut, int full_units,
                                   int k, int lane, float theta, float &tv, int &ti, uint4 *stage, float2 *cand,
                                   bool &empty) {
    for (int b = 0; b < n; b += 32) {
        int first = 0, count = 0;
        if (b + lane < n) sketch_cell(cut, full_units, cells[b + lane], first, count);
        __syncwarp();
#pragma unroll
        for (int t = 0; t < kBatch; ++t)
            if (t < count) cp_async16(stage + t * 32 + lane, row + static_cast<size_t>(first + 32 * t) * 16);
        cp_async_wait_all();
        __syncwarp();
        merge_staged_cells<DT>(stage, first, count, k, lane, theta, tv, ti, cand, empty);
    }
}

// The largest entry of each of this lane's sketch vectors v0 + 32 q + lane
// (-inf past the row's n_vec).
template <int DT>
__device__ __forceinline__ void vector_maxima(float (&vm)[kSketchVecs], const uint4 *sk, int v0, int n_vec, int lane) {
    uint4 w[kSketchVecs];
#pragma unroll
    for (int q = 0; q < kSketchVecs; ++q) {
        const int v = v0 + q * 32 + lane;
        w[q] = v < n_vec ? __ldg(sk + v) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int q = 0; q < kSketchVecs; ++q) vm[q] = v0 + q * 32 + lane < n_vec ? Elem<DT>::unit_max(w[q]) : -INFINITY;
}

// Bit i: entry i of sketch vector *p reaches theta.
template <int DT>
__device__ __forceinline__ uint32_t vector_hits(const uint4 *p, float theta) {
    constexpr int kPerVec = 16 / static_cast<int>(sizeof(typename Elem<DT>::Sketch));
    float y[kPerVec];
    Elem<DT>::unpack(__ldg(p), y);
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < kPerVec; ++i)
        if (y[i] >= theta) m |= 1u << i;
    return m;
}

template <int DT>
__global__ void __launch_bounds__(kTopkWarps * 32, kTopkMinBlocks) topk_rows_kernel(const RowStatsArgs a) {
    using E = Elem<DT>;
    constexpr int kPerVec = 16 / static_cast<int>(sizeof(typename E::Sketch));  // sketch entries per 16 bytes
    __shared__ uint4 stage_all[kTopkWarps][kBatch * 32];
    __shared__ float2 cand_all[kTopkWarps][kCandBatch];
    __shared__ int32_t cells_all[kTopkWarps][kCellCap];

    const int lane = threadIdx.x & 31;
    const int wib = threadIdx.x >> 5;
    uint4 *stage = stage_all[wib];
    float2 *cand = cand_all[wib];
    int32_t *cells = cells_all[wib];
    const int64_t n_slots = static_cast<int64_t>(a.n_seg) * a.cap;
    const int64_t nv = a.units_per_row;
    const int V = static_cast<int>(a.vocab);
    const int full_units = V / Elem<DT>::N;
    const int k = a.k;
    const int n_vec = static_cast<int>(a.sketch_stride / kPerVec);  // the whole slot (-inf past the row's chunks)
    const bool one_batch = n_vec <= 32 * kSketchVecs;
    bool waited = false;

    // One warp per list slot (entry), in slot order: no scan of the list.
    for (int64_t slot = static_cast<int64_t>(blockIdx.x) * kTopkWarps + wib;;
         slot += static_cast<int64_t>(gridDim.x) * kTopkWarps) {
        // The list is an input of the statistics launch, which waited for its
        // producers before letting this launch begin: it is read before the wait.
        Segment s;
        s.slot = slot;
        s.valid = false;
        const bool have = slot < n_slots;
        if (have) {
            const int seg = static_cast<int>(slot / a.cap);
            int cnt = a.cap;
            if (a.seg_cnt) cnt = min(max(__ldcg(a.seg_cnt + seg), 0), a.cap);  // (as the statistics launch clamps)
            if (slot - static_cast<int64_t>(seg) * a.cap < cnt) describe<DT, true>(a, seg, s);
        }
        if (!waited) {  // everything below reads the statistics launch's results
            pdl_wait();
            pdl_launch_next();
            waited = true;
        }
        if (!have) break;
        if (!s.valid) continue;  // skipped entry, or a bad descriptor the statistics launch flagged
        const uint4 *sk = reinterpret_cast<const uint4 *>(static_cast<const typename E::Sketch *>(a.sketch) +
                                                          slot * a.sketch_stride);
        const float zmax = __ldcg(a.zmax + slot);
        const float4 nrm = __ldcg(a.norm + slot);
        const int piece = __ldcg(a.sketch_piece);
        const uint32_t health = __ldcg(a.health);
        // Pass 1: the largest entry of each of this lane's vectors v0 + 32 q + lane.
        float vm[kSketchVecs];
        vector_maxima<DT>(vm, sk, 0, n_vec, lane);
        if (health != 0) {  // the statistics launch gave up, or found the workspace unhealthy
            if (lane == 0) flag_error(a.err, RPS_DEVERR_WORKSPACE);
            break;
        }
        if (zmax != zmax) {  // the statistics launch found no finite row
            if (lane == 0) {
                a.argmax[slot] = -1;
                a.mu[slot] = NAN;
                a.htrunc[slot] = NAN;
            }
            if (lane < k) {
                a.topk_idx[slot * k + lane] = -1;
                a.topk_logit[slot * k + lane] = NAN;
            }
            continue;
        }
        // (clamped: a record or a piece length left by a failed launch never
        // names a unit outside the row)
        const int n_units = static_cast<int>(nv);
        const SketchRow cut = sketch_row(min(max(__float_as_int(nrm.w), 1), n_units), min(max(piece, 1), n_units),
                                         full_units);
        // the k-th largest of the lanes' largest entries
        float lane_max = -INFINITY;
        for (int v0 = 0;;) {
#pragma unroll
            for (int q = 0; q < kSketchVecs; ++q) lane_max = fmaxf(lane_max, vm[q]);
            v0 += 32 * kSketchVecs;
            if (v0 >= n_vec) break;
            vector_maxima<DT>(vm, sk, v0, n_vec, lane);
        }
        const float theta = warp_kth_largest(lane_max, k, lane);

        // Pass 2: the cells that reach it, buffered and reloaded kCellCap at a
        // time. Few vectors hold one; only those are read again (from L1).
        float tv = -INFINITY;
        int ti = INT_MAX;
        bool empty = true;
        int pending = 0;
        for (int v0 = 0; v0 < n_vec; v0 += 32 * kSketchVecs) {
            if (!one_batch) vector_maxima<DT>(vm, sk, v0, n_vec, lane);
            uint32_t hv = 0;  // bit q: vector q holds an entry at or above theta
#pragma unroll
            for (int q = 0; q < kSketchVecs; ++q)
                if (vm[q] >= theta) hv |= 1u << q;
            if (!__any_sync(kFull, hv != 0)) continue;
            int c = 0;
            for (uint32_t b = hv; b; b &= b - 1) c += __popc(vector_hits<DT>(sk + v0 + (__ffs(b) - 1) * 32 + lane, theta));
            int incl = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int n = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += n;
            }
            const int end = pending + __shfl_sync(kFull, incl, 31);
            for (int base = 0;; base += kCellCap) {
                int slot_i = pending + incl - c;
                for (uint32_t b = hv; b; b &= b - 1) {
                    const int q = __ffs(b) - 1;
                    uint32_t m = vector_hits<DT>(sk + v0 + q * 32 + lane, theta);
                    while (m) {
                        const int i = __ffs(m) - 1;
                        m &= m - 1;
                        if (slot_i >= base && slot_i < base + kCellCap)
                            cells[slot_i - base] = (v0 + q * 32 + lane) * kPerVec + i;
                        ++slot_i;
                    }
                }
                __syncwarp();
                if (end - base <= kCellCap) {
                    pending = end - base;
                    break;
                }
                merge_sketch_cells<DT>(s.row, cells, kCellCap, cut, full_units, k, lane, theta, tv, ti, stage, cand,
                                       empty);
                __syncwarp();
            }
            if (pending == kCellCap) {
                merge_sketch_cells<DT>(s.row, cells, kCellCap, cut, full_units, k, lane, theta, tv, ti, stage, cand,
                                       empty);
                pending = 0;
                __syncwarp();
            }
        }
        if (pending > 0)
            merge_sketch_cells<DT>(s.row, cells, pending, cut, full_units, k, lane, theta, tv, ti, stage, cand, empty);
        if (full_units < nv) topk_tail<DT>(s.row, V, k, lane, tv, ti);

        float mu, ht;
        topk_mass(tv, nrm.x, nrm.y, nrm.z, k, lane, mu, ht);
        // rank 0 of T (largest logit, lowest token) is the argmax of Eq. 1
        const int i0 = __shfl_sync(kFull, ti, 0);
        if (lane == 0) {
            a.argmax[slot] = i0;
            a.mu[slot] = mu;
            a.htrunc[slot] = ht;
        }
        if (lane < k) {
            a.topk_idx[slot * k + lane] = ti;
            a.topk_logit[slot * k + lane] = tv;
        }
    }
}

constexpr int kDynSmemBytes = kStatThreads / 32 * kStages * kChunkUnits * static_cast<int>(sizeof(uint4));

template <int DT, bool SKETCH>
cudaError_t prepare_typed() {
    return cudaFuncSetAttribute(row_stats_kernel<DT, SKETCH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kDynSmemBytes);
}

template <int DT, bool SKETCH>
cudaError_t launch_typed(const RowStatsArgs &a, int grid, cudaStream_t stream) {
    return launch_pdl(row_stats_kernel<DT, SKETCH>, dim3(grid), dim3(kStatThreads), kDynSmemBytes, stream, a);
}

// Statistics-only mode: one launch. Top-k mode: statistics with the sketch,
// then the top-k rows.
template <int DT>
cudaError_t launch_dtype(const RowStatsArgs &a, int grid, int topk_grid, cudaStream_t stream) {
    if (a.k == 0) return launch_typed<DT, false>(a, grid, stream);
    RowStatsArgs st = a;
    st.k = 0;
    cudaError_t e = launch_typed<DT, true>(st, grid, stream);
    if (e != cudaSuccess) return e;
    return launch_pdl(topk_rows_kernel<DT>, dim3(topk_grid), dim3(kTopkWarps * 32), 0, stream, a);
}

template <int DT>
cudaError_t occupancy_typed(int *blocks) {
    cudaError_t e = prepare_typed<DT, false>();
    if (e == cudaSuccess) e = prepare_typed<DT, true>();
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, row_stats_kernel<DT, false>, kStatThreads,
                                                         kDynSmemBytes);
}

}  // namespace

cudaError_t launch_row_stats(const RowStatsArgs &a, int dtype, int grid, int topk_grid, cudaStream_t stream) {
    return dtype == RPS_BF16 ? launch_dtype<RPS_BF16>(a, grid, topk_grid, stream)
                             : launch_dtype<RPS_F32>(a, grid, topk_grid, stream);
}

cudaError_t row_stats_occupancy(int dtype, int *blocks_per_sm) {
    return dtype == RPS_BF16 ? occupancy_typed<RPS_BF16>(blocks_per_sm) : occupancy_typed<RPS_F32>(blocks_per_sm);
}

}  // namespace rps
