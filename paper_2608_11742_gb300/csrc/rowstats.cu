// rowstats.cu -- fused single-pass row statistics of logit rows (rps_score_step).
//
// For every listed row z (V logits) one pass over HBM yields
//   zmax, argmax (Eq. 1), lse, H = -sum p log p, P^max (Sec. 2 notation) and,
//   in top-k mode, T_i, mu_i and the truncated entropy of Eq. 3.
//
// Work split. The rows' 16-byte units are laid end to end and cut into equal
// contiguous pieces, one per warp of a persistent grid, so every warp streams
// the same number of bytes whatever the row count. A piece covers the tail of
// one row, whole rows and the head of another; each (warp, row) pair leaves a
// partial record in the workspace and the last warp to finish a row (atomic
// ticket, no waiting) merges the at most kMaxPartials records and writes the row.
//
// Per lane, a row segment is reduced as a base-2 online softmax against an
// exponent reference mref that is raised only when a value exceeds it by more
// than kSlack nats (rare), so the steady state is, per element, one FFMA, one
// MUFU ex2 and two FP32 adds/FMAs:
//   s = sum 2^u, t = sum u 2^u, u = (z - mref) log2(e)
//   H = ln S - ln2 * T / S,  lse = mref + ln S   (after merging lanes / pieces)
// The exact maximum is tracked per 16-byte unit; its token index is resolved
// once per segment by re-reading the unit that holds it.
//
// Top-k (k <= 32) lives in a warp-distributed sorted list, lane j holding rank j
// in the order (logit desc, token asc). Elements below a warp threshold are
// discarded with one compare per unit; the threshold is the list's k-th value,
// seeded after the first batch by the k-th largest lane maximum (a valid lower
// bound: those k lanes each hold an element at least that large).
//
// -inf logits or NaN make the fast path's t NaN; the segment is then rescanned
// with clamped exponents (SAFE), which scores -inf as probability 0 and flags
// NaN input as RPS_DEVERR_NONFINITE.
#include <cfloat>
#include <climits>

#include "rps_internal.cuh"

namespace rps {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kSlack = 8.0f;  // nats the reference may trail the maximum

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
__device__ __forceinline__ f2 sub2(f2 a, f2 b) {
    f2 r;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
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
    __device__ static __forceinline__ float load1(const char *row, int64_t e) {
        return reinterpret_cast<const float *>(row)[e];
    }
    __device__ static __forceinline__ float pick(const uint32_t *words, int i) {
        return __uint_as_float(words[i]);
    }
};

struct LaneState {
    float mref;   // exponent reference, -inf until the first finite value
    f2 s, t;      // pairwise partial sums of 2^u and u 2^u, u = (z - mref) log2(e)
    float mx;     // exact running maximum
    int best;     // first element of the unit where mx was first reached, -1 if none
    bool bad;     // NaN input seen (SAFE scan only)
};

__device__ __forceinline__ void lane_init(LaneState &L) {
    L.mref = -INFINITY;
    L.s = pack2(0.f, 0.f);
    L.t = pack2(0.f, 0.f);
    L.mx = -INFINITY;
    L.best = -1;
    L.bad = false;
}

// Fold one unit of n valid values (n == N except for a ragged row tail). The
// exponent is formed as (z - mref) * log2(e): the difference is exact for
// values near the reference, so large logits lose no absolute precision.
template <int N, bool SAFE>
__device__ __forceinline__ float fold_unit(LaneState &L, const float (&y)[N], int n, int e0) {
    float vmax = -INFINITY;
#pragma unroll
    for (int i = 0; i < N; ++i)
        if (i < n) vmax = fmaxf(vmax, y[i]);
    if (vmax > L.mx) {
        L.mx = vmax;
        L.best = e0;
    }
    if (vmax > L.mref + kSlack) {  // raise the exponent reference (rare)
        float slo, shi;
        unpack2(L.s, slo, shi);
        if (slo + shi > 0.f) {
            const float d = (L.mref - vmax) * kLog2e;
            const float a = ex2(d);
            const f2 a2 = pack2(a, a);
            L.t = mul2(a2, fma2(pack2(d, d), L.s, L.t));
            L.s = mul2(a2, L.s);
        }
        L.mref = vmax;
    }
    const f2 m2 = pack2(L.mref, L.mref);
    const f2 l2 = pack2(kLog2e, kLog2e);
#pragma unroll
    for (int i = 0; i < N; i += 2) {
        const bool v0 = i < n, v1 = i + 1 < n;
        if (!v0) break;
        const f2 u2 = mul2(sub2(pack2(y[i], v1 ? y[i + 1] : y[i]), m2), l2);
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
    return vmax;
}

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

template <int DT, bool TOPK, bool SAFE>
__device__ __forceinline__ void scan_segment(const char *row, int V, int u0, int u1, int k, int lane,
                                             LaneState &L, float &tv, int &ti, uint4 *stage) {
    using E = Elem<DT>;
    constexpr int N = E::N;
    lane_init(L);
    tv = -INFINITY;
    ti = INT_MAX;
    float seed = -INFINITY;  // lower bound on the segment's k-th largest value
    const int full_end = min(u1, V / N);  // units wholly inside the row
    constexpr int step = 32 * kBatch;
    bool first = true;

    uint4 cur[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
        const int u = u0 + j * 32 + lane;
        if (u < full_end) cur[j] = ld_stream(row + static_cast<size_t>(u) * 16);
    }
    for (int b = u0; b < full_end; b += step) {
        uint4 nxt[kBatch];
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int u = b + step + j * 32 + lane;
            if (u < full_end) nxt[j] = ld_stream(row + static_cast<size_t>(u) * 16);
        }
        float bmax = -INFINITY;
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
            const int u = b + j * 32 + lane;
            if (u < full_end) {
                float y[N];
                E::unpack(cur[j], y);
                bmax = fmaxf(bmax, fold_unit<N, SAFE>(L, y, N, u * N));
            }
        }
        if (TOPK) {
            if (first) {
                seed = warp_kth_largest(bmax, k, lane);
                first = false;
            }
            float th = fmaxf(__shfl_sync(kFull, tv, k - 1), seed);
            if (__any_sync(kFull, bmax >= th)) {
                // stage this batch and extract its candidates one at a time
                unsigned cm = 0;
#pragma unroll
                for (int j = 0; j < kBatch; ++j) {
                    const int u = b + j * 32 + lane;
                    if (u < full_end) {
                        stage[lane * kBatch + j] = cur[j];
                        float y[N];
                        E::unpack(cur[j], y);
#pragma unroll
                        for (int i = 0; i < N; ++i)
                            if (y[i] >= th) cm |= 1u << (j * N + i);
                    }
                }
                __syncwarp();
                const uint32_t *words = reinterpret_cast<const uint32_t *>(stage);
                while (true) {
                    const unsigned lanes = __ballot_sync(kFull, cm != 0);
                    if (!lanes) break;
                    const int src = __ffs(lanes) - 1;
                    const int bit = __shfl_sync(kFull, __ffs(cm) - 1, src);
                    if (lane == src) cm &= cm - 1;
                    const int j = bit / N, i = bit % N;
                    const float cv = E::pick(words + (src * kBatch + j) * 4, i);
                    if (cv >= th) {
                        const int ci = (b + j * 32 + src) * N + i;
                        topk_insert(tv, ti, cv, ci, k, lane);
                        th = fmaxf(__shfl_sync(kFull, tv, k - 1), seed);
                    }
                }
                __syncwarp();
            }
        }
#pragma unroll
        for (int j = 0; j < kBatch; ++j) cur[j] = nxt[j];
    }

    // ragged tail: the last unit of the row holds fewer than N values
    if (u1 > full_end && full_end == V / N) {
        const int e0 = full_end * N;
        const int n = V - e0;
        float y[N];
#pragma unroll
        for (int i = 0; i < N; ++i) y[i] = (i < n && lane == 0) ? E::load1(row, e0 + i) : -INFINITY;
        float tmax = -INFINITY;
        if (lane == 0) tmax = fold_unit<N, SAFE>(L, y, n, e0);
        if (TOPK) {
            if (first) seed = warp_kth_largest(tmax, k, lane);
            float th = fmaxf(__shfl_sync(kFull, tv, k - 1), seed);
#pragma unroll
            for (int i = 0; i < N; ++i) {
                const float cv = __shfl_sync(kFull, y[i], 0);
                if (i < n && cv >= th) {
                    topk_insert(tv, ti, cv, e0 + i, k, lane);
                    th = fmaxf(__shfl_sync(kFull, tv, k - 1), seed);
                }
            }
        }
    }
}

// Lowest token index holding value mx among this lane's best unit (INT_MAX if none).
template <int DT>
__device__ __forceinline__ int resolve_argmax(const char *row, int64_t V, const LaneState &L, float MX) {
    using E = Elem<DT>;
    constexpr int N = E::N;
    if (L.best < 0 || !(L.mx == MX)) return INT_MAX;
    const int64_t e0 = L.best;
    const int n = static_cast<int>((V - e0 < N ? V - e0 : static_cast<int64_t>(N)));
    float y[N];
    if (n == N) {
        E::unpack(ld_stream(row + e0 * E::kBytes), y);
    } else {
#pragma unroll
        for (int i = 0; i < N; ++i) y[i] = i < n ? E::load1(row, e0 + i) : -INFINITY;
    }
#pragma unroll
    for (int i = 0; i < N; ++i)
        if (i < n && y[i] == MX) return static_cast<int>(e0 + i);
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
        d = (mref - r.M) * kLog2e;
        a = ex2(d);
    }
    // a NaN s (bad input) must survive the merge
    r.S = warp_sum(live ? a * s : (s != s ? s : 0.f));
    r.T = warp_sum(live ? a * fmaf(d, s, t) : 0.f);
    r.MX = warp_max(mx);
    r.AM = warp_min_int(mx == r.MX ? am : INT_MAX);
    return r;
}

__device__ __forceinline__ void write_row(const RowStatsArgs &a, int64_t slot, const RowTotals &r, float tv, int ti,
                                          int lane) {
    const bool ok = (r.MX > -INFINITY) && (r.S > 0.f) && !(r.S != r.S) && !(r.T != r.T) && (r.AM != INT_MAX);
    // Probabilities are formed relative to the exponent reference M, p_v =
    // exp(z_v - M) / S, never as exp(z_v - lse): with large logits lse carries
    // an absolute rounding error of ulp(lse) that the exponential would amplify.
    float lse = NAN, H = NAN, pmax = NAN, lnS = NAN, invS = NAN;
    if (ok) {
        lnS = logf(r.S);
        invS = 1.f / r.S;
        lse = r.M + lnS;
        H = fmaxf(lnS - kLn2 * r.T * invS, 0.f);
        pmax = expf(r.MX - r.M) * invS;
    }
    if (lane == 0) {
        a.zmax[slot] = ok ? r.MX : NAN;
        a.lse[slot] = lse;
        a.H[slot] = H;
        a.pmax[slot] = pmax;
        a.argmax[slot] = ok ? r.AM : -1;
        if (!ok) flag_error(a.err, RPS_DEVERR_NONFINITE);
    }
    if (a.k > 0) {
        float p = 0.f, h = 0.f;
        if (ok && lane < a.k) {
            const float d = tv - r.M;  // exact for the reference's neighbourhood (Sterbenz)
            p = expf(d) * invS;
            if (p > 0.f) h = -p * (d - lnS);
        }
        const float mu = warp_sum(p), ht = warp_sum(h);
        if (lane == 0) {
            a.mu[slot] = ok ? mu : NAN;
            a.htrunc[slot] = ok ? ht : NAN;
        }
        if (lane < a.k) {
            a.topk_idx[slot * a.k + lane] = ok ? ti : -1;
            a.topk_logit[slot * a.k + lane] = ok ? tv : NAN;
        }
    }
}

template <int DT, bool TOPK>
__global__ void __launch_bounds__(kRowThreads, kRowMinBlocks) row_stats_kernel(const RowStatsArgs a) {
    __shared__ int32_t seg_start[RPS_MAX_SEGMENTS + 1];
    __shared__ uint4 stage_all[TOPK ? (kRowThreads / 32) * 32 * kBatch : 1];
    const int lane = threadIdx.x & 31;
    const int warp_in_block = threadIdx.x >> 5;
    const int warp = blockIdx.x * (kRowThreads / 32) + warp_in_block;
    uint4 *stage = stage_all + (TOPK ? warp_in_block * 32 * kBatch : 0);

    // Exclusive prefix of the segment counts (clamped to capacity), four
    // segments per thread, then a block-wide scan.
    int64_t total_rows;
    if (a.seg_cnt) {
        __shared__ int32_t warp_total[kRowThreads / 32];
        constexpr int kPer = RPS_MAX_SEGMENTS / kRowThreads;
        int32_t c[kPer];
        int32_t local = 0;
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
            const int s = threadIdx.x * kPer + i;
            int32_t v = s < a.n_seg ? a.seg_cnt[s] : 0;
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
        if (lane == 31) warp_total[warp_in_block] = incl;
        __syncthreads();
        int32_t run = incl - local;
        for (int w = 0; w < warp_in_block; ++w) run += warp_total[w];
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
            seg_start[threadIdx.x * kPer + i] = run;
            run += c[i];
        }
        if (threadIdx.x == kRowThreads - 1) seg_start[RPS_MAX_SEGMENTS] = run;
        __syncthreads();
        total_rows = seg_start[a.n_seg];
    } else {
        total_rows = static_cast<int64_t>(a.n_seg) * a.cap;
    }

    const int64_t nv = a.units_per_row;
    const int64_t total = total_rows * nv;
    if (total == 0) return;
    const int64_t piece = max((total + a.warps - 1) / a.warps, a.min_piece);
    const int64_t g_begin = static_cast<int64_t>(warp) * piece;
    if (g_begin >= total) return;
    const int64_t g_end = min(g_begin + piece, total);
    const char *base = static_cast<const char *>(a.data);
    constexpr int kBytes = Elem<DT>::kBytes;

    for (int64_t g = g_begin; g < g_end;) {
        const int64_t r = g / nv;
        const int64_t u0 = g - r * nv;
        const int64_t u1 = min(nv, u0 + (g_end - g));
        g += u1 - u0;

        // row r of the concatenated list -> (segment, entry) -> slot
        int64_t slot;
        int seg;
        if (a.seg_cnt) {
            int lo = 0, hi = a.n_seg;  // find s with seg_start[s] <= r < seg_start[s + 1]
            while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if (seg_start[mid] <= r) lo = mid; else hi = mid;
            }
            seg = lo;
            slot = static_cast<int64_t>(lo) * a.cap + (r - seg_start[lo]);
        } else {
            seg = static_cast<int>(r / a.cap);
            slot = r;
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
        if (pos < 0) continue;
        if (req < 0 || req >= a.n_req || br < 0 || br >= a.n_branch || pos >= a.n_pos) {
            if (lane == 0) flag_error(a.err, RPS_DEVERR_ROW_INDEX);
            continue;
        }
        const char *row = base + (req * a.req_stride + br * a.branch_stride + pos * a.pos_stride) * kBytes;

        LaneState L;
        float tv;
        int ti;
        const int V32 = static_cast<int>(a.vocab);
        scan_segment<DT, TOPK, false>(row, V32, static_cast<int>(u0), static_cast<int>(u1), a.k, lane, L, tv, ti, stage);
        {
            float a0, a1, b0, b1;
            unpack2(L.s, a0, a1);
            unpack2(L.t, b0, b1);
            const float chk = a0 + a1 + b0 + b1;
            if (__any_sync(kFull, chk != chk)) {
                scan_segment<DT, TOPK, true>(row, V32, static_cast<int>(u0), static_cast<int>(u1), a.k, lane, L, tv,
                                             ti, stage);
                if (L.bad) L.s = pack2(NAN, NAN);
            }
        }
        const float MX = warp_max(L.mx);
        const int am = resolve_argmax<DT>(row, a.vocab, L, MX);
        float s_lo, s_hi, t_lo, t_hi;
        unpack2(L.s, s_lo, s_hi);
        unpack2(L.t, t_lo, t_hi);
        RowTotals rt = combine(L.mref, s_lo + s_hi, t_lo + t_hi, L.mx, am);

        const int64_t w_first = (r * nv) / piece;
        const int64_t w_last = ((r + 1) * nv - 1) / piece;
        const int count = static_cast<int>(w_last - w_first + 1);
        if (count == 1) {
            write_row(a, slot, rt, tv, ti, lane);
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
        if (TOPK && lane < a.k)
            a.part_topk[(slot * kMaxPartials + my) * a.k + lane] = make_float2(tv, __int_as_float(ti));
        __threadfence();
        __syncwarp();
        unsigned prior = 0;
        if (lane == 0) prior = atomicAdd(a.ticket + slot, 1u);
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
        if (TOPK) {
            const float2 *lists = a.part_topk + slot * kMaxPartials * a.k;
            float2 e = __ldcg(lists + lane % a.k);  // list 0 seeds the merged list
            tv = lane < a.k ? e.x : -INFINITY;
            ti = lane < a.k ? __float_as_int(e.y) : INT_MAX;
            const int total_entries = count * a.k;
            for (int base_e = a.k; base_e < total_entries; base_e += 32) {
                const int idx = base_e + lane;
                float cv = -INFINITY;
                int ci = INT_MAX;
                if (idx < total_entries) {
                    const float2 f = __ldcg(lists + idx);
                    cv = f.x;
                    ci = __float_as_int(f.y);
                }
                float th = __shfl_sync(kFull, tv, a.k - 1);
                bool has = idx < total_entries && ci != INT_MAX && cv >= th;
                while (true) {
                    const unsigned lanes = __ballot_sync(kFull, has);
                    if (!lanes) break;
                    const int src = __ffs(lanes) - 1;
                    const float v = __shfl_sync(kFull, cv, src);
                    const int i = __shfl_sync(kFull, ci, src);
                    if (lane == src) has = false;
                    topk_insert(tv, ti, v, i, a.k, lane);
                    th = __shfl_sync(kFull, tv, a.k - 1);
                    has = has && cv >= th;
                }
            }
        }
        write_row(a, slot, rt, tv, ti, lane);
    }
}

template <int DT, bool TOPK>
cudaError_t launch_typed(const RowStatsArgs &a, int grid, cudaStream_t stream) {
    row_stats_kernel<DT, TOPK><<<grid, kRowThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

template <int DT, bool TOPK>
cudaError_t occupancy_typed(int *blocks) {
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, row_stats_kernel<DT, TOPK>, kRowThreads, 0);
}

}  // namespace

cudaError_t launch_row_stats(const RowStatsArgs &a, int dtype, int grid, cudaStream_t stream) {
    if (dtype == RPS_BF16)
        return a.k > 0 ? launch_typed<RPS_BF16, true>(a, grid, stream) : launch_typed<RPS_BF16, false>(a, grid, stream);
    return a.k > 0 ? launch_typed<RPS_F32, true>(a, grid, stream) : launch_typed<RPS_F32, false>(a, grid, stream);
}

cudaError_t row_stats_occupancy(int dtype, bool topk, int *blocks_per_sm) {
    if (dtype == RPS_BF16) return topk ? occupancy_typed<RPS_BF16, true>(blocks_per_sm)
                                       : occupancy_typed<RPS_BF16, false>(blocks_per_sm);
    return topk ? occupancy_typed<RPS_F32, true>(blocks_per_sm) : occupancy_typed<RPS_F32, false>(blocks_per_sm);
}

}  // namespace rps
