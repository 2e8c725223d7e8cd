// decide_device.cuh -- the per-request decision steps of one RPS step as
// block-level device functions; the decision kernels of decide.cu run them,
// one block per request.
//
//   select_request        standard commit (Eq. 2 with the fallback of
//                         Algorithm 1), M' = M \ S, pivots (Eq. 3), candidate
//                         tokens (Sec. 3.1) and the lookahead row list
//   score_request         Eq. 4 per (pivot, candidate) and N_tau (Proposition 1)
//   commit_request        commit-or-abstain and the mask after the step
//   score_commit_request  the two above for one request
// Everything here is O(L * k) words, negligible next to the row-statistics
// stream, so the code keeps dependent global-memory round trips few: a block
// first stages what it needs in shared memory with independent loads.
#pragma once

#include <cfloat>
#include <climits>

#include "rps_internal.cuh"

namespace rps {
namespace {

constexpr int kSelectThreads = 256;
constexpr int kScoreThreads = 256;
constexpr int kMaxSlots = RPS_MAX_PIVOTS * (RPS_MAX_K + 1);

// Block-wide exclusive scan of one int per thread; returns the block total.
__device__ __forceinline__ int block_excl_scan(int v, int &excl, int *warp_buf) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += n;
    }
    __syncthreads();  // warp_buf may still be read by a previous call
    if (lane == 31) warp_buf[w] = incl;
    __syncthreads();
    int before = 0, total = 0;
    for (int i = 0; i < nw; ++i) {
        if (i < w) before += warp_buf[i];
        total += warp_buf[i];
    }
    excl = before + incl - v;
    return total;
}

// Best entry of the block by (value desc, position asc); idx -1 when no thread has one.
struct Best {
    float v;
    int pos;
    int idx;
};

// Larger value first, then lower position; the entry index makes the order
// total (positions are distinct in valid input).
__device__ __forceinline__ bool better(const Best &a, const Best &b) {
    if (a.idx < 0) return false;
    if (b.idx < 0) return true;
    return a.v > b.v || (a.v == b.v && (a.pos < b.pos || (a.pos == b.pos && a.idx < b.idx)));
}

__device__ Best block_best(Best mine, Best *buf) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        Best o_;
        o_.v = __shfl_xor_sync(kFull, mine.v, o);
        o_.pos = __shfl_xor_sync(kFull, mine.pos, o);
        o_.idx = __shfl_xor_sync(kFull, mine.idx, o);
        if (better(o_, mine)) mine = o_;
    }
    __syncthreads();
    if (lane == 0) buf[w] = mine;
    __syncthreads();
    Best r = buf[0];
    for (int i = 1; i < nw; ++i)
        if (better(buf[i], r)) r = buf[i];
    return r;
}

// Brings the 128-byte line holding p into L1 (no data is returned).
__device__ __forceinline__ void prefetch_l1(const void *p) { asm volatile("prefetch.global.L1 [%0];" ::"l"(p)); }

// Pivot order as one unsigned key: larger truncated entropy first, then lower
// position (positions are distinct). The float's bits are mapped to an unsigned
// order; 0 is below every key and marks "none".
__device__ __forceinline__ uint64_t pivot_key(float v, int pos) {
    const uint32_t b = __float_as_uint(v + 0.f);  // -0 orders as +0
    const uint32_t hi = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
    return (static_cast<uint64_t>(hi) << 32) | static_cast<uint32_t>(~pos);
}

// The P <= RPS_MAX_PIVOTS largest of n distinct keys (0 = none), into out[0..P)
// in descending order: in every group of 32 (one warp, a key per lane), each
// key counts the larger keys of its group by shuffles and the best P move on,
// until one group is left. With P <= 16 a level takes n to at most n / 2 + 16,
// so the levels end and each one's output fits t_a / t_b of n / 2 + 32 keys.
static_assert(RPS_MAX_PIVOTS <= 16 && RPS_MAX_COMMIT_K <= 16, "block_top_keys halves the keys per level");
__device__ void block_top_keys(const uint64_t *keys, int n, int P, uint64_t *t_a, uint64_t *t_b, uint64_t *out) {
    const int tid = threadIdx.x, lane = tid & 31;
    const uint64_t *cur = keys;
    uint64_t *nxt = t_a;
    for (;;) {
        const int groups = (n + 31) / 32;
        uint64_t *dst = groups <= 1 ? out : nxt;
        const int n_dst = groups <= 1 ? P : groups * P;
        for (int t = tid; t < n_dst; t += blockDim.x) dst[t] = 0ull;
        __syncthreads();
        // (blockDim.x is a multiple of 32: a warp's lanes hold one whole group)
        for (int t0 = tid & ~31; t0 < n; t0 += blockDim.x) {
            const int t = t0 + lane;
            const uint64_t me = t < n ? cur[t] : 0ull;
            int rank = 0;
#pragma unroll
            for (int u = 0; u < 32; ++u) rank += __shfl_sync(kFull, me, u) > me;
            if (me != 0ull && rank < P) dst[(groups <= 1 ? 0 : (t0 >> 5) * P) + rank] = me;
        }
        __syncthreads();
        if (groups <= 1) return;
        cur = nxt;
        nxt = nxt == t_a ? t_b : t_a;
        n = groups * P;
    }
}

// Dynamic shared memory of select_kernel: per masked position, then a constant.
constexpr int kSelectBytesPerPos = sizeof(uint64_t) + sizeof(uint64_t) + 4 * sizeof(float) + 4 * sizeof(int32_t) + 1;
constexpr int kSelectBytesExtra = 2 * 32 * sizeof(uint64_t) + 16;
__host__ __device__ constexpr int half_keys(int L) { return L / 2 + 32; }

// Shared-memory scratch of select_request apart from its per-position arrays.
struct SelectShared {
    uint64_t winners[RPS_MAX_PIVOTS];  // also the commit set's keys (top-k rules)
    Best best_buf[kSelectThreads / 32];
    int warp_buf[kSelectThreads / 32];
    int piv_i[RPS_MAX_PIVOTS];  // index of pivot j in M'
    int piv_nc[RPS_MAX_PIVOTS];
    int n_piv_s;
    int br_off[RPS_MAX_PIVOTS * RPS_MAX_K + 1];
    int16_t valid_b[RPS_MAX_PIVOTS * RPS_MAX_K];  // the m-th valid branch
};
constexpr size_t kSelectSharedBytes = (sizeof(SelectShared) + 15) / 16 * 16;

// Shared memory select_request needs for L masked positions.
__host__ __device__ constexpr size_t select_smem_bytes(int L) {
    return kSelectSharedBytes + static_cast<size_t>(L) * kSelectBytesPerPos + kSelectBytesExtra;
}

// Steps 1-6 of one request (standard commit, M', pivots, candidates, lookahead
// rows) by one block of at most kSelectThreads threads, in `smem` of
// select_smem_bytes(L). The statistics are read through L2 (__ldcg). With
// `wait_inside` the block calls pdl_wait itself after staging the mask and
// writing the defaults: the base statistics are the only input the previous
// launch writes.
__device__ void select_request(const SelectArgs &a, int q, unsigned char *smem, bool wait_inside) {
    const int tid = threadIdx.x;
    const int L = a.L, P = a.P, K = a.K, NB = P * K;
    const int64_t base = static_cast<int64_t>(q) * L;
    const rps_pivots &o = a.out;

    SelectShared &sh = *reinterpret_cast<SelectShared *>(smem);
    int *warp_buf = sh.warp_buf;
    Best *best_buf = sh.best_buf;
    int *piv_i = sh.piv_i;
    int *piv_nc = sh.piv_nc;
    uint64_t *winners = sh.winners;
    int &n_piv_s = sh.n_piv_s;
    int *br_off = sh.br_off;
    int16_t *valid_b = sh.valid_b;
    uint64_t *keys = reinterpret_cast<uint64_t *>(smem + kSelectSharedBytes);  // rank keys (0: none)
    uint64_t *t_a = keys + L;                                 // tournament buffers
    uint64_t *t_b = t_a + half_keys(L);
    float *pm = reinterpret_cast<float *>(t_b + half_keys(L));  // P^max of mask entry k
    float *mu = pm + L;                                         // retained mass
    float *ht = mu + L;                                         // truncated entropy
    float *hh = ht + L;                                         // entropy
    int32_t *pos = reinterpret_cast<int32_t *>(hh + L);         // position
    int32_t *am = pos + L;                                      // argmax token
    int32_t *rk = am + L;                                       // M' entry i -> mask entry
    int32_t *rp = rk + L;                                       // M' entry i -> position
    uint8_t *in_S = reinterpret_cast<uint8_t *>(rp + L);

    // Stage this request's statistics over the whole capacity, so that these
    // loads do not wait for the mask count (entries past it are never used),
    // and write the defaults.
    int cnt = a.mask_cnt[q];
    for (int k = tid; k < L; k += blockDim.x) pos[k] = a.mask_pos[base + k];
    if (cnt < 0 || cnt > L) {
        if (tid == 0) flag_error(a.err, RPS_DEVERR_MASK);
        cnt = cnt < 0 ? 0 : L;
    }
    for (int j = tid; j < P; j += blockDim.x) {
        o.pivot_k[q * P + j] = -1;
        o.pivot_pos[q * P + j] = -1;
        o.n_cand[q * P + j] = 0;
    }
    for (int i = tid; i < P * K; i += blockDim.x) o.cand_tok[static_cast<int64_t>(q) * P * K + i] = -1;
    for (int b = tid; b < NB; b += blockDim.x) {
        o.branch_valid[q * NB + b] = 0;
        o.branch_off[q * NB + b] = 0;
        o.branch_cnt[q * NB + b] = 0;
    }
    if (wait_inside) pdl_wait();
    for (int k = tid; k < L; k += blockDim.x) {
        pm[k] = __ldcg(a.pmax + base + k);
        mu[k] = __ldcg(a.mu + base + k);
        ht[k] = __ldcg(a.htrunc + base + k);
        hh[k] = __ldcg(a.H + base + k);
        am[k] = __ldcg(a.argmax + base + k);
        // the pivots' candidate step reads a row's zmax and top-k list: bring
        // them to L1 now, while the statistics load, instead of a round trip later
        if (k < cnt) {
            prefetch_l1(a.zmax + base + k);
            prefetch_l1(a.topk_logit + (base + k) * a.k_max);
            prefetch_l1(a.topk_idx + (base + k) * a.k_max);
        }
    }
    __syncthreads();

    // Step 1: the commit set S (Eq. 2).
    if (a.commit_rule == RPS_COMMIT_THRESHOLD) {
        // S = {i in M : P^max_i >= tau}; fallback to the most confident row
        int any = 0;
        for (int k = tid; k < cnt; k += blockDim.x) {
            const uint8_t f = pm[k] >= a.tau;
            in_S[k] = f;
            any |= f;
        }
        any = __syncthreads_or(any);
        if (!any && cnt > 0) {
            Best mine{-INFINITY, INT_MAX, -1};
            for (int k = tid; k < cnt; k += blockDim.x) {
                Best c{pm[k], pos[k], k};
                if (!(c.v == c.v)) c.v = -INFINITY;  // NaN statistics never win
                if (better(c, mine)) mine = c;
            }
            const Best b = block_best(mine, best_buf);
            if (tid == 0) in_S[b.idx] = 1;
            __syncthreads();
        }
    } else {
        // S = the commit_k rows of largest P^max (or of smallest H), lower position
        // on ties, NaN statistics last: a tournament on keys over M
        for (int k = tid; k < cnt; k += blockDim.x) {
            float v = a.commit_rule == RPS_COMMIT_TOPK_CONFIDENCE ? pm[k] : -hh[k];
            if (!(v == v)) v = -INFINITY;
            keys[k] = pivot_key(v, pos[k]);
        }
        __syncthreads();
        block_top_keys(keys, cnt, a.commit_k, t_a, t_b, winners);
        for (int k = tid; k < cnt; k += blockDim.x) {
            uint8_t f = 0;
            for (int j = 0; j < a.commit_k; ++j) f |= keys[k] == winners[j];
            in_S[k] = f;
        }
        __syncthreads();
    }

    // Order-preserving split of M into S (committed) and M'.
    int n_commit = 0;
    for (int t0 = 0; t0 < cnt; t0 += blockDim.x) {
        const int k = t0 + tid;
        const int f = k < cnt ? in_S[k] : 0;
        int excl;
        const int tot = block_excl_scan(f, excl, warp_buf);
        if (k < cnt) {
            if (f) {
                o.commit_pos[base + n_commit + excl] = pos[k];
                o.commit_tok[base + n_commit + excl] = am[k];
            } else {
                const int r = k - (n_commit + excl);
                rk[r] = k;
                rp[r] = pos[k];
                if (a.pivot_rule == RPS_PIVOT_TRUNCATED_ENTROPY)
                    keys[r] = mu[k] >= a.tau_pivot && ht[k] == ht[k] ? pivot_key(ht[k], pos[k]) : 0ull;
                else {
                    const float v = a.pivot_rule == RPS_PIVOT_MAX_CONFIDENCE ? pm[k] : hh[k];
                    keys[r] = v == v ? pivot_key(v, pos[k]) : 0ull;
                }
                o.rem_k[base + r] = k;
                o.rem_pos[base + r] = pos[k];
            }
        }
        n_commit += tot;
    }
    const int n_rem = cnt - n_commit;
    if (tid == 0) {
        o.n_commit[q] = n_commit;
        o.rem_cnt[q] = n_rem;
        o.n_branch_rows[q] = 0;
    }
    if (n_rem == 0) {
        if (tid == 0) o.state[q] = RPS_STATE_DONE;
        return;
    }
    __syncthreads();

    // Steps 3-4: the P best feasible rows of M' by their key -- truncated
    // entropy under the mass constraint (Eq. 3), or confidence, or entropy --
    // lower position on ties, by a tournament on the keys.
    {
        block_top_keys(keys, n_rem, P, t_a, t_b, winners);
        if (tid == 0) {
            int c = 0;
            while (c < P && winners[c] != 0ull) ++c;
            n_piv_s = c;
        }
        __syncthreads();
        for (int i = tid; i < n_rem; i += blockDim.x) {
            const uint64_t key = keys[i];
            if (key == 0ull) continue;
            for (int j = 0; j < n_piv_s; ++j) {
                if (key == winners[j]) {
                    piv_i[j] = i;
                    o.pivot_k[q * P + j] = rk[i];
                    o.pivot_pos[q * P + j] = rp[i];
                }
            }
        }
        __syncthreads();
    }
    const int n_piv = n_piv_s;
    if (n_piv == 0) {
        if (tid == 0) o.state[q] = RPS_STATE_NO_FEASIBLE;
        return;
    }

    // Step 5: candidates z_v - zmax >= log r in rank order, at most K: one warp
    // per pivot, lane t tests rank t of T_i (all loads at once).
    {
        const int lane = tid & 31, w = tid >> 5, nw = blockDim.x >> 5;
        for (int j = w; j < n_piv; j += nw) {
            const int64_t row = base + rk[piv_i[j]];
            const double zmax = a.zmax[row];
            bool pass = false;
            int tok = -1;
            if (lane < a.k_max) {
                const double zt = a.topk_logit[row * a.k_max + lane];
                tok = a.topk_idx[row * a.k_max + lane];
                pass = zt - zmax >= a.log_r;
            }
            const unsigned m = __ballot_sync(kFull, pass);
            const int rank = __popc(m & ((1u << lane) - 1u));
            if (pass && rank < K) o.cand_tok[(static_cast<int64_t>(q) * P + j) * K + rank] = tok;
            if (lane == 0) {
                const int nc = min(__popc(m), K);
                piv_nc[j] = nc;
                o.n_cand[q * P + j] = nc;
            }
        }
    }
    __syncthreads();
    int searchable = 0;
    for (int j = 0; j < n_piv; ++j) searchable |= piv_nc[j] >= 2;
    if (!searchable) {
        if (tid == 0) o.state[q] = RPS_STATE_NO_CANDIDATES;
        return;
    }

    // Step 6: branch b = j * K + c lists M' without pivot j; the lists of the
    // valid branches are laid end to end in branch order (one warp, 32
    // branches at a time).
    if (tid < 32) {
        const int lane = tid;
        int off = 0, m = 0;
        for (int b0 = 0; b0 < NB; b0 += 32) {
            const int b = b0 + lane;
            const int j = b / K, c = b % K;
            const bool valid = b < NB && j < n_piv && piv_nc[j] >= 2 && c < piv_nc[j];
            const unsigned vm = __ballot_sync(kFull, valid);
            const int before = __popc(vm & ((1u << lane) - 1u));
            if (b < NB) {
                const int my_off = off + before * (n_rem - 1);
                if (valid) valid_b[m + before] = static_cast<int16_t>(b);
                br_off[b] = my_off;
                o.branch_off[q * NB + b] = my_off;
                o.branch_cnt[q * NB + b] = valid ? n_rem - 1 : 0;
                o.branch_valid[q * NB + b] = valid;
            }
            off += __popc(vm) * (n_rem - 1);
            m += __popc(vm);
        }
        if (lane == 0) {
            br_off[NB] = off;
            o.n_branch_rows[q] = off;
            o.state[q] = RPS_STATE_SEARCH;
        }
    }
    __syncthreads();
    // one warp per valid branch: M' in order, without the branch's pivot
    {
        const int lane = tid & 31, w = tid >> 5, nw = blockDim.x >> 5;
        const int n_valid = n_rem > 1 ? br_off[NB] / (n_rem - 1) : 0;
        for (int m = w; m < n_valid; m += nw) {
            const int b = valid_b[m];
            const int pi = piv_i[b / K];
            int32_t *rows = o.branch_rows + (static_cast<int64_t>(q) * NB * L + br_off[b]) * 3;
            // the (q, 1 + b, pos) triples, one per lane: the warp's three stores
            // cover 384 consecutive bytes
            for (int d = lane; d < n_rem - 1; d += 32) {
                const int i = d < pi ? d : d + 1;
                rows[3 * d] = q;
                rows[3 * d + 1] = 1 + b;
                rows[3 * d + 2] = rp[i];
            }
        }
    }
}

__device__ __forceinline__ float load_logit(const void *data, int dtype, int64_t e) {
    if (dtype == RPS_BF16)
        return __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t *>(data)[e]) << 16);
    return static_cast<const float *>(data)[e];
}

// Pivot-selection facts of one request, staged in shared memory with
// independent loads so that the scoring and the decision need no further
// dependent global round trips.
struct PivotView {
    int state, n_rem;
    int pivot_k[RPS_MAX_PIVOTS];
    int pivot_pos[RPS_MAX_PIVOTS];
    int n_cand[RPS_MAX_PIVOTS];
    int branch_off[RPS_MAX_PIVOTS * RPS_MAX_K];
    int branch_cnt[RPS_MAX_PIVOTS * RPS_MAX_K];
    int cand_tok[RPS_MAX_PIVOTS * RPS_MAX_K];
    uint8_t branch_valid[RPS_MAX_PIVOTS * RPS_MAX_K];
};

// Dynamic shared memory of the score / commit kernels: rem_k and rem_pos of one request.
__host__ __device__ constexpr size_t view_smem_bytes(int L) { return 2 * static_cast<size_t>(L) * sizeof(int32_t); }

__device__ void stage_view(const rps_pivots &pv, int q, int L, int P, int K, PivotView &v, int32_t *rem_k,
                           int32_t *rem_pos) {
    const int NB = P * K;
    const int64_t base = static_cast<int64_t>(q) * L;
    if (threadIdx.x == 0) {
        v.state = pv.state[q];
        v.n_rem = pv.rem_cnt[q];
    }
    for (int j = threadIdx.x; j < P; j += blockDim.x) {
        v.pivot_k[j] = pv.pivot_k[q * P + j];
        v.pivot_pos[j] = pv.pivot_pos[q * P + j];
        v.n_cand[j] = pv.n_cand[q * P + j];
    }
    for (int b = threadIdx.x; b < NB; b += blockDim.x) {
        v.branch_valid[b] = pv.branch_valid[q * NB + b];
        v.branch_off[b] = pv.branch_off[q * NB + b];
        v.branch_cnt[b] = pv.branch_cnt[q * NB + b];
        v.cand_tok[b] = pv.cand_tok[static_cast<int64_t>(q) * NB + b];
    }
    // the whole capacity: entries past rem_cnt are read but never used
    for (int i = threadIdx.x; i < L; i += blockDim.x) {
        rem_k[i] = pv.rem_k[base + i];
        rem_pos[i] = pv.rem_pos[base + i];
    }
}

// Per-slot values of the Eq. 4 score that do not read the lookahead rows'
// statistics: the plausibility term, and for [MASK] the whole sum over D_j.
struct SlotPre {
    float sum;   // [MASK]: sum of the anchor entropies over D_j (tokens: added later)
    int count;   // [MASK]: #{pmax >= tau} over D_j
    float la;    // log a
    int scored;  // the slot is scored
};

// First half of the scores, one warp per (pivot, slot): what comes from the
// pivots, the anchor statistics and the anchor logits.
__device__ void score_prepare(const ScoreArgs &a, int q, const PivotView &v, const int32_t *rem_k, SlotPre *pre) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const int L = a.L, P = a.P, K = a.K;
    const int64_t base = static_cast<int64_t>(q) * L;
    int n_rem = v.n_rem;
    if (n_rem < 0 || n_rem > L) n_rem = 0;  // select flags bad counts; never index past the capacity
    for (int slot = w; slot < P * (K + 1); slot += nw) {
        const int j = slot / (K + 1), c = slot % (K + 1);
        const int pk = v.pivot_k[j];
        bool scored = v.state == RPS_STATE_SEARCH && pk >= 0 && pk < L && v.n_cand[j] >= 2;
        if (scored && c < K) scored = v.branch_valid[j * K + c] != 0;
        float sum = 0.f, la = NAN;
        int count = 0;
        if (scored) {
            if (c < K) {
                const int b = j * K + c;
                const int tok = v.cand_tok[b];
                const int p = v.pivot_pos[j];
                float z = NAN;
                if (tok < 0 || tok >= a.vocab) {
                    if (lane == 0) flag_error(a.err, RPS_DEVERR_TOKEN);
                } else if (p < 0 || p >= a.n_pos) {
                    if (lane == 0) flag_error(a.err, RPS_DEVERR_ROW_INDEX);
                } else {
                    z = load_logit(a.anchor_data, a.dtype, q * a.req_stride + a.branch_offset + p * a.pos_stride + tok);
                }
                la = z - a.a_lse[base + pk];
            } else {
                for (int i = lane; i < n_rem; i += 32) {
                    const int k = rem_k[i];
                    if (k == pk || k < 0 || k >= L) continue;
                    sum += a.a_H[base + k];
                    count += a.a_pmax[base + k] >= a.tau;
                }
                sum = warp_sum(sum);
                count = warp_sum_int(count);
                la = a.a_zmax[base + pk] - a.a_lse[base + pk];
            }
        }
        if (lane == 0) pre[slot] = SlotPre{sum, count, la, scored ? 1 : 0};
    }
}

// Second half, one warp per (pivot, slot): the token slots' sums over the
// lookahead rows, then every slot's score; the scores are also kept in `sc`.
__device__ void score_finish(const ScoreArgs &a, int q, const PivotView &v, const SlotPre *pre, float *sc) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const int L = a.L, P = a.P, K = a.K, NB = P * K;
    int n_rem = v.n_rem;
    if (n_rem < 0 || n_rem > L) n_rem = 0;
    for (int slot = w; slot < P * (K + 1); slot += nw) {
        const int j = slot / (K + 1), c = slot % (K + 1);
        const int64_t o = (static_cast<int64_t>(q) * P + j) * (K + 1) + c;
        const SlotPre sp = pre[slot];
        float mean_H = NAN, log_a = NAN, score = NAN;
        int n_tau = -1;
        if (sp.scored) {
            float sum = sp.sum;
            int count = sp.count;
            if (c < K) {
                const int b = j * K + c;
                const int64_t first = static_cast<int64_t>(q) * NB * L + v.branch_off[b];
                const int n = v.branch_cnt[b];
                // lane's entries lane + 32 t in order; eight at a time in flight
                constexpr int kIn = 8;
                for (int i0 = 0; i0 < n; i0 += 32 * kIn) {
                    float h[kIn], pm[kIn];
#pragma unroll
                    for (int u = 0; u < kIn; ++u) {
                        const int i = i0 + u * 32 + lane;
                        h[u] = i < n ? __ldcg(a.b_H + first + i) : 0.f;
                        pm[u] = i < n ? __ldcg(a.b_pmax + first + i) : 0.f;
                    }
#pragma unroll
                    for (int u = 0; u < kIn; ++u) {
                        if (i0 + u * 32 + lane < n) {
                            sum += h[u];
                            count += pm[u] >= a.tau;
                        }
                    }
                }
                sum = warp_sum(sum);
                count = warp_sum_int(count);
            }
            const int n = n_rem - 1;
            mean_H = n > 0 ? sum / static_cast<float>(n) : 0.f;
            n_tau = count;
            log_a = sp.la;
            score = -mean_H + (a.lambda != 0.f ? a.lambda * sp.la : 0.f);
        }
        if (lane == 0) {
            a.out.mean_H[o] = mean_H;
            a.out.n_tau[o] = n_tau;
            a.out.log_a[o] = log_a;
            a.out.score[o] = score;
            if (sc) sc[slot] = score;
        }
    }
}

// Commit decision of one request by one warp; `s_req` holds the request's scores.
__device__ void commit_request(const CommitArgs &a, int q, const PivotView &v, const int32_t *rem_pos,
                               const float *s_req) {
    const int lane = threadIdx.x & 31;
    const int L = a.L, P = a.P, K = a.K;
    const int64_t base = static_cast<int64_t>(q) * L;
    const int state = v.state;

    // Best slot and gain of the pivot held by this lane.
    int best = -1;
    float gain = NAN;
    int ppos = INT_MAX;
    bool wins = false;
    if (lane < P && state == RPS_STATE_SEARCH && v.pivot_pos[lane] >= 0 && v.n_cand[lane] >= 2) {
        const float *s = s_req + lane * (K + 1);
        best = K;
        for (int c = 0; c < K; ++c) {
            if (!v.branch_valid[lane * K + c]) continue;
            if (s[c] > s[best]) best = c;
        }
        gain = s[best] - s[K];
        ppos = v.pivot_pos[lane];
        wins = best < K && gain > 0.f;
    }
    if (lane < P) {
        a.out.best_slot[q * P + lane] = best;
        a.out.gain[q * P + lane] = gain;
    }
    // Pivot with the largest positive gain, lower position on ties.
    float g = wins ? gain : -INFINITY;
    int p = wins ? ppos : INT_MAX;
    int j = wins ? lane : -1;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float og = __shfl_xor_sync(kFull, g, o);
        const int op = __shfl_xor_sync(kFull, p, o);
        const int oj = __shfl_xor_sync(kFull, j, o);
        if (oj >= 0 && (j < 0 || og > g || (og == g && op < p))) {
            g = og;
            p = op;
            j = oj;
        }
    }
    const int win_best = __shfl_sync(kFull, best, j >= 0 ? j : 0);
    int commit_pos = -1;
    if (lane == 0) {
        int winner, ctok = -1;
        float margin = 0.f;
        if (state == RPS_STATE_DONE) winner = RPS_WIN_DONE;
        else if (state != RPS_STATE_SEARCH) winner = RPS_WIN_SKIP;
        else if (j < 0) winner = RPS_WIN_ANCHOR;
        else {
            winner = j * K + win_best;
            commit_pos = v.pivot_pos[j];
            ctok = v.cand_tok[j * K + win_best];
            margin = g;
        }
        a.out.winner[q] = winner;
        a.out.commit_pos[q] = commit_pos;
        a.out.commit_tok[q] = ctok;
        a.out.margin[q] = margin;
    }
    commit_pos = __shfl_sync(kFull, commit_pos, 0);

    // Mask after the step: M' without the committed pivot, in order.
    int n_rem = state == RPS_STATE_DONE ? 0 : v.n_rem;
    if (n_rem < 0 || n_rem > L) n_rem = 0;
    int kept = 0;
    for (int i0 = 0; i0 < n_rem; i0 += 32) {
        const int i = i0 + lane;
        const int32_t rp = i < n_rem ? rem_pos[i] : -1;
        const bool keep = i < n_rem && rp != commit_pos;
        const unsigned m = __ballot_sync(kFull, keep);
        if (keep) a.out.mask_pos[base + kept + __popc(m & ((1u << lane) - 1u))] = rp;
        kept += __popc(m);
    }
    if (lane == 0) a.out.mask_cnt[q] = kept;
}

// Score and commit of one request by one block, in `smem` of
// score_commit_smem_bytes(L): the view, the per-slot values and scores, then
// rem_k and rem_pos. With `wait_inside`, the block calls pdl_wait itself once
// the first half is done: that half reads nothing the lookahead rows' launch
// (the previous kernel on the stream) writes.
struct ScoreShared {
    PivotView v;
    SlotPre pre[kMaxSlots];
    float sc[kMaxSlots];
};
constexpr size_t kScoreSharedBytes = (sizeof(ScoreShared) + 15) / 16 * 16;

__host__ __device__ constexpr size_t score_commit_smem_bytes(int L) { return kScoreSharedBytes + view_smem_bytes(L); }

__device__ void score_commit_request(const ScoreArgs &s, const CommitArgs &c, int q, unsigned char *smem,
                                     bool wait_inside) {
    ScoreShared &sh = *reinterpret_cast<ScoreShared *>(smem);
    int32_t *view = reinterpret_cast<int32_t *>(smem + kScoreSharedBytes);
    stage_view(s.piv, q, s.L, s.P, s.K, sh.v, view, view + s.L);
    __syncthreads();
    score_prepare(s, q, sh.v, view, sh.pre);
    if (wait_inside) pdl_wait();
    __syncthreads();
    score_finish(s, q, sh.v, sh.pre, sh.sc);
    __syncthreads();
    if (threadIdx.x < 32) commit_request(c, q, sh.v, view + s.L, sh.sc);
}

}  // namespace
}  // namespace rps
