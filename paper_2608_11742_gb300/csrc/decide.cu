// decide.cu -- per-request decision kernels of one RPS step.
//
//   select_kernel        standard commit (Eq. 2 with the fallback of Algorithm 1),
//                        M' = M \ S, pivots (Eq. 3), candidate tokens (Sec. 3.1)
//                        and the lookahead row list       -> rps_select_pivots
//   score_kernel         Eq. 4 per (pivot, candidate) and N_tau (Proposition 1)
//                                                         -> rps_score_branches
//   commit_kernel        commit-or-abstain and the mask after the step
//                                                         -> rps_commit
//   score_commit_kernel  both of the above in one launch  -> rps_score_and_commit
// One block per request; everything here is O(L * k) words, negligible next to
// the row-statistics stream, so the kernels are written to keep dependent
// global-memory round trips few: each block first stages what it needs in
// shared memory with independent loads.
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

__device__ __forceinline__ bool better(const Best &a, const Best &b) {
    if (a.idx < 0) return false;
    if (b.idx < 0) return true;
    return a.v > b.v || (a.v == b.v && a.pos < b.pos);
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

// Dynamic shared memory of select_kernel per masked position.
constexpr int kSelectBytesPerPos = 3 * sizeof(float) + 3 * sizeof(int32_t) + 2;

__global__ void __launch_bounds__(kSelectThreads) select_kernel(const SelectArgs a) {
    pdl_wait();
    pdl_launch_next();
    const int q = blockIdx.x;
    const int tid = threadIdx.x;
    const int L = a.L, P = a.P, K = a.K, NB = P * K;
    const int64_t base = static_cast<int64_t>(q) * L;
    const rps_pivots &o = a.out;

    __shared__ int warp_buf[kSelectThreads / 32];
    __shared__ Best best_buf[kSelectThreads / 32];
    __shared__ int piv_i[RPS_MAX_PIVOTS];  // index of pivot j in M'
    __shared__ int piv_nc[RPS_MAX_PIVOTS];
    extern __shared__ __align__(16) unsigned char sel_smem[];
    float *pm = reinterpret_cast<float *>(sel_smem);  // P^max of mask entry k
    float *mu = pm + L;                                // retained mass
    float *ht = mu + L;                                // truncated entropy
    int32_t *pos = reinterpret_cast<int32_t *>(ht + L);  // position
    int32_t *am = pos + L;                               // argmax token
    int32_t *rk = am + L;                                // M' entry i -> mask entry
    uint8_t *in_S = reinterpret_cast<uint8_t *>(rk + L);
    uint8_t *taken = in_S + L;

    int cnt = a.mask_cnt[q];
    if (cnt < 0 || cnt > L) {
        if (tid == 0) flag_error(a.err, RPS_DEVERR_MASK);
        cnt = cnt < 0 ? 0 : L;
    }

    // Stage this request's statistics (independent loads) and write the defaults.
    for (int k = tid; k < cnt; k += blockDim.x) {
        pm[k] = a.pmax[base + k];
        mu[k] = a.mu[base + k];
        ht[k] = a.htrunc[base + k];
        pos[k] = a.mask_pos[base + k];
        am[k] = a.argmax[base + k];
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
    __syncthreads();

    // Step 1: S = {i in M : P^max_i >= tau}; fallback to the most confident row.
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
    for (int i = tid; i < n_rem; i += blockDim.x) taken[i] = 0;
    __syncthreads();

    // Steps 3-4: feasibility (mu >= tau_pivot) and pivots by truncated entropy.
    int n_piv = 0;
    for (int j = 0; j < P; ++j) {
        Best mine{-INFINITY, INT_MAX, -1};
        for (int i = tid; i < n_rem; i += blockDim.x) {
            const int k = rk[i];
            if (taken[i] || !(mu[k] >= a.tau_pivot)) continue;
            Best c{ht[k], pos[k], i};
            if (!(c.v == c.v)) continue;
            if (better(c, mine)) mine = c;
        }
        const Best b = block_best(mine, best_buf);
        if (b.idx < 0) break;
        if (tid == 0) {
            taken[b.idx] = 1;
            piv_i[j] = b.idx;
            o.pivot_k[q * P + j] = rk[b.idx];
            o.pivot_pos[q * P + j] = b.pos;
        }
        n_piv = j + 1;
        __syncthreads();
    }
    if (n_piv == 0) {
        if (tid == 0) o.state[q] = RPS_STATE_NO_FEASIBLE;
        return;
    }

    // Step 5: candidates z_v - zmax >= log r in rank order, at most K.
    if (tid < n_piv) {
        const int j = tid;
        const int64_t row = base + rk[piv_i[j]];
        const double zmax = a.zmax[row];
        int nc = 0;
        for (int t = 0; t < a.k_max && nc < K; ++t) {
            const double zt = a.topk_logit[row * a.k_max + t];
            if (zt - zmax >= a.log_r)
                o.cand_tok[(static_cast<int64_t>(q) * P + j) * K + nc++] = a.topk_idx[row * a.k_max + t];
        }
        piv_nc[j] = nc;
        o.n_cand[q * P + j] = nc;
    }
    __syncthreads();
    int searchable = 0;
    for (int j = 0; j < n_piv; ++j) searchable |= piv_nc[j] >= 2;
    if (!searchable) {
        if (tid == 0) o.state[q] = RPS_STATE_NO_CANDIDATES;
        return;
    }

    // Step 6: branch b = j * K + c lists M' without pivot j.
    int off = 0;
    for (int j = 0; j < P; ++j) {
        const bool searched = j < n_piv && piv_nc[j] >= 2;
        for (int c = 0; c < K; ++c) {
            const int b = j * K + c;
            const bool valid = searched && c < piv_nc[j];
            const int n = valid ? n_rem - 1 : 0;
            if (tid == 0) {
                o.branch_off[q * NB + b] = off;
                o.branch_cnt[q * NB + b] = n;
                o.branch_valid[q * NB + b] = valid;
            }
            if (valid) {
                const int pi = piv_i[j];
                int32_t *rows = o.branch_rows + (static_cast<int64_t>(q) * NB * L + off) * 3;
                for (int i = tid; i < n_rem; i += blockDim.x) {
                    if (i == pi) continue;
                    const int d = i < pi ? i : i - 1;
                    rows[d * 3 + 0] = q;
                    rows[d * 3 + 1] = 1 + b;
                    rows[d * 3 + 2] = pos[rk[i]];
                }
            }
            off += n;
        }
    }
    if (tid == 0) {
        o.n_branch_rows[q] = off;
        o.state[q] = RPS_STATE_SEARCH;
    }
}

__device__ __forceinline__ float load_logit(const void *data, int dtype, int64_t e) {
    if (dtype == RPS_BF16)
        return __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t *>(data)[e]) << 16);
    return static_cast<const float *>(data)[e];
}

// Pivot-selection facts of one request, staged in shared memory.
struct PivotView {
    int state, n_rem;
    int pivot_k[RPS_MAX_PIVOTS];
    int pivot_pos[RPS_MAX_PIVOTS];
    int n_cand[RPS_MAX_PIVOTS];
};

__device__ void stage_pivots(const rps_pivots &pv, int q, int P, PivotView &v) {
    if (threadIdx.x == 0) {
        v.state = pv.state[q];
        v.n_rem = pv.rem_cnt[q];
    }
    for (int j = threadIdx.x; j < P; j += blockDim.x) {
        v.pivot_k[j] = pv.pivot_k[q * P + j];
        v.pivot_pos[j] = pv.pivot_pos[q * P + j];
        v.n_cand[j] = pv.n_cand[q * P + j];
    }
}

// Eq. 4 scores of one request, one warp per (pivot, slot); also kept in `sc`.
__device__ void score_request(const ScoreArgs &a, int q, const PivotView &v, float *sc) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const int L = a.L, P = a.P, K = a.K, NB = P * K;
    const int64_t base = static_cast<int64_t>(q) * L;
    const rps_pivots &pv = a.piv;
    for (int slot = w; slot < P * (K + 1); slot += nw) {
        const int j = slot / (K + 1), c = slot % (K + 1);
        const int64_t o = (static_cast<int64_t>(q) * P + j) * (K + 1) + c;
        const int pk = v.pivot_k[j];
        float mean_H = NAN, log_a = NAN, score = NAN;
        int n_tau = -1;
        bool scored = v.state == RPS_STATE_SEARCH && pk >= 0 && v.n_cand[j] >= 2;
        if (scored && c < K) scored = pv.branch_valid[q * NB + j * K + c] != 0;
        if (scored) {
            float sum = 0.f;
            int count = 0;
            float la;
            if (c < K) {
                const int b = j * K + c;
                const int64_t first = static_cast<int64_t>(q) * NB * L + pv.branch_off[q * NB + b];
                const int n = pv.branch_cnt[q * NB + b];
                for (int i = lane; i < n; i += 32) {
                    sum += a.b_H[first + i];
                    count += a.b_pmax[first + i] >= a.tau;
                }
                const int tok = pv.cand_tok[(static_cast<int64_t>(q) * P + j) * K + c];
                const int p = v.pivot_pos[j];
                if (tok < 0 || tok >= a.vocab) {
                    if (lane == 0) flag_error(a.err, RPS_DEVERR_TOKEN);
                    la = NAN;
                } else if (p < 0 || p >= a.n_pos) {
                    if (lane == 0) flag_error(a.err, RPS_DEVERR_ROW_INDEX);
                    la = NAN;
                } else {
                    const int64_t e = q * a.req_stride + a.branch_offset + p * a.pos_stride + tok;
                    la = load_logit(a.anchor_data, a.dtype, e) - a.a_lse[base + pk];
                }
            } else {
                for (int i = lane; i < v.n_rem; i += 32) {
                    const int k = pv.rem_k[base + i];
                    if (k == pk) continue;
                    sum += a.a_H[base + k];
                    count += a.a_pmax[base + k] >= a.tau;
                }
                la = a.a_zmax[base + pk] - a.a_lse[base + pk];
            }
            sum = warp_sum(sum);
            count = warp_sum_int(count);
            const int n = v.n_rem - 1;
            mean_H = n > 0 ? sum / static_cast<float>(n) : 0.f;
            n_tau = count;
            log_a = la;
            score = -mean_H + (a.lambda != 0.f ? a.lambda * la : 0.f);
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

// Commit decision of one request by one warp; `s` holds the request's scores.
__device__ void commit_request(const CommitArgs &a, int q, const float *s_req) {
    const int lane = threadIdx.x & 31;
    const int L = a.L, P = a.P, K = a.K, NB = P * K;
    const int64_t base = static_cast<int64_t>(q) * L;
    const rps_pivots &pv = a.piv;
    const int state = pv.state[q];

    // Best slot and gain of the pivot held by this lane.
    int best = -1;
    float gain = NAN;
    int ppos = INT_MAX;
    bool wins = false;
    if (lane < P && state == RPS_STATE_SEARCH && pv.pivot_pos[q * P + lane] >= 0 && pv.n_cand[q * P + lane] >= 2) {
        const float *s = s_req + lane * (K + 1);
        best = K;
        for (int c = 0; c < K; ++c) {
            if (!pv.branch_valid[q * NB + lane * K + c]) continue;
            if (s[c] > s[best]) best = c;
        }
        gain = s[best] - s[K];
        ppos = pv.pivot_pos[q * P + lane];
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
            commit_pos = pv.pivot_pos[q * P + j];
            ctok = pv.cand_tok[(static_cast<int64_t>(q) * P + j) * K + win_best];
            margin = g;
        }
        a.out.winner[q] = winner;
        a.out.commit_pos[q] = commit_pos;
        a.out.commit_tok[q] = ctok;
        a.out.margin[q] = margin;
    }
    commit_pos = __shfl_sync(kFull, commit_pos, 0);

    // Mask after the step: M' without the committed pivot, in order.
    const int n_rem = state == RPS_STATE_DONE ? 0 : pv.rem_cnt[q];
    int kept = 0;
    for (int i0 = 0; i0 < n_rem; i0 += 32) {
        const int i = i0 + lane;
        const int32_t rp = i < n_rem ? pv.rem_pos[base + i] : -1;
        const bool keep = i < n_rem && rp != commit_pos;
        const unsigned m = __ballot_sync(kFull, keep);
        if (keep) a.out.mask_pos[base + kept + __popc(m & ((1u << lane) - 1u))] = rp;
        kept += __popc(m);
    }
    if (lane == 0) a.out.mask_cnt[q] = kept;
}

__global__ void __launch_bounds__(kScoreThreads) score_kernel(const ScoreArgs a) {
    pdl_wait();
    pdl_launch_next();
    __shared__ PivotView v;
    stage_pivots(a.piv, blockIdx.x, a.P, v);
    __syncthreads();
    score_request(a, blockIdx.x, v, nullptr);
}

__global__ void __launch_bounds__(32) commit_kernel(const CommitArgs a) {
    pdl_wait();
    pdl_launch_next();
    const int q = blockIdx.x;
    commit_request(a, q, a.score + static_cast<int64_t>(q) * a.P * (a.K + 1));
}

__global__ void __launch_bounds__(kScoreThreads) score_commit_kernel(const ScoreArgs s, const CommitArgs c) {
    pdl_wait();
    pdl_launch_next();
    __shared__ PivotView v;
    __shared__ float sc[kMaxSlots];
    stage_pivots(s.piv, blockIdx.x, s.P, v);
    __syncthreads();
    score_request(s, blockIdx.x, v, sc);
    __syncthreads();
    if (threadIdx.x < 32) commit_request(c, blockIdx.x, sc);
}

}  // namespace

cudaError_t launch_select(const SelectArgs &a, cudaStream_t stream) {
    const size_t smem = static_cast<size_t>(a.L) * kSelectBytesPerPos + 16;
    if (smem > 48 * 1024) {
        const cudaError_t e =
            cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    return launch_pdl(select_kernel, dim3(a.n_req), dim3(kSelectThreads), smem, stream, a);
}

cudaError_t launch_score(const ScoreArgs &a, cudaStream_t stream) {
    return launch_pdl(score_kernel, dim3(a.n_req), dim3(kScoreThreads), 0, stream, a);
}

cudaError_t launch_commit(const CommitArgs &a, cudaStream_t stream) {
    return launch_pdl(commit_kernel, dim3(a.n_req), dim3(32), 0, stream, a);
}

cudaError_t launch_score_commit(const ScoreArgs &s, const CommitArgs &c, cudaStream_t stream) {
    return launch_pdl(score_commit_kernel, dim3(s.n_req), dim3(kScoreThreads), 0, stream, s, c);
}

}  // namespace rps
