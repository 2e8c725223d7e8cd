/*
 * rps_oracle.c -- CPU oracle of the Ripple-Pivot Search (RPS) scoring path.
 *
 * TEST INFRASTRUCTURE, NOT PART OF THE LIBRARY. Only the test-suite, the
 * package smoke check and the benchmark's CPU-baseline leg load this code. It
 * shares no source, header, table or helper with the CUDA path.
 *
 * Plain, slow and single threaded: every quantity is computed in fp64 straight
 * from its definition in the paper, in the paper's order and notation.
 *
 *   row statistics   notation of Sec. 2 (H(p_i), P_i^max), Eq. 1 (argmax), Eq. 3
 *                    (top-k_max support T_i, retained mass mu_i, truncated entropy)
 *   standard commit  Eq. 2, confidence-aware rule, with the fallback of
 *                    Algorithm 1 when no position passes the threshold
 *   pivot selection  Eq. 3 and the adaptive candidate set C of Sec. 3.1
 *                    ("Lookahead scoring"); skip rules of Algorithm 1
 *   benefit score    Eq. 4, mean downstream entropy and N_tau of Proposition 1
 *   commit decision  argmax of Eq. 4 over C including [MASK]; Algorithm 1
 *
 * Readings of points the paper leaves open (ties, several pivots per step,
 * n = 0, lambda = 0, the layout of several requests) are stated beside the code
 * that applies them.
 *
 * Data layout (shared with the C ABI only by specification, not by code):
 *   base / anchor statistics   [req * L + k], k = index in the request's mask list
 *   pivots                     [req * P + j]
 *   candidate tokens           [(req * P + j) * K + c]
 *   lookahead branches         b = j * K + c, NB = P * K; logits branch 1 + b
 *   branch row lists           per request, capacity NB * L, three int32 each
 *                              (req, 1 + b, pos); branch b's rows start at
 *                              branch_off[req * NB + b]
 *   branch scores              [(req * P + j) * (K + 1) + c], c == K is [MASK]
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { ORACLE_F32 = 0, ORACLE_BF16 = 1 };

/* Per-request state after pivot selection. */
enum {
    STATE_SEARCH = 0,        /* lookahead branches are scored this step */
    STATE_DONE = 1,          /* no masked position left after the standard commit */
    STATE_NO_FEASIBLE = 2,   /* no position satisfies mu_i >= tau_pivot */
    STATE_NO_CANDIDATES = 3  /* every pivot has at most one non-[MASK] candidate */
};

/* Rules for the commit set S (Eq. 2) and for the pivots (Eq. 3 and the
 * ablation strategies of Sec. 4.3). */
enum { COMMIT_THRESHOLD = 0, COMMIT_TOPK_CONFIDENCE = 1, COMMIT_TOPK_LOW_ENTROPY = 2 };
enum { PIVOT_TRUNCATED_ENTROPY = 0, PIVOT_MAX_CONFIDENCE = 1, PIVOT_MAX_ENTROPY = 2 };

/* Winner codes of the commit decision (>= 0: lookahead branch index b). */
enum { WIN_ANCHOR = -1, WIN_SKIP = -2, WIN_DONE = -3 };

/* Element v of a logit row, widened to double (bf16 is the top half of binary32). */
static double logit_at(const void *row, int32_t dtype, int64_t v)
{
    if (dtype == ORACLE_BF16) {
        uint32_t bits = (uint32_t)((const uint16_t *)row)[v] << 16;
        float f;
        memcpy(&f, &bits, sizeof f);
        return (double)f;
    }
    return (double)((const float *)row)[v];
}

typedef struct {
    double z;
    int64_t v;
} ranked_token;

/* Rank order of tokens: higher logit first; equal logits, lower token id first. */
static int rank_before(const void *pa, const void *pb)
{
    const ranked_token *a = (const ranked_token *)pa, *b = (const ranked_token *)pb;
    if (a->z > b->z) return -1;
    if (a->z < b->z) return 1;
    if (a->v < b->v) return -1;
    if (a->v > b->v) return 1;
    return 0;
}

/*
 * Row statistics of n_rows logit rows. Row n starts at element row_off[n] of
 * `logits` and holds V logits z_v. With p_v = exp(z_v - lse):
 *   zmax   = max_v z_v,  argmax = lowest v attaining it                 (Eq. 1)
 *   lse    = zmax + log sum_v exp(z_v - zmax)
 *   H      = -sum_v p_v log p_v, with 0 log 0 = 0                       (H(p_i), Sec. 2)
 *   pmax   = max_v p_v = exp(zmax - lse)                                (P_i^max, Sec. 2)
 *   T      = the k tokens ranked first by (z desc, v asc)               (T_i, Eq. 3)
 *   mu     = sum_{v in T} p_v                                           (mu_i, Eq. 3)
 *   htrunc = -sum_{v in T} p_v log p_v, probabilities not renormalised  (Eq. 3)
 * k == 0 skips T, mu and htrunc. topk_idx / topk_logit receive T in rank order
 * ([n][k]). A row without a finite logit gets NaN statistics and argmax -1.
 * Returns the number of such rows.
 */
int64_t rps_oracle_row_stats(const void *logits, int32_t dtype, int64_t V,
                             const int64_t *row_off, int64_t n_rows, int32_t k,
                             double *zmax, double *lse, double *H, double *pmax,
                             double *mu, double *htrunc, int32_t *argmax,
                             int32_t *topk_idx, double *topk_logit)
{
    const size_t esize = dtype == ORACLE_BF16 ? 2 : 4;
    ranked_token *order = k > 0 ? (ranked_token *)malloc((size_t)V * sizeof *order) : NULL;
    int64_t bad = 0;
    for (int64_t n = 0; n < n_rows; ++n) {
        const void *row = (const char *)logits + (size_t)row_off[n] * esize;

        /* Maximum logit and the lowest token attaining it. */
        double m = -INFINITY;
        int64_t am = -1;
        for (int64_t v = 0; v < V; ++v) {
            double z = logit_at(row, dtype, v);
            if (z > m) { m = z; am = v; }
        }
        if (!isfinite(m)) {
            zmax[n] = lse[n] = H[n] = pmax[n] = NAN;
            if (mu) mu[n] = NAN;
            if (htrunc) htrunc[n] = NAN;
            argmax[n] = -1;
            for (int32_t t = 0; t < k; ++t) { topk_idx[n * k + t] = -1; topk_logit[n * k + t] = NAN; }
            ++bad;
            continue;
        }

        /* log-sum-exp, shifted by the maximum. */
        double sum = 0.0;
        for (int64_t v = 0; v < V; ++v) sum += exp(logit_at(row, dtype, v) - m);
        const double l = m + log(sum);

        /* Shannon entropy of p, with log p_v = z_v - lse. */
        double h = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            double z = logit_at(row, dtype, v);
            double p = exp(z - l);
            if (p > 0.0) h -= p * (z - l);
        }

        zmax[n] = m;
        lse[n] = l;
        H[n] = h;
        pmax[n] = exp(m - l);
        argmax[n] = (int32_t)am;

        if (k > 0) {
            /* T_i: full sort by rank order, keep the first k. */
            for (int64_t v = 0; v < V; ++v) { order[v].z = logit_at(row, dtype, v); order[v].v = v; }
            qsort(order, (size_t)V, sizeof *order, rank_before);
            double mass = 0.0, ht = 0.0;
            for (int32_t t = 0; t < k; ++t) {
                double p = exp(order[t].z - l);
                mass += p;
                if (p > 0.0) ht -= p * (order[t].z - l);
                topk_idx[n * k + t] = (int32_t)order[t].v;
                topk_logit[n * k + t] = order[t].z;
            }
            mu[n] = mass;
            htrunc[n] = ht;
        }
    }
    free(order);
    return bad;
}

/*
 * Standard commit and pivot selection for n_req requests (one decoding step).
 *
 * Inputs: the mask lists (mask_pos[req * L + k], k < mask_cnt[req], distinct
 * positions) and the base statistics of those rows, as produced by
 * rps_oracle_row_stats (topk_* with row stride k_max).
 *
 * 1. S = {i in M : P_i^max >= tau} (Eq. 2, confidence-aware rule). If S is
 *    empty, S = {argmax_{i in M} P_i^max} (Algorithm 1), ties to the lower
 *    position. Each i in S is committed to argmax_v p_i(v) (Eq. 1).
 * 2. M' = M \ S, kept in mask-list order (rem_k / rem_pos). M' empty: DONE.
 * 3. Feasible rows: mu_i >= tau_pivot (Eq. 3). None: NO_FEASIBLE.
 * 4. Pivots: the P feasible rows of largest truncated entropy, taken one at a
 *    time, ties to the lower position. For P = 1 this is i* of Eq. 3.
 *    (Reading: several pivot slots per step are scored side by side; fewer
 *    feasible rows than P leave the last slots empty, pivot_k = -1.)
 * 5. Candidates of a pivot: tokens v of T_{i*} with p(v) >= r * P^max
 *    (Sec. 3.1), evaluated as z_v - zmax >= log r, in rank order, at most K of
 *    them. A pivot with fewer than two candidates is not searched (Algorithm 1
 *    skips when |C \ {MASK}| <= 1). No searchable pivot: NO_CANDIDATES.
 * 6. Lookahead branch b = j * K + c is valid when pivot j is searched and
 *    c < n_cand[j]. Its rows are M' without pivot j, in M' order; they are
 *    listed per request as (req, 1 + b, pos) triples.
 */
void rps_oracle_select_pivots(
    int32_t n_req, int32_t L, const int32_t *mask_pos, const int32_t *mask_cnt,
    const double *zmax, const double *pmax, const int32_t *argmax,
    const double *mu, const double *htrunc, const double *H,
    const int32_t *topk_idx, const double *topk_logit, int32_t k_max,
    double r, double tau_pivot, double tau, int32_t P, int32_t K,
    int32_t commit_rule, int32_t commit_k, int32_t pivot_rule,
    int32_t *n_commit, int32_t *commit_pos, int32_t *commit_tok,
    int32_t *rem_cnt, int32_t *rem_k, int32_t *rem_pos, int32_t *state,
    int32_t *pivot_k, int32_t *pivot_pos, int32_t *n_cand, int32_t *cand_tok,
    uint8_t *branch_valid, int32_t *branch_off, int32_t *branch_cnt,
    int32_t *n_branch_rows, int32_t *branch_rows)
{
    const int32_t NB = P * K;
    const double log_r = log(r);
    unsigned char *in_S = (unsigned char *)malloc((size_t)(L > 0 ? L : 1));
    unsigned char *taken = (unsigned char *)malloc((size_t)(L > 0 ? L : 1));

    for (int32_t q = 0; q < n_req; ++q) {
        const int32_t cnt = mask_cnt[q];
        const int64_t base = (int64_t)q * L;
        n_commit[q] = 0;
        rem_cnt[q] = 0;
        n_branch_rows[q] = 0;
        for (int32_t j = 0; j < P; ++j) {
            pivot_k[q * P + j] = -1;
            pivot_pos[q * P + j] = -1;
            n_cand[q * P + j] = 0;
            for (int32_t c = 0; c < K; ++c) cand_tok[(q * P + j) * K + c] = -1;
        }
        for (int32_t b = 0; b < NB; ++b) {
            branch_valid[q * NB + b] = 0;
            branch_off[q * NB + b] = 0;
            branch_cnt[q * NB + b] = 0;
        }
        if (cnt == 0) { state[q] = STATE_DONE; continue; }

        /* Step 1: the commit set S (Eq. 2). */
        if (commit_rule == COMMIT_THRESHOLD) {
            /* confidence-aware rule, with the fallback of Algorithm 1 */
            int any = 0;
            for (int32_t k = 0; k < cnt; ++k) {
                in_S[k] = pmax[base + k] >= tau;
                any |= in_S[k];
            }
            if (!any) {
                int32_t best = 0;
                for (int32_t k = 1; k < cnt; ++k) {
                    double a = pmax[base + k], b = pmax[base + best];
                    if (a > b || (a == b && mask_pos[base + k] < mask_pos[base + best])) best = k;
                }
                in_S[best] = 1;
            }
        } else {
            /* top-k rules: the commit_k rows of largest P^max, or of smallest H,
             * lower position on ties; NaN statistics rank as -inf */
            for (int32_t k = 0; k < cnt; ++k) in_S[k] = 0;
            for (int32_t m = 0; m < commit_k && m < cnt; ++m) {
                int32_t best = -1;
                double bv = 0.0;
                for (int32_t k = 0; k < cnt; ++k) {
                    if (in_S[k]) continue;
                    double v = commit_rule == COMMIT_TOPK_CONFIDENCE ? pmax[base + k] : -H[base + k];
                    if (v != v) v = -INFINITY;
                    if (best < 0 || v > bv || (v == bv && mask_pos[base + k] < mask_pos[base + best])) {
                        best = k;
                        bv = v;
                    }
                }
                in_S[best] = 1;
            }
        }
        for (int32_t k = 0; k < cnt; ++k) {
            if (in_S[k]) {
                commit_pos[base + n_commit[q]] = mask_pos[base + k];
                commit_tok[base + n_commit[q]] = argmax[base + k];
                n_commit[q]++;
            } else {
                rem_k[base + rem_cnt[q]] = k;
                rem_pos[base + rem_cnt[q]] = mask_pos[base + k];
                rem_cnt[q]++;
            }
        }

        /* Step 2: nothing left to search. */
        if (rem_cnt[q] == 0) { state[q] = STATE_DONE; continue; }

        /* Step 3: the rows a pivot may come from. Eq. 3: the probability-mass
         * constraint; the ablation strategies take every row of M' (NaN
         * statistics excepted). */
        int n_feasible = 0;
        for (int32_t i = 0; i < rem_cnt[q]; ++i) {
            const int32_t k = rem_k[base + i];
            taken[i] = 0;
            if (pivot_rule == PIVOT_TRUNCATED_ENTROPY) {
                if (mu[base + k] >= tau_pivot) n_feasible++;
            } else {
                const double v = pivot_rule == PIVOT_MAX_CONFIDENCE ? pmax[base + k] : H[base + k];
                if (v == v) n_feasible++;
            }
        }
        if (n_feasible == 0) { state[q] = STATE_NO_FEASIBLE; continue; }

        /* Step 4: pivots, the P best feasible rows: by truncated entropy (Eq. 3),
         * by confidence or by entropy; lower position on ties. */
        for (int32_t j = 0; j < P; ++j) {
            int32_t best = -1;
            double bv = 0.0;
            for (int32_t i = 0; i < rem_cnt[q]; ++i) {
                int32_t k = rem_k[base + i];
                if (taken[i]) continue;
                double v;
                if (pivot_rule == PIVOT_TRUNCATED_ENTROPY) {
                    if (!(mu[base + k] >= tau_pivot)) continue;
                    v = htrunc[base + k];
                } else {
                    v = pivot_rule == PIVOT_MAX_CONFIDENCE ? pmax[base + k] : H[base + k];
                    if (v != v) continue;
                }
                if (best < 0 || v > bv || (v == bv && rem_pos[base + i] < rem_pos[base + best])) {
                    best = i;
                    bv = v;
                }
            }
            if (best < 0) break;
            taken[best] = 1;
            pivot_k[q * P + j] = rem_k[base + best];
            pivot_pos[q * P + j] = rem_pos[base + best];
        }

        /* Step 5: adaptive candidate set of each pivot. */
        int searchable = 0;
        for (int32_t j = 0; j < P; ++j) {
            int32_t k = pivot_k[q * P + j];
            if (k < 0) continue;
            int32_t nc = 0;
            for (int32_t t = 0; t < k_max && nc < K; ++t) {
                double zt = topk_logit[(base + k) * k_max + t];
                if (zt - zmax[base + k] >= log_r)
                    cand_tok[(q * P + j) * K + nc++] = topk_idx[(base + k) * k_max + t];
            }
            n_cand[q * P + j] = nc;
            if (nc >= 2) searchable = 1;
        }
        if (!searchable) { state[q] = STATE_NO_CANDIDATES; continue; }
        state[q] = STATE_SEARCH;

        /* Step 6: lookahead branches and their rows. */
        int32_t *rows = branch_rows + (int64_t)q * NB * L * 3;
        int32_t used = 0;
        for (int32_t j = 0; j < P; ++j) {
            int32_t kp = pivot_k[q * P + j];
            int searched = kp >= 0 && n_cand[q * P + j] >= 2;
            for (int32_t c = 0; c < K; ++c) {
                int32_t b = j * K + c;
                branch_off[q * NB + b] = used;
                if (!searched || c >= n_cand[q * P + j]) continue;
                branch_valid[q * NB + b] = 1;
                for (int32_t i = 0; i < rem_cnt[q]; ++i) {
                    if (rem_k[base + i] == kp) continue;
                    rows[used * 3 + 0] = q;
                    rows[used * 3 + 1] = 1 + b;
                    rows[used * 3 + 2] = rem_pos[base + i];
                    used++;
                }
                branch_cnt[q * NB + b] = used - branch_off[q * NB + b];
            }
        }
        n_branch_rows[q] = used;
    }
    free(in_S);
    free(taken);
}

/*
 * Downstream-benefit score of every candidate (Eq. 4) for the requests whose
 * state is SEARCH.
 *
 * For pivot j with downstream set D_j = M' \ {i*_j} and n = |D_j| = |M'| - 1:
 *   mean_H  = (1/n) sum_{i in D_j} H(p_i^c)                (H-bar_c, Sec. 3.2)
 *   n_tau   = #{i in D_j : max_v p_i^c(v) >= tau}          (N_tau(c), Prop. 1)
 *   log_a   = log p_anchor(c) at the pivot, or log P_anchor^max for [MASK]
 *   score   = -mean_H + lambda * log_a                     (Eq. 4)
 * Token candidates read branch b = j * K + c (statistics in the compact
 * per-request layout, capacity NB * L, branch_off / branch_cnt); [MASK] reads the
 * anchor branch, i.e. the anchor statistics of the rows of D_j. p_anchor(c) uses
 * the anchor logit of token c at the pivot (anchor_logits, element strides).
 * Readings: n == 0 gives mean_H = 0 (Prop. 1 assumes n > 0); lambda == 0 drops
 * the plausibility term, so a zero anchor probability cannot produce 0 * -inf.
 * Slots that are not scored get NaN and n_tau = -1.
 */
void rps_oracle_score_branches(
    int32_t n_req, int32_t L, int32_t P, int32_t K,
    const int32_t *state, const int32_t *rem_cnt, const int32_t *rem_k,
    const int32_t *pivot_k, const int32_t *pivot_pos, const int32_t *n_cand,
    const int32_t *cand_tok, const uint8_t *branch_valid,
    const int32_t *branch_off, const int32_t *branch_cnt,
    const double *branch_H, const double *branch_pmax,
    const double *anchor_H, const double *anchor_pmax,
    const double *anchor_lse, const double *anchor_zmax,
    const void *anchor_logits, int32_t dtype,
    int64_t anchor_req_stride, int64_t anchor_pos_stride,
    double lambda, double tau,
    double *mean_H, int32_t *n_tau, double *log_a, double *score)
{
    const int32_t NB = P * K;
    for (int32_t q = 0; q < n_req; ++q) {
        const int64_t base = (int64_t)q * L;
        for (int32_t j = 0; j < P; ++j) {
            for (int32_t c = 0; c <= K; ++c) {
                int64_t o = ((int64_t)q * P + j) * (K + 1) + c;
                mean_H[o] = NAN; n_tau[o] = -1; log_a[o] = NAN; score[o] = NAN;
            }
            int32_t kp = pivot_k[q * P + j];
            if (state[q] != STATE_SEARCH || kp < 0 || n_cand[q * P + j] < 2) continue;
            const int32_t n = rem_cnt[q] - 1;

            for (int32_t c = 0; c <= K; ++c) {
                int64_t o = ((int64_t)q * P + j) * (K + 1) + c;
                double sum_H = 0.0;
                int32_t count = 0;
                double la;
                if (c < K) {
                    int32_t b = j * K + c;
                    if (!branch_valid[q * NB + b]) continue;
                    int64_t first = (int64_t)q * NB * L + branch_off[q * NB + b];
                    for (int32_t i = 0; i < branch_cnt[q * NB + b]; ++i) {
                        sum_H += branch_H[first + i];
                        if (branch_pmax[first + i] >= tau) count++;
                    }
                    int32_t tok = cand_tok[(q * P + j) * K + c];
                    const char *row = (const char *)anchor_logits +
                        ((size_t)q * anchor_req_stride + (size_t)pivot_pos[q * P + j] * anchor_pos_stride) *
                        (dtype == ORACLE_BF16 ? 2 : 4);
                    la = logit_at(row, dtype, tok) - anchor_lse[base + kp];
                } else {
                    for (int32_t i = 0; i < rem_cnt[q]; ++i) {
                        int32_t k = rem_k[base + i];
                        if (k == kp) continue;
                        sum_H += anchor_H[base + k];
                        if (anchor_pmax[base + k] >= tau) count++;
                    }
                    la = anchor_zmax[base + kp] - anchor_lse[base + kp];
                }
                double h_bar = n > 0 ? sum_H / n : 0.0;
                mean_H[o] = h_bar;
                n_tau[o] = count;
                log_a[o] = la;
                score[o] = -h_bar + (lambda != 0.0 ? lambda * la : 0.0);
            }
        }
    }
}

/*
 * Commit decision (Eq. 4 argmax over C including [MASK]; Algorithm 1).
 *
 * For each searched pivot j: c*_j = argmax of score over its valid token slots
 * and [MASK]. Ties favour [MASK] (abstaining is the conservative default that
 * the [MASK] plausibility P^max is meant to give, Sec. 3.1), then the candidate
 * of higher rank. gain_j = score(c*_j) - score([MASK]) >= 0.
 * Reading for several pivots: commit at most one pivot per step, the one with
 * the largest gain_j > 0, ties to the lower position. For P = 1 this is
 * exactly Algorithm 1.
 * Outputs: winner (b = j * K + c when a token is committed, WIN_ANCHOR when
 * every searched pivot keeps [MASK], WIN_SKIP for NO_FEASIBLE / NO_CANDIDATES,
 * WIN_DONE for DONE), the committed (pivot position, token), the margin
 * gain of the winner, per-pivot best slot / gain, and the mask after the step:
 * M' without the committed pivot, in M' order.
 */
void rps_oracle_commit(
    int32_t n_req, int32_t L, int32_t P, int32_t K,
    const int32_t *state, const int32_t *pivot_pos, const int32_t *n_cand,
    const int32_t *cand_tok, const uint8_t *branch_valid, const double *score,
    const int32_t *rem_cnt, const int32_t *rem_pos,
    int32_t *best_slot, double *gain,
    int32_t *winner, int32_t *commit_pos, int32_t *commit_tok, double *margin,
    int32_t *out_mask_cnt, int32_t *out_mask_pos)
{
    const int32_t NB = P * K;
    for (int32_t q = 0; q < n_req; ++q) {
        const int64_t base = (int64_t)q * L;
        int32_t win_j = -1;
        for (int32_t j = 0; j < P; ++j) {
            best_slot[q * P + j] = -1;
            gain[q * P + j] = NAN;
            if (state[q] != STATE_SEARCH || pivot_pos[q * P + j] < 0 || n_cand[q * P + j] < 2) continue;
            const double *s = score + ((int64_t)q * P + j) * (K + 1);
            int32_t best = K; /* [MASK] */
            for (int32_t c = 0; c < K; ++c) {
                if (!branch_valid[q * NB + j * K + c]) continue;
                if (s[c] > s[best]) best = c;
            }
            best_slot[q * P + j] = best;
            gain[q * P + j] = s[best] - s[K];
            if (best < K && gain[q * P + j] > 0.0) {
                if (win_j < 0 || gain[q * P + j] > gain[q * P + win_j] ||
                    (gain[q * P + j] == gain[q * P + win_j] &&
                     pivot_pos[q * P + j] < pivot_pos[q * P + win_j]))
                    win_j = j;
            }
        }

        commit_pos[q] = -1;
        commit_tok[q] = -1;
        margin[q] = 0.0;
        if (state[q] == STATE_DONE) winner[q] = WIN_DONE;
        else if (state[q] != STATE_SEARCH) winner[q] = WIN_SKIP;
        else if (win_j < 0) winner[q] = WIN_ANCHOR;
        else {
            int32_t c = best_slot[q * P + win_j];
            winner[q] = win_j * K + c;
            commit_pos[q] = pivot_pos[q * P + win_j];
            commit_tok[q] = cand_tok[(q * P + win_j) * K + c];
            margin[q] = gain[q * P + win_j];
        }

        int32_t n = 0;
        for (int32_t i = 0; i < rem_cnt[q]; ++i) {
            if (rem_pos[base + i] == commit_pos[q]) continue;
            out_mask_pos[base + n++] = rem_pos[base + i];
        }
        out_mask_cnt[q] = n;
    }
}
