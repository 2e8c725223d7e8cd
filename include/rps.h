/*
 * rps.h -- C ABI of the GB300 scoring path of Ripple-Pivot Search (RPS).
 *
 * One decoding step of RPS (Algorithm 1 of the paper) on logits already in
 * device memory:
 *
 *   rps_score_step      per-row statistics of the masked rows: entropy H(p_i),
 *                       confidence P_i^max, argmax (Eq. 1), top-k_max support
 *                       T_i, retained mass mu_i and truncated entropy (Eq. 3)
 *   rps_select_pivots   confidence-aware standard commit S (Eq. 2, with the
 *                       fallback of Algorithm 1), remaining set M' = M \ S,
 *                       pivot selection (Eq. 3), adaptive candidate tokens
 *                       (Sec. 3.1) and the list of lookahead rows to score
 *   rps_score_step      again, on the lookahead branches' rows
 *   rps_score_branches  downstream-benefit score of every candidate (Eq. 4),
 *                       with the eligible-commit count N_tau (Proposition 1)
 *   rps_commit          commit-or-abstain decision (Eq. 4 argmax over C
 *                       including [MASK]; Algorithm 1) and the mask after the step
 *   rps_run_step        the whole step above in one call
 *
 * Conventions
 *   - Every array pointer is a caller-owned DEVICE pointer unless stated.
 *     The library never allocates device memory; per-call scratch comes from a
 *     caller-owned workspace sized by rps_workspace_bytes.
 *   - Calls are asynchronous on the given stream (NULL = legacy default stream)
 *     and return as soon as the work is enqueued.
 *   - Host-detectable errors (NULL pointers, out-of-range sizes or parameters,
 *     misaligned logits) return an error status before anything is enqueued and
 *     write nothing.
 *   - Bad DATA found by a kernel (a row descriptor outside the logit tensor, a
 *     mask count above capacity, a row without a finite logit) does not trap:
 *     the kernel skips the offending item, writes NaN / -1 where it stands, and
 *     ORs a bit into a sticky per-device error word that rps_poll_device_status
 *     reads and clears.
 *   - Results are deterministic for a given input and launch configuration.
 *   - Layout per request q of n_req, with L positions of capacity:
 *       mask / base statistics      [q * L + k], k = index in q's mask list
 *       pivot slot j of P           [q * P + j]
 *       candidate c of K            [(q * P + j) * K + c]
 *       lookahead branch b          b = j * K + c of NB = P * K; it is branch
 *                                   1 + b of the logit tensor (branch 0 = base)
 *       branch scores               [(q * P + j) * (K + 1) + c], c == K is [MASK]
 */
#ifndef RPS_H
#define RPS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st *rps_stream_t;

typedef enum {
    RPS_OK = 0,
    RPS_ERR_INVALID_ARG = 1, /* rejected on the host; nothing was enqueued */
    RPS_ERR_UNSUPPORTED = 2, /* well-formed request outside this build's limits */
    RPS_ERR_CUDA = 3,        /* a CUDA runtime call (launch, attribute query) failed */
    RPS_ERR_DEVICE = 4,      /* a kernel flagged bad data; see rps_poll_device_status */
    RPS_ERR_TIMEOUT = 5      /* reserved; a kernel wait that gives up is reported as RPS_DEVERR_TIMEOUT */
} rps_status;

/* Bits of the device error word. */
#define RPS_DEVERR_ROW_INDEX 0x1u  /* row descriptor outside the logit tensor */
#define RPS_DEVERR_NONFINITE 0x2u  /* a scored row holds NaN or no finite logit */
#define RPS_DEVERR_MASK 0x4u       /* mask count above capacity or position out of range */
#define RPS_DEVERR_TOKEN 0x8u      /* candidate token outside the vocabulary */
#define RPS_DEVERR_TIMEOUT 0x10u   /* a bounded wait for an asynchronous copy gave up; the call's
                                      outputs are incomplete and its workspace is marked unhealthy */
#define RPS_DEVERR_WORKSPACE 0x20u /* the workspace was marked unhealthy by an earlier call that gave
                                      up (or holds a stale ticket): the call wrote no statistics;
                                      rps_workspace_init makes the workspace usable again */

typedef enum { RPS_F32 = 0, RPS_BF16 = 1 } rps_dtype;

/* Per-request state after rps_select_pivots. */
typedef enum {
    RPS_STATE_SEARCH = 0,       /* lookahead branches are scored this step */
    RPS_STATE_DONE = 1,         /* M' is empty after the standard commit (Algorithm 1 break) */
    RPS_STATE_NO_FEASIBLE = 2,  /* no row has mu_i >= tau_pivot: skip the search (Eq. 3) */
    RPS_STATE_NO_CANDIDATES = 3 /* no pivot has two candidates: skip (|C \ MASK| <= 1) */
} rps_state;

/* Winner codes written by rps_commit (>= 0 is the committed branch b). */
#define RPS_WIN_ANCHOR (-1) /* every searched pivot keeps [MASK]: reuse the anchor's logits */
#define RPS_WIN_SKIP (-2)   /* search skipped: the next step needs a fresh forward pass */
#define RPS_WIN_DONE (-3)   /* nothing left to decode in this block */

/* Commit-set rules (Eq. 2) and pivot rules (Eq. 3; the pivot strategies the
 * paper's ablation compares, Sec. 4.3). */
#define RPS_COMMIT_THRESHOLD 0        /* S = {i : P^max_i >= tau}, else the most confident row */
#define RPS_COMMIT_TOPK_CONFIDENCE 1  /* S = the commit_k rows of largest P^max */
#define RPS_COMMIT_TOPK_LOW_ENTROPY 2 /* S = the commit_k rows of smallest H */
#define RPS_PIVOT_TRUNCATED_ENTROPY 0 /* Eq. 3: largest truncated entropy among mu_i >= tau_pivot */
#define RPS_PIVOT_MAX_CONFIDENCE 1    /* largest P^max in M', no mass constraint */
#define RPS_PIVOT_MAX_ENTROPY 2       /* largest H in M', no mass constraint */

/* Limits of this build. */
#define RPS_MAX_K 32        /* k_max */
#define RPS_MAX_COMMIT_K 16 /* commit_k of the top-k commit rules */
#define RPS_MAX_PIVOTS 16   /* P */
#define RPS_MAX_POS 4096    /* L */
#define RPS_MAX_SEGMENTS 1024

/* Hyper-parameters (Sec. 4 "Implementation details": k_max = 10, r = 0.1,
 * tau_pivot = 0.9 / 0.95, lambda in [0.1, 0.5]; Appendix C: tau = 0.9). */
typedef struct {
    int32_t k_max;            /* |T_i| of Eq. 3, 1..RPS_MAX_K */
    float r;                  /* reachability ratio of the candidate set, (0, 1] */
    float tau_pivot;          /* probability-mass constraint of Eq. 3 */
    float tau;                /* confidence threshold of Eq. 2 (and of N_tau) */
    float lambda;             /* plausibility weight of Eq. 4, >= 0 */
    int32_t n_pivots;         /* P: pivot slots scored side by side, 1..RPS_MAX_PIVOTS */
    int32_t tokens_per_pivot; /* K: candidate tokens per pivot, 1..k_max */
    int32_t pivot_rule;       /* RPS_PIVOT_*; 0 is the paper's rule */
    int32_t commit_rule;      /* RPS_COMMIT_*; 0 is the paper's rule */
    int32_t commit_k;         /* k of the top-k commit rules, 1..RPS_MAX_COMMIT_K (ignored by rule 0) */
} rps_params;

/* A logit tensor [n_req][n_branch][n_pos][vocab] in device memory. The vocab
 * dimension is contiguous; the other strides are in elements. `data` must be
 * 16-byte aligned and every stride a multiple of 16 bytes, so that each row
 * starts on a 16-byte boundary; vocab itself is unrestricted. */
typedef struct {
    const void *data;
    int32_t dtype; /* rps_dtype */
    int32_t n_req, n_branch, n_pos;
    int64_t vocab;
    int64_t req_stride, branch_stride, pos_stride;
} rps_logits;

/* Rows to score, grouped in n_seg segments of capacity cap. Entry i of segment s
 * is rows[(s * cap + i) * 3 + {0,1,2}] = (req, branch, pos) and its statistics go
 * to slot s * cap + i of the output arrays. Only i < seg_cnt[s] is read
 * (seg_cnt is a device array, or NULL for "all cap entries"); pos < 0 marks an
 * entry to skip (its slot is not written).
 * Mask form: with rows == NULL, entry i of segment s is
 * (s, mask_branch, mask_pos[s * cap + i]), so a request's masked rows (seg_cnt =
 * mask_cnt, cap = L) are scored without building a descriptor list. */
typedef struct {
    const int32_t *rows;
    const int32_t *seg_cnt;
    int32_t n_seg;
    int32_t cap;
    const int32_t *mask_pos;
    int32_t mask_branch;
} rps_row_list;

/* Per-row statistics, structure of arrays, one entry per slot. zmax is the
 * largest logit, lse = log sum_v exp(z_v), pmax = exp(zmax - lse). topk_idx /
 * topk_logit hold T_i in rank order (logit descending, then token id
 * ascending), k_max entries per slot; topk_idx == NULL selects the
 * statistics-only mode (mu, htrunc, topk_* untouched). */
typedef struct {
    float *zmax, *lse, *H, *pmax;
    int32_t *argmax;
    float *mu, *htrunc;
    int32_t *topk_idx;
    float *topk_logit;
} rps_row_stats;

/* Outputs of rps_select_pivots (all device arrays). */
typedef struct {
    int32_t *n_commit;      /* [n_req] |S| */
    int32_t *commit_pos;    /* [n_req][L] positions of S in mask order */
    int32_t *commit_tok;    /* [n_req][L] their greedy tokens (Eq. 1) */
    int32_t *rem_cnt;       /* [n_req] |M'| */
    int32_t *rem_k;         /* [n_req][L] mask-list index of each M' entry */
    int32_t *rem_pos;       /* [n_req][L] position of each M' entry */
    int32_t *state;         /* [n_req] rps_state */
    int32_t *pivot_k;       /* [n_req][P] mask-list index of pivot j, -1 if empty */
    int32_t *pivot_pos;     /* [n_req][P] position of pivot j, -1 if empty */
    int32_t *n_cand;        /* [n_req][P] candidate tokens of pivot j */
    int32_t *cand_tok;      /* [n_req][P][K] candidate tokens in rank order, -1 padded */
    uint8_t *branch_valid;  /* [n_req][NB] 1 when branch b is scored */
    int32_t *branch_off;    /* [n_req][NB] first entry of branch b in its request's list */
    int32_t *branch_cnt;    /* [n_req][NB] entries of branch b (|M'| - 1 when valid) */
    int32_t *n_branch_rows; /* [n_req] entries in the request's list */
    int32_t *branch_rows;   /* [n_req][NB * L][3] (q, 1 + b, pos): an rps_row_list with
                               n_seg = n_req, cap = NB * L, seg_cnt = n_branch_rows */
} rps_pivots;

/* Outputs of rps_score_branches, [n_req][P][K + 1] each (slot K is [MASK]);
 * slots that are not scored hold NaN and n_tau = -1. */
typedef struct {
    float *mean_H;  /* mean downstream entropy H-bar_c */
    int32_t *n_tau; /* N_tau(c) of Proposition 1 */
    float *log_a;   /* log p_anchor(c), log P_anchor^max for [MASK] */
    float *score;   /* Eq. 4 */
} rps_branch_scores;

/* Outputs of rps_commit. */
typedef struct {
    int32_t *best_slot; /* [n_req][P] argmax slot of each searched pivot (K = [MASK]) */
    float *gain;        /* [n_req][P] score(best) - score([MASK]) */
    int32_t *winner;    /* [n_req] branch b, or RPS_WIN_ANCHOR / _SKIP / _DONE */
    int32_t *commit_pos, *commit_tok; /* [n_req] committed pivot and token, -1 if none */
    float *margin;      /* [n_req] gain of the committed pivot, 0 if none */
    int32_t *mask_pos;  /* [n_req][L] mask after the step (M' minus the committed pivot) */
    int32_t *mask_cnt;  /* [n_req] */
} rps_commit_out;

/* Bytes of workspace rps_score_step needs for up to max_rows row slots
 * (n_seg * cap) of `vocab` logits of the given rps_dtype with top-k size k_max
 * (0 for statistics only). Returns 0 for invalid arguments. */
size_t rps_workspace_bytes(int64_t max_rows, int64_t vocab, int32_t dtype, int32_t k_max);

/* Zero a workspace (asynchronously on `stream`). A workspace must be zeroed
 * once before its first use; every completed rps_score_step leaves it ready
 * for the next call. One workspace must not serve two calls that can overlap.
 * Its first 256 bytes hold a health word: a call whose kernel gives up on a
 * bounded wait (RPS_DEVERR_TIMEOUT) leaves row tickets unfinished and marks
 * the word, and every later call on that workspace writes no statistics and
 * reports RPS_DEVERR_WORKSPACE until the workspace is zeroed again. */
rps_status rps_workspace_init(void *d_ws, size_t ws_bytes, rps_stream_t stream);

/*
 * Row statistics (Sec. 2 notation; Eq. 1; Eq. 3) of every listed row:
 * zmax, lse, H = -sum_v p_v log p_v, pmax = P^max, argmax (lowest token on
 * ties), and in top-k mode T_i (k_max tokens by logit desc / token asc),
 * mu = sum_{T_i} p_v and htrunc = -sum_{T_i} p_v log p_v (not renormalised).
 * fp32 arithmetic; argmax and T_i are exact (taken on the input values).
 * Top-k mode makes two launches on `stream` (the statistics, then the top-k
 * search over a sketch the first leaves in the workspace); statistics-only
 * mode makes one.
 * Errors: RPS_ERR_INVALID_ARG for NULL pointers, a misaligned tensor, sizes out
 * of range or a workspace smaller than rps_workspace_bytes(n_seg * cap, vocab,
 * dtype, k); RPS_ERR_UNSUPPORTED above RPS_MAX_K / RPS_MAX_SEGMENTS.
 */
rps_status rps_score_step(const rps_logits *logits, const rps_row_list *rows, const rps_params *prm,
                          const rps_row_stats *out, void *d_ws, size_t ws_bytes, rps_stream_t stream);

/*
 * Standard commit and pivot selection for n_req requests (Eq. 2, Eq. 3,
 * Sec. 3.1, Algorithm 1). `base` holds top-k-mode statistics of each request's
 * masked rows in mask order ([q * L + k], k < mask_cnt[q]); mask_pos lists
 * distinct positions. Per request:
 *   S = {i in M : pmax_i >= tau}, or the single most confident row (lowest
 *   position on ties) when that is empty (RPS_COMMIT_THRESHOLD); or the
 *   commit_k rows of largest pmax / smallest H (the other rules of Eq. 2,
 *   lower position on ties, NaN statistics last); S is committed to argmax tokens.
 *   M' = M \ S. Feasible rows: mu_i >= tau_pivot. Pivots: up to P feasible
 *   rows by truncated entropy (descending, lower position on ties); with
 *   RPS_PIVOT_MAX_CONFIDENCE / _MAX_ENTROPY every row of M' is feasible and
 *   pivots are taken by pmax / H instead.
 *   Candidates: tokens of T_{i*} with z_v - zmax >= log r (that is
 *   p(v) >= r P^max), in rank order, at most K; a pivot is searched when it has
 *   at least two. Branch b = j * K + c lists M' without pivot j.
 * Errors: RPS_ERR_INVALID_ARG for NULL pointers or sizes out of range;
 * RPS_ERR_UNSUPPORTED when L > RPS_MAX_POS or P > RPS_MAX_PIVOTS.
 */
rps_status rps_select_pivots(const rps_row_stats *base, int32_t n_req, int32_t L, const int32_t *d_mask_pos,
                             const int32_t *d_mask_cnt, const rps_params *prm, const rps_pivots *out,
                             rps_stream_t stream);

/*
 * Downstream-benefit scores (Eq. 4; N_tau of Proposition 1). For searched pivot
 * j with D_j = M' \ {i*_j} and n = |M'| - 1:
 *   mean_H = (1/n) sum_{i in D_j} H(p_i^c)  (0 when n == 0)
 *   n_tau  = #{i in D_j : pmax_i^c >= tau}
 *   log_a  = z_anchor(i*_j, c) - lse_anchor(i*_j); for [MASK] zmax - lse
 *   score  = -mean_H + lambda * log_a  (the plausibility term is dropped when
 *            lambda == 0)
 * Token candidates read `branch` (statistics-only mode is enough) in the
 * compact layout of piv->branch_rows; [MASK] reads the anchor statistics of
 * the rows of D_j ([q * L + k], like `base`). The anchor's pivot-row logits are
 * read from branch `anchor_branch` of `anchor_logits`.
 */
rps_status rps_score_branches(const rps_logits *anchor_logits, int32_t anchor_branch,
                              const rps_row_stats *anchor, const rps_row_stats *branch, int32_t n_req,
                              int32_t L, const rps_pivots *piv, const rps_params *prm,
                              const rps_branch_scores *out, rps_stream_t stream);

/*
 * Commit decision (Algorithm 1; Eq. 4). Per searched pivot j the best slot is
 * the argmax of score over its valid tokens and [MASK]; ties keep [MASK], then
 * the higher-ranked token. gain_j = score(best) - score([MASK]). The request
 * commits the pivot with the largest gain_j > 0 (lower position on ties) to
 * its best token, or abstains. out->mask_* receives M' minus the committed
 * pivot and may alias the mask arrays given to rps_select_pivots.
 */
rps_status rps_commit(const rps_branch_scores *scores, int32_t n_req, int32_t L, const rps_pivots *piv,
                      const rps_params *prm, const rps_commit_out *out, rps_stream_t stream);

/* rps_score_branches followed by rps_commit in one launch (same arguments and
 * results as the two calls in sequence). */
rps_status rps_score_and_commit(const rps_logits *anchor_logits, int32_t anchor_branch,
                                const rps_row_stats *anchor, const rps_row_stats *branch, int32_t n_req, int32_t L,
                                const rps_pivots *piv, const rps_params *prm, const rps_branch_scores *scores,
                                const rps_commit_out *out, rps_stream_t stream);

/*
 * One whole step in one call: rps_score_step over the base rows (branch 0 of
 * `logits`, mask form d_mask_pos / d_mask_cnt of capacity L, top-k mode into
 * `base`, workspace d_ws_base), rps_select_pivots into `piv`, rps_score_step
 * over piv->branch_rows (statistics-only mode into `branch`, workspace
 * d_ws_branch, a different one), and rps_score_and_commit with branch 0 as the
 * anchor -- five launches with the results of the four calls. Every argument
 * is checked before anything is enqueued. Because the call knows which launch
 * writes what, the select launch stages the mask before waiting for the base
 * statistics, and the score launch computes everything that does not read the
 * lookahead statistics before waiting for them.
 */
rps_status rps_run_step(const rps_logits *logits, int32_t n_req, int32_t L, const int32_t *d_mask_pos,
                        const int32_t *d_mask_cnt, const rps_params *prm, const rps_row_stats *base,
                        const rps_pivots *piv, const rps_row_stats *branch, const rps_branch_scores *scores,
                        const rps_commit_out *out, void *d_ws_base, size_t ws_base_bytes, void *d_ws_branch,
                        size_t ws_branch_bytes, rps_stream_t stream);

/*
 * Outer loop of Algorithm 1 over semi-autoregressive blocks (the response of
 * L_total positions is decoded block by block, B positions each, left to
 * right). Call after rps_commit of a step whose mask arrays are block-local
 * ([n_req][B], positions 0..B-1 of the current block). Per request:
 *   tokens[q][b * B + p] = the token committed at block position p this step
 *     (the standard commit S of `piv` and the pivot committed by `commit`);
 *   the next step's mask (d_mask_pos / d_mask_cnt) is commit->mask_* while
 *     the block has masked positions, else the whole next block (block[q]
 *     advances), else empty with done[q] = 1.
 * Device arrays: d_tokens [n_req][L_total] (-1 while masked, caller-initialised),
 * d_block [n_req], d_mask_pos [n_req][B], d_mask_cnt [n_req], d_done [n_req]
 * (in/out); d_steps [n_req] (optional, NULL to skip) counts the steps each
 * request took before it was done. commit->mask_* may alias d_mask_*. A commit
 * list outside the block sets RPS_DEVERR_MASK.
 * Errors: RPS_ERR_INVALID_ARG for NULL pointers or sizes out of range;
 * RPS_ERR_UNSUPPORTED when B > RPS_MAX_POS.
 */
rps_status rps_decode_advance(const rps_pivots *piv, const rps_commit_out *commit, int32_t n_req, int32_t B,
                              int32_t L_total, int32_t *d_tokens, int32_t *d_block, int32_t *d_mask_pos,
                              int32_t *d_mask_cnt, int32_t *d_done, int32_t *d_steps, rps_stream_t stream);

/*
 * Copy the rows of a row list from src to the same (req, branch, pos) of dst.
 * The paper has no counterpart: it is data movement for callers whose logits
 * sit in host memory, so that a step copies only the rows it scores (the masked
 * base rows, then the lookahead rows rps_select_pivots lists) instead of the
 * whole tensor, with no host synchronisation between the two. `rows` has the
 * meaning of rps_score_step (mask form or explicit list; device arrays).
 * src: device memory, or page-locked host memory (e.g. cudaHostAlloc), which the
 * GPU reads through its device alias over the host link. dst: device memory
 * (written, though rps_logits holds a const pointer).
 * Same dtype, vocab and extents; strides may differ (16-byte multiples, 16-byte
 * aligned bases).
 * Errors: RPS_ERR_INVALID_ARG for NULL pointers, mismatched tensors, misaligned
 * tensors, or src in pageable host memory (which the device cannot read
 * safely); a row descriptor outside the tensors sets RPS_DEVERR_ROW_INDEX.
 */
rps_status rps_gather_rows(const rps_logits *src, const rps_row_list *rows, const rps_logits *dst,
                           rps_stream_t stream);

/* Bytes of scratch the library holds on each device for rps_score_step_noalloc. */
#define RPS_STATIC_SCRATCH_BYTES (8u << 20)

/*
 * rps_score_step without a caller workspace. The paper has no counterpart: this
 * is a deployment variant for callers that cannot allocate device memory, such
 * as plugins of a host runtime that owns every device allocation and forbids
 * others, or bindings from languages with no CUDA allocator. Inputs and outputs
 * are as for rps_score_step; the scratch is a fixed RPS_STATIC_SCRATCH_BYTES
 * array inside the library, which every GPU that loads the library keeps until
 * the process exits.
 *   - Requests whose rps_workspace_bytes(n_seg * cap, vocab, dtype, k) exceeds
 *     RPS_STATIC_SCRATCH_BYTES return RPS_ERR_UNSUPPORTED before anything is
 *     enqueued; argument errors return RPS_ERR_INVALID_ARG likewise.
 *   - No cudaMalloc, cudaFree or other allocating call is made. Each call clears
 *     the part of the array it uses with cudaMemsetAsync on `stream`.
 *   - The first call on each device looks up the array's device address while
 *     that device is current; make that first call before any stream capture.
 *     The address is kept for the life of the process: after cudaDeviceReset
 *     (or anything else that destroys the device's primary context) it no
 *     longer names the array, so do not call this function on that device
 *     again in the same process.
 *   - All calls on a device share the one array: calls that can overlap on the
 *     GPU (different streams without ordering between them) race and corrupt each
 *     other's results. Order them on one stream or serialise them.
 */
rps_status rps_score_step_noalloc(const rps_logits *logits, const rps_row_list *rows, const rps_params *prm,
                                  const rps_row_stats *out, rps_stream_t stream);

/*
 * LM head with the row statistics in its epilogue (Sec. 2 notation: p_i is
 * the softmax of the denoiser's logits for position i; Eq. 1; Eq. 3). For each
 * hidden row h the logits are z = h W^T, W holding one row of d weights per
 * token; the call computes the statistics of rps_score_step (the same
 * definitions, ties and output layout, slot r = hidden row r) without writing
 * the logits to memory: a tensor-core contraction (bf16 x bf16, fp32
 * accumulation) whose epilogue folds each tile of logits into the rows'
 * softmax sums, maxima and top-k lists, then a merge launch.
 * Layout: hidden [n_rows][d] and unembed [vocab][d], bf16, d contiguous, rows
 * hidden_stride / unembed_stride elements apart (multiples of 8); bases 16-byte
 * aligned; d a multiple of 64.
 */
typedef struct {
    const void *hidden;
    const void *unembed;
    int32_t n_rows;
    int32_t d;
    int64_t vocab;
    int64_t hidden_stride, unembed_stride;
    int32_t unembed_packed; /* 0: unembed is [vocab][d] as above; 1: it was written by
                               rps_lmhead_pack_unembed (unembed_stride is then unused) */
} rps_lmhead;

/*
 * The unembedding in the LM head's packed tile layout (no counterpart in the
 * paper; a one-time re-layout of a static weight). Each 256-token x 64-column
 * block becomes one contiguous 32 KB image, so that the LM head reads the
 * unembedding in whole blocks instead of 128 bytes from each of 256 rows; rows
 * past the vocabulary are zero. rps_lmhead_packed_bytes gives the size (0 for
 * invalid arguments: vocab out of range, d not a positive multiple of 64).
 * unembed: [vocab][d] bf16, rows `stride` elements apart (a multiple of 8).
 * One launch on `stream`; packed must not overlap unembed. Errors:
 * RPS_ERR_INVALID_ARG for NULL or misaligned pointers, sizes out of range or a
 * small output.
 */
size_t rps_lmhead_packed_bytes(int64_t vocab, int32_t d);
rps_status rps_lmhead_pack_unembed(const void *unembed, int64_t vocab, int32_t d, int64_t stride, void *packed,
                                   size_t packed_bytes, rps_stream_t stream);

/* Workspace bytes of rps_lmhead_row_stats (k_max 0 for statistics only); 0 for
 * invalid arguments. The workspace needs no zeroing before its first use
 * except its first 256 bytes (the health word of rps_workspace_init), so
 * rps_workspace_init on the whole workspace is the simple rule. */
size_t rps_lmhead_workspace_bytes(int32_t n_rows, int64_t vocab, int32_t k_max);

/*
 * Statistics of every hidden row's logits h W^T into `out` (top-k mode when
 * out->topk_idx != NULL, with k = prm->k_max; prm may be NULL otherwise).
 * d_logits_out: NULL normally; for testing, a device array [n_rows][vocab] of
 * fp32 that also receives the logits the epilogue folds.
 * Two launches on `stream`. Errors: RPS_ERR_INVALID_ARG for NULL pointers,
 * sizes, strides or alignment out of range, or a small workspace;
 * RPS_ERR_UNSUPPORTED for k_max above RPS_MAX_K; RPS_ERR_CUDA when the
 * tensor-map encoder is not available. A bounded device wait that gives up
 * reports RPS_DEVERR_TIMEOUT and leaves the workspace unhealthy, as for
 * rps_score_step.
 */
rps_status rps_lmhead_row_stats(const rps_lmhead *lm, const rps_params *prm, const rps_row_stats *out,
                                float *d_logits_out, void *d_ws, size_t ws_bytes, rps_stream_t stream);

/*
 * Branch-isolating attention of the packed lookahead forward pass (Sec. 3.1
 * "Lookahead scoring"; Fig. 2, right). The lookahead pass scores all branches
 * of a step in one forward pass over a packed sequence of n_tokens =
 * n_context + n_branch * branch_len tokens: the shared context, then the
 * generation region once per branch (branch 0 = the anchor, the normal
 * sequence's own region). A query of branch j attends to the context and to
 * branch j only; a context query attends to the context and branch 0 (the
 * normal sequence). For every (batch, head):
 *   out_i = sum_{k visible from i} softmax_k(scale * q_i . k_k) v_k
 * bf16 inputs and output, fp32 scores and accumulation, probabilities rounded
 * to bf16 before they weight the values. No dense mask is formed.
 * Layout (bf16, contiguous): q, k, out [n_batch][n_heads][n_tokens][head_dim];
 * vt [n_batch][n_heads][head_dim][n_tokens] (the values transposed, tokens
 * contiguous). head_dim must be 128; n_context (>= 0) and branch_len (>= 1)
 * multiples of 8; bases 16-byte aligned.
 */
typedef struct {
    const void *q, *k, *vt;
    void *out;
    int32_t n_batch, n_heads, head_dim;
    int32_t n_context, n_branch, branch_len;
    float scale;
} rps_packed_attention;

/* One launch on `stream`. Errors: RPS_ERR_INVALID_ARG for NULL or misaligned
 * pointers and sizes out of range; RPS_ERR_UNSUPPORTED for head_dim != 128 or
 * tensors above 2^31 rows; RPS_ERR_CUDA when the tensor-map encoder is not
 * available. A bounded device wait that gives up reports RPS_DEVERR_TIMEOUT
 * (the output is then incomplete). */
rps_status rps_packed_attention_fwd(const rps_packed_attention *attn, rps_stream_t stream);

/* Synchronise `stream`, then read and clear the calling device's error word.
 * Returns RPS_OK or RPS_ERR_DEVICE (with the RPS_DEVERR_* bits in *detail when
 * detail != NULL), or RPS_ERR_CUDA if the synchronisation itself failed. */
rps_status rps_poll_device_status(rps_stream_t stream, uint32_t *detail);

/* Testing hook, no counterpart in the paper: sets the limit of the
 * row-statistics kernels' wait for each asynchronous row copy (200 ms by
 * default, restored by UINT64_MAX; 0 makes every such wait give up at once,
 * so that a test can see a timeout reported). It applies to calls enqueued
 * after it, process-wide. The copies already issued are still waited for
 * (200 ms each) before a warp that gave up stops. Returns the previous limit. */
uint64_t rps_debug_set_ring_wait_ns(uint64_t ns);

/* Static description of a status code. */
const char *rps_status_string(rps_status status);

/* ABI version, major * 10000 + minor * 100 + patch. */
int32_t rps_version(void);

#ifdef __cplusplus
}
#endif

#endif /* RPS_H */
