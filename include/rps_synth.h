/*
 * rps_synth.h -- C ABI of the seeded synthetic-logit generator (librps_synth.so).
 *
 * Input generation for tests and benchmarks of the RPS scoring path; it holds
 * none of the scoring arithmetic. It writes the same bits as the host twin in
 * paper_2608_11742_gb300/synth.py: Philox4x32-10 counters (Salmon et al.,
 * SC'11), a scaled Irwin-Hall noise of eight 16-bit uniforms, per-position
 * regimes (one +12 spike, 2-5 distinct +4 spikes, or noise / 0.5), branch spike
 * scaling by a factor in [0.8, 1.6), and bf16 round-to-nearest-even.
 * The paper's workloads are LLaDA / Dream decoding steps (Sec. 4); these logits
 * stand in for them.
 */
#ifndef RPS_SYNTH_H
#define RPS_SYNTH_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/*
 * Fill out[q][b][pos][v] (element strides req_stride, branch_stride, pos_stride;
 * vocab contiguous) for q < n_req, b <= n_branch (b = 0 is the base), pos < L,
 * v < vocab. dtype: 0 = fp32, 1 = bf16 bits. Regime thresholds t_low <= t_mid
 * are compared with a 32-bit draw (values up to 2^32). step keys the branch
 * factors. Optional device arrays [n_req][L] (NULL = defaults): scale (spike
 * scale, 1.0), epoch (noise epoch, 0), valid (0 = write NaN rows). The output
 * must be 16-byte aligned with 16-byte multiple strides.
 * Returns 0 on success, 1 for invalid arguments, 2 for a CUDA launch error.
 */
int32_t rps_synth_fill(void *out, int32_t dtype, int32_t n_req, int32_t n_branch, int32_t L, int64_t vocab,
                       int64_t req_stride, int64_t branch_stride, int64_t pos_stride, uint32_t seed,
                       uint64_t t_low, uint64_t t_mid, uint32_t step, const float *scale, const int32_t *epoch,
                       const uint8_t *valid, void *stream);


/*
 * Decode mode: the current semi-autoregressive block of every request. Row p of
 * request q is response position d_block[q] * B + p (rows past L_total are NaN);
 * the branch factors use the step index *d_step; scale and epoch are
 * [n_req][L_total] device arrays over the response. All pointers are device
 * pointers. Returns as rps_synth_fill.
 */
int32_t rps_synth_fill_blocks(void *out, int32_t dtype, int32_t n_req, int32_t n_branch, int32_t B, int64_t vocab,
                              int64_t req_stride, int64_t branch_stride, int64_t pos_stride, uint32_t seed,
                              uint64_t t_low, uint64_t t_mid, const int32_t *d_step, const int32_t *d_block,
                              int32_t L_total, const float *scale, const int32_t *epoch, void *stream);

/*
 * Apply one step's decisions (d_winner [n_req], the winner codes of rps_commit)
 * to the generator state of each request's current block -- a committed branch b
 * multiplies the spike scale by that branch's factor of the step, a skip (-2)
 * advances the noise epoch -- then advance *d_step. Returns 0, 1 for invalid
 * arguments, 2 for a CUDA launch error.
 */
int32_t rps_synth_advance(const int32_t *d_winner, int32_t n_req, int32_t B, int32_t L_total, const int32_t *d_block,
                          int32_t *d_step, float *scale, int32_t *epoch, uint32_t seed, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* RPS_SYNTH_H */
