// synth.cu -- seeded synthetic logits on the device (librps_synth.so).
//
// Input generation only: the GPU twin of paper_2608_11742_gb300/synth.py, bit
// for bit. Every value is integer arithmetic or one explicitly rounded fp32
// operation (__fmul_rn / __fadd_rn, so nothing is fused into an FMA):
//   Philox4x32-10 (Salmon et al., SC'11) keyed by (seed, 0x52505331);
//   eps = (2 S - 8 * 65535) * sqrt(1.5) / 131072, S = sum of eight 16-bit words;
//   regime from a 32-bit draw: low (+12 on one token), mid (+4 on 2-5 distinct
//   tokens), high (eps * 2); branch b > 0 scales the spike by f in [0.8, 1.6);
//   bf16 by round-to-nearest-even on the fp32 bits.
#include <cstdint>
#include <cuda_runtime.h>

#include "rps_synth.h"

namespace {

constexpr uint32_t kM0 = 0xD2511F53u, kM1 = 0xCD9E8D57u;
constexpr uint32_t kW0 = 0x9E3779B9u, kW1 = 0xBB67AE85u;
constexpr uint32_t kKey1 = 0x52505331u;
constexpr uint32_t kTagNoise = 1, kTagRegime = 2, kTagSpikes = 3, kTagBranch = 4;
constexpr int kMaxSpikeDraws = 16;
constexpr int kPerThread = 8;

struct U4 {
    uint32_t x, y, z, w;
};

__device__ __forceinline__ U4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        if (r) {
            k0 += kW0;
            k1 += kW1;
        }
        const uint32_t hi0 = __umulhi(kM0, c0), lo0 = kM0 * c0;
        const uint32_t hi1 = __umulhi(kM1, c2), lo1 = kM1 * c2;
        const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0;
        c1 = lo1;
        c2 = n2;
        c3 = lo0;
    }
    return U4{c0, c1, c2, c3};
}

__device__ __forceinline__ uint32_t tag(uint32_t t, uint32_t epoch) { return (t & 0xFFu) | ((epoch & 0xFFFFFFu) << 8); }

__device__ __forceinline__ uint16_t to_bf16(float z) {
    const uint32_t b = __float_as_uint(z);
    return static_cast<uint16_t>((b + 0x7FFFu + ((b >> 16) & 1u)) >> 16);
}

struct Args {
    void *out;
    int32_t dtype, n_req, n_branch, L;
    int64_t vocab, req_stride, branch_stride, pos_stride;
    uint32_t seed, step;
    uint64_t t_low, t_mid;
    const float *scale;
    const int32_t *epoch;
    const uint8_t *valid;
    // decode mode (d_block != nullptr): row p of request q is response position
    // d_block[q] * L + p; scale / epoch are [n_req][state_L] over the response;
    // rows past the response end are NaN; the step index is read from d_step
    const int32_t *d_step;
    const int32_t *d_block;
    int32_t state_L;
};

// Spike scale factor in [0.8, 1.6) of branch b >= 1 at (q, pos), drawn per step.
__device__ __forceinline__ float branch_factor(uint32_t seed, int q, int b, int pos, uint32_t step) {
    const U4 bf = philox(b, pos, q, tag(kTagBranch, step), seed, kKey1);
    const float u = __fmul_rn(static_cast<float>(bf.x >> 8), 5.9604644775390625e-8f);
    return __fadd_rn(0.8f, __fmul_rn(0.8f, u));
}

__global__ void fill_kernel(const Args a) {
    const int64_t V = a.vocab;
    const uint32_t step = a.d_step ? static_cast<uint32_t>(*a.d_step) : a.step;
    const int64_t chunks = (V + kPerThread - 1) / kPerThread;
    const int64_t rows = static_cast<int64_t>(a.n_req) * (a.n_branch + 1) * a.L;
    const int64_t total = rows * chunks;
    for (int64_t g = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; g < total;
         g += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t row = g / chunks;
        const int64_t v0 = (g - row * chunks) * kPerThread;
        const int local = static_cast<int>(row % a.L);
        const int b = static_cast<int>((row / a.L) % (a.n_branch + 1));
        const int q = static_cast<int>(row / (static_cast<int64_t>(a.L) * (a.n_branch + 1)));
        const int64_t off = q * a.req_stride + b * a.branch_stride + local * a.pos_stride + v0;
        const int n = static_cast<int>((V - v0 < kPerThread ? V - v0 : static_cast<int64_t>(kPerThread)));
        const int pos = a.d_block ? a.d_block[q] * a.L + local : local;  // position in the response
        const bool is_valid = a.d_block ? pos < a.state_L
                                        : a.valid == nullptr || a.valid[static_cast<int64_t>(q) * a.L + local] != 0;
        const int64_t state_row = static_cast<int64_t>(q) * a.state_L + pos;

        float z[kPerThread];
        if (!is_valid) {
#pragma unroll
            for (int i = 0; i < kPerThread; ++i) z[i] = __int_as_float(0x7FC00000);
        } else {
            // regime and spike tokens of (q, pos)
            const U4 reg = philox(0, pos, q, tag(kTagRegime, 0), a.seed, kKey1);
            int regime, n_spk = 0;
            int toks[5];
            if (reg.x < a.t_low) {
                regime = 0;
                toks[0] = static_cast<int>(reg.y % static_cast<uint32_t>(V));
                n_spk = 1;
            } else if (reg.x < a.t_mid) {
                regime = 1;
                int want = 2 + static_cast<int>(reg.z % 4u);
                if (want > V) want = static_cast<int>(V);
                for (int d = 0; d < kMaxSpikeDraws && n_spk < want; ++d) {
                    const U4 w = philox(d, pos, q, tag(kTagSpikes, 0), a.seed, kKey1);
                    const uint32_t words[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int t = static_cast<int>(words[i] % static_cast<uint32_t>(V));
                        bool dup = false;
                        for (int j = 0; j < n_spk; ++j) dup |= toks[j] == t;
                        if (n_spk < want && !dup) toks[n_spk++] = t;
                    }
                }
            } else {
                regime = 2;
            }
            float amp = 0.f;
            if (regime != 2) {
                const float h = regime == 0 ? 12.0f : 4.0f;
                const float sc = a.scale ? a.scale[state_row] : 1.0f;
                const float f = b > 0 ? branch_factor(a.seed, q, b, pos, step) : 1.0f;
                amp = __fmul_rn(__fmul_rn(h, sc), f);
            }
            const uint32_t ep = a.epoch ? static_cast<uint32_t>(a.epoch[state_row]) : 0u;
#pragma unroll
            for (int i = 0; i < kPerThread; ++i) {
                if (i >= n) {
                    z[i] = 0.f;
                    continue;
                }
                const int64_t v = v0 + i;
                const U4 w = philox(static_cast<uint32_t>(v), pos, q, tag(kTagNoise, ep), a.seed, kKey1);
                const int32_t s = static_cast<int32_t>((w.x & 0xFFFFu) + (w.x >> 16) + (w.y & 0xFFFFu) + (w.y >> 16) +
                                                       (w.z & 0xFFFFu) + (w.z >> 16) + (w.w & 0xFFFFu) + (w.w >> 16));
                const float eps = __fmul_rn(static_cast<float>(2 * s - 8 * 65535), 0x1.3988e2p-17f);
                if (regime == 2) {
                    z[i] = __fmul_rn(eps, 2.0f);
                } else {
                    bool spike = false;
                    for (int j = 0; j < n_spk; ++j) spike |= toks[j] == v;
                    z[i] = spike ? __fadd_rn(eps, amp) : eps;
                }
            }
        }
        if (a.dtype == 1) {
            uint16_t *o = static_cast<uint16_t *>(a.out) + off;
            if (n == kPerThread && !is_valid) {
                *reinterpret_cast<uint4 *>(o) = make_uint4(0x7FC07FC0u, 0x7FC07FC0u, 0x7FC07FC0u, 0x7FC07FC0u);
            } else if (n == kPerThread) {
                uint32_t p[4];
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    p[i] = static_cast<uint32_t>(to_bf16(z[2 * i])) | (static_cast<uint32_t>(to_bf16(z[2 * i + 1])) << 16);
                *reinterpret_cast<uint4 *>(o) = make_uint4(p[0], p[1], p[2], p[3]);
            } else {
                for (int i = 0; i < n; ++i) o[i] = is_valid ? to_bf16(z[i]) : static_cast<uint16_t>(0x7FC0);
            }
        } else {
            float *o = static_cast<float *>(a.out) + off;
            for (int i = 0; i < n; ++i) o[i] = z[i];
        }
    }
}

}  // namespace

extern "C" int32_t rps_synth_fill(void *out, int32_t dtype, int32_t n_req, int32_t n_branch, int32_t L, int64_t vocab,
                                  int64_t req_stride, int64_t branch_stride, int64_t pos_stride, uint32_t seed,
                                  uint64_t t_low, uint64_t t_mid, uint32_t step, const float *scale,
                                  const int32_t *epoch, const uint8_t *valid, void *stream) {
    if (!out || (dtype != 0 && dtype != 1) || n_req < 1 || n_branch < 0 || L < 1 || vocab < 1 ||
        vocab > 0xFFFFFFFFLL || t_low > t_mid || t_mid > (1ull << 32))
        return 1;
    const int64_t esize = dtype == 1 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(out) % 16 || (req_stride * esize) % 16 || (branch_stride * esize) % 16 ||
        (pos_stride * esize) % 16)
        return 1;
    Args a;
    a.out = out;
    a.dtype = dtype;
    a.n_req = n_req;
    a.n_branch = n_branch;
    a.L = L;
    a.vocab = vocab;
    a.req_stride = req_stride;
    a.branch_stride = branch_stride;
    a.pos_stride = pos_stride;
    a.seed = seed;
    a.step = step;
    a.t_low = t_low;
    a.t_mid = t_mid;
    a.scale = scale;
    a.epoch = epoch;
    a.valid = valid;
    a.d_step = nullptr;
    a.d_block = nullptr;
    a.state_L = L;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms < 1) sms = 1;
    fill_kernel<<<sms * 8, 256, 0, static_cast<cudaStream_t>(stream)>>>(a);
    return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

namespace {

// The decision of a step applied to the generator state of the positions of
// each request's current block: a committed branch becomes the next base (its
// spike factor of the step multiplies the spike scale), a skip draws fresh noise
// (the noise epoch advances), an abstain or a finished request changes nothing.
__global__ void advance_kernel(const int32_t *winner, int32_t B, int32_t L_total, const int32_t *d_block,
                               const int32_t *d_step, float *scale, int32_t *epoch, uint32_t seed) {
    const int q = blockIdx.x;
    const int w = winner[q];
    const uint32_t step = static_cast<uint32_t>(*d_step);
    const int base = d_block[q] * B;
    for (int p = threadIdx.x; p < B; p += blockDim.x) {
        const int pos = base + p;
        if (pos >= L_total) break;
        const int64_t i = static_cast<int64_t>(q) * L_total + pos;
        if (w >= 0) scale[i] = __fmul_rn(scale[i], branch_factor(seed, q, 1 + w, pos, step));
        else if (w == -2) epoch[i] += 1;
    }
}

__global__ void step_kernel(int32_t *d_step) { *d_step += 1; }

}  // namespace

extern "C" int32_t rps_synth_fill_blocks(void *out, int32_t dtype, int32_t n_req, int32_t n_branch, int32_t B,
                                         int64_t vocab, int64_t req_stride, int64_t branch_stride, int64_t pos_stride,
                                         uint32_t seed, uint64_t t_low, uint64_t t_mid, const int32_t *d_step,
                                         const int32_t *d_block, int32_t L_total, const float *scale,
                                         const int32_t *epoch, void *stream) {
    if (!out || !d_step || !d_block || !scale || !epoch || (dtype != 0 && dtype != 1) || n_req < 1 || n_branch < 0 ||
        B < 1 || L_total < 1 || vocab < 1 || vocab > 0xFFFFFFFFLL || t_low > t_mid || t_mid > (1ull << 32))
        return 1;
    const int64_t esize = dtype == 1 ? 2 : 4;
    if (reinterpret_cast<uintptr_t>(out) % 16 || (req_stride * esize) % 16 || (branch_stride * esize) % 16 ||
        (pos_stride * esize) % 16)
        return 1;
    Args a;
    a.out = out;
    a.dtype = dtype;
    a.n_req = n_req;
    a.n_branch = n_branch;
    a.L = B;
    a.vocab = vocab;
    a.req_stride = req_stride;
    a.branch_stride = branch_stride;
    a.pos_stride = pos_stride;
    a.seed = seed;
    a.step = 0;
    a.t_low = t_low;
    a.t_mid = t_mid;
    a.scale = scale;
    a.epoch = epoch;
    a.valid = nullptr;
    a.d_step = d_step;
    a.d_block = d_block;
    a.state_L = L_total;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms < 1) sms = 1;
    fill_kernel<<<sms * 8, 256, 0, static_cast<cudaStream_t>(stream)>>>(a);
    return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

extern "C" int32_t rps_synth_advance(const int32_t *d_winner, int32_t n_req, int32_t B, int32_t L_total,
                                     const int32_t *d_block, int32_t *d_step, float *scale, int32_t *epoch,
                                     uint32_t seed, void *stream) {
    if (!d_winner || !d_block || !d_step || !scale || !epoch || n_req < 1 || B < 1 || L_total < 1) return 1;
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    advance_kernel<<<n_req, 256, 0, s>>>(d_winner, B, L_total, d_block, d_step, scale, epoch, seed);
    step_kernel<<<1, 1, 0, s>>>(d_step);
    return cudaGetLastError() == cudaSuccess ? 0 : 2;
}
