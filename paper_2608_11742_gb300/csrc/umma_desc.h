// umma_desc.h -- encoders of the two descriptors a tcgen05.mma reads, in plain
// C++ (host and device), so that every field can be checked on the host.
//
// Instruction descriptor of tcgen05.mma .kind::f16 (32 bits, PTX ISA, "Instruction
// descriptor" of the tcgen05 MMA instructions):
//   [0,2) sparsity selector   [2] sparsity      [3] saturate
//   [4,6) D format (1 = f32)  [7,10) A format   [10,13) B format (kind::f16: 0 = f16, 1 = bf16)
//   [13] negate A  [14] negate B  [15] A major (0 = K)  [16] B major (0 = K)
//   [17,23) N >> 3            [24,29) M >> 4    [30,32) shift (0)
//
// Shared-memory matrix descriptor (64 bits, PTX ISA, "Shared memory descriptor"):
//   [0,14)  start address >> 4
//   [16,30) leading-dimension byte offset >> 4
//   [32,46) stride-dimension byte offset >> 4
//   [46,48) version (1 for tcgen05)
//   [49,52) base offset (0: the swizzle pattern starts on a 1024-byte boundary)
//   [52]    leading-dimension offset mode (0: relative)
//   [61,64) swizzle: 0 none, 1 128-byte with 32-byte atoms, 2 128-byte, 4 64-byte, 6 32-byte
//
// The operands here are K-major tiles written by a TMA load with 128-byte
// swizzle: row r of the tile (an M or N index) holds 64 bf16 of K in 128
// bytes, rows follow each other at 128 bytes, so eight rows form one
// 1024-byte swizzle atom and the atoms of successive 8-row groups are 1024
// bytes apart (the stride-dimension offset). A K-major swizzled operand whose
// K extent per instruction (16 bf16, 32 bytes) lies inside one 128-byte row
// does not use the leading-dimension offset; the next K slice of the same
// 64-wide row starts 32 bytes further.
#pragma once

#include <stdint.h>

#ifdef __CUDACC__
#define UMMA_HD __host__ __device__
#else
#define UMMA_HD
#endif

namespace rps {
namespace umma {

enum : uint32_t { kFmtF16 = 0, kFmtBF16 = 1, kAccF32 = 1 };
enum : uint32_t { kSwizzleNone = 0, kSwizzle128B = 2 };

// kind::f16 with bf16 A and B, f32 accumulator, both operands K-major.
UMMA_HD inline constexpr uint32_t instr_desc_bf16(uint32_t m, uint32_t n) {
    return (kAccF32 << 4) | (kFmtBF16 << 7) | (kFmtBF16 << 10) | ((n >> 3) << 17) | ((m >> 4) << 24);
}

UMMA_HD inline constexpr uint64_t smem_desc(uint32_t smem_addr, uint32_t lbo_bytes, uint32_t sbo_bytes, uint32_t swizzle) {
    return static_cast<uint64_t>((smem_addr >> 4) & 0x3FFFu) |
           (static_cast<uint64_t>((lbo_bytes >> 4) & 0x3FFFu) << 16) |
           (static_cast<uint64_t>((sbo_bytes >> 4) & 0x3FFFu) << 32) | (static_cast<uint64_t>(1) << 46) |
           (static_cast<uint64_t>(swizzle & 7u) << 61);
}

// K-major tile of 64 bf16 per row, 128-byte swizzle, 8-row groups 1024 bytes apart.
UMMA_HD inline constexpr uint64_t smem_desc_kmajor_sw128(uint32_t smem_addr) {
    return smem_desc(smem_addr, 16, 1024, kSwizzle128B);
}

// The descriptor of the K slice `k16` (16 bf16 = 32 bytes further per slice).
UMMA_HD inline constexpr uint64_t advance_k16(uint64_t desc, uint32_t k16) { return desc + static_cast<uint64_t>(2 * k16); }

}  // namespace umma
}  // namespace rps
