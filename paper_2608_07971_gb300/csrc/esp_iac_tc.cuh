// Tensor-core path of the IAC predictor (Sec. 3.3.2, Eq. dnn_pred): the two hidden layers as
// tcgen05 MMAs (kind::tf32, accumulators in tensor memory) with a three-term split that keeps
// fp32-level accuracy.
//
// Tile: 128 pairs (one per TMEM lane and per thread of a warpgroup) x 64 hidden units. Layer 1 is
// D1[128 x 64] = X[128 x 40] * W1'^T (36 inputs padded to 40 = 5 MMA k-steps of 8), layer 2 is
// D2 = H1[128 x 64] * W2'^T (8 k-steps); the output layer (64 terms) and the biases run in the
// epilogue on the CUDA cores. Split: every operand a = a_hi + a_lo with a_hi = a truncated to tf32
// (exact) and a_lo = tf32(a - a_hi) (round to nearest, ties away), and each k-step issues
// a_hi*b_hi + a_hi*b_lo + a_lo*b_hi into the same fp32 accumulator; per product the dropped term
// and the roundings of the low parts are below 2^-19 |a b|.
//
// CTA: two warpgroups, each running its own sequence of tiles (one warpgroup's epilogue overlaps the
// other's MMAs), the split weights W1', W2' staged once per CTA (53,248 bytes), 64 KB of operand A
// per warpgroup, 256 TMEM columns (D1, D2 of each warpgroup). Operands use the canonical
// no-swizzle K-major layout: 8-row x 16-byte core matrices of 128 contiguous bytes, consecutive
// along K (leading offset 128 B), row groups of 8 at a stride of K/4 * 128 B. One elected thread
// per warpgroup issues the MMAs and commits them to the warpgroup's mbarrier; every wait is bounded
// and a timeout ends the warpgroup's loop (the decision is made warpgroup-wide by a reducing
// barrier), flags the error word, and the CTA still frees its tensor memory.
#pragma once

#include <cstdint>

namespace iac_tc {

constexpr int kM = 128;          // pairs per tile
constexpr int kN = 64;           // hidden units (narrower models are zero-padded)
constexpr int kK1 = 40;          // 36 inputs padded to a multiple of the tf32 MMA K (8)
constexpr int kK2 = 64;
constexpr int kWG = 2;           // warpgroups per CTA
constexpr int kThreads = 128 * kWG;
constexpr int kTmemCols = 256;   // D1 and D2 (64 fp32 columns each) per warpgroup

constexpr int kB1Bytes = kN * kK1 * 4;                      // 10,240
constexpr int kB2Bytes = kN * kK2 * 4;                      // 16,384
constexpr int kBImgBytes = 2 * kB1Bytes + 2 * kB2Bytes;     // hi, lo of W1' then of W2'
constexpr int kABytes = kM * kK2 * 4;                       // 32,768 per part (hi or lo)
constexpr int kOffB1Hi = 0, kOffB1Lo = kB1Bytes, kOffB2Hi = 2 * kB1Bytes, kOffB2Lo = 2 * kB1Bytes + kB2Bytes;
constexpr int kOffA = kBImgBytes;                           // warpgroup g: hi at kOffA + 2g kABytes, lo after it
constexpr int kOffBar = kOffA + kWG * 2 * kABytes;
constexpr int kOffSlot = kOffBar + 8 * kWG;
constexpr int kSmemBytes = kOffSlot + 16 + 1024;            // + alignment slack of the dynamic base

// Byte offset of element (row, col) in the canonical no-swizzle K-major layout of a K-wide operand.
__host__ __device__ constexpr int cm_off(int row, int col, int K)
{
    return (row >> 3) * (K / 4 * 128) + (col >> 2) * 128 + (row & 7) * 16 + (col & 3) * 4;
}

__host__ __device__ inline uint32_t tf32_trunc_bits(uint32_t b)
{
    return b & 0xffffe000u;
}

// Round to the nearest tf32 value, ties away from zero (magnitude rounding on the bit pattern).
__host__ __device__ inline uint32_t tf32_round_bits(uint32_t b)
{
    return (b + 0x1000u) & 0xffffe000u;
}

// Instruction descriptor of tcgen05.mma kind::tf32: D fp32 (bits 4-5 = 1), A and B tf32 (bits 7-9,
// 10-12 = 2), both K-major (bits 15, 16 = 0), N >> 3 at bits 17-22, M >> 4 at bits 24-28.
constexpr uint32_t kIdesc = (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(kN >> 3) << 17) |
                            ((uint32_t)(kM >> 4) << 24);

}  // namespace iac_tc
