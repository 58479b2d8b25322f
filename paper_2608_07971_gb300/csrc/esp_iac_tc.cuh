// Tensor-core path of the IAC predictor (Sec. 3.3.2, Eq. dnn_pred): the two hidden layers as
// tcgen05 MMAs (kind::tf32, accumulators in tensor memory) with a three-term split that keeps
// fp32-level accuracy.
//
// Tile: 128 pairs (one per TMEM lane and per thread of a warpgroup) x 64 hidden units. Layer 1 is
// D1[128 x 64] = X[128 x 40] * [W1' | b1']^T: the 36 inputs, a column of ones that carries the bias
// (b1' in column 36 of the weights) and zero padding to 40 = 5 MMA k-steps of 8. Layer 2 is
// D2 = H1[128 x 64] * W2'^T (8 k-steps) issued in two halves of 32 columns of H1; its bias, the
// output layer (64 terms) and the ReLUs run in the epilogues on the CUDA cores. Split: every operand
// a = a_hi + a_lo with a_hi = a truncated to tf32 (exact) and a_lo = tf32(a - a_hi) (round to
// nearest, ties away), and each k-step issues a_hi*b_hi + a_hi*b_lo + a_lo*b_hi into the same fp32
// accumulator; per product the dropped term and the roundings of the low parts are below 2^-19 |a b|.
//
// Operands. An M = 128, N = 64, K = 8 tf32 MMA with both operands in shared memory reads 6 KB, more
// than the tensor core's time for it at 128 B per cycle, so with both layers reading A from shared
// memory the kernel was bound by shared-memory bandwidth. Layer 2 therefore takes its A operand (H1)
// from tensor memory, where the epilogue writes it with tcgen05.st, and reads only B from shared
// memory; layer 1 keeps X in shared memory (X, D1 and a half of H1 do not fit together in a
// warpgroup's columns). Each warpgroup owns two regions of 64 TMEM columns: one holds a tile's
// accumulators (D1, then D2 once D1 has been read into registers), the other a half of H1, hi at its
// column 0 and lo at 32 (lane = row, column = k, the layout of an M = 128 operand in tensor memory);
// the second half is written once the first half's MMAs have completed. The roles swap from one tile
// to the next, so the next tile's layer 1 is issued as soon as layer 2 completes and runs during the
// output epilogue.
//
// CTA: four warpgroups, each running its own sequence of tiles, so that four tiles' dependency
// chains (features, MMA 1, epilogue 1, the two halves of layer 2, epilogue 2) overlap on one SM; the
// next tile's inputs are computed and stored while the current tile's last MMAs run. The split weights
// W1', W2' are staged once per CTA (53,248 bytes); a warpgroup's X buffer holds hi and lo (2 x 20 KB).
// Shared-memory operands use the canonical no-swizzle K-major layout: 8-row x 16-byte core matrices
// of 128 contiguous bytes, consecutive along K (leading offset 128 B), row groups of 8 at a stride of
// K/4 * 128 B. One elected thread per warpgroup, each in a different SM sub-partition, issues the
// MMAs and commits them to the warpgroup's mbarrier; every wait is bounded, agreed warp-wide (the
// tcgen05 loads and stores after it are warp-collective) and warpgroup-wide at the next hand-off
// barrier (a reducing barrier). A timeout ends the warpgroup's loop, flags the error word, makes the
// mbarrier track every MMA still in flight and waits for them (bounded) before the CTA frees its
// tensor memory.
#pragma once

#include <cstdint>

namespace iac_tc {

constexpr int kM = 128;          // pairs per tile
constexpr int kN = 64;           // hidden units (narrower models are zero-padded)
constexpr int kK1 = 40;          // 36 inputs and the bias column, padded to a multiple of the tf32 MMA K (8)
constexpr int kK2 = 64;
constexpr int kKH = 32;          // layer 2 in two halves of 32 columns of H1
constexpr int kWG = 4;           // warpgroups per CTA
constexpr int kThreads = 128 * kWG;
constexpr int kTmemCols = 512;   // two regions of 64 columns per warpgroup (accumulators; a half of H1)

constexpr int kB1Bytes = kN * kK1 * 4;                      // 10,240
constexpr int kB2Bytes = kN * kK2 * 4;                      // 16,384
constexpr int kBImgBytes = 2 * kB1Bytes + 2 * kB2Bytes;     // hi, lo of W1' then of W2'
constexpr int kA1Bytes = kM * kK1 * 4;                      // 20,480: one part (hi or lo) of X
constexpr int kABufBytes = 2 * kA1Bytes;                    // a warpgroup's X: hi at 0, lo at kA1Bytes
constexpr int kOffB1Hi = 0, kOffB1Lo = kB1Bytes, kOffB2Hi = 2 * kB1Bytes, kOffB2Lo = 2 * kB1Bytes + kB2Bytes;
constexpr int kOffA = kBImgBytes;                           // warpgroup g's buffer at kOffA + g kABufBytes
constexpr int kOffBar = kOffA + kWG * kABufBytes;
constexpr int kOffSlot = kOffBar + 8 * kWG;
constexpr int kSmemBytes = kOffSlot + 16 + 1024;            // + alignment slack of the dynamic base
static_assert(2 * kN * kWG <= kTmemCols, "the two regions of every warpgroup");
static_assert(2 * kKH == kN, "a half of H1, hi and lo, fills a region");
static_assert(kSmemBytes <= 232448, "shared memory of one CTA");

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
