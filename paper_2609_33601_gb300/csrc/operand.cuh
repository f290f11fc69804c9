// operand.cuh -- the INT4 code formats the library moves around, and the one conversion
// between them that the GEMM relies on.
//
// Packed codes (the public format): 4-bit two's complement, two per byte, element 2j in the
// low nibble of byte j, rows contiguous along K.
//
// MMA operand bytes (internal): the tensor core has no INT8/INT4 MMA on sm_103a, so codes are
// fed to tcgen05.mma kind::f8f6f4 as E4M3 bytes.  A code q in [-8, 7] is stored as the
// sign-magnitude byte  (q < 0 ? 0x80 : 0) | |q|,  which E4M3 reads as exactly q * 2^-9
// (|q| <= 7 are subnormals m * 2^-9, |q| = 8 is the smallest normal 2^-6).  Products are then
// qa * qb * 2^-18 and every per-group sum is an integer multiple of 2^-18 that fp32 holds
// exactly (|sum| <= 64 * K < 2^24 for K <= 262143); the GEMM epilogue multiplies by 2^18.
//
// Operand byte order: within every run of 8 consecutive elements e0..e7 of a row the bytes
// are stored as [e0 e2 e4 e6 e1 e3 e5 e7].  The dot product is invariant under a permutation
// of K applied identically to both operands, so A and B just have to agree; the order makes
// the nibble -> byte conversion free of shuffles.  Every 16-byte packed chunk (elements
// 32c..32c+31) becomes the two 16-byte operand chunks 2c and 2c+1.
#pragma once
#include <cstdint>

namespace jq {

// 8 packed nibbles (one 32-bit word, elements e0..e7) -> 8 operand bytes in operand order:
// .x = bytes for e0,e2,e4,e6 and .y = bytes for e1,e3,e5,e7.
// Per nibble n (two's complement, sign s = n >> 3): |q| = ((n & 7) ^ 7s) + s, computed for all
// eight nibbles at once (the largest magnitude, 8, still fits a nibble, so no carry crosses
// nibbles); then the magnitudes are spread to bytes and each sign lands on bit 7 of its byte.
__device__ __forceinline__ uint2 nib8_to_operand(uint32_t w) {
  const uint32_t s = (w >> 3) & 0x11111111u;                  // sign of each nibble, at its bit 0
  const uint32_t s8 = s << 3;                                 // the same sign at the nibble's bit 3
  const uint32_t mag = ((w & 0x77777777u) ^ (s8 - s)) + s;     // eight magnitudes in [0, 8]
  const uint32_t lo = (mag & 0x0F0F0F0Fu) | ((s << 7) & 0xF0F0F0F0u);  // even elements
  const uint32_t hi = ((mag >> 4) & 0x0F0F0F0Fu) | (s8 & 0xF0F0F0F0u);  // odd elements
  return make_uint2(lo, hi);
}

// 32 packed codes (16 bytes) -> 32 operand bytes (two 16-byte chunks).
__device__ __forceinline__ void nib32_to_operand(uint4 p, uint4& lo, uint4& hi) {
  const uint2 a = nib8_to_operand(p.x), b = nib8_to_operand(p.y);
  const uint2 c = nib8_to_operand(p.z), d = nib8_to_operand(p.w);
  lo = make_uint4(a.x, a.y, b.x, b.y);
  hi = make_uint4(c.x, c.y, d.x, d.y);
}

// Offset operand bytes (the few-token kernel's weights): the code q becomes the byte q + 8 in
// [0, 15], which E4M3 also reads exactly, as (q + 8) * 2^-9 (0..7 are subnormals, 8..15 have
// exponent field 1: 2^-6 * (1 + m/8) = (8 + m) * 2^-9).  Adding 8 to a 4-bit two's complement
// code is flipping its bit 3, so 8 codes take three operations instead of ten.  A dot product
// with offset weights is sum (qw + 8) qa = sum qw qa + 8 sum qa: the kernel subtracts 8 times the
// activation code sum, exactly, before any scaling.  |sum (qw + 8) qa| <= 120 per element, so a
// run of up to 139808 elements (120 * 139808 < 2^24) accumulates exactly in fp32.
__device__ __forceinline__ uint2 nib8_to_operand_offset(uint32_t w) {
  return make_uint2((w & 0x0F0F0F0Fu) ^ 0x08080808u, ((w >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u);
}
__device__ __forceinline__ void nib32_to_operand_offset(uint4 p, uint4& lo, uint4& hi) {
  const uint2 a = nib8_to_operand_offset(p.x), b = nib8_to_operand_offset(p.y);
  const uint2 c = nib8_to_operand_offset(p.z), d = nib8_to_operand_offset(p.w);
  lo = make_uint4(a.x, a.y, b.x, b.y);
  hi = make_uint4(c.x, c.y, d.x, d.y);
}
// Sum of the 32 signed codes of a 16-byte packed chunk: flip to offset codes q + 8, add the
// nibble pairs of the four words bytewise (at most 4 * 30 = 120 per byte), fold the bytes into
// 16-bit halves and the halves into one sum, and remove the 32 * 8 offset.  Plain logic and
// adds only: the integer dot-product instruction is slow on this part.
__device__ __forceinline__ int nib32_sum(uint4 p) {
  const uint32_t w[4] = {p.x, p.y, p.z, p.w};
  uint32_t bytes = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t u = w[i] ^ 0x88888888u;
    bytes += (u & 0x0F0F0F0Fu) + ((u >> 4) & 0x0F0F0F0Fu);
  }
  const uint32_t halves = (bytes & 0x00FF00FFu) + ((bytes >> 8) & 0x00FF00FFu);
  return (int)((halves & 0xFFFFu) + (halves >> 16)) - 256;
}
constexpr int kOffsetMaxRun = 139808;

// Packed ternary codes (the W1.58A4 weights, 16 codes per 32-bit word, ternary.cu) -> operand
// bytes.  Bits 0-1 of byte j of (word >> 2i) hold c = q + 1 in {0, 1, 2} for elements
// {2j, 2j+1, 8+2j, 9+2j}[i], so the four shifts give the operand chunk of the word's 16 elements
// in operand order with no byte movement.  Sign-magnitude bytes: c = 2 -> 0x01, c = 1 -> 0x00,
// c = 0 -> 0x81; the magnitude bit is the complement of bit 0 of c and the sign is set where
// neither bit of c is.
__device__ __forceinline__ uint32_t tern4_to_operand(uint32_t p) {
  const uint32_t mag = ~p & 0x01010101u;
  const uint32_t neg = ~(p | (p >> 1)) & 0x01010101u;
  return mag | (neg << 7);
}
__device__ __forceinline__ uint4 tern16_to_operand(uint32_t w) {
  return make_uint4(tern4_to_operand(w), tern4_to_operand(w >> 2), tern4_to_operand(w >> 4),
                    tern4_to_operand(w >> 6));
}
// The packed ternary word of 16 zero codes.
constexpr uint32_t kTernaryZeroWord = 0x55555555u;

// A-operand image (the GEMM's activation operand in global memory): for every 128-row tile
// mt and every 128-element K stage kb, one contiguous 16 KB block that is byte for byte the
// shared-memory image the tensor core reads -- 128 rows of 128 operand bytes in the 128-byte
// swizzle (16-byte chunk c of row r at chunk position c ^ (r % 8), 8-row atoms of 1024 bytes).
// Blocks are ordered (mt, kb), so consecutive K stages of a tile are adjacent and one bulk copy
// can fetch several.  Rows past M in the last tile are never written and never used (each output
// row depends only on its own operand row).
constexpr uint32_t kImageRows = 128;
constexpr uint32_t kImageStageK = 128;
constexpr uint32_t kImageBlockBytes = kImageRows * kImageStageK;  // 16 KB

// Byte offset of the 16-byte operand chunk that holds K positions 16*c16 .. 16*c16+15 of stage
// kb for row `row` of the operand.
__host__ __device__ __forceinline__ uint64_t image_chunk_offset(int64_t row, uint32_t kb, uint32_t c16,
                                                               uint32_t k_stages) {
  const uint64_t mt = static_cast<uint64_t>(row) / kImageRows;
  const uint32_t r = static_cast<uint32_t>(row % kImageRows);
  return (mt * k_stages + kb) * kImageBlockBytes + (r >> 3) * 1024u + (r & 7u) * 128u + ((c16 ^ (r & 7u)) << 4);
}

// Factor that turns an fp32 sum of operand products back into the integer partial, and its
// inverse, the value of one integer unit of such a sum.
constexpr float kOperandUnitInv = 262144.0f;  // 2^18
constexpr float kOperandUnit = 1.0f / 262144.0f;  // 2^-18, exact

}  // namespace jq
