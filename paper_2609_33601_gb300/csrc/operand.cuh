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
// Per byte lane with nibble n (two's complement): t = n >> 3 (the sign), and
// (n ^ (t * 0x8F)) + t  maps n < 8 to n and n >= 8 to 0x80 | (16 - n): the sign-magnitude byte.
// No carry crosses a byte lane (every intermediate lane value stays below 0x90).
__device__ __forceinline__ uint2 nib8_to_operand(uint32_t w) {
  const uint32_t te = (w >> 3) & 0x01010101u;
  const uint32_t to = (w >> 7) & 0x01010101u;
  const uint32_t ve = (w & 0x0F0F0F0Fu) ^ (te * 0x8Fu);
  const uint32_t vo = ((w >> 4) & 0x0F0F0F0Fu) ^ (to * 0x8Fu);
  return make_uint2(ve + te, vo + to);
}

// 32 packed codes (16 bytes) -> 32 operand bytes (two 16-byte chunks).
__device__ __forceinline__ void nib32_to_operand(uint4 p, uint4& lo, uint4& hi) {
  const uint2 a = nib8_to_operand(p.x), b = nib8_to_operand(p.y);
  const uint2 c = nib8_to_operand(p.z), d = nib8_to_operand(p.w);
  lo = make_uint4(a.x, a.y, b.x, b.y);
  hi = make_uint4(c.x, c.y, d.x, d.y);
}

// Factor that turns an fp32 sum of operand products back into the integer partial.
constexpr float kOperandUnitInv = 262144.0f;  // 2^18

}  // namespace jq
