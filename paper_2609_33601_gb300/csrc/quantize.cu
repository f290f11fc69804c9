// quantize.cu -- symmetric INT4 quantisers (activations and weights) and the conversion of
// packed codes into the GEMM's E4M3 operand bytes.  Both producers of the GEMM's A operand also
// write the correction the GEMM needs for its offset-code weights (operand.cuh): per row and
// group, corr = 8 * sum_{k in g} qa[row, k] in the accumulator's units (2^-18), exact.
//
// Rule (per row and per run of G consecutive K elements; group64 / group128 as the paper fixes
// them in Sec. 4.2 "FLUX" and the Appendix experimental-detail tables, G = K for per-token):
//     amax = max|x|,  s = fl32(amax / 7),  q = clamp(rint(fl32(x / s)), -8, 7),  s = q = 0 if amax = 0.
//
// Exact division without a division per element: with r = RN(1/s) (one correctly rounded
// reciprocal per group) and y = RN(x * r), |y - x/s| < 2^-20 and |fl(x/s) - x/s| < 2^-21 for
// |x/s| <= 7.5, so rint(y) == rint(fl(x/s)) unless y lies within 2^-19 of a half-integer.
// Those rare elements (and groups whose scale is subnormal, where 1/s may overflow) take the
// IEEE division __fdiv_rn.  rint(y) itself comes from one fp32 add of 1.5*2^23 + 8: the sum is
// an integer 0x4B400008 + rint(y) whose low nibble is the offset code q + 8.
#include <climits>
#include <cstdint>
#include <type_traits>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kernels.cuh"
#include "operand.cuh"
#include "ptx.cuh"

namespace jq {

namespace {

constexpr float kRintMagic = 12582920.0f;  // 1.5 * 2^23 + 8

// Loads 32 consecutive values of a row as fp32.
__device__ __forceinline__ void load32(const __nv_bfloat16* p, float (&x)[32]) {
  const uint4* v = reinterpret_cast<const uint4*>(p);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint4 u = __ldg(v + i);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      x[8 * i + 2 * j] = __uint_as_float(w[j] << 16);
      x[8 * i + 2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
    }
  }
}
__device__ __forceinline__ void load32(const float* p, float (&x)[32]) {
  const float4* v = reinterpret_cast<const float4*>(p);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float4 u = __ldg(v + i);
    x[4 * i] = u.x;
    x[4 * i + 1] = u.y;
    x[4 * i + 2] = u.z;
    x[4 * i + 3] = u.w;
  }
}

__device__ __forceinline__ float amax32(const float (&x)[32]) {
  float m = 0.0f;
#pragma unroll
  for (int i = 0; i < 32; ++i) m = fmaxf(m, fabsf(x[i]));
  return m;
}

// One code by the rule itself, as its offset nibble q + 8 in [0, 15]: the IEEE quotient, rint,
// the clamp (the elements the reciprocal rule cannot settle, and subnormal scales).
__device__ __forceinline__ uint32_t code_exact(float x, float s) {
  const float q = fminf(fmaxf(rintf(__fdiv_rn(x, s)), -8.0f), 7.0f);
  return static_cast<uint32_t>(static_cast<int>(q) + 8);
}

// 8 values of one group (pairs: elements 2e and 2e + 1 in x[e]) -> their offset codes q + 8 as
// the 8 nibbles of one word in packed order (element 2j in the low nibble of byte j), by the
// reciprocal rule above with r = RN(1/s), its fp32 steps in packed pairs (each component rounds as
// the scalar operation would).  `ties` gets bit 8j + 7 for element 2j and bit 8j + 6 for element
// 2j + 1 when that element's y may lie within 2^-19 of a half-integer (its nibble then needs the
// IEEE quotient).  The test is d^2 - c >= 0 with d = y - rint(y) and c just below
// (1/2 - 2^-19)^2, in one fused operation: every element the reciprocal rule may get wrong is
// flagged, and a few more.  The codes are gathered from the sums' low bytes by byte permutes.
constexpr float kTieSq = 0x1.ffffp-3f;  // 2^-2 - 2^-19: (1/2 - 2^-19)^2 = 2^-2 - 2^-19 + 2^-38, rounded down

__device__ __forceinline__ uint32_t codes8_pairs(const float2 (&x)[4], float r, uint32_t& ties) {
  const float2 r2 = make_float2(r, r), m2 = make_float2(kRintMagic, kRintMagic);
  const float2 nm2 = make_float2(-kRintMagic, -kRintMagic), neg1 = make_float2(-1.0f, -1.0f);
  const float2 nc2 = make_float2(-kTieSq, -kTieSq);
  uint32_t t[8], v[8];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 y = __fmul2_rn(x[e], r2);
    const float2 tt = __fadd2_rn(y, m2);         // 1.5 * 2^23 + 8 + rint(y): low byte q + 8
    const float2 rt = __fadd2_rn(tt, nm2);       // rint(y), exact
    const float2 d = __ffma2_rn(rt, neg1, y);    // y - rint(y), exact
    const float2 g = __ffma2_rn(d, d, nc2);      // d^2 - c: sign clear for a (possible) near-tie
    t[2 * e] = __float_as_uint(tt.x);
    t[2 * e + 1] = __float_as_uint(tt.y);
    v[2 * e] = __float_as_uint(g.x);
    v[2 * e + 1] = __float_as_uint(g.y);
  }
  // low bytes of the even elements to bytes 0-3, of the odd elements likewise, then nibbles
  const uint32_t ev = __byte_perm(__byte_perm(t[0], t[2], 0x0040), __byte_perm(t[4], t[6], 0x0040), 0x5410);
  const uint32_t od = __byte_perm(__byte_perm(t[1], t[3], 0x0040), __byte_perm(t[5], t[7], 0x0040), 0x5410);
  // top bytes (signs) of the tie tests likewise
  const uint32_t tv = __byte_perm(__byte_perm(v[0], v[2], 0x0073), __byte_perm(v[4], v[6], 0x0073), 0x5410);
  const uint32_t to = __byte_perm(__byte_perm(v[1], v[3], 0x0073), __byte_perm(v[5], v[7], 0x0073), 0x5410);
  ties = (~tv & 0x80808080u) | ((~to & 0x80808080u) >> 1);
  return ev | (od << 4);
}
// The bit of `ties` that flags element j of the 8.
__host__ __device__ constexpr int tie_bit(int j) { return 8 * (j >> 1) + ((j & 1) ? 6 : 7); }

// 32 values of one group (scale s) -> 4 words of packed two's complement nibbles.
__device__ __forceinline__ void quantize32(const float (&x)[32], float s, uint32_t (&pk)[4]) {
  if (s == 0.0f) {
#pragma unroll
    for (int i = 0; i < 4; ++i) pk[i] = 0u;
    return;
  }
  const bool exact_only = !(s >= 0x1p-126f);  // subnormal scale: 1/s may not be representable
  const float r = __frcp_rn(s);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    uint32_t ties = 0xC0C0C0C0u, w = 0;  // a subnormal scale: every element by division
    if (!exact_only) {
      const float2 xp[4] = {make_float2(x[8 * i], x[8 * i + 1]), make_float2(x[8 * i + 2], x[8 * i + 3]),
                            make_float2(x[8 * i + 4], x[8 * i + 5]), make_float2(x[8 * i + 6], x[8 * i + 7])};
      w = codes8_pairs(xp, r, ties);
    }
    if (ties != 0) {  // the elements near a tie take the IEEE quotient
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if ((ties >> tie_bit(j)) & 1u)
          w = (w & ~(0xFu << (4 * j))) | (code_exact(x[8 * i + j], s) << (4 * j));
    }
    pk[i] = w ^ 0x88888888u;  // offset (q + 8) -> two's complement nibble
  }
}

// The same for 8 bf16 values (one 16-byte unit of a row, element 2e in the low half of word e).
__device__ __forceinline__ uint32_t codes8_offset(uint4 u, float r, uint32_t& ties) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
  float2 x[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) x[e] = make_float2(__uint_as_float(w[e] << 16), __uint_as_float(w[e] & 0xFFFF0000u));
  return codes8_pairs(x, r, ties);
}

// ---------------------------------------------------------------- DiT neighbour operations
// The inputs of a DiT-XL/2 block's linears come from the adaLN modulation (before the attention's
// QKV projection and the MLP's first linear) and from the MLP's tanh GELU (before its second
// linear).  Fusing them here makes the quantiser read the operation's input instead of a bf16
// tensor the operation wrote.  Each yields the bf16 value the linear layer would receive.
enum NeighbourOp : int { kOpNone = 0, kOpModulate = 1, kOpGelu = 2 };

struct OpArgs {
  const float* shift = nullptr;  // modulation: [samples, K]
  const float* scale = nullptr;  // modulation: [samples, K]
  int64_t tokens_per_sample = 1;
};

// bf16( fl32( fl32( x * fl32(1 + scale) ) + shift ) ): IEEE single steps, no contraction, one
// rounding to bf16 (round to nearest even).
__device__ __forceinline__ float modulate_bf16(float x, float shift, float scale) {
  const float z = __fadd_rn(__fmul_rn(x, __fadd_rn(1.0f, scale)), shift);
  return __bfloat162float(__float2bfloat16_rn(z));
}

// e^x for x <= 0 in fp32 steps: Cody and Waite's reduction n = rint(x log2 e), r = x - n ln2 with
// ln2 split into a 15-bit high part (n * ln2_hi exact for |n| <= 150) and a low part, e^r by its
// Taylor polynomial to degree 8 (Horner, fused multiply-adds; |r| <= 0.35, truncation below
// 2^-32), e^x = 2^n e^r by one exact-exponent product (two below the normal range); 0 below
// x = -104.  Every step is one IEEE operation, so the CPU oracle reproduces it bit for bit.
//
// It (and the GELU below) works on a pair of values, the floating-point steps as packed pairs:
// each packed operation rounds every component exactly as the scalar one would (the packed fused
// multiply-add is __fmaf_rn per component), so the values are those of the scalar sequence with
// half the floating-point instructions; the selects are per component.  Branch-free (selects only), so that independent pairs interleave: below -104
// the result is 0, and below the normal range the power of two is applied as 2^(n+64) then 2^-64
// (the second product is by exactly 1 above).
__device__ __forceinline__ float pow2_f32(int n) { return __int_as_float((n + 127) << 23); }
__device__ __forceinline__ float2 f2(float v) { return make_float2(v, v); }

__device__ __forceinline__ float2 exp_neg_f32x2(float2 x) {
  const bool zx = x.x < -104.0f, zy = x.y < -104.0f;
  x = make_float2(fmaxf(x.x, -104.0f), fmaxf(x.y, -104.0f));
  // n = rint(t) by the 1.5 * 2^23 addition (t in [-151, 0]: the sum's unit is 1 and rounds to
  // nearest even, exactly as rint; the subtraction is exact)
  const float2 t = __fmul2_rn(x, f2(0x1.715476p+0f));
  const float2 tm = __fadd2_rn(t, f2(12582912.0f));
  const float2 n = __fadd2_rn(tm, f2(-12582912.0f));
  const float2 nn = make_float2(-n.x, -n.y);
  float2 r = __ffma2_rn(nn, f2(0x1.62e4p-1f), x);
  r = __ffma2_rn(nn, f2(0x1.7f7d1cp-20f), r);
  float2 p = f2(0x1.a01a02p-16f);           // 1/8!
  p = __ffma2_rn(p, r, f2(0x1.a01a02p-13f));  // 1/7!
  p = __ffma2_rn(p, r, f2(0x1.6c16c2p-10f));  // 1/6!
  p = __ffma2_rn(p, r, f2(0x1.111112p-7f));   // 1/5!
  p = __ffma2_rn(p, r, f2(0x1.555556p-5f));   // 1/4!
  p = __ffma2_rn(p, r, f2(0x1.555556p-3f));   // 1/3!
  p = __ffma2_rn(p, r, f2(0x1p-1f));          // 1/2!
  p = __ffma2_rn(p, r, f2(1.0f));
  p = __ffma2_rn(p, r, f2(1.0f));
  const int nx = static_cast<int>(n.x), ny = static_cast<int>(n.y);
  const bool lx = nx < -126, ly = ny < -126;
  const float2 v = __fmul2_rn(__fmul2_rn(p, make_float2(pow2_f32(lx ? nx + 64 : nx), pow2_f32(ly ? ny + 64 : ny))),
                              make_float2(lx ? 0x1p-64f : 1.0f, ly ? 0x1p-64f : 1.0f));
  return make_float2(zx ? 0.0f : v.x, zy ? 0.0f : v.y);
}

// a / d for d in [1, 2] and a in [0, 1] without the division unit: Newton-Raphson division (the
// reciprocal of D = d/2 in [1/2, 1] from the linear estimate 48/17 - 32/17 D, three iterations
// y += y (1 - D y), each squaring the relative error from at most 1/17), then Markstein's
// correction q + (a - q d) y with the exact remainder from a fused multiply-add.  It is not the
// IEEE quotient for every such pair (a = 1, d = 2 - 2^-23 gives 1/2 instead of 1/2 + 2^-24), so
// it stands in for the GELU's division only because the GELU value, rounded to bf16, is the
// oracle's for every one of the 65280 finite bf16 inputs (a GPU test runs all of them).
__device__ __forceinline__ float2 div_1_2(float2 a, float2 d) {
  const float2 D = __fmul2_rn(d, f2(0.5f));
  const float2 nD = make_float2(-D.x, -D.y);
  float2 y = __ffma2_rn(D, f2(-32.0f / 17.0f), f2(48.0f / 17.0f));
#pragma unroll
  for (int i = 0; i < 3; ++i) y = __ffma2_rn(y, __ffma2_rn(nD, y, f2(1.0f)), y);
  const float2 yh = __fmul2_rn(y, f2(0.5f));  // ~ 1/d
  const float2 q = __fmul2_rn(a, yh);
  const float2 r = __ffma2_rn(make_float2(-q.x, -q.y), d, a);  // a - q d, exact
  return __ffma2_rn(r, yh, q);
}

// The tanh GELU evaluated in fp32 by the oracle's fixed sequence of IEEE operations, but for the
// logistic's division (div_1_2 above): u = 0.7978846 (h + 0.044715 h^3), 1 + tanh(u) = 2 sigma(2u) with the logistic as
// 1 / (1 + e^{-2u}) (u >= 0) or e^{2u} / (1 + e^{2u}) (u < 0), g = h sigma(2u); then rounded to
// bf16 as a bf16 model stores it.  Straight-line: the logistic takes one division with a
// selected numerator (e = e^{-2|u|} in both forms); +-0 stays +-0.  On a pair of values, as above.
__device__ __forceinline__ float2 gelu_bf16x2(float2 h) {
  const float2 h3 = __fmul2_rn(__fmul2_rn(h, h), h);
  const float2 p = __fadd2_rn(h, __fmul2_rn(f2(0x1.6e4e26p-5f), h3));
  const float2 u = __fmul2_rn(f2(0x1.988454p-1f), p);
  const float2 e = exp_neg_f32x2(__fmul2_rn(f2(-2.0f), make_float2(fabsf(u.x), fabsf(u.y))));
  const float2 d = __fadd2_rn(f2(1.0f), e);
  const float2 sig = div_1_2(make_float2(u.x >= 0.0f ? 1.0f : e.x, u.y >= 0.0f ? 1.0f : e.y), d);
  const float2 g = __fmul2_rn(h, sig);
  return __bfloat1622float2(__floats2bfloat162_rn(g.x, g.y));
}

// The GELU's input is a bf16 value, so the whole function is a table of 65536 bf16 results: the
// fused quantiser looks each value up instead of evaluating the sequence (about 35 operations an
// element, which made that kernel compute-bound).  The table is filled on the device by
// gelu_bf16x2 itself -- the same values by construction -- once per device before the first
// fused GELU call (launch_gelu_quantize_act).
__device__ uint16_t g_gelu_bf16[65536];

__global__ void __launch_bounds__(256) gelu_table_kernel() {
  const uint32_t i = blockIdx.x * 256u + threadIdx.x;  // entries 2i, 2i + 1
  if (i >= 32768u) return;
  const float2 g = gelu_bf16x2(make_float2(__uint_as_float((2u * i) << 16), __uint_as_float((2u * i + 1u) << 16)));
  g_gelu_bf16[2u * i] = static_cast<uint16_t>(__float_as_uint(g.x) >> 16);
  g_gelu_bf16[2u * i + 1u] = static_cast<uint16_t>(__float_as_uint(g.y) >> 16);
}

// Applies the neighbour operation to 32 consecutive values of row `row` from K index `col`.
template <int kOp>
__device__ __forceinline__ void apply_op(float (&v)[32], int64_t row, int64_t col, int64_t K, const OpArgs& op) {
  if constexpr (kOp == kOpModulate) {
    const int64_t base = (row / op.tokens_per_sample) * K + col;
    const float4* sh = reinterpret_cast<const float4*>(op.shift + base);
    const float4* sc = reinterpret_cast<const float4*>(op.scale + base);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float4 a = __ldg(sh + i), c = __ldg(sc + i);
      v[4 * i] = modulate_bf16(v[4 * i], a.x, c.x);
      v[4 * i + 1] = modulate_bf16(v[4 * i + 1], a.y, c.y);
      v[4 * i + 2] = modulate_bf16(v[4 * i + 2], a.z, c.z);
      v[4 * i + 3] = modulate_bf16(v[4 * i + 3], a.w, c.w);
    }
  } else if constexpr (kOp == kOpGelu) {  // v[i] holds a bf16 value: its bits index the table
#pragma unroll
    for (int i = 0; i < 32; ++i)
      v[i] = __uint_as_float(static_cast<uint32_t>(__ldg(g_gelu_bf16 + (__float_as_uint(v[i]) >> 16))) << 16);
  }
}

// 32 codes of one row starting at K index `col` (a multiple of 32): packed codes go to the
// row-major [rows, K/2] array; operand bytes go to the A-operand image (operand.cuh).
template <bool kOperand>
__device__ __forceinline__ void store32(uint8_t* out, int64_t row, int64_t col, int64_t K, const uint32_t (&pk)[4]) {
  const uint4 p = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  if constexpr (kOperand) {
    uint4 lo, hi;
    nib32_to_operand(p, lo, hi);
    const uint32_t k_stages = static_cast<uint32_t>(K / kImageStageK);
    const uint32_t kb = static_cast<uint32_t>(col / kImageStageK);
    const uint32_t c16 = static_cast<uint32_t>((col % kImageStageK) / 16);
    *reinterpret_cast<uint4*>(out + image_chunk_offset(row, kb, c16, k_stages)) = lo;
    *reinterpret_cast<uint4*>(out + image_chunk_offset(row, kb, c16 + 1, k_stages)) = hi;
  } else {
    *reinterpret_cast<uint4*>(out + row * (K / 2) + col / 2) = p;
  }
}

// The rest of one thread's 32 elements once they are in registers (as the bf16 value the linear
// layer receives): the group amax over the group's L adjacent lanes, the scale, the codes and their
// store, and the group's scale (and, for the operand image, its code-sum correction) from the
// group's first lane.  Every lane of the warp takes part (the shuffles); `valid` lanes hold data.
template <int L, bool kOperand, bool kScaleT>
__device__ __forceinline__ void finish_chunk(const float (&v)[32], bool valid, int64_t row, int64_t col, int64_t M,
                                             int64_t K, uint8_t* __restrict__ out, float* __restrict__ scales,
                                             float* __restrict__ corr) {
  float a = amax32(v);
#pragma unroll
  for (int o = 1; o < L; o <<= 1) a = fmaxf(a, __shfl_xor_sync(0xFFFFFFFFu, a, o));
  const float s = __fdiv_rn(a, 7.0f);
  uint32_t pk[4] = {0x88888888u, 0x88888888u, 0x88888888u, 0x88888888u};  // sums to 0 past the end
  if (valid) {
    quantize32(v, s, pk);
    store32<kOperand>(out, row, col, K, pk);
  }
  int cs = 0;
  if constexpr (kOperand) {  // the group's code sum, over its L lanes
    cs = valid ? nib32_sum(make_uint4(pk[0], pk[1], pk[2], pk[3])) : 0;
#pragma unroll
    for (int o = 1; o < L; o <<= 1) cs += __shfl_xor_sync(0xFFFFFFFFu, cs, o);
  }
  if (valid && (threadIdx.x & (L - 1)) == 0) {
    const int64_t ng = K / (32 * L);
    const int64_t g = col / (32 * L);
    if constexpr (kScaleT) scales[g * M + row] = s;
    else scales[row * ng + g] = s;
    if constexpr (kOperand) corr[row * ng + g] = (float)(8 * cs) * kOperandUnit;
  }
}

// G = 32 * L (L = 2 or 4): each thread quantises 32 consecutive elements; the L threads of a
// group are adjacent lanes and reduce amax with xor-shuffles.
template <typename In, int L, bool kOperand, bool kScaleT, int kOp = kOpNone>
__global__ void __launch_bounds__(256, kOp == kOpModulate ? 4 : 1) quantize_groups_kernel(const In* __restrict__ x, int64_t M, int64_t K,
                                                              int64_t ldx, uint8_t* __restrict__ out,
                                                              float* __restrict__ scales, float* __restrict__ corr,
                                                              const OpArgs op) {
  // The activation quantiser lets the next kernel (the linear layer, which starts by streaming
  // its weights) launch at once; the weight packer does not, so nothing reads weights early.
  if (!kScaleT) pdl_launch_dependents();
  pdl_wait();
  const int64_t chunks_per_row = K / 32;
  const int64_t total = M * chunks_per_row;
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c - (threadIdx.x & 31) < total;
       c += (int64_t)gridDim.x * blockDim.x) {
    const bool valid = c < total;
    const int64_t row = valid ? c / chunks_per_row : 0;
    const int64_t col = valid ? (c % chunks_per_row) * 32 : 0;
    float v[32];
    if (valid) {
      load32(x + row * ldx + col, v);
      apply_op<kOp>(v, row, col, K, op);
    } else {
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = 0.0f;
    }
    finish_chunk<L, kOperand, kScaleT>(v, valid, row, col, M, K, out, scales, corr);
  }
}

// The same quantiser for bf16 activations with many rows, the input staged through shared memory
// by TMA: tiles of 64 rows x 256 elements (32 KB) in a 3-slot ring per CTA, two CTAs per SM, so
// that the bytes in flight are set by the rings (up to 192 KB per SM), not by registers.  Warp 16
// (one thread) issues the tile loads; warps 0-15 take a tile's 512 chunks of 32 elements, one per
// thread (chunk j: row j / 8 of the tile, elements 32 (j % 8) ..), and release the slot.  A chunk
// is read from shared memory twice (the group amax, then the codes) so that few values live in
// registers.  The codes follow the same reciprocal rule as quantize32 with the fp32 steps in
// packed pairs; the elements near a tie are then redone with the IEEE quotient one by one.  Rows past M and columns past
// K arrive as zeros and are skipped.  Tiles are ordered column-fastest.
constexpr int kQtRows = 64, kQtCols = 256, kQtSlots = 3, kQtConsumerWarps = 16;
constexpr int kQtThreads = 32 * (kQtConsumerWarps + 1);
constexpr uint32_t kQtSlotBytes = kQtRows * kQtCols * 2;
constexpr uint32_t kQtSmemBytes = kQtSlots * kQtSlotBytes + 2 * kQtSlots * 8 + 16;
static_assert(32 * kQtConsumerWarps * 32 == kQtRows * kQtCols, "one chunk of 32 elements per consumer thread");

template <int L, bool kOperand>
__global__ void __launch_bounds__(kQtThreads, 2) quantize_tiles_kernel(const __grid_constant__ CUtensorMap tmX,
                                                                       int64_t M, int64_t K,
                                                                       uint8_t* __restrict__ out,
                                                                       float* __restrict__ scales,
                                                                       float* __restrict__ corr, uint32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kQtSlots * kQtSlotBytes);
  uint64_t* empty = full + kQtSlots;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty + kQtSlots);
  const uint32_t warp = warp_id(), lane = lane_id();
  if (threadIdx.x == 0) {
    for (int i = 0; i < kQtSlots; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kQtConsumerWarps);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  pdl_launch_dependents();  // as in quantize_groups_kernel
  pdl_wait();
  const int64_t col_tiles = (K + kQtCols - 1) / kQtCols;
  const int64_t tiles = (M + kQtRows - 1) / kQtRows * col_tiles;
  if (warp == kQtConsumerWarps) {  // TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmX);
      uint32_t it = 0;
      for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x, ++it) {
        const uint32_t slot = it % kQtSlots;
        if (!mbar_wait(&empty[slot], ((it / kQtSlots) & 1u) ^ 1u, abort_flag, status)) break;
        mbar_arrive_expect_tx(&full[slot], kQtSlotBytes);
        tma_load_2d(smem + slot * kQtSlotBytes, &tmX, &full[slot], (int)((t % col_tiles) * kQtCols),
                    (int)((t / col_tiles) * kQtRows));
      }
      // After an abort, let the loads already issued land before the CTA's shared memory goes.
      if (*abort_flag) {
        int dummy = 0;
        const uint32_t issued = it;
        for (uint32_t k = issued > (uint32_t)kQtSlots ? issued - kQtSlots : 0; k < issued; ++k)
          (void)mbar_wait(&full[k % kQtSlots], (k / kQtSlots) & 1u, &dummy, nullptr);
      }
    }
    return;
  }
  const int j = (int)threadIdx.x;  // this thread's chunk of every tile
  uint32_t it = 0;
  for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x, ++it) {
    const uint32_t slot = it % kQtSlots;
    if (!__all_sync(0xFFFFFFFFu, mbar_wait(&full[slot], (it / kQtSlots) & 1u, abort_flag, status))) break;
    const int64_t row = (t / col_tiles) * kQtRows + (j >> 3), col = (t % col_tiles) * kQtCols + 32 * (j & 7);
    const bool valid = row < M && col < K;
    const uint4* src = reinterpret_cast<const uint4*>(smem + slot * kQtSlotBytes + (j >> 3) * (kQtCols * 2) +
                                                      (j & 7) * 64);
    // amax over bf16 pairs (|x| by clearing the signs; finite inputs), then as fp32
    __nv_bfloat162 m2 = __floats2bfloat162_rn(0.0f, 0.0f);  // zeros past the ends
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint4 u = src[q];
      const uint32_t w[4] = {u.x & 0x7FFF7FFFu, u.y & 0x7FFF7FFFu, u.z & 0x7FFF7FFFu, u.w & 0x7FFF7FFFu};
#pragma unroll
      for (int e = 0; e < 4; ++e) m2 = __hmax2(m2, *reinterpret_cast<const __nv_bfloat162*>(&w[e]));
    }
    float a = fmaxf(__low2float(m2), __high2float(m2));
#pragma unroll
    for (int o = 1; o < L; o <<= 1) a = fmaxf(a, __shfl_xor_sync(0xFFFFFFFFu, a, o));
    const float s = __fdiv_rn(a, 7.0f);
    uint32_t pk[4] = {0u, 0u, 0u, 0u};  // an all-zero group (s = 0) has zero codes
    if (valid && s != 0.0f) {
      const bool normal = s >= 0x1p-126f;  // 1/s representable: the reciprocal rule applies
      const float r = __frcp_rn(s);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t ties = 0xC0C0C0C0u, word = 0;  // a subnormal scale: every element by division
        if (normal) word = codes8_offset(src[q], r, ties);
        // the elements near a tie (all of them for a subnormal scale) take the IEEE quotient
        while (ties != 0) {
          const int bit = __ffs(ties) - 1;  // 8j + 7: element 2j, 8j + 6: element 2j + 1
          ties &= ties - 1;
          const int e = 2 * (bit >> 3) + ((bit & 7) == 6 ? 1 : 0);
          const uint16_t b = reinterpret_cast<const uint16_t*>(src + q)[e];
          const uint32_t c = code_exact(__uint_as_float((uint32_t)b << 16), s);
          word = (word & ~(0xFu << (4 * e))) | (c << (4 * e));
        }
        pk[q] = word ^ 0x88888888u;
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[slot]);  // the slot's bytes are no longer read
    if (valid) store32<kOperand>(out, row, col, K, pk);
    int cs = 0;
    if constexpr (kOperand) {  // the group's code sum, over its L lanes
      cs = valid ? nib32_sum(make_uint4(pk[0], pk[1], pk[2], pk[3])) : 0;
#pragma unroll
      for (int o = 1; o < L; o <<= 1) cs += __shfl_xor_sync(0xFFFFFFFFu, cs, o);
    }
    if (valid && (threadIdx.x & (L - 1)) == 0) {
      const int64_t ng = K / (32 * L), g = col / (32 * L);
      scales[row * ng + g] = s;
      if constexpr (kOperand) corr[row * ng + g] = (float)(8 * cs) * kOperandUnit;
    }
  }
}

// G = K: one block per row; pass 1 reduces the row amax, pass 2 quantises (the second read
// of the row hits L1/L2).
template <typename In, bool kOperand, bool kScaleT, int kOp = kOpNone>
__global__ void __launch_bounds__(128) quantize_rows_kernel(const In* __restrict__ x, int64_t M, int64_t K,
                                                            int64_t ldx, uint8_t* __restrict__ out,
                                                            float* __restrict__ scales, float* __restrict__ corr,
                                                            const OpArgs op) {
  __shared__ float red[4];
  __shared__ int red_cs[4];
  if (!kScaleT) pdl_launch_dependents();  // as in quantize_groups_kernel
  pdl_wait();
  for (int64_t row = blockIdx.x; row < M; row += gridDim.x) {
    const In* xr = x + row * ldx;
    float a = 0.0f;
    for (int64_t col = threadIdx.x * 32; col < K; col += 32 * blockDim.x) {
      float v[32];
      load32(xr + col, v);
      apply_op<kOp>(v, row, col, K, op);
      a = fmaxf(a, amax32(v));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) a = fmaxf(a, __shfl_xor_sync(0xFFFFFFFFu, a, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = a;
    __syncthreads();
    a = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
    __syncthreads();
    const float s = __fdiv_rn(a, 7.0f);
    int cs = 0;
    for (int64_t col = threadIdx.x * 32; col < K; col += 32 * blockDim.x) {
      float v[32];
      load32(xr + col, v);
      apply_op<kOp>(v, row, col, K, op);
      uint32_t pk[4];
      quantize32(v, s, pk);
      store32<kOperand>(out, row, col, K, pk);
      if constexpr (kOperand) cs += nib32_sum(make_uint4(pk[0], pk[1], pk[2], pk[3]));
    }
    if constexpr (kOperand) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) cs += __shfl_xor_sync(0xFFFFFFFFu, cs, o);
      if ((threadIdx.x & 31) == 0) red_cs[threadIdx.x >> 5] = cs;
      __syncthreads();
      cs = red_cs[0] + red_cs[1] + red_cs[2] + red_cs[3];
      __syncthreads();
    }
    if (threadIdx.x == 0) {
      if constexpr (kScaleT) scales[row] = s;  // [1, M]
      else scales[row] = s;                    // [M, 1]
      if constexpr (kOperand) corr[row] = (float)(8 * cs) * kOperandUnit;
    }
  }
}

// Packed codes [rows, K/2] -> the A-operand image (16 bytes in, 32 bytes out per thread) and
// the per-group corrections.  G = 32 * L: a group is L adjacent lanes (a row holds a multiple of
// L chunks, so no group straddles a warp).
template <int L>
__global__ void __launch_bounds__(256) expand_operand_kernel(const uint8_t* __restrict__ packed, int64_t rows,
                                                             int64_t K, uint8_t* __restrict__ image,
                                                             float* __restrict__ corr) {
  pdl_launch_dependents();
  pdl_wait();
  const int64_t per_row = K / 32;
  const int64_t chunks = rows * per_row;
  const uint32_t k_stages = static_cast<uint32_t>(K / kImageStageK);
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c - (threadIdx.x & 31) < chunks;
       c += (int64_t)gridDim.x * blockDim.x) {
    const bool valid = c < chunks;
    const int64_t row = valid ? c / per_row : 0;
    const int64_t col = valid ? (c % per_row) * 32 : 0;
    const uint4 p = valid ? __ldg(reinterpret_cast<const uint4*>(packed) + c)
                          : make_uint4(0x88888888u, 0x88888888u, 0x88888888u, 0x88888888u);
    if (valid) {
      uint4 lo, hi;
      nib32_to_operand(p, lo, hi);
      const uint32_t kb = static_cast<uint32_t>(col / kImageStageK);
      const uint32_t c16 = static_cast<uint32_t>((col % kImageStageK) / 16);
      *reinterpret_cast<uint4*>(image + image_chunk_offset(row, kb, c16, k_stages)) = lo;
      *reinterpret_cast<uint4*>(image + image_chunk_offset(row, kb, c16 + 1, k_stages)) = hi;
    }
    int cs = valid ? nib32_sum(p) : 0;
#pragma unroll
    for (int o = 1; o < L; o <<= 1) cs += __shfl_xor_sync(0xFFFFFFFFu, cs, o);
    if (valid && (threadIdx.x & (L - 1)) == 0) corr[row * (per_row / L) + col / (32 * L)] = (float)(8 * cs) * kOperandUnit;
  }
}

// G = K: one block per row (the row's code sum is a block reduction).
__global__ void __launch_bounds__(128) expand_operand_rows_kernel(const uint8_t* __restrict__ packed, int64_t rows,
                                                                  int64_t K, uint8_t* __restrict__ image,
                                                                  float* __restrict__ corr) {
  __shared__ int red_cs[4];
  pdl_launch_dependents();
  pdl_wait();
  const int64_t per_row = K / 32;
  const uint32_t k_stages = static_cast<uint32_t>(K / kImageStageK);
  for (int64_t row = blockIdx.x; row < rows; row += gridDim.x) {
    int cs = 0;
    for (int64_t i = threadIdx.x; i < per_row; i += blockDim.x) {
      const uint4 p = __ldg(reinterpret_cast<const uint4*>(packed) + row * per_row + i);
      uint4 lo, hi;
      nib32_to_operand(p, lo, hi);
      const int64_t col = i * 32;
      const uint32_t kb = static_cast<uint32_t>(col / kImageStageK);
      const uint32_t c16 = static_cast<uint32_t>((col % kImageStageK) / 16);
      *reinterpret_cast<uint4*>(image + image_chunk_offset(row, kb, c16, k_stages)) = lo;
      *reinterpret_cast<uint4*>(image + image_chunk_offset(row, kb, c16 + 1, k_stages)) = hi;
      cs += nib32_sum(p);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cs += __shfl_xor_sync(0xFFFFFFFFu, cs, o);
    if ((threadIdx.x & 31) == 0) red_cs[threadIdx.x >> 5] = cs;
    __syncthreads();
    if (threadIdx.x == 0) corr[row] = (float)(8 * (red_cs[0] + red_cs[1] + red_cs[2] + red_cs[3])) * kOperandUnit;
    __syncthreads();
  }
}

int grid_for(int64_t work_items, int threads, int sms) {
  int64_t blocks = (work_items + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return static_cast<int>(blocks);
}

// bf16 activations (with no neighbour operation) take the TMA-staged kernel when every CTA gets
// at least two tiles (each CTA's first tile waits for its whole copy; smaller inputs are better
// served by the register kernel's many small loads).
constexpr int64_t kQtMinRows = 64;
constexpr int kQtMinTilesPerSm = 4;

template <int L, bool kOperand>
cudaError_t launch_quantize_tiles(const __nv_bfloat16* x, int64_t M, int64_t K, int64_t ldx, uint8_t* out,
                                  float* scales, float* corr, cudaStream_t stream, int sms) {
  // The input as a 2-D tensor [M, K] of row pitch ldx (the callers check that the base and the
  // pitch are 16-byte aligned, as the tensor map needs); boxes of 256 x 64, zeros past the ends.
  CUtensorMap tm;
  if (!encode_2d(&tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, x, (uint64_t)K, (uint64_t)M, (uint64_t)ldx * 2, kQtCols,
                 kQtRows, CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;
  static PerDevice<bool> smem_attr;  // once per device and instantiation
  bool attr_ok = false;
  cudaError_t ae = smem_attr.get(
      [](bool& v) {
        v = true;
        return cudaFuncSetAttribute(quantize_tiles_kernel<L, kOperand>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kQtSmemBytes);
      },
      attr_ok);
  if (ae != cudaSuccess) return ae;
  const int64_t tiles = (M + kQtRows - 1) / kQtRows * ((K + kQtCols - 1) / kQtCols);
  const int64_t cap = 2 * static_cast<int64_t>(sms);  // two CTAs per SM
  const int grid = static_cast<int>(tiles < cap ? tiles : cap);
  return launch_pdl(quantize_tiles_kernel<L, kOperand>, dim3(grid), dim3(kQtThreads), kQtSmemBytes, stream, tm, M, K,
                    out, scales, corr, device_status_word());
}

template <typename In, bool kOperand, bool kScaleT, int kOp = kOpNone>
cudaError_t launch_quantize(const In* x, int64_t M, int64_t K, int64_t ldx, int G, uint8_t* out, float* scales,
                            float* corr, cudaStream_t stream, int sms, const OpArgs& op = OpArgs()) {
  if (M == 0) return cudaSuccess;
  if (G == K) {
    int blocks = static_cast<int>(M < static_cast<int64_t>(sms) * 16 ? M : static_cast<int64_t>(sms) * 16);
    return launch_pdl(quantize_rows_kernel<In, kOperand, kScaleT, kOp>, dim3(blocks), dim3(128), 0, stream, x, M, K,
                      ldx, out, scales, corr, op);
  }
  if constexpr (std::is_same<In, __nv_bfloat16>::value && !kScaleT && kOp == kOpNone) {
    const int64_t tiles = (M + kQtRows - 1) / kQtRows * ((K + kQtCols - 1) / kQtCols);
    if (M >= kQtMinRows && M <= INT32_MAX && tiles >= kQtMinTilesPerSm * static_cast<int64_t>(sms))
      return G == 64 ? launch_quantize_tiles<2, kOperand>(x, M, K, ldx, out, scales, corr, stream, sms)
                     : launch_quantize_tiles<4, kOperand>(x, M, K, ldx, out, scales, corr, stream, sms);
  }
  const int grid = grid_for(M * (K / 32), 256, sms);
  if (G == 64)
    return launch_pdl(quantize_groups_kernel<In, 2, kOperand, kScaleT, kOp>, dim3(grid), dim3(256), 0, stream, x, M,
                      K, ldx, out, scales, corr, op);
  return launch_pdl(quantize_groups_kernel<In, 4, kOperand, kScaleT, kOp>, dim3(grid), dim3(256), 0, stream, x, M, K,
                    ldx, out, scales, corr, op);
}

}  // namespace

cudaError_t launch_quantize_act(const void* x, int64_t M, int64_t K, int64_t ldx, int G, uint8_t* q, float* s_a,
                                cudaStream_t stream, int sms) {
  return launch_quantize<__nv_bfloat16, false, false>(static_cast<const __nv_bfloat16*>(x), M, K, ldx, G, q, s_a,
                                                      nullptr, stream, sms);
}

cudaError_t launch_quantize_act_operand(const void* x, int64_t M, int64_t K, int64_t ldx, int G, uint8_t* op,
                                        float* s_a, float* corr, cudaStream_t stream, int sms) {
  return launch_quantize<__nv_bfloat16, true, false>(static_cast<const __nv_bfloat16*>(x), M, K, ldx, G, op, s_a,
                                                     corr, stream, sms);
}

cudaError_t launch_pack_weight(const float* w, int64_t N, int64_t K, int G, uint8_t* qw, float* s_w,
                               cudaStream_t stream, int sms) {
  return launch_quantize<float, false, true>(w, N, K, K, G, qw, s_w, nullptr, stream, sms);
}

cudaError_t launch_expand_operand(const uint8_t* packed, int64_t rows, int64_t K, int G, uint8_t* op, float* corr,
                                  cudaStream_t stream, int sms) {
  const int64_t chunks = rows * (K / 32);
  if (chunks == 0) return cudaSuccess;
  if (G == K) {
    const int blocks = static_cast<int>(rows < static_cast<int64_t>(sms) * 16 ? rows : static_cast<int64_t>(sms) * 16);
    return launch_pdl(expand_operand_rows_kernel, dim3(blocks), dim3(128), 0, stream, packed, rows, K, op, corr);
  }
  const int grid = grid_for(chunks, 256, sms);
  if (G == 64) return launch_pdl(expand_operand_kernel<2>, dim3(grid), dim3(256), 0, stream, packed, rows, K, op, corr);
  return launch_pdl(expand_operand_kernel<4>, dim3(grid), dim3(256), 0, stream, packed, rows, K, op, corr);
}

}  // namespace jq

namespace jq {

cudaError_t launch_modulate_quantize_act(const void* x, int64_t M, int64_t K, int64_t ldx, const float* shift,
                                         const float* scale, int64_t tokens_per_sample, int G, uint8_t* q, float* s_a,
                                         cudaStream_t stream, int sms) {
  OpArgs op;
  op.shift = shift;
  op.scale = scale;
  op.tokens_per_sample = tokens_per_sample;
  return launch_quantize<__nv_bfloat16, false, false, kOpModulate>(static_cast<const __nv_bfloat16*>(x), M, K, ldx, G, q,
                                                                    s_a, nullptr, stream, sms, op);
}

cudaError_t launch_gelu_quantize_act(const void* h, int64_t M, int64_t K, int64_t ldh, int G, uint8_t* q, float* s_a,
                                     cudaStream_t stream, int sms) {
  // The GELU table: filled once per device and waited for before it counts as ready, so a call
  // on any stream of the device may read it.  A first call made while `stream` is being captured
  // into a graph cannot wait: it puts the filling kernel into the graph ahead of the quantiser
  // (every replay rewrites the same values) and leaves the once-per-device filling to a later
  // call made outside a capture.
  static PerDevice<bool> table;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess) return cudaGetLastError();
  if (cs == cudaStreamCaptureStatusNone) {
    bool ready = false;
    cudaError_t e = table.get(
        [stream](bool& v) {
          gelu_table_kernel<<<128, 256, 0, stream>>>();
          cudaError_t le = cudaGetLastError();
          if (le == cudaSuccess) le = cudaStreamSynchronize(stream);
          v = le == cudaSuccess;
          return le;
        },
        ready);
    if (e != cudaSuccess) return e;
  } else {
    gelu_table_kernel<<<128, 256, 0, stream>>>();
    cudaError_t le = cudaGetLastError();
    if (le != cudaSuccess) return le;
  }
  return launch_quantize<__nv_bfloat16, false, false, kOpGelu>(static_cast<const __nv_bfloat16*>(h), M, K, ldh, G, q,
                                                                s_a, nullptr, stream, sms);
}

}  // namespace jq
