// nvfp4.cu -- the NVFP4 W4A4 linear layer (the format of the paper's LLaDA-8B rows, Appendix
// table "ELF-B and LLaDA-8B experimental details": "NVFP4 W4A4").
//
// The format: FP4 E2M1 elements (magnitudes 0, 0.5, 1, 1.5, 2, 3, 4, 6), one FP8 E4M3 scale per
// block of 16 consecutive reduction-axis elements of a row, one fp32 scale g per tensor.  Per
// block b:  s_b = e4m3(fl32(amax_b / fl32(6 g))),  S_b = fl32(s_b g),  q = e2m1(fl32(x / S_b)),
// both roundings to nearest with ties to the even mantissa and saturating (448, 6); q = 0 where
// g == 0 or S_b == 0.  Weights: g = fl32(amax |w| / 2688); activations: g given by the caller.
// The layer: y = sum_b (sum_{k in b} qa qw) sa_b sw_b ga gw + bias.
//
// Kernels:
//   nvfp4_amax_kernel / nvfp4_finish_g_kernel  the weights' tensor amax and g (three launches
//                      with the quantiser; the packing is offline)
//   nvfp4_quantize_kernel<In>  one thread per block of 16: E4M3 scale byte and 8 bytes of codes
//   nvfp4_expand_kernel  codes and block scales -> a bf16 operand image: every element's exact
//                      value q * s_b (E2M1 x E4M3 needs at most 6 significant bits and lies in
//                      [2^-10, 2688], so bf16 holds it exactly), in the 128-byte-swizzled K-major
//                      layout of the GEMM's operand images with a stage of 64 elements (128 B)
//   nvfp4_gemm_kernel  persistent tcgen05 kind::f16 GEMM with bf16 operands from both images by
//                      TMA, fp32 accumulation in TMEM over the whole K (the block scales are
//                      inside the operands), two accumulators, epilogue y = (acc * ga) * gw + bias
// The products q_a s_a,b * q_w s_w,b are exact in the tensor core; its fp32 sum over K is not,
// and its error is bounded by the fp32 summation bound over K products.
//
// Why bf16 operands and not the FP4 tensor-core kind: kind::mxf4nvf4.block_scale reads the block
// scales from tensor memory in a layout fixed by the instruction (scale-factor tiles copied by
// tcgen05.cp, scale-factor IDs in the instruction descriptor) that could not be checked against
// its documentation here; the bf16 path needs only forms the rest of the library already runs.
#include <cfloat>
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kernels.cuh"
#include "operand.cuh"
#include "ptx.cuh"

namespace jq {

namespace {

// ---------------------------------------------------------------- roundings (the format)
__device__ __forceinline__ float pow2f(int n) { return __int_as_float((n + 127) << 23); }  // n in [-126, 127]

// Nearest E4M3 value to a (finite, >= 0): 3 mantissa bits, exponent bias 7, normals down to 2^-6,
// subnormals in steps of 2^-9, ties to even, saturating at 448.  Scaling by the quantum is exact.
__device__ __forceinline__ float e4m3_round(float a) {
  if (a == 0.0f) return 0.0f;
  const int e = (int)((__float_as_uint(a) >> 23) & 255u) - 127;  // floor(log2 a) for normal a
  int q = e - 3;                                                   // the quantum's exponent
  if (q < -9) q = -9;                                              // subnormal quantum
  const float n = rintf(a * pow2f(-q));                            // ties to even
  const float r = n * pow2f(q);                                    // exact (inf only past 448)
  return r > 448.0f ? 448.0f : r;
}
// The E4M3 byte of a value e4m3_round returned.
__device__ __forceinline__ uint32_t e4m3_byte(float r) {
  if (r == 0.0f) return 0u;
  if (r < 0x1p-6f) return (uint32_t)(r * 512.0f);                // subnormal: m * 2^-9
  const int e = (int)((__float_as_uint(r) >> 23) & 255u) - 127;  // in [-6, 8]
  const uint32_t m = (__float_as_uint(r) >> 20) & 7u;            // 3 mantissa bits
  return ((uint32_t)(e + 7) << 3) | m;
}
__device__ __forceinline__ float e4m3_value(uint32_t b) {
  const uint32_t e = (b >> 3) & 15u, m = b & 7u;
  return e == 0u ? (float)m * 0x1p-9f : (float)(8u + m) * pow2f((int)e - 10);
}
// Nearest E2M1 magnitude to a (>= 0) as its 3-bit index into (0, 0.5, 1, 1.5, 2, 3, 4, 6), ties
// to the even mantissa (the even indices), saturating at 6.
__device__ __forceinline__ uint32_t e2m1_index(float a) {
  if (a <= 0.25f) return 0u;
  if (a < 0.75f) return 1u;
  if (a <= 1.25f) return 2u;
  if (a < 1.75f) return 3u;
  if (a <= 2.5f) return 4u;
  if (a < 3.5f) return 5u;
  if (a <= 5.0f) return 6u;
  return 7u;
}

// ---------------------------------------------------------------- weights' tensor scale
__global__ void __launch_bounds__(256) nvfp4_amax_kernel(const float* __restrict__ w, int64_t n,
                                                        unsigned int* __restrict__ amax_bits) {
  pdl_wait();
  float m = 0.0f;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    m = fmaxf(m, fabsf(__ldg(w + i)));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
  if ((threadIdx.x & 31) == 0) atomicMax(amax_bits, __float_as_uint(m));  // non-negative: bits order as values
}
__global__ void nvfp4_finish_g_kernel(float* g) {
  pdl_wait();
  *g = __fdiv_rn(__uint_as_float(*reinterpret_cast<const unsigned int*>(g)), 2688.0f);
}

// ---------------------------------------------------------------- quantiser
__device__ __forceinline__ void load16(const __nv_bfloat16* p, float (&x)[16]) {
  const uint4* v = reinterpret_cast<const uint4*>(p);
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const uint4 u = __ldg(v + i);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      x[8 * i + 2 * j] = __uint_as_float(w[j] << 16);
      x[8 * i + 2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
    }
  }
}
__device__ __forceinline__ void load16(const float* p, float (&x)[16]) {
  const float4* v = reinterpret_cast<const float4*>(p);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float4 u = __ldg(v + i);
    x[4 * i] = u.x;
    x[4 * i + 1] = u.y;
    x[4 * i + 2] = u.z;
    x[4 * i + 3] = u.w;
  }
}

// One thread per block of 16 elements: codes [rows, K/2] (element 2j in the low nibble of byte
// j), scale bytes [rows, K/16].  g from g_dev when given (the weights' computed scale), else g_host.
template <typename In>
__global__ void __launch_bounds__(256) nvfp4_quantize_kernel(const In* __restrict__ x, int64_t rows, int64_t K,
                                                            int64_t ldx, float g_host, const float* g_dev,
                                                            uint8_t* __restrict__ codes, uint8_t* __restrict__ scales) {
  if (sizeof(In) == 2) pdl_launch_dependents();
  pdl_wait();
  const float g = g_dev != nullptr ? *g_dev : g_host;
  const int64_t nb = K / 16;
  const int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;  // the block of 16 within the row
  if (b >= nb) return;
  for (int64_t r = blockIdx.y; r < rows; r += gridDim.y) {
    float v[16];
    load16(x + r * ldx + b * 16, v);
    float amax = 0.0f;
#pragma unroll
    for (int i = 0; i < 16; ++i) amax = fmaxf(amax, fabsf(v[i]));
    float s = 0.0f, S = 0.0f;
    if (g != 0.0f) {
      s = e4m3_round(__fdiv_rn(amax, 6.0f * g));
      S = s * g;
    }
    uint32_t lo = 0u, hi = 0u;
    if (S != 0.0f) {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const float q = __fdiv_rn(v[i], S);
        const uint32_t idx = e2m1_index(fabsf(q));
        const uint32_t c = idx | ((q < 0.0f && idx != 0u) ? 8u : 0u);
        if (i < 8) lo |= c << (4 * i);
        else hi |= c << (4 * (i - 8));
      }
    }
    *reinterpret_cast<uint2*>(codes + r * (K / 2) + b * 8) = make_uint2(lo, hi);
    scales[r * nb + b] = (uint8_t)e4m3_byte(s);
  }
}

// ---------------------------------------------------------------- bf16 operand images
constexpr int kStageK = 64;  // bf16 elements per 128-byte operand row of a stage

// One thread per 32 elements of a row (four 16-byte chunks of the image, all in one stage); grid
// x over the row's 32-element units, y over rows.  rows may be short of a whole 128-row tile:
// the image's rows past them are never written (their outputs are never kept).
// 8 E2M1 codes (one 32-bit word, element i in bits 4i..4i+3) -> their values as 4 bf16 pairs
// (elements 2k, 2k+1 in word k), without conversions: byte permutes look up the low and high
// bytes of each magnitude's bf16 bits in 8-entry tables (0, 0.5, 1, 1.5, 2, 3, 4, 6 are 0000,
// 3F00, 3F80, 3FC0, 4000, 4040, 4080, 40C0), a third permute turns each sign bit into 0x00 or
// 0x80 for the high byte, and two more interleave low and high bytes into pairs.
__device__ __forceinline__ uint4 e2m1x8_bf16(uint32_t w) {
  constexpr uint32_t kLoA = 0xC0800000u, kLoB = 0xC0804000u;  // low bytes of idx 0-3, 4-7
  constexpr uint32_t kHiA = 0x3F3F3F00u, kHiB = 0x40404040u;  // high bytes of idx 0-3, 4-7
  const uint32_t mag = w & 0x77777777u;                        // magnitude index per nibble
  const uint32_t sgn = (w >> 3) & 0x11111111u;                 // sign per nibble: byte 0 or 1
  uint32_t out[4];
#pragma unroll
  for (int h = 0; h < 2; ++h) {  // elements 4h .. 4h + 3
    const uint32_t sel = (mag >> (16 * h)) & 0xFFFFu, ssel = (sgn >> (16 * h)) & 0xFFFFu;
    const uint32_t lo = __byte_perm(kLoA, kLoB, sel);
    const uint32_t hi = __byte_perm(kHiA, kHiB, sel) | __byte_perm(0x8000u, 0u, ssel);
    out[2 * h] = __byte_perm(lo, hi, 0x5140);
    out[2 * h + 1] = __byte_perm(lo, hi, 0x7362);
  }
  return make_uint4(out[0], out[1], out[2], out[3]);
}

// A bf16 pair times the block scale (an E4M3 value, exact in bf16): every product has at most 6
// significant bits and lies in [2^-10, 2688], so the bf16 multiply is exact.
__device__ __forceinline__ uint32_t bf16x2_scale(uint32_t v, __nv_bfloat162 s2) {
  const __nv_bfloat162 p = __hmul2(*reinterpret_cast<const __nv_bfloat162*>(&v), s2);
  return *reinterpret_cast<const uint32_t*>(&p);
}

__global__ void __launch_bounds__(128) nvfp4_expand_kernel(const uint8_t* __restrict__ codes,
                                                          const uint8_t* __restrict__ scales, int64_t rows, int64_t K,
                                                          uint8_t* __restrict__ image) {
  pdl_launch_dependents();
  pdl_wait();
  const int64_t u = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;  // 32-element unit of the row
  if (u >= K / 32) return;
  const uint32_t k_stages = (uint32_t)(K / kStageK);
  const int64_t k0 = u * 32;
  const uint32_t kb = (uint32_t)(k0 / kStageK), c16 = (uint32_t)((k0 % kStageK) / 8);
  for (int64_t r = blockIdx.y; r < rows; r += gridDim.y) {
    const uint4 c = __ldg(reinterpret_cast<const uint4*>(codes + r * (K / 2) + k0 / 2));
    const uint8_t* sr = scales + r * (K / 16) + k0 / 16;  // byte loads: the scales carry no alignment rule
    const __nv_bfloat162 s0 = __float2bfloat162_rn(e4m3_value(__ldg(sr)));      // elements 0-15
    const __nv_bfloat162 s1 = __float2bfloat162_rn(e4m3_value(__ldg(sr + 1)));  // elements 16-31
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {  // chunk q: elements 8q .. 8q + 7 (4 code bytes)
      const __nv_bfloat162 sq = q < 2 ? s0 : s1;
      const uint4 m = e2m1x8_bf16(w[q]);
      *reinterpret_cast<uint4*>(image + image_chunk_offset(r, kb, c16 + (uint32_t)q, k_stages)) =
          make_uint4(bf16x2_scale(m.x, sq), bf16x2_scale(m.y, sq), bf16x2_scale(m.z, sq), bf16x2_scale(m.w, sq));
    }
  }
}

// ---------------------------------------------------------------- GEMM
constexpr int kTileM = 128, kTileN = 256, kStages = 4, kThreadsG = 192, kAccBufs = 2;
constexpr uint32_t kABytes = kTileM * 128, kBBytes = kTileN * 128, kStageBytes = kABytes + kBBytes;  // 48 KB
constexpr uint32_t kOffBars = kStages * kStageBytes;
constexpr uint32_t kNumBarsG = 2 * kStages + 2 * kAccBufs;
constexpr uint32_t kSmemG = kOffBars + kNumBarsG * 8 + 16;
constexpr uint32_t kTmemColsG = kAccBufs * kTileN;  // 512: two accumulators
// kind::f16, bf16 A and B (both K-major), fp32 accumulator: D format [4,6) = 1, A format [7,10)
// = 1 (BF16), B format [10,13) = 1 (BF16), N >> 3 at [17,23), M >> 4 at [24,29).
constexpr uint32_t kIdescBf16 = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kTileN >> 3) << 17) |
                                ((uint32_t)(kTileM >> 4) << 24);

__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

struct NvArgs {
  int M, N, k_stages, num_m, num_tiles;
  float ga;
  const float* gw;   // device scalar
  const float* bias;  // [N] or nullptr
  __nv_bfloat16* y;   // [M, N]
  uint32_t* status;
};

// Persistent: CTA c computes 128 x 256 output tiles c, c + grid, ... (tiles M-fastest, so that the
// tiles in flight at once share weight tiles), with two TMEM accumulators so that a tile's
// epilogue runs under the next tile's MMAs.  Warp 0: TMA producer (A: one 128-row box, B: two,
// per 64-element stage, into a 4-stage ring that runs on across tiles).  Warp 1: TMEM owner and
// MMA issuer (four 128x256x16 MMAs per stage, one commit per stage to free the slot, one per tile
// for the drain).  Warps 2-5: drain, one accumulator row per thread, handing the accumulator back
// once its last columns are in registers.
__global__ void __launch_bounds__(kThreadsG, 1)
    nvfp4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const NvArgs a) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0) {
    if (threadIdx.x == 0 && a.status != nullptr) atomicExch(a.status, (uint32_t)kDevSmemAlign);
    return;
  }
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kOffBars);
  uint64_t* empty = full + kStages;
  uint64_t* acc_full = empty + kStages;
  uint64_t* acc_empty = acc_full + kAccBufs;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + kAccBufs);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const uint32_t warp = warp_id(), lane = lane_id();
  const int ks = a.k_stages;
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < kAccBufs; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 4);  // the four drain warps
    }
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemColsG);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_launch_dependents();
  pdl_wait();  // the images come from the kernels before this one

  uint32_t issued = 0;  // producer: stages issued (ring position)
  if (warp == 0) {
    if (lane == 0) {
      bool ok = true;
      for (int t = (int)blockIdx.x; ok && t < a.num_tiles; t += (int)gridDim.x) {
        const int mt = t % a.num_m, nt = t / a.num_m;
        for (int kb = 0; kb < ks; ++kb, ++issued) {
          const uint32_t s = issued % kStages;
          if (!(ok = mbar_wait(&empty[s], ((issued / kStages) & 1u) ^ 1u, abort_flag, a.status))) break;
          uint8_t* st = smem + s * kStageBytes;
          mbar_arrive_expect_tx(&full[s], kStageBytes);
          tma_load_2d(st, &tmA, &full[s], 0, (mt * ks + kb) * kTileM);
          tma_load_2d(st + kABytes, &tmB, &full[s], 0, ((2 * nt) * ks + kb) * 128);
          tma_load_2d(st + kABytes + kBBytes / 2, &tmB, &full[s], 0, ((2 * nt + 1) * ks + kb) * 128);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = true;
      uint32_t it = 0, tile_it = 0;
      for (int t = (int)blockIdx.x; ok && t < a.num_tiles; t += (int)gridDim.x, ++tile_it) {
        const uint32_t ab = tile_it % kAccBufs;
        // the drain has emptied this accumulator (tile_it - 2's)
        if (!(ok = mbar_wait(&acc_empty[ab], ((tile_it / kAccBufs) & 1u) ^ 1u, abort_flag, a.status))) break;
        tc_fence_after();
        const uint32_t d = tmem_base + ab * (uint32_t)kTileN;
        for (int kb = 0; kb < ks; ++kb, ++it) {
          const uint32_t s = it % kStages;
          if (!(ok = mbar_wait(&full[s], (it / kStages) & 1u, abort_flag, a.status))) break;
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + s * kStageBytes);
          const uint64_t ad = sdesc_kmajor_sw128(sa), bd = sdesc_kmajor_sw128(sa + kABytes);
#pragma unroll
          for (int k4 = 0; k4 < 4; ++k4)  // 16 bf16 (32 bytes) of K per MMA: +2 in the descriptor's 16-byte units
            umma_bf16(d, ad + 2u * (uint32_t)k4, bd + 2u * (uint32_t)k4, kIdescBf16, (kb | k4) != 0 ? 1u : 0u);
          umma_commit(&empty[s]);
        }
        if (ok) umma_commit(&acc_full[ab]);
      }
    }
  } else {  // drain: warp w reads TMEM lanes 32 (w % 4) .. (all four quarters over warps 2-5)
    const uint32_t quarter = warp & 3u;
    const float gw = *a.gw;
    uint32_t tile_it = 0;
    for (int t = (int)blockIdx.x; t < a.num_tiles; t += (int)gridDim.x, ++tile_it) {
      const int mt = t % a.num_m, nt = t / a.num_m;
      const uint32_t ab = tile_it % kAccBufs;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[ab], (tile_it / kAccBufs) & 1u, abort_flag, a.status));
      if (!ok) break;
      tc_fence_after();
      const int row = mt * kTileM + (int)(quarter * 32u + lane);
      const uint32_t taddr = tmem_base + ((quarter * 32u) << 16) + ab * (uint32_t)kTileN;
#pragma unroll 1
      for (int c = 0; c < kTileN; c += 32) {
        uint32_t r[32];
        tmem_ld32(taddr + (uint32_t)c, r);
        tmem_ld_wait();
        if (c + 32 == kTileN) {  // every column of this accumulator is in registers: hand it back
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[ab]);
        }
        const int col0 = nt * kTileN + c;
        if (row < a.M) {
#pragma unroll
          for (int v8 = 0; v8 < 4; ++v8) {
            const int col = col0 + 8 * v8;
            if (col < a.N) {  // N % 8 == 0: a chunk of 8 is wholly inside or outside
              uint32_t o[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const int cc = 8 * v8 + 2 * i;
                const float b0 = a.bias != nullptr ? __ldg(a.bias + col + 2 * i) : 0.0f;
                const float b1 = a.bias != nullptr ? __ldg(a.bias + col + 2 * i + 1) : 0.0f;
                const float y0 = (__uint_as_float(r[cc]) * a.ga) * gw + b0;
                const float y1 = (__uint_as_float(r[cc + 1]) * a.ga) * gw + b1;
                const __nv_bfloat162 p = __floats2bfloat162_rn(y0, y1);
                o[i] = *reinterpret_cast<const uint32_t*>(&p);
              }
              *reinterpret_cast<uint4*>(a.y + (int64_t)row * a.N + col) = make_uint4(o[0], o[1], o[2], o[3]);
            }
          }
        }
      }
    }
  }
  // Every TMA copy issued has landed (the MMA waited for each, or the abort path below waits),
  // every MMA has completed (the drain waited for each tile's last commit, or all gave up).
  tc_fence_before();
  __syncthreads();
  if (warp == 0 && lane == 0 && *abort_flag) {  // unwinding: wait (bounded) for copies in flight
    for (uint32_t i = (issued > (uint32_t)kStages ? issued - kStages : 0u); i < issued; ++i) {
      int dummy = 0;
      mbar_wait(&full[i % kStages], (i / kStages) & 1u, &dummy, a.status);
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemColsG);
  }
}

// Grid of (units of a row / threads) x rows, the rows capped at the grid's y limit (the kernels
// stride over the rest).
dim3 grid_rows(int64_t units, int threads, int64_t rows) {
  const int64_t gx = (units + threads - 1) / threads;
  return dim3((unsigned)gx, (unsigned)(rows < 65535 ? rows : 65535), 1);
}

int grid_cap(int64_t items, int threads, int sms) {
  int64_t b = (items + threads - 1) / threads;
  const int64_t cap = (int64_t)sms * 8;
  return (int)(b < 1 ? 1 : (b > cap ? cap : b));
}

}  // namespace

size_t nvfp4_image_bytes(int64_t rows, int64_t K) { return (size_t)((rows + 127) / 128 * 128) * (size_t)K * 2; }

cudaError_t launch_nvfp4_quantize_act(const void* x, int64_t M, int64_t K, int64_t ldx, float g, uint8_t* codes,
                                      uint8_t* scales, cudaStream_t stream, int sms) {
  if (M == 0) return cudaSuccess;
  return launch_pdl(nvfp4_quantize_kernel<__nv_bfloat16>, grid_rows(K / 16, 128, M), dim3(128), 0, stream,
                    static_cast<const __nv_bfloat16*>(x), M, K, ldx, g, (const float*)nullptr, codes, scales);
}

cudaError_t launch_nvfp4_pack_weight(const float* w, int64_t N, int64_t K, uint8_t* codes, uint8_t* scales, float* g,
                                     cudaStream_t stream, int sms) {
  if (N == 0) return cudaSuccess;
  cudaError_t e = cudaMemsetAsync(g, 0, sizeof(float), stream);
  if (e != cudaSuccess) return e;
  if ((e = launch_pdl(nvfp4_amax_kernel, dim3(grid_cap(N * K, 256, sms)), dim3(256), 0, stream, w, N * K,
                      reinterpret_cast<unsigned int*>(g))) != cudaSuccess)
    return e;
  if ((e = launch_pdl(nvfp4_finish_g_kernel, dim3(1), dim3(1), 0, stream, g)) != cudaSuccess) return e;
  return launch_pdl(nvfp4_quantize_kernel<float>, grid_rows(K / 16, 128, N), dim3(128), 0, stream, w, N, K, K, 0.0f,
                    (const float*)g, codes, scales);
}

cudaError_t launch_nvfp4_linear(const uint8_t* qa, const uint8_t* sa, float ga, const uint8_t* qw, const uint8_t* sw,
                                const float* gw, const float* bias, void* y, int64_t M, int64_t N, int64_t K,
                                uint8_t* workspace, uint32_t* status, cudaStream_t stream, int sms) {
  if (M == 0 || N == 0) return cudaSuccess;
  uint8_t* img_a = workspace;
  uint8_t* img_b = workspace + nvfp4_image_bytes(M, K);
  cudaError_t e;
  if ((e = launch_pdl(nvfp4_expand_kernel, grid_rows(K / 32, 128, M), dim3(128), 0, stream, qa, sa, M, K, img_a)) !=
      cudaSuccess)
    return e;
  if ((e = launch_pdl(nvfp4_expand_kernel, grid_rows(K / 32, 128, N), dim3(128), 0, stream, qw, sw, N, K, img_b)) !=
      cudaSuccess)
    return e;
  // The set-up CUDA keeps per device: the dynamic shared-memory size of the GEMM kernel.
  static PerDevice<bool> attr;
  bool done = false;
  if ((e = attr.get(
           [](bool& v) {
             v = true;
             return cudaFuncSetAttribute(nvfp4_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemG);
           },
           done)) != cudaSuccess)
    return e;
  // Both images as rows of 128 bytes; one box = one 128-row block of a stage, copied as it is
  // (already in the 128-byte swizzle).
  const int ks = (int)(K / kStageK);
  const int64_t rows_a = (M + 127) / 128 * 128 * ks, rows_b = (N + 127) / 128 * 128 * ks;
  CUtensorMap tmA, tmB;
  if (!encode_2d(&tmA, CU_TENSOR_MAP_DATA_TYPE_UINT8, img_a, 128, (uint64_t)rows_a, 128, 128, 128,
                 CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !encode_2d(&tmB, CU_TENSOR_MAP_DATA_TYPE_UINT8, img_b, 128, (uint64_t)rows_b, 128, 128, 128,
                 CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;
  NvArgs a;
  a.M = (int)M;
  a.N = (int)N;
  a.k_stages = ks;
  a.num_m = (int)((M + kTileM - 1) / kTileM);
  a.num_tiles = a.num_m * (int)((N + kTileN - 1) / kTileN);
  a.ga = ga;
  a.gw = gw;
  a.bias = bias;
  a.y = static_cast<__nv_bfloat16*>(y);
  a.status = status;
  const int grid = a.num_tiles < sms ? a.num_tiles : sms;  // persistent: one CTA per SM
  return launch_pdl(nvfp4_gemm_kernel, dim3(grid), dim3(kThreadsG), kSmemG, stream, tmA, tmB, a);
}

}  // namespace jq
