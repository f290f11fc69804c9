// fakequant.cu -- training side: fake quantisation of bf16 activations and the straight-through
// backward.  Stage 1 of Theseus QAD (Sec. 3, Algorithm 1) trains the quantised student blocks by
// gradient descent, and the paper names the straight-through estimator as the gradient rule of
// 4-bit activations (Sec. 3, "Why QAT fails").  The forward is the deployed quantiser's code
// dequantised, xhat = q * s, rounded once to bf16; the backward passes the gradient where the
// unclamped code rint(fl32(x / s)) lies in [-8, 7] and writes +0 where the clamp acted.
//
// The same forward serves the student's fp32 weights (xhat = q * s rounded once to fp32).
// Both kernels stream HBM: the bf16 forward reads 2 bytes and writes 2 (xhat) + 1 (mask) per
// element plus 4 bytes per group for the scales (fp32: 4 + 4 + 1); the backward reads 2 + 1 and
// writes 2.
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kernels.cuh"

namespace jq {
namespace {

constexpr int kFqThreads = 256;             // 8 elements per thread per chunk

// bf16 of the exact product q * s, rounded once (nearest even).  The product of a 4-bit integer
// and a 24-bit significand needs up to 28 bits; rounding it to fp32 and then to bf16 could round
// twice.  Round to odd in fp32 instead (truncate, then set the last bit when the truncation was
// inexact): with 24 >= 8 + 2 bits the final bf16 rounding of a round-to-odd value equals the
// single rounding of the exact value (Boldo and Melquiond, "When double rounding is odd", 2005).
// The fma residual q*s - rz(q*s) is exact; products here are never below the fp32 normal range
// unless they are multiples of the subnormal quantum, hence exact.
__device__ __forceinline__ uint16_t bf16_of_exact_product(float qf, float s) {
  const float p = __fmul_rz(qf, s);
  const float e = __fmaf_rn(qf, s, -p);
  uint32_t b = __float_as_uint(p);
  if (e != 0.0f) b |= 1u;
  return __bfloat16_as_ushort(__float2bfloat16_rn(__uint_as_float(b)));
}

__device__ __forceinline__ float bf16_bits_to_f32(uint32_t b) { return __uint_as_float(b << 16); }

// 8 consecutive elements (k % 8 == 0) widened to fp32, and xhat written back in the input's type.
__device__ __forceinline__ void load8(const uint16_t* p, float v[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int j = 0; j < 8; ++j) v[j] = bf16_bits_to_f32((w[j / 2] >> (16 * (j & 1))) & 0xFFFFu);
}
__device__ __forceinline__ void load8(const float* p, float v[8]) {
  const float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void store8(uint16_t* p, const int q[8], float s) {
  uint32_t out[4];
#pragma unroll
  for (int j = 0; j < 4; ++j)
    out[j] = bf16_of_exact_product(static_cast<float>(q[2 * j]), s) |
             (static_cast<uint32_t>(bf16_of_exact_product(static_cast<float>(q[2 * j + 1]), s)) << 16);
  *reinterpret_cast<uint4*>(p) = make_uint4(out[0], out[1], out[2], out[3]);
}
// fp32 output: the IEEE product of the (exact) code and the scale is the single rounding of q*s.
__device__ __forceinline__ void store8(float* p, const int q[8], float s) {
  float o[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) o[j] = __fmul_rn(static_cast<float>(q[j]), s);
  reinterpret_cast<float4*>(p)[0] = make_float4(o[0], o[1], o[2], o[3]);
  reinterpret_cast<float4*>(p)[1] = make_float4(o[4], o[5], o[6], o[7]);
}

// T = uint16_t: bf16 activations -> bf16 xhat; T = float: fp32 weights -> fp32 xhat.  R rows per
// block, kFqThreads / R threads per row (R = 1 or 4: with many short rows, four at a time per
// block so that each thread keeps more loads in flight between the block's barriers);
// the per-row group scales live in dynamic shared memory [R][K/G].
template <typename T, int R>
__global__ void __launch_bounds__(kFqThreads) fake_quant_kernel(const T* __restrict__ x, int64_t M, int64_t K, int G,
                                                                 const float* __restrict__ s_in, T* __restrict__ xhat,
                                                                 uint8_t* __restrict__ mask,
                                                                 float* __restrict__ s_out) {
  extern __shared__ float s_rows[];  // [R][K/G]: per group of each row, amax bits, then the scale
  constexpr int kRowThreads = kFqThreads / R;
  constexpr int kChunk = kRowThreads * 8;  // elements of a row one pass of its threads covers
  const int sub = threadIdx.x / kRowThreads, tid = threadIdx.x % kRowThreads;
  const int lane = threadIdx.x & 31;
  const int ng = static_cast<int>(K / G);
  float* s_grp = s_rows + sub * ng;
  // lanes that share a group within one 256-element warp span: G/8 for G = 64, 128; the warp
  // for one group per row (G = K >= 256, where every lane of a warp lies in the same group)
  const int seg = G >= 256 ? 32 : G / 8;
  // uniform trip count across the block: every thread takes the same number of row rounds
  for (int64_t row0 = static_cast<int64_t>(blockIdx.x) * R; row0 < M; row0 += static_cast<int64_t>(gridDim.x) * R) {
    const int64_t row = row0 + sub;
    const bool row_ok = row < M;
    const T* xr = x + (row_ok ? row : 0) * K;
    if (s_in != nullptr) {
      if (row_ok)
        for (int g = tid; g < ng; g += kRowThreads) s_grp[g] = s_in[row * ng + g];
      __syncthreads();
    } else {
      for (int g = tid; g < ng; g += kRowThreads) reinterpret_cast<uint32_t*>(s_grp)[g] = 0u;
      __syncthreads();
      for (int64_t base = 0; base < K; base += kChunk) {  // uniform trip count across the block
        const int64_t k = base + static_cast<int64_t>(tid) * 8;
        const bool valid = row_ok && k < K;
        float m = 0.0f;
        if (valid) {
          float v[8];
          load8(xr + k, v);
#pragma unroll
          for (int j = 0; j < 8; ++j) m = fmaxf(m, fabsf(v[j]));
        }
        for (int off = seg / 2; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, off));
        // the segment's first lane holds its smallest k: if any lane of the segment is in the row,
        // that one is
        if (valid && (lane % seg) == 0)
          atomicMax(reinterpret_cast<unsigned int*>(s_grp) + k / G, __float_as_uint(m));  // m >= 0
      }
      __syncthreads();
      for (int g = tid; g < ng; g += kRowThreads) {
        const float amax = __uint_as_float(reinterpret_cast<uint32_t*>(s_grp)[g]);
        s_grp[g] = amax == 0.0f ? 0.0f : __fdiv_rn(amax, 7.0f);
      }
      __syncthreads();
    }
    if (row_ok) {
      for (int g = tid; g < ng; g += kRowThreads) s_out[row * ng + g] = s_grp[g];
      for (int64_t k = static_cast<int64_t>(tid) * 8; k < K; k += kChunk) {
        const float s = s_grp[k / G];  // the 8 elements lie in one group: G % 8 == 0, k % 8 == 0
        float v[8];
        load8(xr + k, v);
        int q[8];
        uint32_t mlo = 0, mhi = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          uint32_t pass = 1;
          q[j] = 0;  // an all-zero group (s = 0): xhat = +0, mask 1
          if (s != 0.0f) {
            const float r = rintf(__fdiv_rn(v[j], s));  // IEEE division, then half to even
            pass = (r >= -8.0f && r <= 7.0f) ? 1u : 0u;
            q[j] = static_cast<int>(fminf(fmaxf(r, -8.0f), 7.0f));  // code 0 gives +0 below
          }
          if (j < 4) mlo |= pass << (8 * j); else mhi |= pass << (8 * (j - 4));
        }
        store8(xhat + row * K + k, q, s);
        *reinterpret_cast<uint2*>(mask + row * K + k) = make_uint2(mlo, mhi);
      }
    }
    __syncthreads();  // s_grp is reused by the next round of rows
  }
}

__global__ void __launch_bounds__(kFqThreads) ste_backward_kernel(const uint16_t* __restrict__ grad,
                                                                   const uint8_t* __restrict__ mask, int64_t n,
                                                                   uint16_t* __restrict__ grad_x) {
  const int64_t nvec = n / 8;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kFqThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kFqThreads + threadIdx.x; i < nvec; i += stride) {
    const uint4 g = reinterpret_cast<const uint4*>(grad)[i];
    const uint2 mk = reinterpret_cast<const uint2*>(mask)[i];
    const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
    uint32_t out[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t mb = j < 2 ? mk.x >> (16 * j) : mk.y >> (16 * (j - 2));  // two mask bytes
      const uint32_t lo = (mb & 0xFFu) ? (gw[j] & 0xFFFFu) : 0u;
      const uint32_t hi = ((mb >> 8) & 0xFFu) ? (gw[j] & 0xFFFF0000u) : 0u;
      out[j] = lo | hi;
    }
    reinterpret_cast<uint4*>(grad_x)[i] = make_uint4(out[0], out[1], out[2], out[3]);
  }
  // the ragged tail (n % 8 elements), by the first threads of the grid
  const int64_t t = nvec * 8 + static_cast<int64_t>(blockIdx.x) * kFqThreads + threadIdx.x;
  if (t < n) grad_x[t] = mask[t] ? grad[t] : static_cast<uint16_t>(0);
}

}  // namespace

// Rows per block: 4 (64 threads a row) when there are many rows (at least 4 such blocks per SM)
// of up to 16384 elements, else 1.  Measured: fp32 weights 21504 x 3072, 3494 -> 4355 GB/s with 4;
// bf16 activations 1024 x 4096, 1669 GB/s with 1 against 1325 with 2 rows per block.
template <typename T>
cudaError_t launch_fake_quant(const T* x, int64_t M, int64_t K, int G, const float* s_in, T* xhat, uint8_t* mask,
                              float* s_out, cudaStream_t stream, int sms) {
  if (M == 0) return cudaSuccess;
  const int R = (K <= 16384 && M >= 16 * static_cast<int64_t>(sms)) ? 4 : 1;
  const int64_t need = (M + R - 1) / R;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  const unsigned blocks = static_cast<unsigned>(need < cap ? need : cap);
  const size_t smem = static_cast<size_t>(R) * static_cast<size_t>(K / G) * sizeof(float);
  if (R == 4)
    fake_quant_kernel<T, 4><<<blocks, kFqThreads, smem, stream>>>(x, M, K, G, s_in, xhat, mask, s_out);
  else
    fake_quant_kernel<T, 1><<<blocks, kFqThreads, smem, stream>>>(x, M, K, G, s_in, xhat, mask, s_out);
  return cudaGetLastError();
}

cudaError_t launch_fake_quant_act(const void* x, int64_t M, int64_t K, int G, const float* s_in, void* xhat,
                                  uint8_t* mask, float* s_out, cudaStream_t stream, int sms) {
  return launch_fake_quant(static_cast<const uint16_t*>(x), M, K, G, s_in, static_cast<uint16_t*>(xhat), mask, s_out,
                           stream, sms);
}

cudaError_t launch_fake_quant_weight(const float* w, int64_t N, int64_t K, int G, const float* s_in, float* what,
                                     uint8_t* mask, float* s_out, cudaStream_t stream, int sms) {
  return launch_fake_quant(w, N, K, G, s_in, what, mask, s_out, stream, sms);
}

cudaError_t launch_ste_backward(const void* grad, const uint8_t* mask, int64_t n, void* grad_x, cudaStream_t stream,
                                int sms) {
  const int64_t want = (n / 8 + kFqThreads - 1) / kFqThreads;
  int64_t blocks = want < static_cast<int64_t>(sms) * 8 ? want : static_cast<int64_t>(sms) * 8;
  if (blocks < 1) blocks = 1;  // the tail alone (n < 8) still needs one block
  ste_backward_kernel<<<static_cast<unsigned>(blocks), kFqThreads, 0, stream>>>(
      static_cast<const uint16_t*>(grad), mask, n, static_cast<uint16_t*>(grad_x));
  return cudaGetLastError();
}

}  // namespace jq
