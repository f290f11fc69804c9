// ternary.cu -- ternary weights for the W1.58A4 setting (ternary weights, INT4 activations,
// group128: Appendix table "DiT-XL/2 experimental details"; the ELF-B table likewise).
//
// Packer.  The paper prints no ternary rule; the reading is the absmean rule of 1.58-bit weight
// quantisation per row and group of G consecutive K elements:
//   s = fl32(mean |w|)   (the mean in fp64, the group summed in index order, one division by G)
//   q = clamp(rint(fl32(w / s)), -1, 1)      (ties to even; s = q = 0 for an all-zero group)
// One thread per group: the fp64 sum has to follow index order to be reproducible bit for bit.
//
// Packed ternary format: q + 1 in {0, 1, 2}, 2 bits per code; every 16 consecutive elements of a
// row fill one little-endian 32-bit word whose byte j (j = 0..3) holds elements 2j, 2j+1, 8+2j
// and 9+2j in bits 0-1, 2-3, 4-5 and 6-7.  So (word >> 2i) & 0x03030303, i = 0..3, are directly
// the MMA operand bytes of elements {0,2,4,6}, {1,3,5,7}, {8,10,12,14}, {9,11,13,15}: the byte
// order the INT4 operand uses (operand.cuh), in offset form q + 1, which E4M3 reads exactly.
// Both the few-token kernel and the GEMM read this format directly (operand.cuh).
#include <cstdint>
#include <cuda_runtime.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace jq {

namespace {

// bit offset of element e (0..15) within its 32-bit word
__host__ __device__ constexpr int tern_bit(int e) { return 8 * ((e & 7) >> 1) + 2 * (e & 1) + 4 * (e >> 3); }

__global__ void __launch_bounds__(128) pack_ternary_kernel(const float* __restrict__ w, int64_t N, int64_t K, int G,
                                                           uint8_t* __restrict__ qw, float* __restrict__ s_w) {
  pdl_wait();
  const int64_t groups = K / G;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < N * groups;
       t += (int64_t)gridDim.x * blockDim.x) {
    // consecutive threads take consecutive rows of the same group: their scale stores coalesce
    const int64_t g = t / N, n = t % N;
    const float* wg = w + n * K + g * G;
    double sum = 0.0;
    for (int k = 0; k < G; k += 4) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(wg + k));
      sum += fabs((double)v.x);
      sum += fabs((double)v.y);
      sum += fabs((double)v.z);
      sum += fabs((double)v.w);
    }
    const float s = __double2float_rn(sum / (double)G);
    s_w[g * N + n] = s;
    uint32_t* out = reinterpret_cast<uint32_t*>(qw + n * (K / 4) + g * (G / 4));
    for (int k0 = 0; k0 < G; k0 += 16) {
      uint32_t word = 0;
#pragma unroll
      for (int e = 0; e < 16; e += 4) {
        const float4 v = __ldg(reinterpret_cast<const float4*>(wg + k0 + e));
        const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          int q = 0;
          if (s != 0.0f) {
            const float r = rintf(__fdiv_rn(vv[i], s));
            q = r > 1.0f ? 1 : (r < -1.0f ? -1 : static_cast<int>(r));
          }
          word |= static_cast<uint32_t>(q + 1) << tern_bit(e + i);
        }
      }
      out[k0 / 16] = word;
    }
  }
}

int grid_cap(int64_t items, int threads, int sms) {
  int64_t blocks = (items + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(sms) * 8;
  return static_cast<int>(blocks < 1 ? 1 : (blocks > cap ? cap : blocks));
}

}  // namespace

cudaError_t launch_pack_weight_ternary(const float* w, int64_t N, int64_t K, int G, uint8_t* qw, float* s_w,
                                       cudaStream_t stream, int sms) {
  if (N == 0) return cudaSuccess;
  return launch_pdl(pack_ternary_kernel, dim3(grid_cap(N * (K / G), 128, sms)), dim3(128), 0, stream, w, N, K, G, qw,
                    s_w);
}

}  // namespace jq
