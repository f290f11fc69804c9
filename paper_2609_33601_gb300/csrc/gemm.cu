// gemm.cu -- the W4A4 GEMM with exact per-group integer accumulation and a fused fp32
// dequantise + bias epilogue (the deployed "naive W4A4" linear: Sec. 1, Appendix FAQ Q7; group
// sizes from Sec. 4.2 "FLUX" and the Appendix experimental-detail tables).
//
//   acc[m,n,g] = sum_{k in group g} qa[m,k] * qw[n,k]
//   y[m,n]     = bf16( sum_g acc[m,n,g] * s_a[m,g] * s_w[g,n] + bias[n] )
//
// sm_103a has no INT8 tensor-core MMA, so codes run through tcgen05.mma kind::f8f6f4 as E4M3
// operand bytes (operand.cuh): every product and every per-group sum is exactly representable,
// so the fp32 TMEM accumulator holds acc[m,n,g] * 2^-18 exactly.
//
// Persistent kernel, one 128x256 output tile at a time per CTA, 16 warps:
//   warp 0      TMA producer: A operand bytes (128x128, 128B swizzle) straight into the MMA
//               stage ring; packed B codes (256 x 64 bytes) into a packed ring; one row of
//               weight scales s_w[g, n0:n0+256] per group into a scale ring.
//   warp 1      MMA issuer (one thread): 4 x (128x256x32) MMAs per K stage into one of two TMEM
//               accumulators; a fresh accumulator starts at every group boundary and is handed
//               to the drain warps with tcgen05.commit when the group ends.
//   warps 2-7   unpack: packed B nibbles -> operand bytes in the 128B-swizzled K-major layout.
//   warps 8-15  drain: per group, tcgen05.ld the partials, y += acc * (s_a * 2^18) * s_w in
//               fp32 registers (warp w owns TMEM lanes 32*(w%4).. and columns 128*((w-8)/4)..);
//               after the last group, + bias, round to bf16, store.
// Every mbarrier wait is bounded; a timeout records a status and unwinds the whole CTA.
#include <cfloat>
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "kernels.cuh"
#include "operand.cuh"
#include "ptx.cuh"

namespace jq {

namespace {

constexpr int kBM = 128, kBN = 256, kBK = 128;
constexpr int kStagesOp = 3;    // operand ring (A via TMA + B via unpack)
constexpr int kStagesPk = 4;    // packed-B ring
constexpr int kScaleSlots = 12;  // weight-scale ring (one slot per group; deep enough not to gate loads)
constexpr int kThreads = 512;
constexpr int kUnpackWarp0 = 2, kNumUnpackWarps = 6;
constexpr int kDrainWarp0 = 8, kNumDrainWarps = 8;
constexpr int kUnpackThreads = kNumUnpackWarps * 32;
constexpr int kDrainThreads = kNumDrainWarps * 32;
constexpr uint32_t kTmemCols = 512;  // two 256-column fp32 accumulators

constexpr uint32_t kOpABytes = kBM * kBK;
constexpr uint32_t kOpBBytes = kBN * kBK;
constexpr uint32_t kPkBBytes = kBN * kBK / 2;
constexpr uint32_t kScaleBytes = kBN * 4;

constexpr uint32_t kOffOpA = 0;
constexpr uint32_t kOffOpB = kOffOpA + kStagesOp * kOpABytes;
constexpr uint32_t kOffPkB = kOffOpB + kStagesOp * kOpBBytes;
constexpr uint32_t kOffSw = kOffPkB + kStagesPk * kPkBBytes;
constexpr uint32_t kOffBar = kOffSw + kScaleSlots * kScaleBytes;
constexpr uint32_t kNumBars = 3 * kStagesOp + 2 * kStagesPk + 2 * kScaleSlots + 4 + 1;
constexpr uint32_t kOffMisc = kOffBar + kNumBars * 8;
constexpr uint32_t kSmemBytes = kOffMisc + 16 + 1024;  // + slack to align the base to 1024

static_assert(kSmemBytes <= 232448, "shared memory budget");

struct Args {
  int M, N, K, G;
  int num_m_tiles, num_tiles;
  const float* s_a;
  const float* bias;
  __nv_bfloat16* y;
  int32_t* partials;
  uint32_t* status;
};

__device__ __forceinline__ uint32_t ring_parity(uint32_t it, uint32_t stages) { return (it / stages) & 1u; }

// A bounded wait that ignores the CTA abort flag (used while draining in-flight async work).
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, uint32_t* status) {
  int dummy = 0;
  mbar_wait(bar, parity, &dummy, status);
}

template <bool kExport>
__device__ __forceinline__ void drain_role(const Args& args, uint32_t tmem_base, const float* sw, uint64_t* full_s,
                                           uint64_t* empty_s, uint64_t* acc_full, uint64_t* acc_empty,
                                           volatile int* abort_flag) {
  const uint32_t warp = warp_id(), lane = lane_id();
  const int M = args.M, N = args.N, K = args.K, G = args.G;
  const int groups = K / G;
    // ------------------------------------------------------------------ drain + epilogue
    const uint32_t quarter = warp & 3u, half = (warp - kDrainWarp0) >> 2;
    const uint32_t lane_base = (quarter * 32u) << 16;
    uint32_t chunk_it = 0, it_s = 0;
    bool ok = true;
    for (int tile = blockIdx.x; ok && tile < args.num_tiles; tile += gridDim.x) {
      const int mt = tile % args.num_m_tiles, nt = tile / args.num_m_tiles;
      const int row = mt * kBM + quarter * 32 + lane;
      const int col0 = nt * kBN + half * 128;
      const bool row_ok = row < M;
      float y[128];
#pragma unroll
      for (int i = 0; i < 128; ++i) y[i] = 0.0f;
      for (int g = 0; g < groups; ++g) {
        const uint32_t ab = chunk_it & 1u, s = it_s % kScaleSlots;
        const float sa = (!kExport && row_ok) ? __ldg(args.s_a + (int64_t)row * groups + g) : 0.0f;
        if (!(ok = mbar_wait(&full_s[s], ring_parity(it_s, kScaleSlots), abort_flag, args.status))) break;
        if (!(ok = mbar_wait(&acc_full[ab], (chunk_it >> 1) & 1u, abort_flag, args.status))) break;
        tc_fence_after();
        const uint32_t taddr = tmem_base + lane_base + ab * kBN + half * 128;
        const float* sws = sw + s * kBN + half * 128;
        if constexpr (kExport) {
#pragma unroll 1
          for (int cc = 0; cc < 4; ++cc) {
            uint32_t r[32];
            tmem_ld32(taddr + cc * 32, r);
            tmem_ld_wait();
            if (cc == 3) {
              tc_fence_before();
              mbar_arrive(&acc_empty[ab]);
            }
            if (row_ok) {
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                const int col = col0 + cc * 32 + j;
                if (col < N)
                  args.partials[((int64_t)row * N + col) * groups + g] =
                      static_cast<int32_t>(__uint_as_float(r[j]) * kOperandUnitInv);
              }
            }
          }
        } else {
          const float f = sa * kOperandUnitInv;  // s_a * 2^18
          const bool f_finite = f <= FLT_MAX;
#pragma unroll
          for (int cc = 0; cc < 4; ++cc) {
            uint32_t r[32];
            tmem_ld32(taddr + cc * 32, r);
            tmem_ld_wait();
            if (cc == 3) {
              tc_fence_before();
              mbar_arrive(&acc_empty[ab]);
            }
            if (f_finite) {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                y[cc * 32 + j] = fmaf(__uint_as_float(r[j]) * f, sws[cc * 32 + j], y[cc * 32 + j]);
            } else {  // |s_a| > 2^110: apply 2^18 to the exact partial first
#pragma unroll
              for (int j = 0; j < 32; ++j)
                y[cc * 32 + j] =
                    fmaf((__uint_as_float(r[j]) * kOperandUnitInv) * sa, sws[cc * 32 + j], y[cc * 32 + j]);
            }
          }
        }
        mbar_arrive(&empty_s[s]);
        ++chunk_it;
        ++it_s;
      }
      if (!ok) break;
      if constexpr (!kExport) {
        if (row_ok) {
          __nv_bfloat16* yrow = args.y + (int64_t)row * N;
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int col = col0 + 8 * i;
            if (col < N) {
              float v[8];
#pragma unroll
              for (int j = 0; j < 8; ++j) v[j] = y[8 * i + j];
              if (args.bias != nullptr) {
                const float4 b0 = __ldg(reinterpret_cast<const float4*>(args.bias + col));
                const float4 b1 = __ldg(reinterpret_cast<const float4*>(args.bias + col + 4));
                v[0] += b0.x; v[1] += b0.y; v[2] += b0.z; v[3] += b0.w;
                v[4] += b1.x; v[5] += b1.y; v[6] += b1.z; v[7] += b1.w;
              }
              uint4 out;
              __nv_bfloat162 t0 = __floats2bfloat162_rn(v[0], v[1]);
              __nv_bfloat162 t1 = __floats2bfloat162_rn(v[2], v[3]);
              __nv_bfloat162 t2 = __floats2bfloat162_rn(v[4], v[5]);
              __nv_bfloat162 t3 = __floats2bfloat162_rn(v[6], v[7]);
              out.x = *reinterpret_cast<uint32_t*>(&t0);
              out.y = *reinterpret_cast<uint32_t*>(&t1);
              out.z = *reinterpret_cast<uint32_t*>(&t2);
              out.w = *reinterpret_cast<uint32_t*>(&t3);
              *reinterpret_cast<uint4*>(yrow + col) = out;
            }
          }
        }
      }
    }
}

template <bool kExport>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ CUtensorMap tmS, const Args args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* opA = smem + kOffOpA;
  uint8_t* opB = smem + kOffOpB;
  uint8_t* pkB = smem + kOffPkB;
  float* sw = reinterpret_cast<float*>(smem + kOffSw);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* full_a = bars;                  // A operand bytes landed (TMA)
  uint64_t* full_b = full_a + kStagesOp;    // B operand bytes written (unpack warps)
  uint64_t* empty_op = full_b + kStagesOp;  // MMAs of the stage finished
  uint64_t* full_pk = empty_op + kStagesOp;
  uint64_t* empty_pk = full_pk + kStagesPk;
  uint64_t* full_s = empty_pk + kStagesPk;
  uint64_t* empty_s = full_s + kScaleSlots;
  uint64_t* acc_full = empty_s + kScaleSlots;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* mma_done = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + kOffMisc + 4);

  const uint32_t warp = warp_id(), lane = lane_id();
  const int M = args.M, N = args.N, K = args.K, G = args.G;
  const int k_stages = K / kBK;
  const int groups = K / G;

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < kStagesOp; ++i) {
      mbar_init(&full_a[i], 1);
      mbar_init(&full_b[i], kUnpackThreads);
      mbar_init(&empty_op[i], 1);
    }
    for (int i = 0; i < kStagesPk; ++i) {
      mbar_init(&full_pk[i], 1);
      mbar_init(&empty_pk[i], kUnpackThreads);
    }
    for (int i = 0; i < kScaleSlots; ++i) {
      mbar_init(&full_s[i], 1);
      mbar_init(&empty_s[i], kDrainThreads);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kDrainThreads);
    }
    mbar_init(mma_done, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    tma_prefetch_desc(&tmS);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp >= kDrainWarp0) {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 216;\n" ::: "memory");
    drain_role<kExport>(args, tmem_base, sw, full_s, empty_s, acc_full, acc_empty, abort_flag);
  } else {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 40;\n" ::: "memory");
  if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t it_op = 0, it_pk = 0, it_s = 0;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < args.num_tiles; tile += gridDim.x) {
        const int mt = tile % args.num_m_tiles, nt = tile / args.num_m_tiles;
        for (int kb = 0; ok && kb < k_stages; ++kb) {
          const int k0 = kb * kBK;
          for (int kk = 0; kk < kBK; kk += (G < kBK ? G : kBK)) {
            if ((k0 + kk) % G != 0) continue;
            const uint32_t s = it_s % kScaleSlots;
            if (!(ok = mbar_wait(&empty_s[s], ring_parity(it_s, kScaleSlots) ^ 1u, abort_flag, args.status))) break;
            mbar_arrive_expect_tx(&full_s[s], kScaleBytes);
            tma_load_2d(sw + s * kBN, &tmS, &full_s[s], nt * kBN, (k0 + kk) / G);
            ++it_s;
          }
          if (!ok) break;
          const uint32_t p = it_pk % kStagesPk;
          if (!(ok = mbar_wait(&empty_pk[p], ring_parity(it_pk, kStagesPk) ^ 1u, abort_flag, args.status))) break;
          mbar_arrive_expect_tx(&full_pk[p], kPkBBytes);
          tma_load_2d(pkB + p * kPkBBytes, &tmB, &full_pk[p], kb * (kBK / 2), nt * kBN);
          ++it_pk;
          const uint32_t o = it_op % kStagesOp;
          if (!(ok = mbar_wait(&empty_op[o], ring_parity(it_op, kStagesOp) ^ 1u, abort_flag, args.status))) break;
          mbar_arrive_expect_tx(&full_a[o], kOpABytes);
          tma_load_2d(opA + o * kOpABytes, &tmA, &full_a[o], k0, mt * kBM);
          ++it_op;
        }
      }
      // Let every issued copy land before the CTA can exit (they complete on their own).
      for (uint32_t i = (it_s > kScaleSlots ? it_s - kScaleSlots : 0); i < it_s; ++i)
        drain_wait(&full_s[i % kScaleSlots], ring_parity(i, kScaleSlots), args.status);
      for (uint32_t i = (it_pk > kStagesPk ? it_pk - kStagesPk : 0); i < it_pk; ++i)
        drain_wait(&full_pk[i % kStagesPk], ring_parity(i, kStagesPk), args.status);
      for (uint32_t i = (it_op > kStagesOp ? it_op - kStagesOp : 0); i < it_op; ++i)
        drain_wait(&full_a[i % kStagesOp], ring_parity(i, kStagesOp), args.status);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_e4m3_f32(kBM, kBN);
      uint32_t it_op = 0, chunk_it = 0, acc_flag = 0, d_tmem = tmem_base;
      uint32_t ab = 0;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < args.num_tiles; tile += gridDim.x) {
        for (int kb = 0; ok && kb < k_stages; ++kb) {
          const uint32_t o = it_op % kStagesOp;
          if (!(ok = mbar_wait(&full_a[o], ring_parity(it_op, kStagesOp), abort_flag, args.status))) break;
          if (!(ok = mbar_wait(&full_b[o], ring_parity(it_op, kStagesOp), abort_flag, args.status))) break;
          tc_fence_after();
          const uint32_t a_base = smem_u32(opA + o * kOpABytes);
          const uint32_t b_base = smem_u32(opB + o * kOpBBytes);
#pragma unroll
          for (int k4 = 0; k4 < kBK / 32; ++k4) {
            const int kg = kb * kBK + k4 * 32;
            if (kg % G == 0) {
              ab = chunk_it & 1u;
              if (!(ok = mbar_wait(&acc_empty[ab], ((chunk_it >> 1) & 1u) ^ 1u, abort_flag, args.status))) break;
              tc_fence_after();
              d_tmem = tmem_base + ab * kBN;
              acc_flag = 0;
            }
            umma_f8f6f4(d_tmem, sdesc_kmajor_sw128(a_base + k4 * 32), sdesc_kmajor_sw128(b_base + k4 * 32), idesc,
                        acc_flag);
            acc_flag = 1;
            if ((kg + 32) % G == 0) {
              umma_commit(&acc_full[ab]);
              ++chunk_it;
            }
          }
          if (!ok) break;
          umma_commit(&empty_op[o]);
          ++it_op;
        }
      }
      // Every MMA this thread issued has finished once mma_done flips.
      umma_commit(mma_done);
      drain_wait(mma_done, 0, args.status);
    }
  } else if (warp < kDrainWarp0) {
    // ------------------------------------------------------------------ unpack
    const uint32_t ut = threadIdx.x - kUnpackWarp0 * 32;
    uint32_t it_pk = 0, it_op = 0;
    bool ok = true;
    for (int tile = blockIdx.x; ok && tile < args.num_tiles; tile += gridDim.x) {
      for (int kb = 0; ok && kb < k_stages; ++kb) {
        const uint32_t p = it_pk % kStagesPk, o = it_op % kStagesOp;
        if (!(ok = mbar_wait(&full_pk[p], ring_parity(it_pk, kStagesPk), abort_flag, args.status))) break;
        if (!(ok = mbar_wait(&empty_op[o], ring_parity(it_op, kStagesOp) ^ 1u, abort_flag, args.status))) break;
        const uint32_t src = smem_u32(pkB + p * kPkBBytes);
        const uint32_t dst = smem_u32(opB + o * kOpBBytes);
        for (uint32_t c = ut; c < kBN * 4; c += kUnpackThreads) {
          const uint32_t r = c >> 2, j = c & 3u, r7 = r & 7u;
          const uint4 pk = ld_shared_v4(src + r * 64 + j * 16);
          uint4 lo, hi;
          nib32_to_operand(pk, lo, hi);
          const uint32_t row_base = dst + (r >> 3) * 1024 + r7 * 128;
          st_shared_v4(row_base + (((2 * j) ^ r7) << 4), lo.x, lo.y, lo.z, lo.w);
          st_shared_v4(row_base + (((2 * j + 1) ^ r7) << 4), hi.x, hi.y, hi.z, hi.w);
        }
        fence_proxy_async_smem();
        mbar_arrive(&empty_pk[p]);
        mbar_arrive(&full_b[o]);
        ++it_pk;
        ++it_op;
      }
    }
  }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

bool encode_2d(CUtensorMap* map, CUtensorMapDataType dtype, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swizzle) {
  auto fn = tensor_map_encoder();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {row_bytes};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, dtype, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <bool kExport>
cudaError_t launch_impl(const GemmProblem& p, cudaStream_t stream, int sms) {
  CUtensorMap tmA, tmB, tmS;
  if (!encode_2d(&tmA, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.a_operand, p.K, p.M, p.K, kBK, kBM,
                 CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_2d(&tmB, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.qw, p.K / 2, p.N, p.K / 2, kBK / 2, kBN,
                 CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !encode_2d(&tmS, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, p.s_w, p.N, p.K / p.G, (uint64_t)p.N * 4, kBN, 1,
                 CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;
  static bool attr_set[2] = {false, false};
  if (!attr_set[kExport]) {
    cudaError_t e = cudaFuncSetAttribute(w4a4_gemm_kernel<kExport>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set[kExport] = true;
  }
  Args a;
  a.M = p.M;
  a.N = p.N;
  a.K = p.K;
  a.G = p.G;
  a.num_m_tiles = (p.M + kBM - 1) / kBM;
  const int num_n_tiles = (p.N + kBN - 1) / kBN;
  a.num_tiles = a.num_m_tiles * num_n_tiles;
  a.s_a = p.s_a;
  a.bias = p.bias;
  a.y = static_cast<__nv_bfloat16*>(p.y);
  a.partials = p.partials;
  a.status = p.status;
  const int grid = a.num_tiles < sms ? a.num_tiles : sms;
  w4a4_gemm_kernel<kExport><<<grid, kThreads, kSmemBytes, stream>>>(tmA, tmB, tmS, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_w4a4_gemm(const GemmProblem& p, cudaStream_t stream, int sms) {
  if (p.M == 0 || p.N == 0) return cudaSuccess;
  return p.partials != nullptr ? launch_impl<true>(p, stream, sms) : launch_impl<false>(p, stream, sms);
}

}  // namespace jq
