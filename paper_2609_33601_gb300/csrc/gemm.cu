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
// Persistent kernel on CTA pairs (clusters of two SMs, tcgen05 cta_group::2).  A pair owns a
// 256 x kBN output tile at a time: CTA r of the pair holds A rows 128r..128r+127 and B rows
// (output columns) r*kBN/2.. of the tile, and the even CTA issues 256 x kBN x 32 MMAs that read
// both CTAs' shared memory and write 128 rows x kBN columns into each CTA's TMEM (two
// accumulators of 256 columns fill its 512).  Per SM this halves the B bytes the tensor core
// reads and the B nibbles each SM unpacks, against a one-SM tile.  The tile width is a parameter
// of the layout (Tile): 256 normally; with several groups, 224 or 128 when their tile count
// leaves the pairs' last round of tiles fuller (grouped_tile_width).  K stages of 128;
// 16 warps per CTA:
//   warp 0      A producer: one 2-D TMA per two K stages (256 rows x 128 bytes of the
//               pre-swizzled A-operand image, 32 KB) -> A ring, completing on the even CTA's
//               barrier
//   warp 1      TMEM owner; in the even CTA also the MMA issuer (one thread): 4 MMAs per K stage
//               into one of the TMEM accumulators; a new accumulator starts at every group
//               boundary and is handed to both CTAs' drain warps when the group ends
//   warp 2      scale producer: weight (and activation) scales of 4 groups per TMA box into a
//               ring for the drain
//   warps 4-7   unpack: packed nibbles straight from global memory (two stages in flight in
//               registers) -> E4M3 operand bytes in the 128B-swizzled K-major layout -> B ring
//   warps 8-15  drain: per group, the group's scales, then the accumulator from TMEM and
//               y += (acc * s_w) * (s_a * 2^18) in fp32 registers (warp w owns TMEM lanes
//               32*(w%4).. and columns (kBN/2)*((w-8)/4)..); after the last group, + bias, round to
//               bf16, store
// Every mbarrier wait is bounded; a timeout records a status and unwinds the CTA, and both CTAs
// of a pair meet at a final cluster barrier before the pair's TMEM is released.
#include <cfloat>
#include <cstdint>
#include <type_traits>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "kernels.cuh"
#include "operand.cuh"
#include "ptx.cuh"

namespace jq {

namespace {

constexpr int kBM = 128;            // A rows per CTA (a pair covers 256)
constexpr int kPairM = 2 * kBM;
constexpr int kBK = 128;
constexpr int kStagesPerSlot = 2;   // K stages per ring slot (one A transfer, two unpacked B stages)
constexpr int kThreads = 512;
constexpr int kWarpProdA = 0, kWarpMma = 1, kWarpScale = 2;
constexpr int kUnpackWarp0 = 4, kUnpackThreads = 128;
constexpr int kUnpackGroups = 2, kUnpackGroupThreads = kUnpackThreads / kUnpackGroups;  // alternate K stages
constexpr int kUnpackGroupWarps = kUnpackGroupThreads / 32;
constexpr int kDrainWarp0 = 8, kNumDrainWarps = 8;
constexpr uint32_t kTmemCols = 512;
constexpr int kRegsCtl = 32, kRegsUnpack = 96, kRegsDrain = 192;
static_assert(4 * 32 * (kRegsCtl + kRegsUnpack + 2 * kRegsDrain) == 65536, "register split must use the launch budget");

constexpr uint32_t kOpABytes = kBM * kBK;                     // 16 KB per K stage per CTA
constexpr uint32_t kSlotABytes = kStagesPerSlot * kOpABytes;  // 32 KB

// Scale ring: each slot holds the weight scales of kScGroups groups for the tile's kBN columns
// ([group][column] fp32) and, when they come by TMA, the activation scales of those groups for
// this CTA's 128 rows ([row][group] fp32).
constexpr int kScGroups = 4, kScSlots = 4;
constexpr uint32_t kScSaBytes = kScGroups * kBM * 4;  // 2 KB

// Everything that depends on the tile width kBN (output columns per pair tile).
template <int kBN_>
struct Tile {
  static constexpr int kBN = kBN_;
  static constexpr int kBNHalf = kBN / 2;                    // B rows per CTA
  static constexpr int kAccBufs = kTmemCols / kBN;           // TMEM accumulators (2 or 4)
  static constexpr int kDrainCols = kBN / 2;                 // accumulator columns per drain warp
  static constexpr int kSlots = kBN > 128 ? 3 : 4;           // operand ring slots (what fits in shared memory)
  static constexpr uint32_t kOpBBytes = kBNHalf * kBK;       // B bytes per K stage per CTA
  static constexpr uint32_t kSlotBBytes = kStagesPerSlot * kOpBBytes;
  static constexpr int kChunksPerThread = kBNHalf * (kBK / 2) / 16 / kUnpackGroupThreads;  // packed 16-byte chunks
  static constexpr uint32_t kScSwBytes = kScGroups * kBN * 4;
  static constexpr uint32_t kScSlotBytes = kScSwBytes + kScSaBytes;
  static constexpr uint32_t kOffA = 0;
  static constexpr uint32_t kOffB = kOffA + kSlots * kSlotABytes;
  static constexpr uint32_t kOffSc = kOffB + kSlots * kSlotBBytes;
  static constexpr uint32_t kOffBar = kOffSc + kScSlots * kScSlotBytes;
  static constexpr uint32_t kNumBars = 2 * kSlots + 2 * kAccBufs + 1 + 2 * kScSlots;
  static constexpr uint32_t kOffMisc = kOffBar + kNumBars * 8;
  static constexpr uint32_t kSmemBytes = kOffMisc + 16;
  static_assert(kBN % 32 == 0 && kBN >= 128 && kBN <= 256, "tile widths (the MMA's N, a multiple of 16 per CTA)");
  static_assert(kDrainCols % 16 == 0, "the drain reads 16 columns at a time");
  static_assert(kChunksPerThread * kUnpackGroupThreads * 16 == kBNHalf * (kBK / 2), "unpack covers the B half");
  static_assert(kOffBar % 8 == 0 && kOffMisc % 8 == 0, "mbarriers need 8-byte alignment");
  static_assert(kOffSc % 128 == 0 && kScSlotBytes % 128 == 0 && kScSwBytes % 128 == 0,
                "TMA destinations need 128 bytes");
  static_assert(kOffA % 1024 == 0 && kOffB % 1024 == 0 && kOpABytes % 1024 == 0 && kOpBBytes % 1024 == 0,
                "128B-swizzled operand slots need 1024-byte alignment");
  // The rings need a 1024-byte aligned base (128B swizzle atoms); the dynamic shared memory
  // window is declared with that alignment and the kernel checks it before touching anything.
  static_assert(kSmemBytes <= 232448, "shared memory budget");
};

struct Args {
  int M, N, K, G;
  int num_m2, num_tiles, k_stages, slots_per_tile;
  int groups, sc_boxes;  // K / G, and scale-ring slots per tile (ceil(groups / kScGroups))
  int sa_tma;            // activation scales come through the scale ring (groups % 4 == 0)
  int ternary;           // qw holds 2-bit ternary codes [N, K/4] (ternary.cu), not INT4 [N, K/2]
  int prefetch_slots;    // L2 prefetch distance of the packed weights, in ring slots (producer_a)
  const uint8_t* qw;
  const float* s_a;
  const float* corr;     // [M, K/G]: 8 * the group's activation code sum in 2^-18 units (offset codes)
  const float* s_w;
  const float* bias;
  __nv_bfloat16* y;
  int32_t* partials;
  uint32_t* status;
};

struct Bars {
  uint64_t *full, *empty;  // operand ring: A and B of a slot arrive on full, leave on empty
  uint64_t *acc_full, *acc_empty, *mma_done;  // TMEM accumulators (T::kAccBufs of each)
  uint64_t *sc_full, *sc_empty;  // scale ring
};

// Accumulator hand-offs: the i-th group accumulated by the pair uses buffer i % kAccBufs, and
// that buffer's phase parity is (i / kAccBufs) & 1.
template <class T>
__device__ __forceinline__ uint32_t acc_buf(uint32_t i) { return i % T::kAccBufs; }
template <class T>
__device__ __forceinline__ uint32_t acc_parity(uint32_t i) { return (i / T::kAccBufs) & 1u; }

struct Pair {
  uint32_t rank;     // 0 = the CTA that issues the MMAs
  int cluster;       // pair index
  int num_clusters;  // pairs in the grid
};

__device__ __forceinline__ uint32_t ring_parity(uint32_t it, uint32_t slots) { return (it / slots) & 1u; }
// Address of a barrier of this CTA's layout in the even CTA of the pair.
__device__ __forceinline__ uint32_t leader_bar(uint64_t* bar) { return mapa_shared(smem_u32(bar), 0); }

// A bounded wait that ignores the CTA abort flag (used while draining in-flight async work).
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, uint32_t* status) {
  int dummy = 0;
  mbar_wait(bar, parity, &dummy, status);
}

// ------------------------------------------------------------------ drain + epilogue
// Export path (jq_w4a4_group_partials, 256-column tiles): each thread owns one TMEM lane (row) and
// 128 columns (32x32b loads) and writes the exact integer partials of every group.
template <class T, bool kOffset>
__device__ __forceinline__ void drain_export(const Args& args, const Pair& pr, uint32_t tmem_base, const Bars& b,
                                             volatile int* abort_flag) {
  const uint32_t warp = warp_id(), lane = lane_id();
  const int M = args.M, N = args.N, groups = args.groups;
  const uint32_t quarter = warp & 3u, half = (warp - kDrainWarp0) >> 2;
  const uint32_t lane_base = (quarter * 32u) << 16;
  uint32_t chunk_it = 0;
  bool ok = true;
  for (int tile = pr.cluster; ok && tile < args.num_tiles; tile += pr.num_clusters) {
    const int mt2 = tile % args.num_m2, nt = tile / args.num_m2;
    const int row = mt2 * kPairM + (int)pr.rank * kBM + (int)(quarter * 32u + lane);
    const int col0 = nt * T::kBN + half * T::kDrainCols;
    const bool row_ok = row < M;
    for (int g = 0; g < groups; ++g) {
      const uint32_t ab = acc_buf<T>(chunk_it);
      const float cr = (kOffset && row_ok) ? -__ldg(args.corr + (int64_t)row * groups + g) : 0.0f;
      // Warp-collective tcgen05.ld follows: the whole warp proceeds or none of it.
      ok = __all_sync(0xffffffffu, mbar_wait(&b.acc_full[ab], acc_parity<T>(chunk_it), abort_flag, args.status));
      if (!ok) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + lane_base + ab * T::kBN + half * T::kDrainCols;
#pragma unroll 1
      for (int cc = 0; cc < T::kDrainCols / 32; ++cc) {
        uint32_t r[32];
        tmem_ld32(taddr + cc * 32, r);
        tmem_ld_wait();
        if (row_ok) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int col = col0 + cc * 32 + j;
            if (col < N)
              args.partials[((int64_t)row * N + col) * groups + g] =
                  static_cast<int32_t>((__uint_as_float(r[j]) + cr) * kOperandUnitInv);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote_cta(leader_bar(&b.acc_empty[ab]));
      ++chunk_it;
    }
  }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// The epilogue of the row-layout drain.  Lane l holds output row row0 + l; written as it is held,
// each 16-byte store instruction would touch 32 rows (32 memory lines).  Instead the lanes of each
// aligned group of W exchange 16-byte chunks (a W x W transpose by xor-shuffle butterflies: at
// distance d a lane swaps chunk k | d or k, by bit d of its lane index, with its partner's other
// one), after which lane g + j holds chunk j of rows g .. g + W - 1, and each store instruction
// writes W consecutive chunks (16 W contiguous bytes) of each of 32 / W rows.
template <int W>
__device__ __forceinline__ void transpose_chunks(uint4 (&o)[W], uint32_t lane) {
#pragma unroll
  for (int d = 1; d < W; d <<= 1) {
    const bool up = (lane & (uint32_t)d) != 0;
#pragma unroll
    for (int k = 0; k < W; ++k) {
      if (k & d) continue;
      const uint4 send = up ? o[k] : o[k | d];
      uint4 recv;
      recv.x = __shfl_xor_sync(0xffffffffu, send.x, d);
      recv.y = __shfl_xor_sync(0xffffffffu, send.y, d);
      recv.z = __shfl_xor_sync(0xffffffffu, send.z, d);
      recv.w = __shfl_xor_sync(0xffffffffu, send.w, d);
      if (up)
        o[k] = recv;
      else
        o[k | d] = recv;
    }
  }
}

// Columns C0 .. C0 + 8W - 1 of the warp's D (relative to col0): + bias, bf16, transposed, stored.
// Rows at or past M and chunks at or past N (N % 8 == 0: a chunk is wholly inside or outside)
// are not written.
template <int W, int D, int C0>
__device__ __forceinline__ void store_block(const Args& args, const float2 (&y)[D / 2], int row0, int col0,
                                            uint32_t lane) {
  uint4 o[W];
#pragma unroll
  for (int k = 0; k < W; ++k) {
    const int c = C0 + 8 * k, col = col0 + c;
    float4 b0 = make_float4(0.f, 0.f, 0.f, 0.f), b1 = b0;
    if (args.bias != nullptr && col < args.N) {
      b0 = __ldg(reinterpret_cast<const float4*>(args.bias + col));
      b1 = __ldg(reinterpret_cast<const float4*>(args.bias + col + 4));
    }
    const float2* yy = y + (c >> 1);
    o[k].x = pack_bf16x2(yy[0].x + b0.x, yy[0].y + b0.y);
    o[k].y = pack_bf16x2(yy[1].x + b0.z, yy[1].y + b0.w);
    o[k].z = pack_bf16x2(yy[2].x + b1.x, yy[2].y + b1.y);
    o[k].w = pack_bf16x2(yy[3].x + b1.z, yy[3].y + b1.w);
  }
  transpose_chunks<W>(o, lane);
  const uint32_t j = lane & (uint32_t)(W - 1);
  const int col = col0 + C0 + 8 * (int)j;
  const int rg = row0 + (int)(lane - j);
#pragma unroll
  for (int t = 0; t < W; ++t) {
    const int r = rg + t;
    if (r < args.M && col < args.N) *reinterpret_cast<uint4*>(args.y + (int64_t)r * args.N + col) = o[t];
  }
}

// Columns C0 .. D - 1: blocks of 8W columns while they fit, the rest (D % 16 == 0) in narrower
// blocks.
template <int W, int D, int C0>
__device__ __forceinline__ void store_rows(const Args& args, const float2 (&y)[D / 2], int row0, int col0,
                                           uint32_t lane) {
  static_assert(D % 16 == 0 && W >= 2, "16-column blocks at the least");
  if constexpr (C0 + 8 * W <= D) {
    store_block<W, D, C0>(args, y, row0, col0, lane);
    store_rows<W, D, C0 + 8 * W>(args, y, row0, col0, lane);
  } else if constexpr (C0 < D) {
    store_rows<W / 2, D, C0>(args, y, row0, col0, lane);
  }
}
// Lanes per row segment of the epilogue's stores: groups of 4 (64-byte segments, two shuffle
// rounds) measured faster than groups of 2 or 8 on the FLUX QKV and dLLM shapes.
constexpr int kStoreLanes = 4;

// Linear path, several groups (sign-magnitude weight codes): warp w (drain index d = w - 8) owns
// one row per thread -- TMEM lane 32*(w%4) + lane -- and columns D*(d/4).. of each accumulator
// (D = kBN/2: 128 for the 256-column tile), read 16 at a time with the 32x32b shape: two loads in
// flight, the next 16 columns arriving while the current ones are scaled.  The running sums are float2 pairs, the operand form of the packed fp32 instructions,
// so y += (acc * s_w) * (s_a * 2^18) costs one FMUL2 and one FFMA2 per two outputs.  The weight
// scales are the same for every lane (broadcast LDS.128 from the scale ring); the activation
// scale is one value per thread and group.  (Per group the lanes of a warp fill 16 KB of registers
// with weight scales this way, four times the 16x256b layout's share, but its 8 wide TMEM loads
// per group against 32 narrow ones make it the faster of the two when every group is drained.)
template <class T, bool kOffset>
__device__ __forceinline__ void drain_linear_rows(const Args& args, const Pair& pr, uint32_t tmem_base,
                                                  const Bars& b, uint8_t* sSc, volatile int* abort_flag) {
  constexpr int D = T::kDrainCols, kBatches = D / 16;
  static_assert(kBatches >= 2, "the load pipeline needs two batches");
  const uint32_t warp = warp_id(), lane = lane_id();
  const int M = args.M, groups = args.groups;
  const uint32_t quarter = warp & 3u, half = (warp - kDrainWarp0) >> 2;
  const uint32_t trow = quarter * 32u + lane;  // row within the CTA's 128
  uint32_t chunk_it = 0, sc_it = 0;
  bool ok = true;
  bool next_full = false;  // the next accumulator was seen complete during the current group
  for (int tile = pr.cluster; ok && tile < args.num_tiles; tile += pr.num_clusters) {
    const int mt2 = tile % args.num_m2, nt = tile / args.num_m2;
    const int row = mt2 * kPairM + (int)pr.rank * kBM + (int)trow;
    const int col0 = nt * T::kBN + half * D;
    const bool row_ok = row < M;
    float2 y[D / 2];
#pragma unroll
    for (int i = 0; i < D / 2; ++i) y[i] = make_float2(0.0f, 0.0f);
    for (int g = 0; g < groups; ++g) {
      const uint32_t ab = acc_buf<T>(chunk_it);
      const int gi = g % kScGroups;
      const uint32_t sslot = sc_it % kScSlots;
      if (gi == 0) {
        ok = __all_sync(0xffffffffu, mbar_wait(&b.sc_full[sslot], ring_parity(sc_it, kScSlots), abort_flag, args.status));
        if (!ok) break;
      }
      const uint8_t* slot = sSc + sslot * T::kScSlotBytes;
      const float4* sw4 = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(slot) + gi * T::kBN + half * D);
      float sa;
      if (args.sa_tma)
        sa = reinterpret_cast<const float*>(slot + T::kScSwBytes)[trow * kScGroups + gi];
      else
        sa = row_ok ? __ldg(args.s_a + (int64_t)row * groups + g) : 0.0f;
      // one-group offset-code weights: the exact partial is the accumulator less 8 * the code sum
      const float cr = (kOffset && row_ok) ? -__ldg(args.corr + (int64_t)row * groups + g) : 0.0f;
      // Warp-collective tcgen05.ld follows: the whole warp proceeds or none of it (a timeout in
      // one lane must not leave the others in an aligned instruction).
      if (!__all_sync(0xffffffffu, next_full)) {
        ok = __all_sync(0xffffffffu, mbar_wait(&b.acc_full[ab], acc_parity<T>(chunk_it), abort_flag, args.status));
        if (!ok) break;
      }
      next_full = false;
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((quarter * 32u) << 16) + ab * T::kBN + half * D;
      auto release = [&]() {  // every column of this accumulator is in registers: hand it back
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote_cta(leader_bar(&b.acc_empty[ab]));
      };
      // Both arithmetic forms are exact-partial * scales in fp32; the second is needed when
      // s_a * 2^18 would overflow.  The choice is made for the whole warp: both issue
      // warp-collective tcgen05.ld / __syncwarp, which every lane must reach.
      if (__all_sync(0xffffffffu, sa * kOperandUnitInv <= FLT_MAX)) {
        const float2 f = make_float2(sa * kOperandUnitInv, sa * kOperandUnitInv);
        const float2 c2 = make_float2(cr, cr);
        auto scale16 = [&](int c, const uint32_t (&r)[16]) {
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float4 w = sw4[(c >> 2) + q];
            float2 d0 = make_float2(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]));
            float2 d1 = make_float2(__uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3]));
            if (kOffset) {  // integers below 2^24: exact
              d0 = __fadd2_rn(d0, c2);
              d1 = __fadd2_rn(d1, c2);
            }
            float2& y0 = y[(c >> 1) + 2 * q];
            float2& y1 = y[(c >> 1) + 2 * q + 1];
            y0 = __ffma2_rn(__fmul2_rn(d0, make_float2(w.x, w.y)), f, y0);
            y1 = __ffma2_rn(__fmul2_rn(d1, make_float2(w.z, w.w)), f, y1);
          }
        };
        uint32_t ra[16], rb[16];
        tmem_ld16(taddr, ra);
        tmem_ld_wait();
#pragma unroll
        for (int bi = 0; bi < kBatches; ++bi) {  // batch bi is in ra (even) or rb (odd)
          uint32_t(&cur)[16] = (bi & 1) ? rb : ra;
          uint32_t(&nxt)[16] = (bi & 1) ? ra : rb;
          if (bi + 1 < kBatches) tmem_ld16(taddr + 16 * (bi + 1), nxt);
          if (bi == kBatches / 2 + 1)  // the next accumulator: seen complete yet?
            next_full = mbar_test_wait(&b.acc_full[acc_buf<T>(chunk_it + 1)], acc_parity<T>(chunk_it + 1));
          scale16(16 * bi, cur);
          if (bi + 1 < kBatches) tmem_ld_wait();
          if (bi + 2 == kBatches) release();  // the last batch is in registers
        }
      } else {  // some |s_a| > 2^110: apply 2^18 to the exact partials first so nothing overflows
#pragma unroll
        for (int c = 0; c < D; c += 16) {
          uint32_t r[16];
          tmem_ld16(taddr + c, r);
          tmem_ld_wait();
          if (c == D - 16) release();
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float4 w = sw4[(c >> 2) + q];
            const float wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              float& yv = (e & 1) ? y[(c >> 1) + 2 * q + (e >> 1)].y : y[(c >> 1) + 2 * q + (e >> 1)].x;
              yv = fmaf(((__uint_as_float(r[4 * q + e]) + cr) * kOperandUnitInv) * sa, wv[e], yv);
            }
          }
        }
      }
      if (gi == kScGroups - 1 || g == groups - 1) {  // done with this scale slot
        __syncwarp();
        if (lane == 0) mbar_arrive(&b.sc_empty[sslot]);
        ++sc_it;
      }
      ++chunk_it;
    }
    if (!ok) break;
    // + bias, round to bf16, store (whole-warp shuffles: every lane takes part)
    store_rows<kStoreLanes, D, 0>(args, y, row - (int)lane, col0, lane);
  }
}
// Linear path, 256-column tiles, one group (offset weight codes, drained once per tile): warp w
// (drain index d = w - 8) owns TMEM lanes 32*(w%4).. (32 rows) and columns 128*(d/4).. of each
// accumulator, read with the 16x256b shape: thread t holds rows t/4 + {0, 8, 16, 24} of those 32
// and columns 8j + 2(t%4) + {0, 1}, j = 0..15, so it needs only 32 weight scales and 4 activation
// scales, loaded at the start of the group, and its bf16 stores are 4-byte pairs of neighbouring
// lanes (the row layout's 16-byte stores per row measured slower here, where the epilogue runs
// after every group).
template <class T, bool kOffset>
__device__ __forceinline__ void drain_linear_quads(const Args& args, const Pair& pr, uint32_t tmem_base,
                                                   const Bars& b, uint8_t* sSc, volatile int* abort_flag) {
  static_assert(T::kBN == 256, "drain layout for 256-column tiles");
  const uint32_t warp = warp_id(), lane = lane_id();
  const int M = args.M, N = args.N, groups = args.groups;
  const uint32_t quarter = warp & 3u, half = (warp - kDrainWarp0) >> 2;
  const uint32_t tq = lane & 3u, t4 = lane >> 2;
  uint32_t chunk_it = 0, sc_it = 0;
  bool ok = true;
  bool next_full = false;
  for (int tile = pr.cluster; ok && tile < args.num_tiles; tile += pr.num_clusters) {
    const int mt2 = tile % args.num_m2, nt = tile / args.num_m2;
    const int row0 = mt2 * kPairM + (int)pr.rank * kBM + (int)(quarter * 32u + t4);  // + 8 * rr
    const int col0 = nt * T::kBN + half * 128 + 2 * (int)tq;                           // + 8 * j
    float2 y[64];  // y[rr * 16 + j]
#pragma unroll
    for (int i = 0; i < 64; ++i) y[i] = make_float2(0.0f, 0.0f);
    for (int g = 0; g < groups; ++g) {
      const uint32_t ab = acc_buf<T>(chunk_it);
      const int gi = g % kScGroups;
      const uint32_t sslot = sc_it % kScSlots;
      if (gi == 0) {
        ok = __all_sync(0xffffffffu, mbar_wait(&b.sc_full[sslot], ring_parity(sc_it, kScSlots), abort_flag, args.status));
        if (!ok) break;
      }
      const uint8_t* slot = sSc + sslot * T::kScSlotBytes;
      const float* sws = reinterpret_cast<const float*>(slot) + gi * T::kBN + half * 128 + 2 * tq;
      float2 w[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) w[j] = *reinterpret_cast<const float2*>(sws + 8 * j);
      float sa[4], cr[4];
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        const int row = row0 + 8 * rr;
        if (args.sa_tma)
          sa[rr] = reinterpret_cast<const float*>(slot + T::kScSwBytes)[(quarter * 32u + t4 + 8u * rr) * kScGroups + gi];
        else
          sa[rr] = row < M ? __ldg(args.s_a + (int64_t)row * groups + g) : 0.0f;
        cr[rr] = (kOffset && row < M) ? -__ldg(args.corr + (int64_t)row * groups + g) : 0.0f;
      }
      if (!__all_sync(0xffffffffu, next_full)) {
        ok = __all_sync(0xffffffffu, mbar_wait(&b.acc_full[ab], acc_parity<T>(chunk_it), abort_flag, args.status));
        if (!ok) break;
      }
      next_full = false;
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((quarter * 32u) << 16) + ab * T::kBN + half * 128;
      auto release = [&]() {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote_cta(leader_bar(&b.acc_empty[ab]));
      };
      auto load = [&](int j, uint32_t (&r)[8]) {
        tmem_ld16x256b_x1(taddr + j * 8, *reinterpret_cast<uint32_t(*)[4]>(&r[0]));
        tmem_ld16x256b_x1(taddr + (16u << 16) + j * 8, *reinterpret_cast<uint32_t(*)[4]>(&r[4]));
      };
      bool finite = true;
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) finite = finite && (sa[rr] * kOperandUnitInv <= FLT_MAX);
      if (__all_sync(0xffffffffu, finite)) {
        float2 f[4], c2[4];
#pragma unroll
        for (int rr = 0; rr < 4; ++rr) {
          f[rr] = make_float2(sa[rr] * kOperandUnitInv, sa[rr] * kOperandUnitInv);
          c2[rr] = make_float2(cr[rr], cr[rr]);
        }
        auto scale = [&](int j, const uint32_t (&r)[8]) {  // r[0..3]: rows +0 / +8; r[4..7]: +16 / +24
#pragma unroll
          for (int rr = 0; rr < 4; ++rr) {
            const int e = 4 * (rr >> 1) + 2 * (rr & 1);
            float2 d = make_float2(__uint_as_float(r[e]), __uint_as_float(r[e + 1]));
            if (kOffset) d = __fadd2_rn(d, c2[rr]);
            y[rr * 16 + j] = __ffma2_rn(__fmul2_rn(d, w[j]), f[rr], y[rr * 16 + j]);
          }
        };
        uint32_t ra[8], rb[8];
        load(0, ra);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 16; j += 2) {
          load(j + 1, rb);
          scale(j, ra);
          tmem_ld_wait();
          if (j == 14) release();
          if (j < 14) load(j + 2, ra);
          if (j == 8)
            next_full = mbar_test_wait(&b.acc_full[acc_buf<T>(chunk_it + 1)], acc_parity<T>(chunk_it + 1));
          scale(j + 1, rb);
          if (j < 14) tmem_ld_wait();
        }
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          uint32_t r[8];
          load(j, r);
          tmem_ld_wait();
          if (j == 15) release();
#pragma unroll
          for (int rr = 0; rr < 4; ++rr) {
            const int e = 4 * (rr >> 1) + 2 * (rr & 1);
            float2& yy = y[rr * 16 + j];
            yy.x = fmaf(((__uint_as_float(r[e]) + cr[rr]) * kOperandUnitInv) * sa[rr], w[j].x, yy.x);
            yy.y = fmaf(((__uint_as_float(r[e + 1]) + cr[rr]) * kOperandUnitInv) * sa[rr], w[j].y, yy.y);
          }
        }
      }
      if (gi == kScGroups - 1 || g == groups - 1) {
        __syncwarp();
        if (lane == 0) mbar_arrive(&b.sc_empty[sslot]);
        ++sc_it;
      }
      ++chunk_it;
    }
    if (!ok) break;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const int col = col0 + 8 * j;
      if (col < N) {
        float2 bj = make_float2(0.f, 0.f);
        if (args.bias != nullptr) bj = __ldg(reinterpret_cast<const float2*>(args.bias + col));
#pragma unroll
        for (int rr = 0; rr < 4; ++rr) {
          const int row = row0 + 8 * rr;
          if (row < M)
            *reinterpret_cast<__nv_bfloat162*>(args.y + (int64_t)row * N + col) =
                __floats2bfloat162_rn(y[rr * 16 + j].x + bj.x, y[rr * 16 + j].y + bj.y);
        }
      }
    }
  }
}

// ------------------------------------------------------------------ scale producer
// Streams the scales the drain needs into the scale ring, kScGroups groups per slot: one TMA box
// of weight scales (kScGroups rows of kBN columns) and, when aligned, one of this CTA's
// activation scales (128 rows of kScGroups groups).  Boxes past the tensors' ends read zeros.
template <class T>
__device__ __forceinline__ void scale_producer(const Args& args, const Pair& pr, const CUtensorMap* tmSW,
                                               const CUtensorMap* tmSA, uint8_t* sSc, const Bars& b,
                                               volatile int* abort_flag) {
  const uint32_t bytes = T::kScSwBytes + (args.sa_tma ? kScSaBytes : 0u);
  uint32_t it = 0;
  bool ok = true;
  for (int tile = pr.cluster; ok && tile < args.num_tiles; tile += pr.num_clusters) {
    const int mt2 = tile % args.num_m2, nt = tile / args.num_m2;
    const int row0 = mt2 * kPairM + (int)pr.rank * kBM;
    for (int bi = 0; bi < args.sc_boxes; ++bi) {
      const uint32_t s = it % kScSlots;
      if (!(ok = mbar_wait(&b.sc_empty[s], ring_parity(it, kScSlots) ^ 1u, abort_flag, args.status))) break;
      uint8_t* slot = sSc + s * T::kScSlotBytes;
      mbar_arrive_expect_tx(&b.sc_full[s], bytes);
      tma_load_2d(slot, tmSW, &b.sc_full[s], nt * T::kBN, bi * kScGroups);
      if (args.sa_tma) tma_load_2d(slot + T::kScSwBytes, tmSA, &b.sc_full[s], bi * kScGroups, row0);
      ++it;
    }
  }
  for (uint32_t i = (it > kScSlots ? it - kScSlots : 0); i < it; ++i)
    drain_wait(&b.sc_full[i % kScSlots], ring_parity(i, kScSlots), args.status);
}

// ------------------------------------------------------------------ A producer
// Both CTAs load their own 128 rows of a slot's two K stages; the transfers complete on the even
// CTA's full barrier, which the even CTA arms with the bytes of both.
// The same thread prefetches into L2 this CTA's packed weight rows of the slot args.prefetch_slots
// ahead of the one it loads A for: the unpack warps fetch weights with plain loads only two slots
// ahead, which left slots waiting for DRAM when a weight tile serves few M tiles.  Measured over
// one-group problems 4096 -> 12288 (linear alone, weight sets larger than L2), with 0 / 2 / 4
// slots: M = 1024 1568 / 1720 / 1703 TFLOP/s, M = 4096 1988 / 2076 / 2077, but M = 16384 2377 /
// 2327 / 2274 (there the weights stay in L2 for the 64 M tiles that share them) and M = 256
// 942 / 922 / 877; so two slots, for 2 to 16 pair tiles along M (launch_impl).
constexpr int kPrefetchSlots = 2;

template <class T>
__device__ __forceinline__ void producer_a(const Args& args, const Pair& pr, const CUtensorMap* tmA,
                                           const CUtensorMap* tmW, uint8_t* sA, const Bars& b,
                                           volatile int* abort_flag) {
  uint32_t it = 0;
  bool ok = true;
  const int wslot_bytes = kStagesPerSlot * kBK / (args.ternary ? 4 : 2);  // packed weight bytes of a slot
  int ptile = pr.cluster, pj = 0;  // the slot whose weights are prefetched next
  auto prefetch_next = [&]() {
    if (ptile >= args.num_tiles) return;
    tma_prefetch_l2_2d(tmW, pj * wslot_bytes, (ptile / args.num_m2) * T::kBN + (int)pr.rank * T::kBNHalf);
    if (++pj == args.slots_per_tile) {
      pj = 0;
      ptile += pr.num_clusters;
    }
  };
  for (int i = 0; i < args.prefetch_slots; ++i) prefetch_next();
  for (int tile = pr.cluster; ok && tile < args.num_tiles; tile += pr.num_clusters) {
    const int mt = (tile % args.num_m2) * 2 + (int)pr.rank;  // 128-row block of the operand image
    for (int j = 0; j < args.slots_per_tile; ++j) {
      const uint32_t s = it % T::kSlots;
      if (!(ok = mbar_wait(&b.empty[s], ring_parity(it, T::kSlots) ^ 1u, abort_flag, args.status))) break;
      if (pr.rank == 0) mbar_arrive_expect_tx(&b.full[s], 2 * kSlotABytes);
      const int image_row = (mt * args.k_stages + j * kStagesPerSlot) * kBM;
      tma_load_2d_pair(sA + s * kSlotABytes, tmA, leader_bar(&b.full[s]), 0, image_row);
      if (args.prefetch_slots > 0) prefetch_next();
      ++it;
    }
  }
  // Let the pair's last copies land before the CTA can leave (the even CTA sees both CTAs' bytes;
  // on an early exit the unpack arrivals may be missing, and the bounded wait ends it).
  if (pr.rank == 0)
    for (uint32_t i = (it > T::kSlots ? it - T::kSlots : 0); i < it; ++i)
      drain_wait(&b.full[i % T::kSlots], ring_parity(i, T::kSlots), args.status);
}

// ------------------------------------------------------------------ MMA issuer (even CTA)
// The tensor core accepts only about one MMA ahead of the one it is executing, so every scalar
// instruction or branch between two MMAs can leave it idle.  All decisions are therefore taken
// once per K stage (a group of 128 or more elements starts and ends on stage boundaries; a
// group of 64 is exactly half a stage), ring positions are wrapping counters, and each stage's
// descriptors come from two precomputed bases by one add (the low field of a descriptor is the
// shared-memory address >> 4, and no slot crosses its 14-bit range).
struct MmaState {
  uint32_t chunk_it = 0;  // accumulator hand-offs so far (selects buffer and parity)
};

// Opens a new accumulator: waits until the drain has emptied it.
template <class T>
__device__ __forceinline__ bool mma_open_acc(const Args& args, const Bars& b, uint32_t tmem_base, MmaState& st,
                                             uint32_t& d_tmem, volatile int* abort_flag) {
  const uint32_t ab = acc_buf<T>(st.chunk_it);
  if (!mbar_wait_cluster(&b.acc_empty[ab], acc_parity<T>(st.chunk_it) ^ 1u, abort_flag, args.status)) return false;
  tc_fence_after();
  d_tmem = tmem_base + ab * T::kBN;
  return true;
}

// One K stage (4 MMAs of K = 32) at descriptor offsets aoff / boff (shared-memory bytes >> 4
// from the rings' bases).  kHalf: group64, two groups per stage, each in a fresh accumulator;
// otherwise a group spans stages_per_group whole stages.  With `wait_next`, the wait for the next
// ring slot's operands sits between the second and third MMA, while the tensor core still has
// queued work.
template <class T, bool kHalf>
__device__ __forceinline__ bool mma_stage(const Args& args, const Bars& b, uint32_t tmem_base, MmaState& st,
                                          uint32_t& d_tmem, int& kg, int stages_per_group, uint64_t adesc0,
                                          uint64_t bdesc0, uint32_t aoff, uint32_t boff, uint32_t idesc,
                                          bool wait_next, uint32_t nslot, uint32_t nphase, volatile int* abort_flag) {
  constexpr uint16_t kBoth = 0x3;
  const uint64_t ad = adesc0 + aoff, bd = bdesc0 + boff;
  if (kHalf) {
    if (!mma_open_acc<T>(args, b, tmem_base, st, d_tmem, abort_flag)) return false;
    umma_f8f6f4_pair(d_tmem, ad, bd, idesc, 0u);
    umma_f8f6f4_pair(d_tmem, ad + 2u, bd + 2u, idesc, 1u);
    umma_commit_pair(&b.acc_full[acc_buf<T>(st.chunk_it)], kBoth);
    ++st.chunk_it;
    if (!mma_open_acc<T>(args, b, tmem_base, st, d_tmem, abort_flag)) return false;
    umma_f8f6f4_pair(d_tmem, ad + 4u, bd + 4u, idesc, 0u);
    if (wait_next && !mbar_wait_cluster(&b.full[nslot], nphase, abort_flag, args.status)) return false;
    umma_f8f6f4_pair(d_tmem, ad + 6u, bd + 6u, idesc, 1u);
    umma_commit_pair(&b.acc_full[acc_buf<T>(st.chunk_it)], kBoth);
    ++st.chunk_it;
  } else {
    if (kg == 0 && !mma_open_acc<T>(args, b, tmem_base, st, d_tmem, abort_flag)) return false;
    umma_f8f6f4_pair(d_tmem, ad, bd, idesc, kg == 0 ? 0u : 1u);
    umma_f8f6f4_pair(d_tmem, ad + 2u, bd + 2u, idesc, 1u);
    if (wait_next && !mbar_wait_cluster(&b.full[nslot], nphase, abort_flag, args.status)) return false;
    umma_f8f6f4_pair(d_tmem, ad + 4u, bd + 4u, idesc, 1u);
    umma_f8f6f4_pair(d_tmem, ad + 6u, bd + 6u, idesc, 1u);
    if (++kg == stages_per_group) {
      umma_commit_pair(&b.acc_full[acc_buf<T>(st.chunk_it)], kBoth);
      ++st.chunk_it;
      kg = 0;
    }
  }
  return true;
}

// The issue loop runs straight through each ring slot: the MMAs of its two stages, the wait for
// the next slot in the middle of the second stage, one commit that frees the slot.  The only
// data-dependent branch per slot is the odd K-stage tail (a slot with one stage).
template <class T, bool kHalf>
__device__ __forceinline__ void mma_role(const Args& args, const Pair& pr, uint32_t tmem_base, uint8_t* sA,
                                         uint8_t* sB, const Bars& b, volatile int* abort_flag) {
  const uint32_t idesc = idesc_e4m3_f32(kPairM, T::kBN);
  constexpr uint16_t kBoth = 0x3;
  const uint64_t adesc0 = sdesc_kmajor_sw128(smem_u32(sA));
  const uint64_t bdesc0 = sdesc_kmajor_sw128(smem_u32(sB));
  const int stages_per_group = kHalf ? 1 : args.G / kBK;
  const int odd_slot = (args.k_stages & 1) != 0 ? args.slots_per_tile - 1 : -1;  // the one-stage slot, if any
  const int my_tiles =
      pr.cluster < args.num_tiles ? (args.num_tiles - 1 - pr.cluster) / pr.num_clusters + 1 : 0;
  const uint32_t total = static_cast<uint32_t>(my_tiles) * static_cast<uint32_t>(args.slots_per_tile);
  uint32_t slot = 0, phase = 0;
  MmaState st;
  uint32_t d_tmem = tmem_base;
  int j = 0, kg = 0;  // slot within the tile, K stage within the group
  bool ok = total > 0 && mbar_wait_cluster(&b.full[0], 0, abort_flag, args.status);
  for (uint32_t q = 0; ok && q < total; ++q) {
    const uint32_t nslot = slot + 1 == (uint32_t)T::kSlots ? 0 : slot + 1;
    const uint32_t nphase = slot + 1 == (uint32_t)T::kSlots ? phase ^ 1u : phase;
    const uint32_t aoff = (slot * kSlotABytes) >> 4, boff = (slot * T::kSlotBBytes) >> 4;
    const bool wait_next = q + 1 < total;
    if (j != odd_slot) {
      ok = mma_stage<T, kHalf>(args, b, tmem_base, st, d_tmem, kg, stages_per_group, adesc0, bdesc0, aoff, boff, idesc,
                               false, 0u, 0u, abort_flag) &&
           mma_stage<T, kHalf>(args, b, tmem_base, st, d_tmem, kg, stages_per_group, adesc0, bdesc0,
                               aoff + (kOpABytes >> 4), boff + (T::kOpBBytes >> 4), idesc, wait_next, nslot, nphase,
                               abort_flag);
    } else {
      ok = mma_stage<T, kHalf>(args, b, tmem_base, st, d_tmem, kg, stages_per_group, adesc0, bdesc0, aoff, boff, idesc,
                               wait_next, nslot, nphase, abort_flag);
    }
    if (!ok) break;
    umma_commit_pair(&b.empty[slot], kBoth);
    slot = nslot;
    phase = nphase;
    if (++j == args.slots_per_tile) j = 0;
  }
  // Every MMA this thread issued has finished once mma_done flips (in both CTAs).
  umma_commit_pair(b.mma_done, kBoth);
  drain_wait(b.mma_done, 0, args.status);
}

// ------------------------------------------------------------------ unpack
// Two groups of two warps take alternate K stages.  Per stage, thread u of a group converts
// packed chunks t = u + 64 i (i < kChunksPerThread): 16-byte chunk t % 4 of the 64 packed bytes
// of B row t / 4 (this CTA's half of the tile's columns).  Each chunk becomes two 16-byte operand
// chunks of the 128B-swizzled row; a quarter-warp's stores cover two rows whose chunk positions
// differ in parity, so they never share a bank.
//
// Each round's global loads are issued two rounds ahead.
// Cursor over the (tile, slot) sequence of this pair; a group's stage in slot j is 2j + group.
struct UnpackCursor {
  int tile, j;
};

// One stage's packed chunks of one thread: 16 bytes of INT4 codes, or the same 32 codes as 8 bytes
// of ternary codes (W1.58A4, qw [N, K/4]).
template <bool kTernary>
using PackedChunk = typename std::conditional<kTernary, uint2, uint4>::type;

template <class T, bool kTernary>
__device__ __forceinline__ void unpack_load(const Args& args, const Pair& pr, const UnpackCursor& c, uint32_t ug,
                                            uint32_t u, PackedChunk<kTernary> (&buf)[T::kChunksPerThread]) {
  const int kb = c.j * kStagesPerSlot + (int)ug;
  if (c.tile < args.num_tiles && kb < args.k_stages) {
    const int n0 = (c.tile / args.num_m2) * T::kBN + (int)pr.rank * T::kBNHalf;
    constexpr int kRowDiv = kTernary ? 4 : 2;  // K elements per packed byte
    constexpr int kChunk = (int)sizeof(PackedChunk<kTernary>);
    const int row_bytes = args.K / kRowDiv;
    const uint8_t* src = args.qw + kb * (kBK / kRowDiv) + (u & 3u) * kChunk;
#pragma unroll
    for (int i = 0; i < T::kChunksPerThread; ++i) {
      const int n = n0 + (int)(u >> 2) + 16 * i;
      if constexpr (kTernary)  // rows past N: zero codes
        buf[i] = n < args.N ? __ldg(reinterpret_cast<const uint2*>(src + (int64_t)n * row_bytes))
                            : make_uint2(kTernaryZeroWord, kTernaryZeroWord);
      else
        buf[i] = n < args.N ? __ldg(reinterpret_cast<const uint4*>(src + (int64_t)n * row_bytes))
                            : make_uint4(0u, 0u, 0u, 0u);
    }
  }
}

__device__ __forceinline__ void unpack_advance(const Args& args, const Pair& pr, UnpackCursor& c) {
  if (++c.j == args.slots_per_tile) {
    c.j = 0;
    c.tile += pr.num_clusters;
  }
}

// Converts this group's stage of ring slot (q % kSlots) into the slot's B half for that stage
// (or, for the missing second stage of an odd K-stage count, only signals the slot).
template <class T, bool kOffset, bool kTernary>
__device__ __forceinline__ bool unpack_store(const Args& args, uint8_t* sB, const Bars& b, uint32_t ug, uint32_t u,
                                             uint32_t q, bool has_stage,
                                             const PackedChunk<kTernary> (&buf)[T::kChunksPerThread],
                                             volatile int* abort_flag) {
  const uint32_t o = q % T::kSlots;
  if (!__all_sync(0xffffffffu, mbar_wait(&b.empty[o], ring_parity(q, T::kSlots) ^ 1u, abort_flag, args.status)))
    return false;
  if (has_stage) {
    const uint32_t dst = smem_u32(sB + o * T::kSlotBBytes + ug * T::kOpBBytes);
    const uint32_t jc = u & 3u;
#pragma unroll
    for (int i = 0; i < T::kChunksPerThread; ++i) {
      const uint32_t r = (u >> 2) + 16u * i, r7 = r & 7u;
      uint4 lo, hi;
      if constexpr (kTernary) {  // operand.cuh: each 16-code word is one operand chunk
        static_assert(!kOffset, "ternary weights enter the MMA in sign-magnitude form only");
        lo = tern16_to_operand(buf[i].x);
        hi = tern16_to_operand(buf[i].y);
      } else if constexpr (kOffset) {
        nib32_to_operand_offset(buf[i], lo, hi);  // offset weight codes (operand.cuh)
      } else {
        nib32_to_operand(buf[i], lo, hi);
      }
      const uint32_t row_base = dst + (r >> 3) * 1024u + r7 * 128u;
      st_shared_v4(row_base + (((2u * jc) ^ r7) << 4), lo.x, lo.y, lo.z, lo.w);
      st_shared_v4(row_base + (((2u * jc + 1u) ^ r7) << 4), hi.x, hi.y, hi.z, hi.w);
    }
    // The stores went to this CTA's own shared memory.  Each thread makes its stores visible to
    // the async proxy (the tensor core reads them there), the warp converges, and one lane
    // arrives on the even CTA's full barrier -- the thread-producer -> pair-MMA hand-off of the
    // SM100 pipelines: a CTA-scope release, which (unlike a cluster-scope one) does not wait for
    // the thread's loads of later rounds that are still in flight.
    fence_proxy_async_smem();
  }
  __syncwarp();
  if ((u & 31u) == 0) mbar_arrive_remote_cta(leader_bar(&b.full[o]));
  return true;
}

template <class T, bool kOffset, bool kTernary>
__device__ __forceinline__ void unpack_role(const Args& args, const Pair& pr, uint8_t* sB, const Bars& b,
                                            volatile int* abort_flag) {
  const uint32_t ut = threadIdx.x - kUnpackWarp0 * 32;
  const uint32_t ug = ut / kUnpackGroupThreads, u = ut % kUnpackGroupThreads;
  const int my_tiles =
      pr.cluster < args.num_tiles ? (args.num_tiles - 1 - pr.cluster) / pr.num_clusters + 1 : 0;
  const uint32_t total = static_cast<uint32_t>(my_tiles) * static_cast<uint32_t>(args.slots_per_tile);
  UnpackCursor sc{pr.cluster, 0};  // the slot being stored
  UnpackCursor lc = sc;            // the slot being loaded (two ahead)
  PackedChunk<kTernary> b0[T::kChunksPerThread], b1[T::kChunksPerThread];
  unpack_load<T, kTernary>(args, pr, lc, ug, u, b0);
  unpack_advance(args, pr, lc);
  unpack_load<T, kTernary>(args, pr, lc, ug, u, b1);
  unpack_advance(args, pr, lc);
  for (uint32_t q = 0; q < total; q += 2) {
    bool has = sc.j * kStagesPerSlot + (int)ug < args.k_stages;
    if (!unpack_store<T, kOffset, kTernary>(args, sB, b, ug, u, q, has, b0, abort_flag)) return;
    unpack_advance(args, pr, sc);
    unpack_load<T, kTernary>(args, pr, lc, ug, u, b0);
    unpack_advance(args, pr, lc);
    if (q + 1 < total) {
      has = sc.j * kStagesPerSlot + (int)ug < args.k_stages;
      if (!unpack_store<T, kOffset, kTernary>(args, sB, b, ug, u, q + 1, has, b1, abort_flag)) return;
      unpack_advance(args, pr, sc);
      unpack_load<T, kTernary>(args, pr, lc, ug, u, b1);
      unpack_advance(args, pr, lc);
    }
  }
}

// kOffset: the weights enter the MMA as offset codes (operand.cuh) and the drain removes the
// activation-sum correction -- used for one-group problems (G = K), where the drain's exact
// subtraction runs once per tile; with several groups the drain is the busier role and the
// weights keep the sign-magnitude form.
template <bool kExport, bool kOffset, int kBN>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmSW,
                     const __grid_constant__ CUtensorMap tmSA, const __grid_constant__ CUtensorMap tmW,
                     const Args args) {
  using T = Tile<kBN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if ((smem_u32(smem_raw) & 1023u) != 0) {  // uniform across the grid: nothing has been touched yet
    if (threadIdx.x == 0 && args.status != nullptr) atomicExch(args.status, (uint32_t)kDevSmemAlign);
    return;
  }
  uint8_t* smem = smem_raw;
  uint8_t* sA = smem + T::kOffA;
  uint8_t* sB = smem + T::kOffB;
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + T::kOffBar);
  Bars b;
  b.full = bar;
  b.empty = b.full + T::kSlots;
  b.acc_full = b.empty + T::kSlots;
  b.acc_empty = b.acc_full + T::kAccBufs;
  b.mma_done = b.acc_empty + T::kAccBufs;
  b.sc_full = b.mma_done + 1;
  b.sc_empty = b.sc_full + kScSlots;
  uint8_t* sSc = smem + T::kOffSc;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + T::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + T::kOffMisc + 4);

  Pair pr;
  pr.rank = cluster_ctarank();
  pr.cluster = static_cast<int>(blockIdx.x >> 1);
  pr.num_clusters = static_cast<int>(gridDim.x >> 1);

  const uint32_t warp = warp_id(), lane = lane_id();
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < T::kSlots; ++i) {
      // the even CTA's expect_tx (both CTAs' A bytes) + every unpack warp of both CTAs
      mbar_init(&b.full[i], 1 + 2 * kUnpackGroups * kUnpackGroupWarps);
      mbar_init(&b.empty[i], 1);  // one pair commit
    }
    for (int i = 0; i < T::kAccBufs; ++i) {
      mbar_init(&b.acc_full[i], 1);
      mbar_init(&b.acc_empty[i], 2 * kNumDrainWarps);  // every drain warp of both CTAs
    }
    mbar_init(b.mma_done, 1);
    for (int i = 0; i < kScSlots; ++i) {
      mbar_init(&b.sc_full[i], 1);                 // the scale producer's expect_tx
      mbar_init(&b.sc_empty[i], kNumDrainWarps);  // every drain warp
    }
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmW);
    if (!kExport) {
      tma_prefetch_desc(&tmSW);
      if (args.sa_tma) tma_prefetch_desc(&tmSA);
    }
  }
  if (warp == kWarpMma) {
    tmem_alloc_pair(tmem_slot, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // the peer's barriers exist before anything signals them
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  // The next kernel in the stream may launch now; it waits for this one before it touches our
  // inputs or outputs.  Every role except the weight unpack reads data the previous kernel may
  // write (the A operand, scales, corrections) or writes the output, so it waits for that kernel
  // first; the unpack reads only the packed weights and starts at once.
  pdl_launch_dependents();
  if (warp < kUnpackWarp0 || warp >= kDrainWarp0) pdl_wait();

  // Register split per warpgroup (totals the 512 x 128 registers of the launch): producer and
  // MMA (warps 0-3) 32, unpack (warps 4-7) 96, drain (warps 8-15, the running sums) 192.
  if (warp >= kDrainWarp0) {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(kRegsDrain) : "memory");
    if constexpr (kExport)
      drain_export<T, kOffset>(args, pr, tmem_base, b, abort_flag);
    else if constexpr (kOffset)
      drain_linear_quads<T, kOffset>(args, pr, tmem_base, b, sSc, abort_flag);
    else
      drain_linear_rows<T, kOffset>(args, pr, tmem_base, b, sSc, abort_flag);
  } else if (warp >= kUnpackWarp0) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegsUnpack) : "memory");
    bool done = false;
    if constexpr (!kExport && !kOffset) {  // W1.58A4 weights (the host never pairs them with offset codes)
      if (args.ternary) {
        unpack_role<T, kOffset, true>(args, pr, sB, b, abort_flag);
        done = true;
      }
    }
    if (!done) unpack_role<T, kOffset, false>(args, pr, sB, b, abort_flag);
  } else {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegsCtl) : "memory");
    if (warp == kWarpProdA) {
      if (lane == 0) producer_a<T>(args, pr, &tmA, &tmW, sA, b, abort_flag);
    } else if (warp == kWarpScale) {
      if (!kExport && lane == 0) scale_producer<T>(args, pr, &tmSW, &tmSA, sSc, b, abort_flag);
    } else if (warp == kWarpMma && lane == 0) {
      if (pr.rank == 0) {
        if (args.G < kBK)
          mma_role<T, true>(args, pr, tmem_base, sA, sB, b, abort_flag);
        else
          mma_role<T, false>(args, pr, tmem_base, sA, sB, b, abort_flag);
      }
      else  // the even CTA's MMAs read this CTA's shared memory and write its TMEM until here
        drain_wait(b.mma_done, 0, args.status);
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

// ---------------------------------------------------------------- host side
template <bool kExport, bool kOffset, int kBN>
cudaError_t launch_impl(const GemmProblem& p, cudaStream_t stream, int sms) {
  using T = Tile<kBN>;
  // The A-operand image seen as rows of 128 bytes: block (mt, kb) is rows (mt*k_stages + kb)*128..
  // One box is two consecutive blocks (two K stages of one 128-row tile).  Boxes that reach past
  // the image (the odd CTA of a pair whose rows all lie beyond M, or the second stage of an odd
  // K-stage count at the very end) read zeros.
  const int k_stages = p.K / kBK;
  const uint64_t image_rows = (uint64_t)((p.M + kBM - 1) / kBM) * k_stages * kBM;
  CUtensorMap tmA;
  if (!encode_2d(&tmA, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.a_operand, kBK, image_rows, kBK, kBK,
                 kStagesPerSlot * kBM, CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;
  // The packed weights as rows of bytes, for the L2 prefetch of a slot's rows (producer_a): one
  // box is one slot's bytes (two K stages) of this CTA's half of the tile's columns.
  CUtensorMap tmW;
  {
    const uint64_t wrow = p.ternary ? (uint64_t)p.K / 4 : (uint64_t)p.K / 2;
    if (!encode_2d(&tmW, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.qw, wrow, (uint64_t)p.N, wrow,
                   (uint32_t)(kStagesPerSlot * kBK / (p.ternary ? 4 : 2)), (uint32_t)T::kBNHalf,
                   CU_TENSOR_MAP_SWIZZLE_NONE))
      return cudaErrorInvalidValue;
  }
  // Scale maps (the export path reads no scales: it passes the A map in their place, unused).
  const int groups = p.K / p.G;
  const bool sa_tma = !kExport && groups % kScGroups == 0;
  CUtensorMap tmSW = tmA, tmSA = tmA;
  if (!kExport) {
    if (!encode_2d(&tmSW, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, p.s_w, p.N, groups, (uint64_t)p.N * 4, kBN, kScGroups,
                   CU_TENSOR_MAP_SWIZZLE_NONE))
      return cudaErrorInvalidValue;
    if (sa_tma && !encode_2d(&tmSA, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, p.s_a, groups, p.M, (uint64_t)groups * 4,
                             kScGroups, kBM, CU_TENSOR_MAP_SWIZZLE_NONE))
      return cudaErrorInvalidValue;
  }
  // Once per device: the shared-memory attribute, and how many pairs can be resident at once.
  static PerDevice<int> setup;
  int max_pairs = 0;
  cudaError_t se = setup.get(
      [sms](int& pairs) {
        cudaError_t e = cudaFuncSetAttribute(w4a4_gemm_kernel<kExport, kOffset, kBN>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)T::kSmemBytes);
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2 * (sms / 2), 1, 1);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cfg.dynamicSmemBytes = T::kSmemBytes;
        int clusters = 0;
        if (cudaOccupancyMaxActiveClusters(&clusters, w4a4_gemm_kernel<kExport, kOffset, kBN>, &cfg) !=
                cudaSuccess ||
            clusters <= 0) {
          (void)cudaGetLastError();
          clusters = sms / 2;
        }
        pairs = clusters < sms / 2 ? clusters : sms / 2;
        return cudaSuccess;
      },
      max_pairs);
  if (se != cudaSuccess) return se;
  Args a;
  a.M = p.M;
  a.N = p.N;
  a.K = p.K;
  a.G = p.G;
  a.num_m2 = (p.M + kPairM - 1) / kPairM;
  const int num_n_tiles = (p.N + kBN - 1) / kBN;
  a.num_tiles = a.num_m2 * num_n_tiles;
  a.k_stages = k_stages;
  a.slots_per_tile = (k_stages + kStagesPerSlot - 1) / kStagesPerSlot;
  a.groups = groups;
  a.sc_boxes = (groups + kScGroups - 1) / kScGroups;
  a.sa_tma = sa_tma ? 1 : 0;
  a.ternary = p.ternary ? 1 : 0;
  a.prefetch_slots = (a.num_m2 >= 2 && a.num_m2 <= 16) ? kPrefetchSlots : 0;
  a.qw = p.qw;
  a.s_a = p.s_a;
  a.corr = p.corr;
  a.s_w = p.s_w;
  a.bias = p.bias;
  a.y = static_cast<__nv_bfloat16*>(p.y);
  a.partials = p.partials;
  a.status = p.status;
  const int pairs = a.num_tiles < max_pairs ? a.num_tiles : max_pairs;
  return launch_pdl(w4a4_gemm_kernel<kExport, kOffset, kBN>, dim3(2 * pairs), dim3(kThreads), T::kSmemBytes, stream,
                    tmA, tmSW, tmSA, tmW, a);
}

}  // namespace

namespace {
// The driver's tensor-map encoder (one entry point per process; the initialisation of a
// function-local static is thread-safe).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = []() -> PFN_cuTensorMapEncodeTiled_v12000 {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return nullptr;
  }();
  return fn;
}
}  // namespace

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

// Tile width of the grouped (sign-magnitude, several groups) linear path.  Every pair of CTAs
// takes ceil(tiles / pairs) tiles at most, each costing time in proportion to its width, so the
// width with the smallest ceil(tiles / pairs) * width finishes first; a narrower tile is taken
// only when it wins by 3 % (it re-reads the A operand more often).  E.g. 1024 x 4096 -> 12288:
// 192 tiles of 256 on 76 pairs (3 rounds, the last half full) against 220 of 224 (3 rounds, nearly
// full); 4096 x 4608 -> 1152: 80 tiles of 256 (2 rounds, the second with 4 tiles) against 144
// of 128 (2 full rounds).
int grouped_tile_width(const GemmProblem& p, int sms) {
  const int64_t num_m2 = (p.M + kPairM - 1) / kPairM, pairs = sms / 2 > 0 ? sms / 2 : 1;
  auto cost = [&](int64_t bn) {
    const int64_t tiles = num_m2 * ((p.N + bn - 1) / bn);
    return ((tiles + pairs - 1) / pairs) * bn;
  };
  int best = 256;
  int64_t c_best = cost(256);
  for (int bn : {224, 128}) {
    const int64_t c = cost(bn);
    if (c * 100 < c_best * 97) {
      best = bn;
      c_best = c;
    }
  }
  return best;
}

cudaError_t launch_w4a4_gemm(const GemmProblem& p, cudaStream_t stream, int sms) {
  if (p.M == 0 || p.N == 0) return cudaSuccess;
  // One group: offset-code weights (see w4a4_gemm_kernel), exact while the whole K run fits the
  // offset form's fp32 range (operand.cuh); longer one-group runs keep the sign-magnitude form,
  // whose sums stay below 2^24 for every K the library accepts.  Group scales: 128-column tiles.
  // Ternary weights keep the sign-magnitude form in every mode (one form keeps the unpack role's
  // registers within the kernel's budget).
  const bool offset = p.G == p.K && p.K <= kOffsetMaxRun && !p.ternary;
  if (p.partials != nullptr)
    return offset ? launch_impl<true, true, 256>(p, stream, sms) : launch_impl<true, false, 256>(p, stream, sms);
  // One group: 256-column tiles always (their 16x256b drain; the row drain on narrower tiles
  // measured slower there: 1024 x 4096 -> 12288 with G = K, 1615 -> 1557 TFLOP/s at width 224).
  if (offset) return launch_impl<false, true, 256>(p, stream, sms);
  switch (grouped_tile_width(p, sms)) {
    case 224:
      return launch_impl<false, false, 224>(p, stream, sms);
    case 128:
      return launch_impl<false, false, 128>(p, stream, sms);
    default:
      return launch_impl<false, false, 256>(p, stream, sms);
  }
}

}  // namespace jq
