// skinny.cu -- the W4A4 linear layer for few tokens (M <= 64), where the layer is bound by
// streaming the packed weights from HBM rather than by the tensor core.
//
// Same arithmetic as gemm.cu (Sec. 1, Appendix FAQ Q7): acc[m,n,g] = sum_{k in g} qa*qw exactly
// (E4M3 operand bytes through tcgen05.mma kind::f8f6f4, operand.cuh), y = sum_g acc*s_a*s_w +
// bias in fp32, rounded to bf16.  The shape of the work is different:
//   - the operands are swapped: each CTA unpacks 128 output channels of the weights into the
//     MMA's M operand and the (at most 64) tokens are its N operand, so the MMA, the TMEM
//     accumulators and the drain all scale with the real token count;
//   - packed weight and activation codes stream in by TMA (two K stages per box, 128-byte
//     swizzle) into a ring in shared memory: the TMA unit keeps far more bytes in flight per SM
//     than per-thread loads, which is what a weight-streaming kernel needs;
//   - no workspace and no separate activation expansion;
//   - K is split across the CTAs of a cluster (up to 8) so that enough SMs stream weights; the
//     partial outputs are summed through distributed shared memory in a fixed tree order, so
//     the result does not depend on timing.  For G = K (one group) the CTAs sum exact integer
//     partials and scale once; otherwise each CTA scales its whole groups and the fp32 partial
//     outputs are summed (the order of the fp32 sum over groups is free).
// CTA layout, 16 warps:
//   warp 0      TMEM owner and MMA issuer (one thread): 4 x (128 x Mp x 32) MMAs per K stage
//   warp 1      activation scales: streams s_a into a ring for the drain, 8 groups per batch
//   warp 2      TMA producer (one thread): per two K stages, one box of 128 weight rows and one
//               of the Mp token rows, 128 packed bytes each
//   warps 4-11  unpack, two groups of four warps on alternate K stages: packed codes from the
//               packed ring -> E4M3 operand rows (128B swizzle) in the operand ring
//   warps 12-15 drain: per group, tcgen05.ld 32x32b (thread = output channel, every token
//               column), y[m] += (acc * s_w) * (s_a[m] * 2^18)
// Every mbarrier wait is bounded; a timeout records a status and unwinds the CTA.
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

constexpr int kRows = 128;       // output channels per CTA (the MMA's M)
constexpr int kBK = 128;         // K elements per stage
constexpr int kStPerSlot = 2;    // K stages per packed slot (one TMA box of 128 packed bytes per row)
constexpr int kPkSlots = 4;      // packed ring (slots of two stages)
constexpr int kOpSlots = 4;      // operand ring (stages)
constexpr int kThreads = 512;
constexpr int kWarpMma = 0, kWarpScale = 1, kWarpTma = 2;
constexpr int kUnpackWarp0 = 4, kUnpackGroups = 2, kUnpackGroupThreads = 128;
constexpr int kUnpackGroupWarps = kUnpackGroupThreads / 32;
constexpr int kWChunks = kRows * 4 / kUnpackGroupThreads;  // packed 16-byte weight chunks per thread per stage
constexpr int kDrainWarp0 = 12, kNumDrainWarps = 4;
constexpr int kSaRing = 16, kSaBatch = 8;  // activation-scale ring (groups), groups per load batch
constexpr int kMaxSplit = 8;
static_assert(kWChunks == 4, "unpack assumes four weight chunks per thread per stage");
static_assert(kDrainWarp0 % 4 == 0, "drain warp w reads TMEM lanes 32 * (w % 4)");

template <int kMp>
struct Layout {
  static constexpr uint32_t kPkW = kRows * kBK;           // packed weights of a slot: 128 rows x 128 B
  static constexpr uint32_t kPkX = kMp * kBK;             // packed tokens of a slot: kMp rows x 128 B
  static constexpr uint32_t kPkSlot = kPkW + kPkX;
  static constexpr uint32_t kOpA = kRows * kBK;           // weight operand bytes of a stage
  static constexpr uint32_t kOpB = kMp * kBK;             // token operand bytes of a stage
  static constexpr uint32_t kOpSlot = kOpA + kOpB;
  static constexpr uint32_t kOffPk = 0;
  static constexpr uint32_t kOffOp = kOffPk + kPkSlots * kPkSlot;
  static constexpr uint32_t kOffSa = kOffOp + kOpSlots * kOpSlot;  // [kSaRing][kMp] fp32
  static constexpr uint32_t kOffBar = kOffSa + kSaRing * kMp * 4;
  static constexpr uint32_t kNumBars = 2 * kPkSlots + 2 * kOpSlots + 4 + 1 + 2 * kSaRing;
  static constexpr uint32_t kOffMisc = kOffBar + kNumBars * 8;
  static constexpr uint32_t kSmemBytes = kOffMisc + 16;
  static constexpr uint32_t kRedBytes = kMp * kRows * 4;  // fp32 partials [kMp][128], reuse the operand ring
  static constexpr uint32_t kTmemCols = 2 * kMp < 32 ? 32 : 2 * kMp;  // two accumulators
  static_assert(kPkW % 1024 == 0 && kPkX % 1024 == 0 && kOpA % 1024 == 0 && kOpB % 1024 == 0,
                "128B-swizzle atoms need 1024-byte alignment");
  static_assert(kOffSa % 16 == 0 && kOffBar % 8 == 0, "alignment");
  static_assert(kRedBytes <= kOpSlots * kOpSlot, "the reduction buffer reuses the operand ring");
  static_assert(kSmemBytes <= 232448, "shared memory budget");
};

struct SkArgs {
  int M, N, K, G;
  int groups;         // K / G
  int k_stages;       // K / 128
  int split;          // CTAs per cluster, each one a K range of the same 128 channels
  const float* s_a;   // [M, K/G]
  const float* s_w;   // [K/G, N]
  const float* bias;  // [N] or nullptr
  __nv_bfloat16* y;   // [M, N]
  uint32_t* status;
};

struct SkBars {
  uint64_t *pk_full, *pk_empty;  // packed ring
  uint64_t *op_full, *op_empty;  // operand ring
  uint64_t *acc_full, *acc_empty, *mma_done;
  uint64_t *sa_full, *sa_empty;  // activation-scale ring
};

__device__ __forceinline__ uint32_t ring_parity(uint32_t it, uint32_t slots) { return (it / slots) & 1u; }

// This CTA's K stages: an even split of the K stages over the ranks of the cluster.
struct Range {
  int st0, nst;  // first stage, number of stages
};
__device__ __forceinline__ Range k_range(const SkArgs& a, uint32_t rank) {
  const int s0 = (int)((int64_t)a.k_stages * rank / a.split);
  const int s1 = (int)((int64_t)a.k_stages * (rank + 1) / a.split);
  return Range{s0, s1 - s0};
}
__device__ __forceinline__ int groups_per_stage(const SkArgs& a) { return a.G < kBK ? kBK / a.G : 1; }
// Groups this CTA drains: G = K is one group however K is split; otherwise whole groups.
__device__ __forceinline__ int drain_groups(const SkArgs& a, const Range& r) {
  if (a.groups == 1) return r.nst > 0 ? 1 : 0;
  return r.nst * groups_per_stage(a);
}

// Row r of a 128B-swizzled K-major tile at `base`: 16-byte chunk c sits at chunk c ^ (r % 8).
__device__ __forceinline__ uint32_t sw128_row(uint32_t base, uint32_t r) { return base + (r >> 3) * 1024u + (r & 7u) * 128u; }

// Within each group of 8 rows, pairs rows r and r + 4 on consecutive indices q: a quarter-warp
// reading two such rows at the same four logical chunks hits 8 distinct physical chunks.
__device__ __forceinline__ uint32_t row_of(uint32_t q) { return (q & ~7u) + ((q & 1u) << 2) + ((q >> 1) & 3u); }

// ------------------------------------------------------------------ TMA producer
template <int kMp>
__device__ __forceinline__ void tma_role(const SkArgs& a, const Range& rg, int n0, const CUtensorMap* tmW,
                                         const CUtensorMap* tmX, uint8_t* smem, const SkBars& b,
                                         volatile int* abort_flag) {
  using L = Layout<kMp>;
  const int nslots = (rg.nst + kStPerSlot - 1) / kStPerSlot;
  for (int j = 0; j < nslots; ++j) {
    const uint32_t s = (uint32_t)j % kPkSlots;
    if (!mbar_wait(&b.pk_empty[s], ring_parity(j, kPkSlots) ^ 1u, abort_flag, a.status)) break;
    uint8_t* slot = smem + L::kOffPk + s * L::kPkSlot;
    const int x = (rg.st0 + j * kStPerSlot) * (kBK / 2);  // packed byte offset along K
    mbar_arrive_expect_tx(&b.pk_full[s], L::kPkSlot);
    tma_load_2d(slot, tmW, &b.pk_full[s], x, n0);
    tma_load_2d(slot + L::kPkW, tmX, &b.pk_full[s], x, 0);
  }
  // let the last copies land before the CTA can leave
  for (int j = nslots > kPkSlots ? nslots - kPkSlots : 0; j < nslots; ++j) {
    int dummy = 0;
    mbar_wait(&b.pk_full[j % kPkSlots], ring_parity(j, kPkSlots), &dummy, a.status);
  }
}

// ------------------------------------------------------------------ unpack
// Group ug converts stage 2j + ug of packed slot j: the 64-byte half ug of every packed row.
// Thread u takes logical chunks t = u + 128 i: row q = t / 4 (paired by row_of), chunk t % 4.
template <int kMp>
__device__ __forceinline__ void unpack_role(const SkArgs& a, const Range& rg, uint8_t* smem, const SkBars& b,
                                            volatile int* abort_flag) {
  using L = Layout<kMp>;
  constexpr int kXChunks = (kMp * 4 + kUnpackGroupThreads - 1) / kUnpackGroupThreads;  // token chunks per thread
  const uint32_t ut = threadIdx.x - kUnpackWarp0 * 32;
  const uint32_t ug = ut / kUnpackGroupThreads, u = ut % kUnpackGroupThreads;
  const uint32_t jc = u & 3u, lc = ug * 4u + jc;  // chunk within the stage / within the 128-byte row
  const int nslots = (rg.nst + kStPerSlot - 1) / kStPerSlot;
  // the packed 16-byte chunk of row r in a packed tile
  auto load = [&](uint32_t src, uint32_t r) { return ld_shared_v4(sw128_row(src, r) + ((lc ^ (r & 7u)) << 4)); };
  // stores it as two operand chunks (rows with bit 2 set store their chunks in the other order,
  // which keeps a quarter-warp's stores on distinct banks)
  auto convert = [&](uint4 p, uint32_t dst, uint32_t r) {
    uint4 lo, hi;
    nib32_to_operand(p, lo, hi);
    const uint32_t row_base = sw128_row(dst, r), r7 = r & 7u;
    const uint32_t c_lo = (2u * jc) ^ r7, c_hi = (2u * jc + 1u) ^ r7;
    if (r & 4u) {
      st_shared_v4(row_base + (c_hi << 4), hi.x, hi.y, hi.z, hi.w);
      st_shared_v4(row_base + (c_lo << 4), lo.x, lo.y, lo.z, lo.w);
    } else {
      st_shared_v4(row_base + (c_lo << 4), lo.x, lo.y, lo.z, lo.w);
      st_shared_v4(row_base + (c_hi << 4), hi.x, hi.y, hi.z, hi.w);
    }
  };
  for (int j = 0; j < nslots; ++j) {
    const uint32_t p = (uint32_t)j % kPkSlots;
    const int st = j * kStPerSlot + (int)ug;  // this group's stage (within the CTA's range)
    if (!__all_sync(0xffffffffu, mbar_wait(&b.pk_full[p], ring_parity(j, kPkSlots), abort_flag, a.status))) return;
    if (st < rg.nst) {
      const uint32_t o = (uint32_t)st % kOpSlots;
      if (!__all_sync(0xffffffffu, mbar_wait(&b.op_empty[o], ring_parity(st, kOpSlots) ^ 1u, abort_flag, a.status)))
        return;
      const uint32_t src = smem_u32(smem + L::kOffPk + p * L::kPkSlot);
      const uint32_t dst = smem_u32(smem + L::kOffOp + o * L::kOpSlot);
      // all loads first: the shared-memory accessors are ordered, so interleaving loads with the
      // previous chunk's stores would expose a load latency per chunk
      uint4 pw[kWChunks], px[kXChunks];
#pragma unroll
      for (int i = 0; i < kWChunks; ++i) pw[i] = load(src, row_of((u + kUnpackGroupThreads * i) >> 2));
#pragma unroll
      for (int i = 0; i < kXChunks; ++i) {
        const uint32_t t = u + kUnpackGroupThreads * i;
        if (t < kMp * 4) px[i] = load(src + L::kPkW, row_of(t >> 2));
      }
#pragma unroll
      for (int i = 0; i < kWChunks; ++i) convert(pw[i], dst, row_of((u + kUnpackGroupThreads * i) >> 2));
#pragma unroll
      for (int i = 0; i < kXChunks; ++i) {
        const uint32_t t = u + kUnpackGroupThreads * i;
        if (t < kMp * 4) convert(px[i], dst + L::kOpA, row_of(t >> 2));
      }
      fence_proxy_async_smem();
      __syncwarp();
      if ((u & 31u) == 0) mbar_arrive(&b.op_full[o]);
    }
    __syncwarp();
    if ((u & 31u) == 0) mbar_arrive(&b.pk_empty[p]);
  }
}

// ------------------------------------------------------------------ activation scales
// One warp (lane m = token): the scales of this CTA's groups into the ring, kSaBatch groups per
// batch of loads so that one load latency covers several groups.  Rows >= M get 0.
template <int kMp>
__device__ __forceinline__ void scale_role(const SkArgs& a, const Range& rg, uint8_t* smem, const SkBars& b,
                                           volatile int* abort_flag) {
  using L = Layout<kMp>;
  constexpr int kPer = kMp / 32 > 0 ? kMp / 32 : 1;  // tokens per lane
  const uint32_t lane = lane_id();
  float* sa_ring = reinterpret_cast<float*>(smem + L::kOffSa);
  const int ng = drain_groups(a, rg);
  if (ng == 0 || a.groups == 1) return;  // G = K: the final pass reads s_a itself
  const int g0 = rg.st0 * groups_per_stage(a);
  for (int gb = 0; gb < ng; gb += kSaBatch) {
    const int nb = ng - gb < kSaBatch ? ng - gb : kSaBatch;
    float v[kSaBatch][kPer];
#pragma unroll
    for (int j = 0; j < kSaBatch; ++j) {
#pragma unroll
      for (int h = 0; h < kPer; ++h) {
        const int m = (int)lane + 32 * h;
        v[j][h] = (j < nb && m < kMp && m < a.M) ? __ldg(a.s_a + (int64_t)m * a.groups + g0 + gb + j) : 0.0f;
      }
    }
#pragma unroll
    for (int j = 0; j < kSaBatch; ++j) {
      if (j >= nb) break;
      const uint32_t it = (uint32_t)(gb + j), o = it % kSaRing;
      if (!__all_sync(0xffffffffu, mbar_wait(&b.sa_empty[o], ring_parity(it, kSaRing) ^ 1u, abort_flag, a.status)))
        return;
#pragma unroll
      for (int h = 0; h < kPer; ++h) {
        const int m = (int)lane + 32 * h;
        if (m < kMp) sa_ring[o * kMp + m] = v[j][h];
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&b.sa_full[o]);
    }
  }
}

// ------------------------------------------------------------------ MMA issuer
template <int kMp>
__device__ __forceinline__ void mma_role(const SkArgs& a, const Range& rg, uint32_t tmem_base, uint8_t* smem,
                                         const SkBars& b, volatile int* abort_flag) {
  using L = Layout<kMp>;
  const uint32_t idesc = idesc_e4m3_f32(kRows, kMp);
  const uint64_t adesc0 = sdesc_kmajor_sw128(smem_u32(smem + L::kOffOp));
  const uint64_t bdesc0 = sdesc_kmajor_sw128(smem_u32(smem + L::kOffOp + L::kOpA));
  const bool single = a.groups == 1;
  const bool half_groups = a.G < kBK;
  uint32_t chunk_it = 0, d_tmem = tmem_base;
  auto open_acc = [&]() -> bool {
    const uint32_t ab = chunk_it & 1u;
    if (!mbar_wait(&b.acc_empty[ab], ((chunk_it >> 1) & 1u) ^ 1u, abort_flag, a.status)) return false;
    tc_fence_after();
    d_tmem = tmem_base + ab * kMp;
    return true;
  };
  auto close_acc = [&]() {
    umma_commit(&b.acc_full[chunk_it & 1u]);
    ++chunk_it;
  };
  bool ok = rg.nst > 0 && (!single || open_acc());
  for (int s = 0; ok && s < rg.nst; ++s) {
    const uint32_t o = (uint32_t)s % kOpSlots;
    if (!(ok = mbar_wait(&b.op_full[o], ring_parity(s, kOpSlots), abort_flag, a.status))) break;
    const uint64_t ad = adesc0 + ((o * L::kOpSlot) >> 4), bd = bdesc0 + ((o * L::kOpSlot) >> 4);
    if (single) {
      umma_f8f6f4(d_tmem, ad, bd, idesc, s == 0 ? 0u : 1u);
      umma_f8f6f4(d_tmem, ad + 2u, bd + 2u, idesc, 1u);
      umma_f8f6f4(d_tmem, ad + 4u, bd + 4u, idesc, 1u);
      umma_f8f6f4(d_tmem, ad + 6u, bd + 6u, idesc, 1u);
    } else if (half_groups) {
      if (!(ok = open_acc())) break;
      umma_f8f6f4(d_tmem, ad, bd, idesc, 0u);
      umma_f8f6f4(d_tmem, ad + 2u, bd + 2u, idesc, 1u);
      close_acc();
      if (!(ok = open_acc())) break;
      umma_f8f6f4(d_tmem, ad + 4u, bd + 4u, idesc, 0u);
      umma_f8f6f4(d_tmem, ad + 6u, bd + 6u, idesc, 1u);
      close_acc();
    } else {
      if (!(ok = open_acc())) break;
      umma_f8f6f4(d_tmem, ad, bd, idesc, 0u);
      umma_f8f6f4(d_tmem, ad + 2u, bd + 2u, idesc, 1u);
      umma_f8f6f4(d_tmem, ad + 4u, bd + 4u, idesc, 1u);
      umma_f8f6f4(d_tmem, ad + 6u, bd + 6u, idesc, 1u);
      close_acc();
    }
    umma_commit(&b.op_empty[o]);
  }
  if (ok && single && rg.nst > 0) close_acc();
  umma_commit(b.mma_done);
  int dummy = 0;
  mbar_wait(b.mma_done, 0, &dummy, a.status);
}

// ------------------------------------------------------------------ drain
// Warp w: TMEM lanes 32 * (w % 4).. (output channels), every token column (kH = kMp of them;
// hf, the column-half index of a wider layout, is 0).  For G = K the accumulator is the exact
// integer partial of this CTA's K range and is kept unscaled.  At the end the partials go to
// the reduction buffer, which reuses the operand ring: the last group's accumulator being full
// means every MMA has finished, and so every stage stored there has been consumed.
template <int kMp>
__device__ __forceinline__ void drain_role(const SkArgs& a, const Range& rg, int n0, uint32_t tmem_base, uint8_t* smem,
                                           const SkBars& b, volatile int* abort_flag) {
  using L = Layout<kMp>;
  constexpr int kH = kMp;  // token columns per thread
  const uint32_t warp = warp_id(), lane = lane_id();
  const uint32_t quarter = warp & 3u, hf = 0;
  const uint32_t ch = quarter * 32u + lane;
  const int n = n0 + (int)ch;
  const bool single = a.groups == 1;
  const float* sa_ring = reinterpret_cast<const float*>(smem + L::kOffSa);
  const int ng = drain_groups(a, rg);
  const int g0 = single ? 0 : rg.st0 * groups_per_stage(a);
  float y[kH];
#pragma unroll
  for (int i = 0; i < kH; ++i) y[i] = 0.0f;
  float sw_next = (!single && ng > 0 && n < a.N) ? __ldg(a.s_w + (int64_t)g0 * a.N + n) : 0.0f;
  for (int gi = 0; gi < ng; ++gi) {
    const uint32_t ab = (uint32_t)gi & 1u;
    const float sw = sw_next;
    if (!single && gi + 1 < ng && n < a.N) sw_next = __ldg(a.s_w + (int64_t)(g0 + gi + 1) * a.N + n);
    const uint32_t so = (uint32_t)gi % kSaRing;
    bool ok = true;
    if (!single) ok = mbar_wait(&b.sa_full[so], ring_parity(gi, kSaRing), abort_flag, a.status);
    ok = ok && mbar_wait(&b.acc_full[ab], ((uint32_t)gi >> 1) & 1u, abort_flag, a.status);
    // warp-collective tcgen05.ld follows: the whole warp proceeds or none of it
    if (!__all_sync(0xffffffffu, ok)) break;
    tc_fence_after();
    const uint32_t taddr = tmem_base + ((quarter * 32u) << 16) + ab * kMp + hf * kH;
    const float* sas = sa_ring + so * kMp + hf * kH;
    // overflow-safe form needed only if some s_a * 2^18 of these columns overflows; the choice
    // is the warp's (no lane may skip the warp-collective loads below)
    bool finite = true;
    if (!single) {
#pragma unroll
      for (int i = 0; i < kH; i += 4) {
        const float4 s4 = *reinterpret_cast<const float4*>(sas + i);
        finite = finite && fmaxf(fmaxf(s4.x, s4.y), fmaxf(s4.z, s4.w)) * kOperandUnitInv <= FLT_MAX;
      }
    }
    finite = __all_sync(0xffffffffu, finite);
#pragma unroll
    for (int c = 0; c < kH / 8; ++c) {
      uint32_t r[8];
      tmem_ld8(taddr + c * 8, r);
      tmem_ld_wait();
      if (c == kH / 8 - 1) {  // the accumulator is in registers: hand it back
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&b.acc_empty[ab]);
      }
      if (single) {
#pragma unroll
        for (int i = 0; i < 8; ++i) y[c * 8 + i] += __uint_as_float(r[i]);  // exact integer partials
      } else if (finite) {
#pragma unroll
        for (int i = 0; i < 8; i += 2) {
          const float2 s2 = *reinterpret_cast<const float2*>(sas + c * 8 + i);
          const float2 t = __fmul2_rn(make_float2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])), make_float2(sw, sw));
          const float2 v = __ffma2_rn(t, make_float2(s2.x * kOperandUnitInv, s2.y * kOperandUnitInv),
                                      make_float2(y[c * 8 + i], y[c * 8 + i + 1]));
          y[c * 8 + i] = v.x;
          y[c * 8 + i + 1] = v.y;
        }
      } else {  // |s_a| > 2^110 somewhere: apply 2^18 to the exact partials first
#pragma unroll
        for (int i = 0; i < 8; ++i)
          y[c * 8 + i] = fmaf((__uint_as_float(r[i]) * kOperandUnitInv) * sas[c * 8 + i], sw, y[c * 8 + i]);
      }
    }
    if (!single) {
      __syncwarp();
      if (lane == 0) mbar_arrive(&b.sa_empty[so]);
    }
  }
  float* red = reinterpret_cast<float*>(smem + L::kOffOp);  // [kMp][128]
#pragma unroll
  for (int i = 0; i < kH; ++i) red[(hf * kH + i) * kRows + ch] = y[i];
}

template <int kMp>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_skinny_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                       const SkArgs a) {
  using L = Layout<kMp>;
  constexpr int kH = kMp;  // token columns per drain thread
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0) {  // uniform across the grid: nothing has been touched yet
    if (threadIdx.x == 0 && a.status != nullptr) atomicExch(a.status, (uint32_t)kDevSmemAlign);
    return;
  }
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + L::kOffBar);
  SkBars b;
  b.pk_full = bar;
  b.pk_empty = b.pk_full + kPkSlots;
  b.op_full = b.pk_empty + kPkSlots;
  b.op_empty = b.op_full + kOpSlots;
  b.acc_full = b.op_empty + kOpSlots;
  b.acc_empty = b.acc_full + 2;
  b.mma_done = b.acc_empty + 2;
  b.sa_full = b.mma_done + 1;
  b.sa_empty = b.sa_full + kSaRing;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::kOffMisc + 4);

  const uint32_t rank = cluster_ctarank();
  const int n0 = (int)(blockIdx.x / a.split) * kRows;
  const Range rg = k_range(a, rank);
  const uint32_t warp = warp_id(), lane = lane_id();
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < kPkSlots; ++i) {
      mbar_init(&b.pk_full[i], 1);                                  // the producer's expect_tx
      mbar_init(&b.pk_empty[i], kUnpackGroups * kUnpackGroupWarps);  // every unpack warp
    }
    for (int i = 0; i < kOpSlots; ++i) {
      mbar_init(&b.op_full[i], kUnpackGroupWarps);  // the stage's unpack group
      mbar_init(&b.op_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&b.acc_full[i], 1);
      mbar_init(&b.acc_empty[i], kNumDrainWarps);
    }
    mbar_init(b.mma_done, 1);
    for (int i = 0; i < kSaRing; ++i) {
      mbar_init(&b.sa_full[i], 1);
      mbar_init(&b.sa_empty[i], kNumDrainWarps);
    }
    fence_mbar_init();
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
  }
  if (warp == kWarpMma) {
    tmem_alloc(tmem_slot, L::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const bool drain = warp >= kDrainWarp0;
  if (drain) {
    drain_role<kMp>(a, rg, n0, tmem_base, smem, b, abort_flag);
  } else if (warp >= kUnpackWarp0) {
    unpack_role<kMp>(a, rg, smem, b, abort_flag);
  } else if (warp == kWarpScale) {
    scale_role<kMp>(a, rg, smem, b, abort_flag);
  } else if (warp == kWarpTma && lane == 0) {
    tma_role<kMp>(a, rg, n0, &tmW, &tmX, smem, b, abort_flag);
  } else if (warp == kWarpMma && lane == 0) {
    mma_role<kMp>(a, rg, tmem_base, smem, b, abort_flag);
  }

  // every role is done; the drain threads have written their partials to the reduction buffer
  tc_fence_before();
  __syncthreads();
  float* red = reinterpret_cast<float*>(smem + L::kOffOp);  // [kMp][128]
  const uint32_t ch = (warp & 3u) * 32u + lane, hf = 0;
  // Fixed-order tree over the cluster: at step d, rank r (r % 2d == 0) adds rank r + d's buffer.
  for (int d = 1; d < a.split; d <<= 1) {
    cluster_sync_all();
    if (drain && (rank % (2u * d)) == 0 && rank + d < (uint32_t)a.split) {
      const uint32_t peer = mapa_shared(smem_u32(red), rank + d);
      float v[kH];
#pragma unroll
      for (int i = 0; i < kH; ++i)  // all loads first: one remote latency, not kH of them
        asm volatile("ld.shared::cluster.f32 %0, [%1];"
                     : "=f"(v[i])
                     : "r"(peer + (uint32_t)((hf * kH + i) * kRows + ch) * 4u));
#pragma unroll
      for (int i = 0; i < kH; ++i) red[(hf * kH + i) * kRows + ch] += v[i];
    }
  }
  cluster_sync_all();  // no CTA leaves while a peer may still read its buffer
  if (drain && rank == 0) {
    const int n = n0 + (int)ch;
    if (n < a.N) {
      const float bn = a.bias != nullptr ? __ldg(a.bias + n) : 0.0f;
      const float swn = a.groups == 1 ? __ldg(a.s_w + n) : 0.0f;
      for (int i = 0; i < kH; ++i) {
        const int m = (int)hf * kH + i;
        if (m >= a.M) break;
        float v = red[m * kRows + ch];
        if (a.groups == 1) {  // exact integer partial: scale once
          const float sa = __ldg(a.s_a + m), f = sa * kOperandUnitInv;
          v = f <= FLT_MAX ? (v * swn) * f : ((v * kOperandUnitInv) * sa) * swn;
        }
        a.y[(int64_t)m * a.N + n] = __float2bfloat16_rn(v + bn);
      }
    }
  }
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem_base, L::kTmemCols);
  }
}

template <int kMp>
cudaLaunchConfig_t make_config(int grid, int split, cudaStream_t stream, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = Layout<kMp>::kSmemBytes;
  cfg.stream = stream;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = split;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

// The split (CTAs per cluster) for `tiles` channel tiles: the largest one up to kMaxSplit, and
// up to the K stages, for which every cluster is resident at once (one wave) and the CTAs do
// not outnumber the SMs.  Cluster residency is asked of the runtime once per size.
template <int kMp>
int choose_split(int tiles, int k_stages, int sms) {
  static int max_clusters[kMaxSplit + 1] = {0};
  static bool probed = false;
  if (!probed) {
    probed = true;
    for (int s = 1; s <= kMaxSplit; ++s) {
      cudaLaunchAttribute attr[1];
      cudaLaunchConfig_t cfg = make_config<kMp>(s * (sms / s), s, nullptr, attr);
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, w4a4_skinny_kernel<kMp>, &cfg) != cudaSuccess) {
        (void)cudaGetLastError();
        n = 0;
      }
      max_clusters[s] = n;
    }
  }
  int best = 1;
  for (int s = 2; s <= kMaxSplit && s <= k_stages; ++s)
    if (tiles * s <= sms && tiles <= max_clusters[s]) best = s;
  return best;
}

template <int kMp>
cudaError_t launch_mp(SkArgs a, const SkinnyProblem& p, int tiles, int sms, cudaStream_t stream) {
  using L = Layout<kMp>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(w4a4_skinny_kernel<kMp>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)L::kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  // Packed codes as byte matrices: weights [N, K/2], tokens [M, K/2]; one box = 128 packed bytes
  // (two K stages) x 128 weight rows or x kMp token rows, 128-byte swizzle.  Rows past N or M
  // and columns past K/2 read zeros.
  CUtensorMap tmW, tmX;
  if (!encode_2d(&tmW, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.qw, p.K / 2, p.N, p.K / 2, kBK, kRows,
                 CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_2d(&tmX, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.q, p.K / 2, p.M, p.K / 2, kBK, kMp, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  a.split = choose_split<kMp>(tiles, a.k_stages, sms);
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_config<kMp>(tiles * a.split, a.split, stream, attr);
  return cudaLaunchKernelEx(&cfg, w4a4_skinny_kernel<kMp>, tmW, tmX, a);
}

}  // namespace

cudaError_t launch_w4a4_skinny(const SkinnyProblem& p, cudaStream_t stream, int sms) {
  if (p.M <= 0 || p.N <= 0) return cudaSuccess;
  if (p.M > kSkinnyMaxM) return cudaErrorInvalidValue;
  SkArgs a;
  a.M = p.M;
  a.N = p.N;
  a.K = p.K;
  a.G = p.G;
  a.groups = p.K / p.G;
  a.k_stages = p.K / kBK;
  a.split = 1;
  a.s_a = p.s_a;
  a.s_w = p.s_w;
  a.bias = p.bias;
  a.y = static_cast<__nv_bfloat16*>(p.y);
  a.status = p.status;
  const int tiles = (p.N + kRows - 1) / kRows;
  if (p.M <= 16) return launch_mp<16>(a, p, tiles, sms, stream);
  if (p.M <= 32) return launch_mp<32>(a, p, tiles, sms, stream);
  return launch_mp<64>(a, p, tiles, sms, stream);
}

}  // namespace jq
