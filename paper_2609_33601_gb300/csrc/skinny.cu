// skinny.cu -- the W4A4 linear layer for few tokens (M <= 64), where the layer is bound by
// streaming the packed weights from HBM rather than by the tensor core.
//
// Same arithmetic as gemm.cu (Sec. 1, Appendix FAQ Q7): acc[m,n,g] = sum_{k in g} qa*qw exactly
// (E4M3 operand bytes through tcgen05.mma kind::f8f6f4, operand.cuh), y = sum_g acc*s_a*s_w +
// bias in fp32, rounded to bf16.  The weights enter the MMA as offset codes qw + 8 (three ALU
// operations per 8 codes instead of ten); the MMA's sum (qw + 8) qa less 8 sum qa, formed
// exactly from the activation codes, is acc.  The shape of the work is different:
//   - the operands are swapped: each CTA unpacks 128 output channels of the weights into the
//     MMA's M operand and the (at most 64) tokens are its N operand, so the MMA, the TMEM
//     accumulators and the drain all scale with the real token count;
//   - packed weight and activation codes stream in by TMA (two K stages per box, 128-byte
//     swizzle) into a ring in shared memory: the TMA unit keeps far more bytes in flight per SM
//     than per-thread loads, which is what a weight-streaming kernel needs;
//   - the unpacked weight operand goes to tensor memory (tcgen05.st), and the MMA reads its A
//     operand from there: a weight byte then crosses shared memory twice (the TMA write and the
//     unpack's load of the packed code, half a byte each) instead of three times more for the
//     operand's store and the tensor core's read, which would make shared-memory bandwidth, not
//     HBM, the limit;
//   - no workspace and no separate activation expansion;
//   - K is split across the CTAs of a cluster (up to 8) so that enough SMs stream weights; the
//     partial outputs are summed through distributed shared memory in a fixed tree order, so
//     the result does not depend on timing.  For G = K (one group) the CTAs sum exact integer
//     partials and scale once; otherwise each CTA scales its whole groups and the fp32 partial
//     outputs are summed (the order of the fp32 sum over groups is free).
// CTA layout, 16 warps:
//   warps 0, 3  MMA issuers (one thread each) of the even / odd packed slots, each into its own
//               accumulators: one issuing thread keeps the tensor core barely one MMA ahead, two
//               keep it fed; 4 x (128 x Mp x 32) MMAs per K stage.  Warp 0 owns TMEM.
//   warp 1      activation scales: s_a of every group into a ring for the drain (with the
//               corrections, when the tokens come pre-expanded); first, the final pass's
//               per-token operands into shared memory
//   warp 2      barrier setup, then TMA producer (one thread): it issues the first pass of
//               weight boxes before the CTA-wide setup barrier; per two K stages, one box of 128
//               weight rows (128 packed bytes of INT4 codes, or 64 of 2-bit ternary codes) and
//               one of the Mp token rows (128 packed bytes), or, for more than 16 tokens, the
//               tokens' pre-expanded operand bytes straight into the operand ring
//   warps 4-11  unpack, two groups of four warps on alternate packed slots (two K stages each,
//               so that one round of waits and fences covers 32 KB of weight operand): thread =
//               weight row (TMEM lane), packed codes -> E4M3 operand bytes in the TMEM A ring;
//               up to 16 tokens also the token rows -> E4M3 operand rows (128B swizzle) in
//               shared memory, and each token group's exact code sum (for the drain)
//   warps 12-15 drain: per group, tcgen05.ld 32x32b (thread = output channel, every token
//               column), y[m] += (acc * s_w) * (s_a[m] * 2^18); for one-group problems they
//               unpack as a third group first
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
constexpr int kOpSlots = 4;      // operand ring (slots of two stages): weights in TMEM, tokens in shared memory
constexpr int kThreads = 512;
constexpr int kWarpMma = 0, kWarpScale = 1, kWarpTma = 2, kWarpMma1 = 3;  // MMA issuers of even / odd slots
constexpr int kUnpackWarp0 = 4, kUnpackGroups = 2, kUnpackGroupThreads = 128;
constexpr int kUnpackGroupWarps = kUnpackGroupThreads / 32;
constexpr int kDrainWarp0 = 12, kNumDrainWarps = 4;
constexpr int kSaRing = 32;  // activation-scale ring (groups)
// Register split per warpgroup while the roles run (totals the 512 x 128 registers of the launch):
// warps 0-3 (MMA issuers, scales, TMA) 80, unpack 128, drain 176; with 64 tokens the drain's 64
// running sums take 8 more from warps 0-3.  Every warpgroup returns to 128 for the reduction
// that all warps take part in.
constexpr int kRegsUnpack = 128, kRegsLaunch = 128;
template <int kMp>
constexpr int kRegsCtl = kMp == 64 ? 72 : 80;
template <int kMp>
constexpr int kRegsDrain = kMp == 64 ? 184 : 176;
static_assert(kRegsCtl<64> + 2 * kRegsUnpack + kRegsDrain<64> == 4 * kRegsLaunch &&
                  kRegsCtl<32> + 2 * kRegsUnpack + kRegsDrain<32> == 4 * kRegsLaunch,
              "register split must use the launch budget");
constexpr int kMaxSplit = 8;
constexpr int kMinSplitSlots = 6;  // K ring slots (two stages each) a CTA keeps at the least
static_assert(kDrainWarp0 % 4 == 0, "drain warp w reads TMEM lanes 32 * (w % 4)");
static_assert(kSkinnyMaxKOneGroup <= kOffsetMaxRun && kSkinnyMaxKOneGroup % kBK == 0, "exact one-group ranges");

template <int kMp>
struct Layout {
  static constexpr int kPkSlots = kMp == 64 ? 6 : 8;      // packed ring (slots of two stages)
  static constexpr uint32_t kPkW = kRows * kBK;           // packed weights of a slot: 128 rows x 128 B
  static constexpr uint32_t kPkX = kMp * kBK;             // packed tokens of a slot: kMp rows x 128 B
  static constexpr uint32_t kPkSlot = kPkW + kPkX;
  static constexpr uint32_t kOpB = kMp * kBK;             // token operand bytes of a stage
  static constexpr uint32_t kOpSlot = kStPerSlot * kOpB;  // the two stages of a slot, one after the other
  static constexpr uint32_t kOffPk = 0;
  static constexpr uint32_t kOffOp = kOffPk + kPkSlots * kPkSlot;
  // scale ring: per group and token the pair (s_a * 2^18 -- or s_a where that overflows --,
  // 8 sum qa in 2^-18 units) [kSaRing][kMp], then one flag per group (1: s_a * 2^18 is finite)
  static constexpr uint32_t kOffSa = kOffOp + kOpSlots * kOpSlot;
  static constexpr uint32_t kOffSaFlag = kOffSa + 2 * kSaRing * kMp * 4;
  static constexpr uint32_t kOffCorr = kOffSaFlag + kSaRing * 4;  // G = K: 8 sum qa per unpack group [3][kMp]
  // the final pass's per-token operands (G = K), staged by the scale warp at the start: the
  // scale and the whole-K correction [2][kMp]
  static constexpr uint32_t kOffFin = kOffCorr + (kUnpackGroups + 1) * kMp * 4;
  static constexpr uint32_t kOffBar = kOffFin + 2 * kMp * 4;
  static constexpr uint32_t kNumBars = 2 * kPkSlots + 3 * kOpSlots + 8 + 2 + 2 * kSaRing + 1;
  static constexpr uint32_t kOffMisc = kOffBar + kNumBars * 8;
  static constexpr uint32_t kSmemBytes = kOffMisc + 16;
  static constexpr uint32_t kRedBytes = kMp * kRows * 4;  // fp32 partials [kMp][128], reuse the packed ring
  // TMEM columns: four fp32 accumulators of kMp columns at 0 (issuer e, buffer ab at column
  // (2e + ab) kMp), the weight operand ring at kACol0 (a stage of 128 E4M3 bytes per lane is 32
  // columns, a slot 64)
  static constexpr uint32_t kACol0 = 256, kAStageCols = kBK / 4, kASlotCols = kStPerSlot * kAStageCols;
  static constexpr uint32_t kTmemCols = 512;
  static_assert(4 * kMp <= kACol0 && kACol0 + kOpSlots * kASlotCols <= kTmemCols, "TMEM columns");
  static_assert(kPkW % 1024 == 0 && kPkX % 1024 == 0 && kOpB % 1024 == 0,
                "128B-swizzle atoms need 1024-byte alignment");
  static_assert(kOffSa % 16 == 0 && kOffBar % 8 == 0, "alignment");
  static_assert(kRedBytes <= kPkSlots * kPkSlot, "the reduction buffer reuses the packed ring");
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
  int image;          // token operand from the pre-expanded A-operand image (see tma_role)
  int ternary;        // 2-bit ternary weights (ternary.cu) instead of 4-bit INT4 codes
  const float* corr;  // image mode: [M, K/G] 8 * the group's activation code sum, 2^-18 units
};

struct SkBars {
  uint64_t *pk_full, *pk_empty;  // packed ring
  uint64_t *op_full, *op_empty;  // operand ring
  uint64_t *acc_full, *acc_empty, *mma_done;  // [2 issuers x 2 buffers], [2 issuers]
  uint64_t *sa_full, *sa_empty;  // activation-scale ring
  uint64_t* corr_full;           // G = K: the range's code sums are in place
  uint64_t* tk_full;             // image mode: the token operand of an operand-ring slot has landed
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


// ------------------------------------------------------------------ TMA producer
template <int kMp>
__device__ __forceinline__ int tma_pre_slots(const Range& rg) {
  const int nslots = (rg.nst + kStPerSlot - 1) / kStPerSlot;
  return nslots < Layout<kMp>::kPkSlots ? nslots : Layout<kMp>::kPkSlots;
}
// packed weight bytes per K stage and per slot (2-bit ternary codes fill half the weight area)
__device__ __forceinline__ int weight_stage_bytes(const SkArgs& a) { return a.ternary ? kBK / 4 : kBK / 2; }

// The weight boxes of the packed ring's first pass (a fresh ring: every slot is free).
template <int kMp>
__device__ __forceinline__ void tma_first_weights(const SkArgs& a, const Range& rg, int n0, const CUtensorMap* tmW,
                                                  uint8_t* smem, const SkBars& b) {
  using L = Layout<kMp>;
  const int wst = weight_stage_bytes(a);
  const uint32_t wslot = a.ternary ? L::kPkW / 2 : L::kPkW;
  const uint32_t wbytes = a.image ? wslot : wslot + L::kPkX;
  for (int j = 0; j < tma_pre_slots<kMp>(rg); ++j) {
    mbar_arrive_expect_tx(&b.pk_full[j], wbytes);
    tma_load_2d(smem + L::kOffPk + (uint32_t)j * L::kPkSlot, tmW, &b.pk_full[j], (rg.st0 + j * kStPerSlot) * wst,
                n0);
  }
}

template <int kMp>
__device__ __forceinline__ void tma_role(const SkArgs& a, const Range& rg, int n0, const CUtensorMap* tmW,
                                         const CUtensorMap* tmX, uint8_t* smem, const SkBars& b,
                                         volatile int* abort_flag) {
  using L = Layout<kMp>;
  constexpr int kPkSlots = L::kPkSlots;
  const int nslots = (rg.nst + kStPerSlot - 1) / kStPerSlot;
  // The weight boxes of the first pass went out during setup (tma_first_weights): they do not
  // depend on the previous kernel in the stream (programmatic launch, ptx.cuh); the token boxes
  // and everything after wait for it.
  const int pre = tma_pre_slots<kMp>(rg);
  const int wst = weight_stage_bytes(a);
  const uint32_t wslot = a.ternary ? L::kPkW / 2 : L::kPkW;
  const uint32_t wbytes = a.image ? wslot : wslot + L::kPkX;
  pdl_wait();
  int jt = 0, jw = pre;  // token slots issued (image mode), weight slots issued
  if (!a.image) {
    for (int j = 0; j < pre; ++j)
      tma_load_2d(smem + L::kOffPk + (uint32_t)j * L::kPkSlot + L::kPkW, tmX, &b.pk_full[j],
                  (rg.st0 + j * kStPerSlot) * (kBK / 2), 0);
    for (; jw < nslots; ++jw) {
      const uint32_t s = (uint32_t)jw % kPkSlots;
      if (!mbar_wait(&b.pk_empty[s], ring_parity(jw, kPkSlots) ^ 1u, abort_flag, a.status)) break;
      uint8_t* slot = smem + L::kOffPk + s * L::kPkSlot;
      const int st = rg.st0 + jw * kStPerSlot;  // first K stage of the slot
      mbar_arrive_expect_tx(&b.pk_full[s], wbytes);
      tma_load_2d(slot, tmW, &b.pk_full[s], st * wst, n0);
      tma_load_2d(slot + L::kPkW, tmX, &b.pk_full[s], st * (kBK / 2), 0);
    }
  } else {
    // Image mode: the tokens arrive as operand bytes (the A-operand image of the GEMM path: per
    // K stage a 128-row block in the 128-byte swizzle, of which the first kMp rows are a stage of
    // this kernel's token operand) and go straight into the operand ring, completing on tk_full;
    // the weights keep streaming into the packed ring.  The two rings advance at different paces
    // (the operand ring frees a slot only when its MMAs are done), so this thread polls both
    // instead of blocking on either.
    long long t0 = clock64();
    while (jw < nslots || jt < nslots) {
      bool moved = false;
      if (jt < nslots) {
        const uint32_t os = (uint32_t)jt % kOpSlots;
        if (mbar_test_wait(&b.op_empty[os], ring_parity(jt, kOpSlots) ^ 1u)) {
          const int nst_j = rg.nst - jt * kStPerSlot < kStPerSlot ? rg.nst - jt * kStPerSlot : kStPerSlot;
          uint8_t* dst = smem + L::kOffOp + os * L::kOpSlot;
          mbar_arrive_expect_tx(&b.tk_full[os], (uint32_t)nst_j * L::kOpB);
          for (int h = 0; h < nst_j; ++h)
            tma_load_2d(dst + (uint32_t)h * L::kOpB, tmX, &b.tk_full[os], 0, (rg.st0 + jt * kStPerSlot + h) * kBK);
          ++jt;
          moved = true;
        }
      }
      if (jw < nslots) {
        const uint32_t s = (uint32_t)jw % kPkSlots;
        if (mbar_test_wait(&b.pk_empty[s], ring_parity(jw, kPkSlots) ^ 1u)) {
          mbar_arrive_expect_tx(&b.pk_full[s], wbytes);
          tma_load_2d(smem + L::kOffPk + s * L::kPkSlot, tmW, &b.pk_full[s], (rg.st0 + jw * kStPerSlot) * wst, n0);
          ++jw;
          moved = true;
        }
      }
      if (moved) {
        t0 = clock64();
        continue;
      }
      __nanosleep(32);  // leave the issue slots to the unpack warps of this SM sub-partition
      if (*abort_flag) break;
      if (clock64() - t0 > (1ll << 31)) {  // bounded, like every other wait here
        *abort_flag = 1;
        if (a.status) atomicExch(a.status, (uint32_t)kDevTimeout);
        break;
      }
    }
  }
  // let the last copies land before the CTA can leave
  for (int j = jw > kPkSlots ? jw - kPkSlots : 0; j < jw; ++j) {
    int dummy = 0;
    mbar_wait(&b.pk_full[j % kPkSlots], ring_parity(j, kPkSlots), &dummy, a.status);
  }
  for (int j = jt > kOpSlots ? jt - kOpSlots : 0; j < jt; ++j) {  // image mode: the token copies
    int dummy = 0;
    mbar_wait(&b.tk_full[j % kOpSlots], ring_parity(j, kOpSlots), &dummy, a.status);
  }
}

// ------------------------------------------------------------------ unpack
// Group ug (of ngroups: 2, or 3 for G = K where the drain warps join in while they have nothing
// to drain) converts packed slots j = ug, ug + ngroups, ...: both K stages of the slot.
// Code sums: the 8 chunks of a token row sit in 8 consecutive lanes, so a group's sum (2 chunks
// for G = 64, 4 for G = 128, all 8 and then all slots for G = K) is a butterfly over 1-3 lanes.
// The drain removes 8 * sum qa, in the accumulator's units (2^-18), from the offset-code MMA;
// G < K: into the scale ring next to s_a (a ring slot is full once the scale warp and the
// group's four warps have written it); G = K: per unpack group, handed over at the end.
// Weights: thread u is weight row u, the TMEM lane its warp may write; its 256 offset operand
// bytes go to 64 columns of the A ring by two tcgen05.st.  Tokens: thread u takes packed chunks
// t = u + 128 i of the token tile, row t / 8, chunk t % 8 (stage (t % 8) / 4), and stores
// each as two operand chunks into the shared-memory operand ring.
template <int kMp>
__device__ __forceinline__ void unpack_role(const SkArgs& a, const Range& rg, uint8_t* smem, uint32_t tmem_base,
                                            const SkBars& b, int ngroups, volatile int* abort_flag) {
  using L = Layout<kMp>;
  constexpr int kPkSlots = L::kPkSlots;
  constexpr int kXChunks = kMp * 8 / kUnpackGroupThreads;  // token chunks per thread per slot
  static_assert(kUnpackWarp0 % 4 == 0 && kUnpackGroupThreads == kRows, "thread u of a group is TMEM lane u");
  static_assert(kMp * 8 % kUnpackGroupThreads == 0, "token chunks divide evenly");
  const uint32_t ut = threadIdx.x - kUnpackWarp0 * 32;
  const uint32_t ug = ut / kUnpackGroupThreads, u = ut % kUnpackGroupThreads;
  const uint32_t r7 = u & 7u;
  const uint32_t a_lane = tmem_base + ((u & ~31u) << 16) + L::kACol0;
  const int nslots = (rg.nst + kStPerSlot - 1) / kStPerSlot;
  const bool single = a.groups == 1;
  const int gpst = groups_per_stage(a), gps = kStPerSlot * gpst;
  const uint32_t c8 = u & 7u;  // the chunk of its token row this thread holds
  float* sc_ring = reinterpret_cast<float*>(smem + L::kOffSa);  // pairs (s_a', c): c is the second
  const int woff = a.ternary ? 1 : 8;  // the weights' operand offset: the correction is woff * sum qa
  int tot[kXChunks];  // G = K: running code sums of this thread's token rows
#pragma unroll
  for (int i = 0; i < kXChunks; ++i) tot[i] = 0;
  for (int j = (int)ug; j < nslots; j += ngroups) {
    const int nst_j = rg.nst - j * kStPerSlot < kStPerSlot ? rg.nst - j * kStPerSlot : kStPerSlot;
    const uint32_t p = (uint32_t)j % kPkSlots, os = (uint32_t)j % kOpSlots;
    if (!__all_sync(0xffffffffu, mbar_wait(&b.pk_full[p], ring_parity(j, kPkSlots), abort_flag, a.status))) return;
    if (!__all_sync(0xffffffffu, mbar_wait(&b.op_empty[os], ring_parity(j, kOpSlots) ^ 1u, abort_flag, a.status)))
      return;
    tc_fence_after();  // the MMAs that read this A slot have finished
    const uint32_t src = smem_u32(smem + L::kOffPk + p * L::kPkSlot);
    const uint32_t dst = smem_u32(smem + L::kOffOp + os * L::kOpSlot);
    // loads in batches ahead of their use: the shared-memory accessors are ordered, so
    // interleaving loads with stores would expose a load latency per chunk.  A quarter-warp reads
    // 8 consecutive rows at one logical chunk (weights) or the 8 chunks of one row (tokens): 8
    // distinct physical chunks.
    uint4 px[kXChunks];
    if (!a.ternary) {
      uint4 pw[8];
      const uint32_t wrow = sw128_row(src, u);
#pragma unroll
      for (int c = 0; c < 8; ++c) pw[c] = ld_shared_v4(wrow + (((uint32_t)c ^ r7) << 4));
#pragma unroll
      for (int h = 0; h < kStPerSlot; ++h) {
        uint32_t v[32];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint4 lo, hi;
          nib32_to_operand_offset(pw[4 * h + c], lo, hi);
          v[8 * c + 0] = lo.x; v[8 * c + 1] = lo.y; v[8 * c + 2] = lo.z; v[8 * c + 3] = lo.w;
          v[8 * c + 4] = hi.x; v[8 * c + 5] = hi.y; v[8 * c + 6] = hi.z; v[8 * c + 7] = hi.w;
        }
        tmem_st32(a_lane + os * L::kASlotCols + (uint32_t)h * L::kAStageCols, v);
      }
    } else {
      // 2-bit ternary weights: 64 packed bytes per row and slot, 64-byte swizzle (16-byte chunk c
      // of row r at chunk c ^ ((r / 2) % 4)); each 32-bit word is 16 codes, and its four 2-bit
      // planes are the operand bytes (q + 1) of elements {0,2,4,6}, {1,3,5,7}, {8,..,14}, {9,..,15}
      uint4 pw[4];
      const uint32_t wrow = src + u * 64u, sw = (u >> 1) & 3u;
#pragma unroll
      for (int c = 0; c < 4; ++c) pw[c] = ld_shared_v4(wrow + (((uint32_t)c ^ sw) << 4));
#pragma unroll
      for (int h = 0; h < kStPerSlot; ++h) {
        uint32_t v[32];
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const uint32_t wd[4] = {pw[2 * h + c].x, pw[2 * h + c].y, pw[2 * h + c].z, pw[2 * h + c].w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
#pragma unroll
            for (int k = 0; k < 4; ++k) v[16 * c + 4 * i + k] = (wd[i] >> (2 * k)) & 0x03030303u;
          }
        }
        tmem_st32(a_lane + os * L::kASlotCols + (uint32_t)h * L::kAStageCols, v);
      }
    }
    // token rows: only the M real ones (rows >= M stay zero in the operand ring); in image mode
    // the producer has copied them as operand bytes and the corrections come from global memory
    const uint32_t mx = a.image ? 0u : (uint32_t)a.M;
#pragma unroll
    for (int i = 0; i < kXChunks; ++i) {
      const uint32_t t = u + kUnpackGroupThreads * i, r = t >> 3;
      px[i] = r < mx ? ld_shared_v4(sw128_row(src + L::kPkW, r) + (((t & 7u) ^ (r & 7u)) << 4))
                     : make_uint4(0x88888888u, 0x88888888u, 0x88888888u, 0x88888888u);
    }
    int xs[kXChunks];  // code sums of the token chunks (chunks of a stage past the range count 0)
#pragma unroll
    for (int i = 0; i < kXChunks; ++i) {
      const uint32_t r = (u + kUnpackGroupThreads * (uint32_t)i) >> 3;
      xs[i] = (r < mx && c8 < 4u * (uint32_t)nst_j) ? nib32_sum(px[i]) : 0;
    }
#pragma unroll
    for (int i = 0; i < kXChunks; ++i) {
      const uint32_t t = u + kUnpackGroupThreads * i, r = t >> 3, h = (t >> 2) & 1u, jc = t & 3u;
      if (r >= mx) continue;
      uint4 lo, hi;
      nib32_to_operand(px[i], lo, hi);
      const uint32_t row_base = sw128_row(dst + h * L::kOpB, r), rr = r & 7u;
      const uint32_t c_lo = (2u * jc) ^ rr, c_hi = (2u * jc + 1u) ^ rr;
      // the two stage tiles sit a multiple of 128 bytes apart (same banks): the stage-1 half of
      // the quarter-warp stores its chunks in the other order
      if (h) {
        st_shared_v4(row_base + (c_hi << 4), hi.x, hi.y, hi.z, hi.w);
        st_shared_v4(row_base + (c_lo << 4), lo.x, lo.y, lo.z, lo.w);
      } else {
        st_shared_v4(row_base + (c_lo << 4), lo.x, lo.y, lo.z, lo.w);
        st_shared_v4(row_base + (c_hi << 4), hi.x, hi.y, hi.z, hi.w);
      }
    }
    tmem_st_wait();
    fence_proxy_async_smem();
    tc_fence_before();
    __syncwarp();
    if ((u & 31u) == 0) {
      mbar_arrive(&b.op_full[os]);
      mbar_arrive(&b.pk_empty[p]);
    }
    if (a.image) continue;
    // group sums: lanes whose chunk opens a group hold that group's sum after the butterfly
#pragma unroll
    for (int i = 0; i < kXChunks; ++i) {
      xs[i] += __shfl_xor_sync(0xffffffffu, xs[i], 1);
      if (gpst == 1) xs[i] += __shfl_xor_sync(0xffffffffu, xs[i], 2);
      if (single) {
        xs[i] += __shfl_xor_sync(0xffffffffu, xs[i], 4);
        tot[i] += xs[i];
      }
    }
    if (single) continue;
    const int cpg = 4 / gpst;  // chunks per group
    for (int q = 0; q < nst_j * gpst; ++q) {
      const int gi = j * gps + q;
      const uint32_t so = (uint32_t)gi % kSaRing;
      if (!__all_sync(0xffffffffu, mbar_wait(&b.sa_empty[so], ring_parity(gi, kSaRing) ^ 1u, abort_flag, a.status)))
        return;
#pragma unroll
      for (int i = 0; i < kXChunks; ++i) {
        const uint32_t r = (u + kUnpackGroupThreads * (uint32_t)i) >> 3;
        if (c8 == (uint32_t)(q * cpg)) sc_ring[2 * (so * kMp + r) + 1] = (float)(woff * xs[i]) * kOperandUnit;
      }
      __syncwarp();
      if ((u & 31u) == 0) mbar_arrive(&b.sa_full[so]);
    }
  }
  if (single && !a.image) {  // this group's share of the range's code sums (zero if it had no slot)
    float* corr = reinterpret_cast<float*>(smem + L::kOffCorr) + ug * kMp;
#pragma unroll
    for (int i = 0; i < kXChunks; ++i) {
      const uint32_t r = (u + kUnpackGroupThreads * (uint32_t)i) >> 3;
      if (c8 == 0u) corr[r] = (float)(woff * tot[i]) * kOperandUnit;
    }
    __syncwarp();
    if ((u & 31u) == 0) mbar_arrive(b.corr_full);
  }
}

// ------------------------------------------------------------------ activation scales
// One warp (lane m = token): the scales of this CTA's groups into the ring, kSaBatch groups per
// batch of loads so that one load latency covers several groups.  Rows >= M get 0.  Each group's
// s_a go in already multiplied by 2^18 unless that overflows for one of them (|s_a| > 2^110),
// with a flag saying which, so the drain neither re-checks nor re-scales.  A ring slot is full
// once this warp and the unpack warps (the code sums) have written it.
template <int kMp>
__device__ __forceinline__ void scale_role(const SkArgs& a, const Range& rg, uint8_t* smem, const SkBars& b,
                                           volatile int* abort_flag) {
  using L = Layout<kMp>;
  constexpr int kPer = kMp > 32 ? kMp / 32 : 1;  // tokens per lane
  constexpr int kSaBatch = 8;
  const uint32_t lane = lane_id();
  float* sc_ring = reinterpret_cast<float*>(smem + L::kOffSa);  // pairs (s_a', c): s_a' is the first
  int* flags = reinterpret_cast<int*>(smem + L::kOffSaFlag);
  const int ng = drain_groups(a, rg);
  {
    // The final pass's per-token operands, fetched at the start: under the weight stream a
    // global load takes microseconds, which the final pass would otherwise wait for after the
    // last MMA.  (Read after the CTA barrier that precedes the reduction.)
    float* fin = reinterpret_cast<float*>(smem + L::kOffFin);
    for (int m = (int)lane; m < kMp; m += 32) {
      const bool in = a.groups == 1 && m < a.M;
      fin[m] = in ? __ldg(a.s_a + m) : 0.0f;
      // whole-K correction (image mode): 8 sum qa, or sum qa for ternary weights (offset 1)
      fin[kMp + m] = (in && a.image) ? __ldg(a.corr + m) * (a.ternary ? 0.125f : 1.0f) : 0.0f;
    }
  }
  if (ng == 0 || a.groups == 1) return;  // G = K: no per-group scales
  const int g0 = rg.st0 * groups_per_stage(a);
  for (int gb = 0; gb < ng; gb += kSaBatch) {
    const int nb = ng - gb < kSaBatch ? ng - gb : kSaBatch;
    float v[kSaBatch][kPer], cv[kSaBatch][kPer];
#pragma unroll
    for (int j = 0; j < kSaBatch; ++j) {
#pragma unroll
      for (int h = 0; h < kPer; ++h) {
        const int m = (int)lane + 32 * h;
        const bool in = j < nb && m < kMp && m < a.M;
        v[j][h] = in ? __ldg(a.s_a + (int64_t)m * a.groups + g0 + gb + j) : 0.0f;
        cv[j][h] = (in && a.image) ? __ldg(a.corr + (int64_t)m * a.groups + g0 + gb + j) : 0.0f;
      }
    }
#pragma unroll
    for (int j = 0; j < kSaBatch; ++j) {
      if (j >= nb) break;
      const uint32_t it = (uint32_t)(gb + j), o = it % kSaRing;
      if (!__all_sync(0xffffffffu, mbar_wait(&b.sa_empty[o], ring_parity(it, kSaRing) ^ 1u, abort_flag, a.status)))
        return;
      bool finite = true;
#pragma unroll
      for (int h = 0; h < kPer; ++h) finite = finite && fabsf(v[j][h]) * kOperandUnitInv <= FLT_MAX;
      finite = __all_sync(0xffffffffu, finite);
#pragma unroll
      for (int h = 0; h < kPer; ++h) {
        const int m = (int)lane + 32 * h;
        if (m < kMp) sc_ring[2 * (o * kMp + m)] = finite ? v[j][h] * kOperandUnitInv : v[j][h];
        // 8 sum qa in 2^-18 units; ternary weights are offset by 1, not 8: sum qa (exact)
        if (m < kMp && a.image) sc_ring[2 * (o * kMp + m) + 1] = a.ternary ? cv[j][h] * 0.125f : cv[j][h];
      }
      if (lane == 0) flags[o] = finite ? 1 : 0;
      __syncwarp();
      if (lane == 0) mbar_arrive(&b.sa_full[o]);
    }
  }
}

// ------------------------------------------------------------------ MMA issuer
// The tensor core accepts the next MMA only about one instruction ahead, so anything the issuing
// thread executes between two MMAs (a branch, address arithmetic) leaves the pipe idle: each
// slot's operand addresses are computed before its MMAs, which then issue straight-line, and the
// group layout is a template parameter rather than a branch.
//   kGroups = 0: one group over all of K (G = K), one accumulator for the CTA's whole range;
//   kGroups = 1: one group per K stage (G = 128);  kGroups = 2: two groups per stage (G = 64).
template <int kMp, int kGroups>
__device__ __forceinline__ void mma_role(const SkArgs& a, const Range& rg, uint32_t e, uint32_t tmem_base,
                                         uint8_t* smem, const SkBars& b, volatile int* abort_flag) {
  using L = Layout<kMp>;
  const uint32_t idesc = idesc_e4m3_f32(kRows, kMp);
  const uint32_t a_tmem0 = tmem_base + L::kACol0;
  const uint64_t bdesc0 = sdesc_kmajor_sw128(smem_u32(smem + L::kOffOp));
  uint32_t chunk_it = 0, d_tmem = tmem_base;  // this issuer's accumulators, in order
  auto open_acc = [&]() -> bool {
    const uint32_t idx = 2u * e + (chunk_it & 1u);
    if (!mbar_wait(&b.acc_empty[idx], ((chunk_it >> 1) & 1u) ^ 1u, abort_flag, a.status)) return false;
    tc_fence_after();
    d_tmem = tmem_base + idx * kMp;
    return true;
  };
  auto close_acc = [&]() {
    umma_commit(&b.acc_full[2u * e + (chunk_it & 1u)]);
    ++chunk_it;
  };
  // the four K slices of one stage: A columns +8, B descriptor +2 (32 bytes) per slice
  auto stage4 = [&](uint32_t ad, uint64_t bd, uint32_t acc_first) {
    umma_f8f6f4_ts(d_tmem, ad, bd, idesc, acc_first);
    umma_f8f6f4_ts(d_tmem, ad + 8u, bd + 2u, idesc, 1u);
    umma_f8f6f4_ts(d_tmem, ad + 16u, bd + 4u, idesc, 1u);
    umma_f8f6f4_ts(d_tmem, ad + 24u, bd + 6u, idesc, 1u);
  };
  const int nslots = (rg.nst + kStPerSlot - 1) / kStPerSlot;
  bool ok = (int)e < nslots && (kGroups != 0 || open_acc());
  for (int j = (int)e; ok && j < nslots; j += 2) {
    const uint32_t os = (uint32_t)j % kOpSlots;
    const uint32_t ad0 = a_tmem0 + os * L::kASlotCols, ad1 = ad0 + L::kAStageCols;
    const uint64_t bd0 = bdesc0 + ((os * L::kOpSlot) >> 4), bd1 = bd0 + (L::kOpB >> 4);
    const bool both = j * kStPerSlot + 1 < rg.nst;  // false only for the last slot of an odd range
    if (!(ok = mbar_wait(&b.op_full[os], ring_parity(j, kOpSlots), abort_flag, a.status))) break;
    if (a.image && !(ok = mbar_wait(&b.tk_full[os], ring_parity(j, kOpSlots), abort_flag, a.status))) break;
    tc_fence_after();  // the unpack's tcgen05.st of this A slot is complete
    if (kGroups == 0) {
      const uint32_t acc0 = j > (int)e ? 1u : 0u;
      if (both) {
        stage4(ad0, bd0, acc0);
        stage4(ad1, bd1, 1u);
      } else {
        stage4(ad0, bd0, acc0);
      }
    } else if (kGroups == 1) {
      if (!(ok = open_acc())) break;
      stage4(ad0, bd0, 0u);
      close_acc();
      if (both) {
        if (!(ok = open_acc())) break;
        stage4(ad1, bd1, 0u);
        close_acc();
      }
    } else {
#pragma unroll
      for (int h = 0; h < kStPerSlot; ++h) {
        if (h == 1 && !both) break;
        const uint32_t ad = h ? ad1 : ad0;
        const uint64_t bd = h ? bd1 : bd0;
        if (!(ok = open_acc())) break;
        umma_f8f6f4_ts(d_tmem, ad, bd, idesc, 0u);
        umma_f8f6f4_ts(d_tmem, ad + 8u, bd + 2u, idesc, 1u);
        close_acc();
        if (!(ok = open_acc())) break;
        umma_f8f6f4_ts(d_tmem, ad + 16u, bd + 4u, idesc, 0u);
        umma_f8f6f4_ts(d_tmem, ad + 24u, bd + 6u, idesc, 1u);
        close_acc();
      }
      if (!ok) break;
    }
    umma_commit(&b.op_empty[os]);
  }
  if (ok && kGroups == 0 && (int)e < nslots) close_acc();
  umma_commit(&b.mma_done[e]);
  int dummy = 0;
  mbar_wait(&b.mma_done[e], 0, &dummy, a.status);
}

// ------------------------------------------------------------------ drain
// Warp w: TMEM lanes 32 * (w % 4).. (output channels), every token column (kH = kMp of them;
// hf, the column-half index of a wider layout, is 0).  For G = K the accumulator is the exact
// integer partial of this CTA's K range and is kept unscaled.  At the end the partials go to
// the reduction buffer, which reuses the packed ring: the last group's accumulator being full
// means every MMA has finished, so every unpack has read its packed slot, and every TMA copy
// into the ring has landed (the unpack waited for each one).
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
  const float* sc_ring = reinterpret_cast<const float*>(smem + L::kOffSa);  // pairs (s_a', c)
  const int* flags = reinterpret_cast<const int*>(smem + L::kOffSaFlag);
  const int ng = drain_groups(a, rg);
  const int g0 = single ? 0 : rg.st0 * groups_per_stage(a);
  float y[kH];
#pragma unroll
  for (int i = 0; i < kH; ++i) y[i] = 0.0f;
  // G = K: both issuers hold a part of the one group (the second only if the range has more
  // than one slot), in their first accumulators.
  const int nslots = (rg.nst + kStPerSlot - 1) / kStPerSlot;
  const int gps = kStPerSlot * groups_per_stage(a);
  const int parts = single ? (nslots > 1 ? 2 : 1) : 1;
  if (single) {
    for (int it = 0; ng > 0 && it < parts; ++it) {
      const uint32_t ab = 2u * (uint32_t)it;  // issuer it's first accumulator
      const bool ok = mbar_wait(&b.acc_full[ab], 0, abort_flag, a.status);
      // warp-collective tcgen05.ld follows: the whole warp proceeds or none of it
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((quarter * 32u) << 16) + ab * kMp + hf * kH;
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
#pragma unroll
        for (int i = 0; i < 8; ++i) y[c * 8 + i] += __uint_as_float(r[i]);  // exact integer partials
      }
    }
  } else {
    // Two groups per round (one for Mp = 64, for registers): one round of waits and one TMEM
    // round trip for both.  Group gi was
    // accumulated by the issuer of its slot js (e = js % 2) as that issuer's chunk
    // (js / 2) * gps + gi % gps (gps = groups per slot); the position is stepped, not divided.
    int gq = 0, js = 0;
    auto next_acc = [&](uint32_t& ab, uint32_t& parity) {
      const uint32_t chunk = (uint32_t)(js >> 1) * (uint32_t)gps + (uint32_t)gq;
      ab = 2u * ((uint32_t)js & 1u) + (chunk & 1u);
      parity = (chunk >> 1) & 1u;
      if (++gq == gps) {
        gq = 0;
        ++js;
      }
    };
    float swa = (ng > 0 && n < a.N) ? __ldg(a.s_w + (int64_t)g0 * a.N + n) : 0.0f;
    constexpr int kPer = kMp <= 32 ? 2 : 1;  // groups per round
    float swb = (kPer == 2 && ng > 1 && n < a.N) ? __ldg(a.s_w + (int64_t)(g0 + 1) * a.N + n) : 0.0f;
    for (int gi = 0; gi < ng; gi += kPer) {
      const bool two = kPer == 2 && gi + 1 < ng;  // the same for every lane
      uint32_t ab0, p0, ab1 = 0, p1 = 0;
      next_acc(ab0, p0);
      if (two) next_acc(ab1, p1);
      const float sw0 = swa, sw1 = swb;  // and the next round's weight scales, a round early
      if (gi + kPer < ng && n < a.N) swa = __ldg(a.s_w + (int64_t)(g0 + gi + kPer) * a.N + n);
      if (kPer == 2 && gi + 3 < ng && n < a.N) swb = __ldg(a.s_w + (int64_t)(g0 + gi + 3) * a.N + n);
      const uint32_t so0 = (uint32_t)gi % kSaRing, so1 = (uint32_t)(gi + 1) % kSaRing;
      bool ok = mbar_wait(&b.sa_full[so0], ring_parity(gi, kSaRing), abort_flag, a.status);
      if (two) ok = ok && mbar_wait(&b.sa_full[so1], ring_parity(gi + 1, kSaRing), abort_flag, a.status);
      ok = ok && mbar_wait(&b.acc_full[ab0], p0, abort_flag, a.status);
      if (two) ok = ok && mbar_wait(&b.acc_full[ab1], p1, abort_flag, a.status);
      // warp-collective tcgen05.ld follows: the whole warp proceeds or none of it
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const uint32_t lanes = tmem_base + ((quarter * 32u) << 16) + hf * kH;
      const float* sc0 = sc_ring + 2 * (so0 * kMp + hf * kH);  // (s_a', c) of the groups' tokens
      const float* sc1 = sc_ring + 2 * (so1 * kMp + hf * kH);
      // the overflow-safe form is needed only if some s_a * 2^18 of a group overflows (the scale
      // warp's flags; the same for every lane, so no lane skips the warp-collective loads below)
      const bool finite = __all_sync(0xffffffffu, flags[so0] != 0 && (!two || flags[so1] != 0));
      auto accumulate = [&](const uint32_t (&r)[8], const float* scs, float sw, int c) {
        if (finite) {
#pragma unroll
          for (int i = 0; i < 8; i += 2) {
            const float4 sc = *reinterpret_cast<const float4*>(scs + 2 * (c * 8 + i));  // s_a'0, c0, s_a'1, c1
            // exact: both are integers below 2^24 (in units of 2^-18)
            const float2 d = make_float2(__uint_as_float(r[i]) - sc.y, __uint_as_float(r[i + 1]) - sc.w);
            const float2 t = __fmul2_rn(d, make_float2(sw, sw));
            const float2 v = __ffma2_rn(t, make_float2(sc.x, sc.z), make_float2(y[c * 8 + i], y[c * 8 + i + 1]));
            y[c * 8 + i] = v.x;
            y[c * 8 + i + 1] = v.y;
          }
        } else {  // |s_a| > 2^110 somewhere: apply 2^18 to the exact partials first
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float2 sc = *reinterpret_cast<const float2*>(scs + 2 * (c * 8 + i));  // s_a (unscaled), c
            y[c * 8 + i] = fmaf(((__uint_as_float(r[i]) - sc.y) * kOperandUnitInv) * sc.x, sw, y[c * 8 + i]);
          }
        }
      };
#pragma unroll
      for (int c = 0; c < kH / 8; ++c) {
        uint32_t r0[8], r1[8];
        tmem_ld8(lanes + ab0 * kMp + c * 8, r0);
        if (two) tmem_ld8(lanes + ab1 * kMp + c * 8, r1);
        tmem_ld_wait();
        if (c == kH / 8 - 1) {  // both accumulators are in registers: hand them back
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&b.acc_empty[ab0]);
            if (two) mbar_arrive(&b.acc_empty[ab1]);
          }
        }
        accumulate(r0, sc0, sw0, c);
        if (two) accumulate(r1, sc1, sw1, c);
      }
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&b.sa_empty[so0]);
        if (two) mbar_arrive(&b.sa_empty[so1]);
      }
    }
  }
  if (single && ng > 0 && !a.image) {  // the exact partial: the offset-code sum less 8 * the range's code sums
    const bool ok = mbar_wait(b.corr_full, 0, abort_flag, a.status);
    const float* corr = reinterpret_cast<const float*>(smem + L::kOffCorr);
#pragma unroll
    for (int i = 0; i < kH; ++i)  // the shares and the difference are exact integers (units 2^-18)
      y[i] = ok ? y[i] - (corr[hf * kH + i] + corr[kMp + hf * kH + i] + corr[2 * kMp + hf * kH + i]) : 0.0f;
  }
  float* red = reinterpret_cast<float*>(smem + L::kOffPk);  // [kMp][128]
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
  b.pk_empty = b.pk_full + L::kPkSlots;
  b.op_full = b.pk_empty + L::kPkSlots;
  b.op_empty = b.op_full + kOpSlots;
  b.acc_full = b.op_empty + kOpSlots;
  b.acc_empty = b.acc_full + 4;
  b.mma_done = b.acc_empty + 4;
  b.sa_full = b.mma_done + 2;
  b.sa_empty = b.sa_full + kSaRing;
  b.corr_full = b.sa_empty + kSaRing;
  b.tk_full = b.corr_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::kOffMisc + 4);

  const uint32_t rank = cluster_ctarank();
  const int n0 = (int)(blockIdx.x / a.split) * kRows;
  const Range rg = k_range(a, rank);
  const uint32_t warp = warp_id(), lane = lane_id();
  const bool single = a.groups == 1;
  const int ngroups = single ? kUnpackGroups + 1 : kUnpackGroups;  // G = K: the drain warps unpack too
  if (warp == kWarpTma) {  // barrier setup, spread over one warp: the TMA warp, which starts streaming right after
    if (lane == 0) *abort_flag = 0;
    for (int i = (int)lane; i < L::kPkSlots; i += 32) {
      mbar_init(&b.pk_full[i], 1);                   // the producer's expect_tx
      mbar_init(&b.pk_empty[i], kUnpackGroupWarps);  // the slot's unpack group
    }
    for (int i = (int)lane; i < kOpSlots; i += 32) {
      mbar_init(&b.op_full[i], kUnpackGroupWarps);  // the slot's unpack group
      mbar_init(&b.op_empty[i], 1);
      mbar_init(&b.tk_full[i], 1);  // image mode: the producer's expect_tx for the token operand
    }
    if (lane < 4) {
      mbar_init(&b.acc_full[lane], 1);
      mbar_init(&b.acc_empty[lane], kNumDrainWarps);
    }
    if (lane < 2) mbar_init(&b.mma_done[lane], 1);
    for (int i = (int)lane; i < kSaRing; i += 32) {
      // the scale warp and one unpack group (the code sums); image mode: the scale warp alone
      mbar_init(&b.sa_full[i], a.image ? 1 : 1 + kUnpackGroupWarps);
      mbar_init(&b.sa_empty[i], kNumDrainWarps);
    }
    if (lane == 0) mbar_init(b.corr_full, ngroups * kUnpackGroupWarps);
    fence_mbar_init();
    __syncwarp();
    if (lane == 0) {
      tma_prefetch_desc(&tmW);
      tma_prefetch_desc(&tmX);
      // The weight boxes of the ring's first pass depend neither on the previous kernel in the
      // stream nor on the rest of this CTA's setup (TMEM, the zeroed token rows): they go out
      // now, before the CTA-wide barrier and before waiting for that kernel.
      tma_first_weights<kMp>(a, rg, n0, &tmW, smem, b);
    }
  }
  if (warp == kWarpMma) {
    tmem_alloc(tmem_slot, L::kTmemCols);
    tmem_relinquish();
  }
  // Token rows >= M of the operand ring are zero codes for good: store them once here, and the
  // unpack converts only the M real rows of every slot.
  if (a.M < kMp && !a.image) {
    const uint32_t row_bytes = (uint32_t)(kMp - a.M) * kBK, tile0 = smem_u32(smem + L::kOffOp);
    for (uint32_t i = threadIdx.x; i < kOpSlots * kStPerSlot * (row_bytes / 16u); i += kThreads) {
      const uint32_t tile = i / (row_bytes / 16u), off = (uint32_t)a.M * kBK + (i % (row_bytes / 16u)) * 16u;
      st_shared_v4(tile0 + tile * L::kOpB + off, 0u, 0u, 0u, 0u);  // whole rows: the swizzle only permutes within a row
    }
    fence_proxy_async_smem();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const bool drain = warp >= kDrainWarp0;
  static_assert(kDrainWarp0 == 12 && kUnpackWarp0 == 4, "the register split is per warpgroup");
  // The next kernel in the stream may launch now; it waits for this one before it touches our
  // inputs or outputs.  Here the TMA producer waits for the previous kernel after its first
  // weight boxes, the scale warp and the drain before their first access to activation data or
  // the output; the unpack and MMA roles touch only shared and tensor memory.
  pdl_launch_dependents();
  // drain threads: this channel's bias and (G = K) weight scale for the final pass, fetched now
  // (weight-side data: no need to wait for the previous kernel) so that no one waits for them later
  float fin_bn = 0.0f, fin_swn = 0.0f;
  if (drain && rank == 0) {
    const int n = n0 + (int)((warp & 3u) * 32u + lane);
    fin_bn = (n < a.N && a.bias != nullptr) ? __ldg(a.bias + n) : 0.0f;
    fin_swn = (n < a.N && a.groups == 1) ? __ldg(a.s_w + n) : 0.0f;
  }
  if (drain) {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(kRegsDrain<kMp>) : "memory");
    if (single) unpack_role<kMp>(a, rg, smem, tmem_base, b, ngroups, abort_flag);  // group 2 (warps 12-15)
    pdl_wait();
    drain_role<kMp>(a, rg, n0, tmem_base, smem, b, abort_flag);
    __syncwarp();
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegsLaunch) : "memory");
  } else if (warp >= kUnpackWarp0) {
    unpack_role<kMp>(a, rg, smem, tmem_base, b, ngroups, abort_flag);
  } else {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegsCtl<kMp>) : "memory");
    if (warp == kWarpScale) {
      pdl_wait();
      scale_role<kMp>(a, rg, smem, b, abort_flag);
    } else if (warp == kWarpTma) {
      if (lane == 0) tma_role<kMp>(a, rg, n0, &tmW, &tmX, smem, b, abort_flag);
    } else if (lane == 0 && (warp == kWarpMma || warp == kWarpMma1)) {
      const uint32_t e = warp == kWarpMma ? 0u : 1u;
      if (a.groups == 1)
        mma_role<kMp, 0>(a, rg, e, tmem_base, smem, b, abort_flag);
      else if (a.G >= kBK)
        mma_role<kMp, 1>(a, rg, e, tmem_base, smem, b, abort_flag);
      else
        mma_role<kMp, 2>(a, rg, e, tmem_base, smem, b, abort_flag);
    }
    __syncwarp();
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(kRegsLaunch) : "memory");
  }

  // every role is done; the drain threads have written their partials to the reduction buffer
  tc_fence_before();
  __syncthreads();
  float* red = reinterpret_cast<float*>(smem + L::kOffPk);  // [kMp][128]
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
  if (a.split > 1) cluster_sync_all();  // no CTA leaves while a peer may still read its buffer
  if (drain && rank == 0) {
    const int n = n0 + (int)ch;
    const float* fin = reinterpret_cast<const float*>(smem + L::kOffFin);  // staged by the scale warp
    if (n < a.N) {
#pragma unroll 8
      for (int i = 0; i < kH; ++i) {
        const int m = (int)hf * kH + i;
        if (m < a.M) {
          float v = red[m * kRows + ch];
          if (a.groups == 1) {  // exact integer partial (less the whole-K correction): scale once
            v -= fin[kMp + m];  // exact: integers below 2^24 (units 2^-18)
            const float sa = fin[m], f = sa * kOperandUnitInv;
            v = f <= FLT_MAX ? (v * fin_swn) * f : ((v * kOperandUnitInv) * sa) * fin_swn;
          }
          a.y[(int64_t)m * a.N + n] = __float2bfloat16_rn(v + fin_bn);
        }
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
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // programmatic launch (ptx.cuh)
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;  // the cluster shape; launches add the programmatic attribute
  return cfg;
}

// The split (CTAs per cluster) for `tiles` channel tiles: the largest one up to kMaxSplit for
// which every cluster is resident at once (one wave), the CTAs do not outnumber the SMs, and
// every CTA keeps at least kMinSplitSlots ring slots of K: below that a CTA's fixed costs (setup,
// first-byte latency, the cluster reduction) outweigh the bandwidth of the extra SMs (measured on
// K=3072 -> N=3072, 24 tiles: split 2 beats 6 by 18 % at one token and 27 % at 64).  Cluster
// residency is asked of the runtime once per device and size.
struct SplitProbe {
  int max_clusters[kMaxSplit + 1];
};

template <int kMp>
cudaError_t choose_split(int tiles, int k_stages, int sms, int& best) {
  // Cluster residency per split, asked of the runtime once per device and tile height.
  static PerDevice<SplitProbe> probes;
  SplitProbe pr;
  cudaError_t e = probes.get(
      [sms](SplitProbe& v) {
        v.max_clusters[0] = 0;
        for (int s = 1; s <= kMaxSplit; ++s) {
          cudaLaunchAttribute attr[2];
          cudaLaunchConfig_t cfg = make_config<kMp>(s * (sms / s), s, nullptr, attr);
          int n = 0;
          if (cudaOccupancyMaxActiveClusters(&n, w4a4_skinny_kernel<kMp>, &cfg) != cudaSuccess) {
            (void)cudaGetLastError();
            n = 0;
          }
          v.max_clusters[s] = n;
        }
        return cudaSuccess;
      },
      pr);
  if (e != cudaSuccess) return e;
  const int slots = (k_stages + kStPerSlot - 1) / kStPerSlot;
  best = 1;
  for (int s = 2; s <= kMaxSplit && s <= k_stages; ++s)
    if (tiles * s <= sms && tiles <= pr.max_clusters[s] && slots / s >= kMinSplitSlots) best = s;
  return cudaSuccess;
}

template <int kMp>
cudaError_t launch_mp(SkArgs a, const SkinnyProblem& p, int tiles, int sms, cudaStream_t stream) {
  using L = Layout<kMp>;
  // The shared-memory attribute is per device: set once for each device, before its first
  // occupancy probe (choose_split) and launch.
  static PerDevice<bool> smem_attr;
  bool attr_ok = false;
  cudaError_t ae = smem_attr.get(
      [](bool& v) {
        v = true;
        return cudaFuncSetAttribute(w4a4_skinny_kernel<kMp>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)L::kSmemBytes);
      },
      attr_ok);
  if (ae != cudaSuccess) return ae;
  // Packed codes as byte matrices: weights [N, K/2], tokens [M, K/2]; one box = 128 packed bytes
  // (two K stages) x 128 weight rows or x kMp token rows, 128-byte swizzle.  Rows past N or M
  // and columns past K/2 read zeros.  Image mode: the tokens come from the A-operand image seen
  // as rows of 128 bytes (block (0, kb) = rows 128 kb ..), one box = the first kMp rows of a
  // block, copied as they are (the image is already in the 128-byte swizzle).
  CUtensorMap tmW, tmX;
  // (ternary weights [N, K/4]: one box = 64 packed bytes (two K stages) x 128 rows, 64-byte swizzle)
  const bool ok_w = a.ternary ? encode_2d(&tmW, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.qw, p.K / 4, p.N, p.K / 4, kBK / 2,
                                          kRows, CU_TENSOR_MAP_SWIZZLE_64B)
                              : encode_2d(&tmW, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.qw, p.K / 2, p.N, p.K / 2, kBK, kRows,
                                          CU_TENSOR_MAP_SWIZZLE_128B);
  const bool ok_x = a.image ? encode_2d(&tmX, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.a_image, kBK,
                                        (uint64_t)a.k_stages * kBK, kBK, kBK, kMp, CU_TENSOR_MAP_SWIZZLE_NONE)
                            : encode_2d(&tmX, CU_TENSOR_MAP_DATA_TYPE_UINT8, p.q, p.K / 2, p.M, p.K / 2, kBK, kMp,
                                        CU_TENSOR_MAP_SWIZZLE_128B);
  if (!ok_w || !ok_x) return cudaErrorInvalidValue;
  cudaError_t se = choose_split<kMp>(tiles, a.k_stages, sms, a.split);
  if (se != cudaSuccess) return se;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = make_config<kMp>(tiles * a.split, a.split, stream, attr);
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, w4a4_skinny_kernel<kMp>, tmW, tmX, a);
}

}  // namespace

cudaError_t launch_w4a4_skinny(const SkinnyProblem& p, cudaStream_t stream, int sms) {
  if (p.M <= 0 || p.N <= 0) return cudaSuccess;
  if (!skinny_supports(p.M, p.K, p.G)) return cudaErrorInvalidValue;
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
  // More than 16 tokens: converting the token rows in every CTA would cost more than the weights'
  // conversion, so they come pre-expanded (operand image + corrections) when the caller has them.
  a.image = (p.a_image != nullptr && p.corr != nullptr && p.M > 16) ? 1 : 0;
  a.ternary = p.ternary ? 1 : 0;
  a.corr = p.corr;
  const int tiles = (p.N + kRows - 1) / kRows;
  if (p.M <= 16) return launch_mp<16>(a, p, tiles, sms, stream);
  if (p.M <= 32) return launch_mp<32>(a, p, tiles, sms, stream);
  return launch_mp<64>(a, p, tiles, sms, stream);
}

}  // namespace jq
