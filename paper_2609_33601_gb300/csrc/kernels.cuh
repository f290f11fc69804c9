// kernels.cuh -- internal launchers behind the C ABI (no argument checking here; api.cu does it).
#pragma once
#include <cstdint>
#include <mutex>

#include <cuda.h>
#include <cuda_runtime.h>

namespace jq {

// Highest device ordinal (+1) the library serves in one process.
constexpr int kMaxDevices = 64;

// Launch set-up that has to happen once per device: kernel attributes (the dynamic shared-memory
// size) and occupancy probes are properties of a kernel on one device, so a value found with
// device 0 current says nothing about device 1.  get() runs `init` for the current device the
// first time that device asks, under a mutex, and records the result only when `init` succeeded
// (a failed set-up is retried on the next call).  Safe to call from several host threads.
template <typename T>
class PerDevice {
 public:
  template <typename F>
  cudaError_t get(F&& init, T& out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu_);
    if (!done_[dev]) {
      T v{};
      e = init(v);
      if (e != cudaSuccess) return e;
      vals_[dev] = v;
      done_[dev] = true;
    }
    out = vals_[dev];
    return cudaSuccess;
  }

 private:
  std::mutex mu_;
  bool done_[kMaxDevices] = {};
  T vals_[kMaxDevices] = {};
};

// Launches `kernel` with programmatic stream serialisation: it may begin while the previous
// kernel of the stream is still running, as soon as that kernel allows it (ptx.cuh,
// pdl_launch_dependents); the kernel itself waits (pdl_wait) before it touches anything the
// previous kernel may write or read.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Largest K the library accepts: every exact group sum of sign-magnitude codes, |acc| <= 64 K,
// stays below 2^24, so the fp32 accumulators hold it exactly (operand.cuh).
constexpr int64_t kMaxK = 262016;  // 2047 * 128
static_assert(64 * kMaxK < (int64_t{1} << 24) && kMaxK % 128 == 0, "exact group sums up to kMaxK");

// bf16 activations [M, ldx] -> packed codes [M, K/2] + scales [M, K/G].
cudaError_t launch_quantize_act(const void* x, int64_t M, int64_t K, int64_t ldx, int G, uint8_t* q, float* s_a,
                                cudaStream_t stream, int sms);
// bf16 activations -> GEMM operand bytes [M, K] + scales [M, K/G] + corrections [M, K/G]
// (fused path; the corrections are 8 * the group's code sum in 2^-18 units, operand.cuh).
cudaError_t launch_quantize_act_operand(const void* x, int64_t M, int64_t K, int64_t ldx, int G, uint8_t* op,
                                        float* s_a, float* corr, cudaStream_t stream, int sms);
// DiT neighbour operations fused with the activation quantiser (quantize.cu): the adaLN
// modulation bf16(x (1 + scale[b]) + shift[b]) of token m of sample b = m / tokens_per_sample,
// shift / scale fp32 [samples, K]; the tanh GELU of h.  Output as launch_quantize_act.
cudaError_t launch_modulate_quantize_act(const void* x, int64_t M, int64_t K, int64_t ldx, const float* shift,
                                         const float* scale, int64_t tokens_per_sample, int G, uint8_t* q, float* s_a,
                                         cudaStream_t stream, int sms);
cudaError_t launch_gelu_quantize_act(const void* h, int64_t M, int64_t K, int64_t ldh, int G, uint8_t* q, float* s_a,
                                     cudaStream_t stream, int sms);
// fp32 weights [N, K] -> packed codes [N, K/2] + scales [K/G, N].
cudaError_t launch_pack_weight(const float* w, int64_t N, int64_t K, int G, uint8_t* qw, float* s_w,
                               cudaStream_t stream, int sms);
// fp32 weights [N, K] -> packed ternary codes [N, K/4] + scales [K/G, N] (ternary.cu).
cudaError_t launch_pack_weight_ternary(const float* w, int64_t N, int64_t K, int G, uint8_t* qw, float* s_w,
                                       cudaStream_t stream, int sms);
// bf16 activations [M, K] (dense rows) -> fake-quantised bf16 [M, K] + pass-through mask u8 [M, K]
// + scales fp32 [M, K/G]; s_in (nullable) gives the scales instead of the amax rule (fakequant.cu).
cudaError_t launch_fake_quant_act(const void* x, int64_t M, int64_t K, int G, const float* s_in, void* xhat,
                                  uint8_t* mask, float* s_out, cudaStream_t stream, int sms);
// fp32 weights [N, K] -> fake-quantised fp32 [N, K] + mask u8 [N, K] + scales fp32 [N, K/G] (fakequant.cu).
cudaError_t launch_fake_quant_weight(const float* w, int64_t N, int64_t K, int G, const float* s_in, float* what,
                                     uint8_t* mask, float* s_out, cudaStream_t stream, int sms);
// straight-through backward: grad_x = grad where mask != 0, +0 elsewhere, n bf16 elements (fakequant.cu).
cudaError_t launch_ste_backward(const void* grad, const uint8_t* mask, int64_t n, void* grad_x, cudaStream_t stream,
                                int sms);
// packed codes [rows, K/2] -> operand bytes [rows, K] + corrections [rows, K/G].
cudaError_t launch_expand_operand(const uint8_t* packed, int64_t rows, int64_t K, int G, uint8_t* op, float* corr,
                                  cudaStream_t stream, int sms);

// NVFP4 (nvfp4.cu): activations bf16 [M, ldx] -> E2M1 codes [M, K/2] + E4M3 block-scale bytes
// [M, K/16] with the caller's tensor scale g; weights fp32 [N, K] -> the same, with g computed
// into the device scalar *g; the linear layer from both (workspace: two bf16 operand images).
size_t nvfp4_image_bytes(int64_t rows, int64_t K);
cudaError_t launch_nvfp4_quantize_act(const void* x, int64_t M, int64_t K, int64_t ldx, float g, uint8_t* codes,
                                      uint8_t* scales, cudaStream_t stream, int sms);
cudaError_t launch_nvfp4_pack_weight(const float* w, int64_t N, int64_t K, uint8_t* codes, uint8_t* scales, float* g,
                                     cudaStream_t stream, int sms);
cudaError_t launch_nvfp4_linear(const uint8_t* qa, const uint8_t* sa, float ga, const uint8_t* qw, const uint8_t* sw,
                                const float* gw, const float* bias, void* y, int64_t M, int64_t N, int64_t K,
                                uint8_t* workspace, uint32_t* status, cudaStream_t stream, int sms);

// Workspace of the GEMM path, each part on a 256-byte boundary: the A-operand image (whole
// 128-row tiles of K operand bytes), the corrections fp32 [M, K/G], and for the fused path the
// activation scales fp32 [M, K/G].
inline size_t ws_image_bytes(int64_t M, int64_t K) {
  return static_cast<size_t>((M + 127) / 128 * 128) * static_cast<size_t>(K);
}
inline size_t ws_per_group_bytes(int64_t M, int64_t K, int32_t G) {
  return (static_cast<size_t>(M) * static_cast<size_t>(K / G) * sizeof(float) + 255) / 256 * 256;
}

struct GemmProblem {
  int M, N, K, G;
  const uint8_t* a_operand;  // [M, K] operand bytes (workspace)
  const float* s_a;          // [M, K/G]
  const float* corr;         // [M, K/G]: 8 * sum of the group's activation codes, in 2^-18 units
  const uint8_t* qw;         // [N, K/2] packed INT4 (or [N, K/4] ternary, below)
  const float* s_w;          // [K/G, N]
  const float* bias;         // [N] or nullptr
  void* y;                   // bf16 [M, N] (or nullptr when exporting partials)
  int32_t* partials;         // int32 [M, N, K/G] or nullptr
  uint32_t* status;          // device status word
  int ternary = 0;           // qw holds packed ternary codes [N, K/4] (ternary.cu) instead of INT4
};

// Device address of the library's status word on the current device, or nullptr.
uint32_t* device_status_word();

// 2-D tiled tensor map (row-major, `inner` elements per row of `row_bytes`), box
// box_inner x box_outer; boxes past the ends read zeros.  False if the driver rejects it.
bool encode_2d(CUtensorMap* map, CUtensorMapDataType dtype, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swizzle);

// Encodes the tensor maps and launches the persistent tcgen05 GEMM.
cudaError_t launch_w4a4_gemm(const GemmProblem& p, cudaStream_t stream, int sms);

// Few-token linear layer (skinny.cu): reads the packed activation codes directly and needs no
// scratch, or, when the caller sets a_image / corr (jq_w4a4_linear does for M > 16), takes the
// tokens pre-expanded from the caller's workspace.  Used for M <= kSkinnyMaxM.  With one group
// (G = K) a CTA accumulates offset-code products over its whole K range in fp32, exact while
// 120 * K < 2^24 (operand.cuh): larger one-group problems take the GEMM, which keeps
// sign-magnitude weights for them.
constexpr int kSkinnyMaxM = 64;
constexpr int kSkinnyMaxKOneGroup = 139776;  // 1092 * 128
inline bool skinny_supports(int64_t M, int64_t K, int32_t G) {
  return M <= kSkinnyMaxM && (G != K || K <= kSkinnyMaxKOneGroup);
}
struct SkinnyProblem {
  int M, N, K, G;
  const uint8_t* q;    // [M, K/2] packed activation codes
  const float* s_a;    // [M, K/G]
  const uint8_t* qw;   // [N, K/2] packed weight codes
  const float* s_w;    // [K/G, N]
  const float* bias;   // [N] or nullptr
  void* y;             // bf16 [M, N]
  uint32_t* status;    // device status word
  // Optional, for M > 16: the tokens as the A-operand image (operand.cuh) and their corrections
  // [M, K/G] (8 * the group's code sum, 2^-18 units), as launch_expand_operand writes them.
  const uint8_t* a_image = nullptr;
  const float* corr = nullptr;
  // Ternary weights: qw is [N, K/4] in the packed ternary format (ternary.cu).
  int ternary = 0;
};
cudaError_t launch_w4a4_skinny(const SkinnyProblem& p, cudaStream_t stream, int sms);

}  // namespace jq
