// noalloc.cu -- jq_w4a4_linear_noalloc: the W4A4 linear layer for callers that cannot allocate
// device memory.
//
// jq_w4a4_linear needs a caller-provided workspace to hold the activation operand bytes
// between its two kernels.  Some callers cannot provide one: code running where cudaMalloc is
// off limits (inside a host callback, in a plug-in whose host framework owns every allocation,
// in a hard-real-time serving loop that must not allocate after start-up), or code that has no
// allocator handle at all.  For them this entry point keeps that scratch in a fixed
// file-scope device array instead.  Everything else -- the inputs, the scales, the output --
// is still passed in by the caller, and the kernels are the same ones jq_w4a4_linear runs.
//
// The array is a program-scope __device__ variable: every GPU that loads this library holds
// its kNoAllocScratchBytes for the life of the process, and every call on a device shares it.
#include <cstdint>
#include <mutex>

#include <cuda_runtime.h>

#include "jq.h"
#include "kernels.cuh"

namespace {

constexpr size_t kNoAllocScratchBytes = JQ_NOALLOC_MAX_SCRATCH_BYTES;
using jq::kMaxDevices;
using jq::kMaxK;

// The scratch: the E4M3 operand image of the activations, whole 128-row tiles of K bytes.  The
// expansion kernel of the same call writes every row below M; rows past M in the last tile are
// read by the GEMM but only feed accumulator rows that are never stored, so no byte of the array
// has to start at zero.
static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

struct NoAllocDevice {
  bool ready = false;
  bool ok = false;
  int sms = 0;
  uint8_t* scratch = nullptr;  // device address of g_noalloc_scratch on this device
  uint32_t* status = nullptr;  // the library's device status word (read by jq_device_status)
};
NoAllocDevice g_noalloc_devices[kMaxDevices];
std::mutex g_noalloc_mutex;

// Set-up, once per device, with that device current.  In host code the name g_noalloc_scratch
// is only a host-side stand-in for the symbol, never a device address, so the address the
// kernels get comes from cudaGetSymbolAddress.
const NoAllocDevice* noalloc_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_noalloc_mutex);
  NoAllocDevice& d = g_noalloc_devices[dev];
  if (!d.ready) {
    d.ready = true;
    cudaDeviceProp prop;
    void* p = nullptr;
    if (cudaGetDeviceProperties(&prop, dev) == cudaSuccess && prop.major == 10 && prop.minor == 3 &&
        cudaGetSymbolAddress(&p, g_noalloc_scratch) == cudaSuccess && p != nullptr) {
      d.sms = prop.multiProcessorCount;
      d.scratch = static_cast<uint8_t*>(p);
      d.status = jq::device_status_word();
      d.ok = d.status != nullptr;
    }
  }
  return d.ok ? &d : nullptr;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" jq_status jq_w4a4_linear_noalloc(const uint8_t* q, const float* s_a, const uint8_t* qw, const float* s_w,
                                           const float* bias, void* y_bf16, int64_t M, int64_t N, int64_t K,
                                           int32_t group, void* stream) {
  if (M < 0 || N < 0) return JQ_ERR_INVALID_ARG;
  if (M == 0 || N == 0) return JQ_OK;
  if (K <= 0 || K % 128 != 0 || K > kMaxK || !(group == 64 || group == 128 || group == K) || N % 8 != 0 ||
      M > INT32_MAX || N > INT32_MAX)
    return JQ_ERR_INVALID_ARG;
  if (q == nullptr || s_a == nullptr || qw == nullptr || s_w == nullptr || y_bf16 == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(s_a) || !aligned16(qw) || !aligned16(s_w) || !aligned16(y_bf16) ||
      (bias != nullptr && !aligned16(bias)))
    return JQ_ERR_MISALIGNED;
  const NoAllocDevice* d0 = nullptr;
  if (jq::skinny_supports(M, K, group)) {  // few tokens: the weight-streaming kernel needs no scratch at all
    if ((d0 = noalloc_device()) == nullptr) return JQ_ERR_UNSUPPORTED;
    jq::SkinnyProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, q, s_a, qw, s_w, bias,
                        y_bf16, d0->status};
    return jq::launch_w4a4_skinny(p, static_cast<cudaStream_t>(stream), d0->sms) == cudaSuccess ? JQ_OK : JQ_ERR_CUDA;
  }
  // the operand image (whole 128-row tiles) and the per-group corrections
  if (jq::ws_image_bytes(M, K) + jq::ws_per_group_bytes(M, K, group) > kNoAllocScratchBytes) return JQ_ERR_WORKSPACE;
  const NoAllocDevice* d = noalloc_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* corr = reinterpret_cast<float*>(d->scratch + jq::ws_image_bytes(M, K));
  if (jq::launch_expand_operand(q, M, K, group, d->scratch, corr, s, d->sms) != cudaSuccess) return JQ_ERR_CUDA;
  jq::GemmProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, d->scratch, s_a, corr, qw,
                    s_w, bias, y_bf16, nullptr, d->status};
  return jq::launch_w4a4_gemm(p, s, d->sms) == cudaSuccess ? JQ_OK : JQ_ERR_CUDA;
}
