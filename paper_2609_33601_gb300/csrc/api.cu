// api.cu -- the C ABI declared in include/jq.h: synchronous argument checks, then kernel
// launches on the caller's stream.  No allocation, no synchronisation (except in
// jq_device_status), no exceptions.
#include <cfloat>
#include <cstdint>
#include <mutex>

#include <cuda_runtime.h>

#include "jq.h"
#include "kernels.cuh"
#include "operand.cuh"
#include "ptx.cuh"

namespace {

using jq::kMaxDevices;
using jq::kMaxK;
// The offset-code form (one group, in the few-token kernel and the GEMM) sums |(q_w + 8) q_a| <= 120
// per element, exact in fp32 over runs of up to kOffsetMaxRun elements; the few-token kernel's
// one-group limit stays inside that run.
static_assert(120 * static_cast<int64_t>(jq::kOffsetMaxRun) < (int64_t{1} << 24), "offset-code runs are exact");
static_assert(jq::kSkinnyMaxKOneGroup <= jq::kOffsetMaxRun, "one-group few-token problems are exact");

// One status word per device, written by kernels that give up a bounded wait.
__device__ uint32_t g_device_status = 0;

struct DeviceInfo {
  bool probed = false;
  bool ok = false;
  int sms = 0;
  uint32_t* status = nullptr;
};
DeviceInfo g_devices[kMaxDevices];
std::mutex g_devices_mutex;

// Resolves the current device once: it must be an sm_103 part.  The probe runs under a mutex and
// is recorded only once it has an answer, so a first call from several host threads at once sees
// either the finished probe or runs it itself, never a half-written entry.
const DeviceInfo* current_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_devices_mutex);
  DeviceInfo& d = g_devices[dev];
  if (!d.probed) {
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) return nullptr;  // not recorded: asked again
    void* p = nullptr;
    const bool sm103 = prop.major == 10 && prop.minor == 3;
    if (sm103 && cudaGetSymbolAddress(&p, g_device_status) != cudaSuccess) return nullptr;
    d.sms = prop.multiProcessorCount;
    d.status = static_cast<uint32_t*>(p);
    d.ok = sm103 && p != nullptr;
    d.probed = true;
  }
  return d.ok ? &d : nullptr;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool group_ok(int64_t K, int32_t group) {
  if (K <= 0 || K % 128 != 0 || K > kMaxK) return false;
  return group == 64 || group == 128 || group == K;
}

size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

jq_status from_cuda(cudaError_t e) { return e == cudaSuccess ? JQ_OK : JQ_ERR_CUDA; }

// Failure-handling probe: one thread waits, with the bounded wait every kernel of the library
// uses, on an mbarrier phase that nothing completes.  The wait gives up after ~2^31 cycles,
// records kDevTimeout in the status word and the block returns: no trap, no fault, no hang.
__global__ void __launch_bounds__(32) wait_timeout_probe_kernel(uint32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    jq::mbar_init(&bar, 1);  // one arrival would complete phase 0; none comes
    abort_flag = 0;
  }
  __syncthreads();
  if (threadIdx.x == 0) (void)jq::mbar_wait(&bar, 0, &abort_flag, status);
  __syncthreads();
}

}  // namespace

namespace jq {
// Device address of the library's status word on the current device (nullptr if the device is
// not supported); kernels launched from other files report bounded-wait timeouts into it.
uint32_t* device_status_word() {
  const DeviceInfo* d = current_device();
  return d == nullptr ? nullptr : d->status;
}
}  // namespace jq

extern "C" {

const char* jq_status_string(jq_status s) {
  switch (s) {
    case JQ_OK: return "JQ_OK";
    case JQ_ERR_INVALID_ARG: return "JQ_ERR_INVALID_ARG";
    case JQ_ERR_MISALIGNED: return "JQ_ERR_MISALIGNED";
    case JQ_ERR_UNSUPPORTED: return "JQ_ERR_UNSUPPORTED";
    case JQ_ERR_CUDA: return "JQ_ERR_CUDA";
    case JQ_ERR_TIMEOUT: return "JQ_ERR_TIMEOUT";
    case JQ_ERR_WORKSPACE: return "JQ_ERR_WORKSPACE";
  }
  return "JQ_ERR_UNKNOWN";
}

jq_status jq_quantize_act(const void* x_bf16, int64_t M, int64_t K, int64_t ldx, int32_t group, uint8_t* q,
                          float* s_a, void* stream) {
  if (M < 0 || !group_ok(K, group) || ldx < K) return JQ_ERR_INVALID_ARG;
  if (M == 0) return JQ_OK;
  if (x_bf16 == nullptr || q == nullptr || s_a == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(x_bf16) || !aligned16(q) || !aligned16(s_a) || (ldx * 2) % 16 != 0) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_quantize_act(x_bf16, M, K, ldx, group, q, s_a, static_cast<cudaStream_t>(stream),
                                           d->sms));
}

jq_status jq_modulate_quantize_act(const void* x_bf16, int64_t M, int64_t K, int64_t ldx, const float* shift,
                                   const float* scale, int64_t tokens_per_sample, int32_t group, uint8_t* q, float* s_a,
                                   void* stream) {
  if (M < 0 || !group_ok(K, group) || ldx < K || tokens_per_sample <= 0) return JQ_ERR_INVALID_ARG;
  if (M == 0) return JQ_OK;
  if (x_bf16 == nullptr || shift == nullptr || scale == nullptr || q == nullptr || s_a == nullptr)
    return JQ_ERR_INVALID_ARG;
  if (!aligned16(x_bf16) || !aligned16(shift) || !aligned16(scale) || !aligned16(q) || !aligned16(s_a) ||
      (ldx * 2) % 16 != 0)
    return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_modulate_quantize_act(x_bf16, M, K, ldx, shift, scale, tokens_per_sample, group, q, s_a,
                                                    static_cast<cudaStream_t>(stream), d->sms));
}

jq_status jq_gelu_quantize_act(const void* h_bf16, int64_t M, int64_t K, int64_t ldh, int32_t group, uint8_t* q,
                               float* s_a, void* stream) {
  if (M < 0 || !group_ok(K, group) || ldh < K) return JQ_ERR_INVALID_ARG;
  if (M == 0) return JQ_OK;
  if (h_bf16 == nullptr || q == nullptr || s_a == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(h_bf16) || !aligned16(q) || !aligned16(s_a) || (ldh * 2) % 16 != 0) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_gelu_quantize_act(h_bf16, M, K, ldh, group, q, s_a, static_cast<cudaStream_t>(stream),
                                                d->sms));
}

jq_status jq_pack_weight(const float* w, int64_t N, int64_t K, int32_t group, uint8_t* qw, float* s_w,
                         void* stream) {
  if (N < 0 || !group_ok(K, group)) return JQ_ERR_INVALID_ARG;
  if (N == 0) return JQ_OK;
  if (w == nullptr || qw == nullptr || s_w == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(w) || !aligned16(qw) || !aligned16(s_w)) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_pack_weight(w, N, K, group, qw, s_w, static_cast<cudaStream_t>(stream), d->sms));
}

size_t jq_workspace_size(int64_t M, int64_t N, int64_t K, int32_t group, int32_t fused) {
  (void)N;
  if (M <= 0 || K <= 0 || group <= 0 || K % group != 0) return 0;
  // A-operand image: whole 128-row tiles of K operand bytes (operand.cuh)
  size_t bytes = jq::ws_image_bytes(M, K) + jq::ws_per_group_bytes(M, K, group);  // A image, corrections
  if (fused) bytes += jq::ws_per_group_bytes(M, K, group);                           // activation scales
  return bytes;
}

namespace {

jq_status check_linear(int64_t M, int64_t N, int64_t K, int32_t group, const void* qw, const float* s_w,
                       const float* bias, const void* y, size_t ws_need, const void* ws, size_t ws_bytes) {
  if (M < 0 || N < 0 || N % 8 != 0 || N > INT32_MAX || M > INT32_MAX || !group_ok(K, group))
    return JQ_ERR_INVALID_ARG;
  if (qw == nullptr || s_w == nullptr || y == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(qw) || !aligned16(s_w) || !aligned16(y) || (bias != nullptr && !aligned16(bias)))
    return JQ_ERR_MISALIGNED;
  if (ws == nullptr || !aligned16(ws) || ws_bytes < ws_need) return JQ_ERR_WORKSPACE;
  return JQ_OK;
}

}  // namespace

jq_status jq_w4a4_linear(const uint8_t* q, const float* s_a, const uint8_t* qw, const float* s_w, const float* bias,
                         void* y_bf16, int64_t M, int64_t N, int64_t K, int32_t group, void* workspace,
                         size_t workspace_bytes, void* stream) {
  if (M == 0 || N == 0) return (M < 0 || N < 0) ? JQ_ERR_INVALID_ARG : JQ_OK;
  if (q == nullptr || s_a == nullptr) return JQ_ERR_INVALID_ARG;
  jq_status st = check_linear(M, N, K, group, qw, s_w, bias, y_bf16, jq_workspace_size(M, N, K, group, 0),
                              workspace, workspace_bytes);
  if (st != JQ_OK) return st;
  if (!aligned16(q) || !aligned16(s_a)) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* a_op = static_cast<uint8_t*>(workspace);
  float* corr = reinterpret_cast<float*>(a_op + jq::ws_image_bytes(M, K));
  if (jq::skinny_supports(M, K, group)) {  // few tokens: the weight-streaming kernel
    jq::SkinnyProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, q, s_a, qw, s_w, bias,
                        y_bf16, d->status};
    if (M > 16) {  // expand the tokens once here rather than in every CTA of the kernel
      if (jq::launch_expand_operand(q, M, K, group, a_op, corr, s, d->sms) != cudaSuccess) return JQ_ERR_CUDA;
      p.a_image = a_op;
      p.corr = corr;
    }
    return from_cuda(jq::launch_w4a4_skinny(p, s, d->sms));
  }
  cudaError_t e = jq::launch_expand_operand(q, M, K, group, a_op, corr, s, d->sms);
  if (e != cudaSuccess) return JQ_ERR_CUDA;
  jq::GemmProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, a_op, s_a, corr, qw, s_w, bias,
                    y_bf16, nullptr, d->status};
  return from_cuda(jq::launch_w4a4_gemm(p, s, d->sms));
}

jq_status jq_fused_quant_linear(const void* x_bf16, int64_t ldx, const uint8_t* qw, const float* s_w,
                                const float* bias, void* y_bf16, int64_t M, int64_t N, int64_t K, int32_t group,
                                void* workspace, size_t workspace_bytes, void* stream) {
  if (M == 0 || N == 0) return (M < 0 || N < 0) ? JQ_ERR_INVALID_ARG : JQ_OK;
  if (x_bf16 == nullptr || ldx < K) return JQ_ERR_INVALID_ARG;
  jq_status st = check_linear(M, N, K, group, qw, s_w, bias, y_bf16, jq_workspace_size(M, N, K, group, 1),
                              workspace, workspace_bytes);
  if (st != JQ_OK) return st;
  if (!aligned16(x_bf16) || (ldx * 2) % 16 != 0) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* a_op = static_cast<uint8_t*>(workspace);
  float* corr = reinterpret_cast<float*>(a_op + jq::ws_image_bytes(M, K));
  float* s_a = reinterpret_cast<float*>(a_op + jq::ws_image_bytes(M, K) + jq::ws_per_group_bytes(M, K, group));
  if (jq::skinny_supports(M, K, group)) {  // few tokens: the weight-streaming kernel
    jq::SkinnyProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, a_op, s_a, qw, s_w,
                        bias, y_bf16, d->status};
    // up to 16 tokens: packed codes in the workspace; more: the operand image and corrections
    cudaError_t e = M > 16 ? jq::launch_quantize_act_operand(x_bf16, M, K, ldx, group, a_op, s_a, corr, s, d->sms)
                           : jq::launch_quantize_act(x_bf16, M, K, ldx, group, a_op, s_a, s, d->sms);
    if (e != cudaSuccess) return JQ_ERR_CUDA;
    if (M > 16) {
      p.a_image = a_op;
      p.corr = corr;
    }
    return from_cuda(jq::launch_w4a4_skinny(p, s, d->sms));
  }
  cudaError_t e = jq::launch_quantize_act_operand(x_bf16, M, K, ldx, group, a_op, s_a, corr, s, d->sms);
  if (e != cudaSuccess) return JQ_ERR_CUDA;
  jq::GemmProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, a_op, s_a, corr, qw, s_w, bias,
                    y_bf16, nullptr, d->status};
  return from_cuda(jq::launch_w4a4_gemm(p, s, d->sms));
}

jq_status jq_pack_weight_ternary(const float* w, int64_t N, int64_t K, int32_t group, uint8_t* qw2, float* s_w,
                                 void* stream) {
  if (N < 0 || !group_ok(K, group)) return JQ_ERR_INVALID_ARG;
  if (N == 0) return JQ_OK;
  if (w == nullptr || qw2 == nullptr || s_w == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(w) || !aligned16(qw2) || !aligned16(s_w)) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_pack_weight_ternary(w, N, K, group, qw2, s_w, static_cast<cudaStream_t>(stream),
                                                  d->sms));
}

size_t jq_w158a4_workspace_size(int64_t M, int64_t N, int64_t K, int32_t group) {
  // as jq_w4a4_linear: both kernels read the 2-bit codes directly
  return jq_workspace_size(M, N, K, group, 0);
}

jq_status jq_w158a4_linear(const uint8_t* q, const float* s_a, const uint8_t* qw2, const float* s_w, const float* bias,
                           void* y_bf16, int64_t M, int64_t N, int64_t K, int32_t group, void* workspace,
                           size_t workspace_bytes, void* stream) {
  if (M == 0 || N == 0) return (M < 0 || N < 0) ? JQ_ERR_INVALID_ARG : JQ_OK;
  if (q == nullptr || s_a == nullptr) return JQ_ERR_INVALID_ARG;
  jq_status st = check_linear(M, N, K, group, qw2, s_w, bias, y_bf16, jq_w158a4_workspace_size(M, N, K, group),
                              workspace, workspace_bytes);
  if (st != JQ_OK) return st;
  if (!aligned16(q) || !aligned16(s_a)) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* a_op = static_cast<uint8_t*>(workspace);
  float* corr = reinterpret_cast<float*>(a_op + jq::ws_image_bytes(M, K));
  if (jq::skinny_supports(M, K, group)) {  // few tokens: stream the 2-bit codes
    jq::SkinnyProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, q, s_a, qw2, s_w, bias,
                        y_bf16, d->status};
    p.ternary = 1;
    if (M > 16) {
      if (jq::launch_expand_operand(q, M, K, group, a_op, corr, s, d->sms) != cudaSuccess) return JQ_ERR_CUDA;
      p.a_image = a_op;
      p.corr = corr;
    }
    return from_cuda(jq::launch_w4a4_skinny(p, s, d->sms));
  }
  // many tokens: the compute-bound GEMM, its weight-unpack warps reading the 2-bit codes
  if (jq::launch_expand_operand(q, M, K, group, a_op, corr, s, d->sms) != cudaSuccess) return JQ_ERR_CUDA;
  jq::GemmProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, a_op, s_a, corr, qw2, s_w,
                    bias, y_bf16, nullptr, d->status};
  p.ternary = 1;
  return from_cuda(jq::launch_w4a4_gemm(p, s, d->sms));
}

jq_status jq_w4a4_group_partials(const uint8_t* q, const uint8_t* qw, int32_t* acc, int64_t M, int64_t N, int64_t K,
                                 int32_t group, void* workspace, size_t workspace_bytes, void* stream) {
  if (M == 0 || N == 0) return (M < 0 || N < 0) ? JQ_ERR_INVALID_ARG : JQ_OK;
  if (q == nullptr || acc == nullptr) return JQ_ERR_INVALID_ARG;
  if (M < 0 || N < 0 || N % 8 != 0 || !group_ok(K, group) || qw == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(qw) || !aligned16(acc)) return JQ_ERR_MISALIGNED;
  if (workspace == nullptr || !aligned16(workspace) || workspace_bytes < jq_workspace_size(M, N, K, group, 0))
    return JQ_ERR_WORKSPACE;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* a_op = static_cast<uint8_t*>(workspace);
  float* corr = reinterpret_cast<float*>(a_op + jq::ws_image_bytes(M, K));
  cudaError_t e = jq::launch_expand_operand(q, M, K, group, a_op, corr, s, d->sms);
  if (e != cudaSuccess) return JQ_ERR_CUDA;
  // The export path needs scale tensors only for their layout; it never reads their values,
  // but the weight-scale tensor map must point at valid memory: reuse the packed weights.
  jq::GemmProblem p{static_cast<int>(M), static_cast<int>(N), static_cast<int>(K), group, a_op, nullptr, corr, qw,
                    reinterpret_cast<const float*>(qw), nullptr, nullptr, acc, d->status};
  return from_cuda(jq::launch_w4a4_gemm(p, s, d->sms));
}

jq_status jq_fake_quant_act(const void* x_bf16, int64_t M, int64_t K, int32_t group, const float* s_in,
                            void* xhat_bf16, uint8_t* mask, float* s_out, void* stream) {
  if (M < 0 || !group_ok(K, group)) return JQ_ERR_INVALID_ARG;
  if (M == 0) return JQ_OK;
  if (x_bf16 == nullptr || xhat_bf16 == nullptr || mask == nullptr || s_out == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(x_bf16) || !aligned16(xhat_bf16) || !aligned16(mask) || !aligned16(s_out) ||
      (s_in != nullptr && !aligned16(s_in)))
    return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_fake_quant_act(x_bf16, M, K, group, s_in, xhat_bf16, mask, s_out,
                                             static_cast<cudaStream_t>(stream), d->sms));
}

jq_status jq_fake_quant_weight(const float* w, int64_t N, int64_t K, int32_t group, const float* s_in, float* what,
                               uint8_t* mask, float* s_out, void* stream) {
  if (N < 0 || !group_ok(K, group)) return JQ_ERR_INVALID_ARG;
  if (N == 0) return JQ_OK;
  if (w == nullptr || what == nullptr || mask == nullptr || s_out == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(w) || !aligned16(what) || !aligned16(mask) || !aligned16(s_out) ||
      (s_in != nullptr && !aligned16(s_in)))
    return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_fake_quant_weight(w, N, K, group, s_in, what, mask, s_out,
                                                static_cast<cudaStream_t>(stream), d->sms));
}

jq_status jq_ste_backward(const void* grad_bf16, const uint8_t* mask, int64_t n, void* grad_x_bf16, void* stream) {
  if (n < 0) return JQ_ERR_INVALID_ARG;
  if (n == 0) return JQ_OK;
  if (grad_bf16 == nullptr || mask == nullptr || grad_x_bf16 == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(grad_bf16) || !aligned16(mask) || !aligned16(grad_x_bf16)) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_ste_backward(grad_bf16, mask, n, grad_x_bf16, static_cast<cudaStream_t>(stream), d->sms));
}

jq_status jq_debug_wait_timeout(void* stream) {
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  wait_timeout_probe_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(d->status);
  return from_cuda(cudaGetLastError());
}

// ---- NVFP4 W4A4 (nvfp4.cu)
namespace {
bool nvfp4_k_ok(int64_t K) { return K > 0 && K % 64 == 0 && K <= kMaxK; }
}  // namespace

jq_status jq_nvfp4_quantize_act(const void* x_bf16, int64_t M, int64_t K, int64_t ldx, float g_a, uint8_t* codes,
                                uint8_t* scales, void* stream) {
  if (M < 0 || !nvfp4_k_ok(K) || ldx < K || !(g_a >= 0.0f && g_a <= FLT_MAX)) return JQ_ERR_INVALID_ARG;
  if (M == 0) return JQ_OK;
  if (x_bf16 == nullptr || codes == nullptr || scales == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(x_bf16) || !aligned16(codes) || (ldx * 2) % 16 != 0) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_nvfp4_quantize_act(x_bf16, M, K, ldx, g_a, codes, scales,
                                                 static_cast<cudaStream_t>(stream), d->sms));
}

jq_status jq_nvfp4_pack_weight(const float* w, int64_t N, int64_t K, uint8_t* codes, uint8_t* scales, float* g_w,
                               void* stream) {
  if (N < 0 || !nvfp4_k_ok(K)) return JQ_ERR_INVALID_ARG;
  if (N == 0) return JQ_OK;
  if (w == nullptr || codes == nullptr || scales == nullptr || g_w == nullptr) return JQ_ERR_INVALID_ARG;
  if (!aligned16(w) || !aligned16(codes) || !aligned16(g_w)) return JQ_ERR_MISALIGNED;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_nvfp4_pack_weight(w, N, K, codes, scales, g_w, static_cast<cudaStream_t>(stream),
                                                d->sms));
}

size_t jq_nvfp4_workspace_size(int64_t M, int64_t N, int64_t K) {
  if (M <= 0 || N <= 0 || !nvfp4_k_ok(K)) return 0;
  return jq::nvfp4_image_bytes(M, K) + jq::nvfp4_image_bytes(N, K);
}

jq_status jq_nvfp4_linear(const uint8_t* codes_a, const uint8_t* scales_a, float g_a, const uint8_t* codes_w,
                          const uint8_t* scales_w, const float* g_w, const float* bias, void* y_bf16, int64_t M,
                          int64_t N, int64_t K, void* workspace, size_t workspace_bytes, void* stream) {
  if (M < 0 || N < 0 || N % 8 != 0 || M > INT32_MAX || N > INT32_MAX || !nvfp4_k_ok(K) ||
      !(g_a >= 0.0f && g_a <= FLT_MAX))
    return JQ_ERR_INVALID_ARG;
  if (M == 0 || N == 0) return JQ_OK;
  if (codes_a == nullptr || scales_a == nullptr || codes_w == nullptr || scales_w == nullptr || g_w == nullptr ||
      y_bf16 == nullptr)
    return JQ_ERR_INVALID_ARG;
  if (!aligned16(codes_a) || !aligned16(codes_w) || !aligned16(y_bf16) || (bias != nullptr && !aligned16(bias)) ||
      (reinterpret_cast<uintptr_t>(g_w) & 3u) != 0)
    return JQ_ERR_MISALIGNED;
  if (workspace == nullptr || !aligned16(workspace) || workspace_bytes < jq_nvfp4_workspace_size(M, N, K))
    return JQ_ERR_WORKSPACE;
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  return from_cuda(jq::launch_nvfp4_linear(codes_a, scales_a, g_a, codes_w, scales_w, g_w, bias, y_bf16, M, N, K,
                                           static_cast<uint8_t*>(workspace), d->status,
                                           static_cast<cudaStream_t>(stream), d->sms));
}

jq_status jq_device_status(void* stream, int32_t reset) {
  const DeviceInfo* d = current_device();
  if (d == nullptr) return JQ_ERR_UNSUPPORTED;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return JQ_ERR_CUDA;
  uint32_t v = 0;
  if (cudaMemcpy(&v, d->status, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return JQ_ERR_CUDA;
  if (reset && v != 0) {
    const uint32_t zero = 0;
    if (cudaMemcpy(d->status, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess) return JQ_ERR_CUDA;
  }
  // 1: a bounded wait gave up; 2: the GEMM found its shared-memory window misaligned and did nothing
  return v == 0 ? JQ_OK : (v == 1 ? JQ_ERR_TIMEOUT : JQ_ERR_UNSUPPORTED);
}

}  // extern "C"
