/*
 * jq.h -- C ABI of libjq: the naive W4A4 linear layer of JustQuant (arxiv 2609.33601)
 * on one GB300 (sm_103a).
 *
 * The paper deploys a "plain low-bit operator graph": activations and weights are quantised
 * to INT4 with per-group scales, packed, and multiplied by a low-bit GEMM, with no smoothing,
 * rotation, normalisation or SVD branch (Sec. 1; Appendix FAQ Q7: low-bit execution "still
 * requires suitable quantization, packing, and matrix-multiplication kernels").  Group sizes
 * are fixed by the paper: group64 for FLUX transformer-block linears (Sec. 4.2 "FLUX";
 * Appendix table "FLUX experimental details"), group128 for DiT-XL/2 and ELF-B (Appendix
 * tables "DiT-XL/2 experimental details", "ELF-B and LLaDA-8B experimental details").
 * Per-token / per-channel scaling is the special case group == K.
 *
 * Quantiser (the paper prints no formula; this is the symmetric INT4 reading):
 *     per row and per run of `group` consecutive K elements:
 *     amax = max|x|,  s = fl32(amax / 7),  q = clamp(rint(fl32(x / s)), -8, 7)
 *     (IEEE fp32 division, round half to even; s = 0 and q = 0 when amax == 0).
 * Linear layer:
 *     acc[m,n,g] = sum_{k in group g} qa[m,k] * qw[n,k]            (exact integers)
 *     y[m,n]     = bf16_rne( sum_g acc[m,n,g] * s_a[m,g] * s_w[g,n] + bias[n] )  (fp32 math)
 *
 * Conventions shared by every entry point
 *   - Matrices are row-major with K contiguous.  Packed codes: 4-bit two's complement, two per
 *     byte, element 2j in the low nibble of byte j; a row of K codes is K/2 bytes.
 *   - Activation scales s_a: fp32 [M, K/group] (one per token and K-group).
 *     Weight scales s_w:     fp32 [K/group, N] (group-major: one row of N channel scales per
 *     K-group).  bias: fp32 [N] or NULL.  Outputs y: bf16 [M, N].
 *   - All data pointers are DEVICE pointers owned by the caller.  The library allocates
 *     nothing, never synchronises (one exception: jq_gelu_quantize_act, below, once per
 *     device), and enqueues its kernels on `stream` (a cudaStream_t passed as void*; NULL =
 *     legacy default stream).
 *   - Supported shapes: group in {64, 128, K}; K % 128 == 0; K <= 262016 (so every exact
 *     per-group sum, |acc| <= 64*K, stays below 2^24); N % 8 == 0; M >= 0 (M == 0 is a no-op).
 *   - Pointers must be 16-byte aligned and ldx*2 a multiple of 16 bytes.
 *   - Arguments are checked synchronously before any launch; a failed check returns an error
 *     status and launches nothing.  A failed launch returns JQ_ERR_CUDA.  No exception
 *     crosses the ABI.
 *   - Every on-GPU wait is bounded (about a second).  A kernel that gives up records
 *     JQ_ERR_TIMEOUT in a device status word read by jq_device_status().
 *   - Devices and threads: kernels launch on the CURRENT device (cudaGetDevice) and all
 *     pointers must belong to it.  Per-device launch set-up (kernel attributes, occupancy
 *     probes, the device status word) happens on a device's first call, under a mutex, so a
 *     process may drive several GPUs and call from several host threads, first calls included.
 *   - Kernels are launched with programmatic dependent launch: one of this library's kernels may
 *     start while the previous kernel on the stream is still running, when that kernel is also
 *     one of this library's (the linear layers start streaming their weights early), and waits
 *     for it before touching any data it writes or reads.  Stream order holds for all data;
 *     other kernels on the stream, yours included, order with these as with any kernel.
 */
#ifndef JQ_H
#define JQ_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define JQ_API __attribute__((visibility("default")))
#else
#define JQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  JQ_OK = 0,
  JQ_ERR_INVALID_ARG = 1,  /* null pointer, bad size, unsupported group/K/N combination */
  JQ_ERR_MISALIGNED = 2,   /* a pointer or a row pitch breaks the 16-byte rule */
  JQ_ERR_UNSUPPORTED = 3,  /* no CUDA device of the required architecture (sm_103) */
  JQ_ERR_CUDA = 4,         /* a CUDA runtime/driver call or kernel launch failed */
  JQ_ERR_TIMEOUT = 5,      /* a kernel gave up a bounded wait (reported by jq_device_status) */
  JQ_ERR_WORKSPACE = 6     /* workspace pointer NULL/misaligned or smaller than required */
} jq_status;

/* Human-readable name of a status code (static string, never NULL; no counterpart in the paper). */
JQ_API const char* jq_status_string(jq_status s);

/*
 * Activation quantiser (per token and K-group; rule above).  The paper quantises the activations
 * of the transformer-block linears to INT4 with group64 (Sec. 4.2 "FLUX"; Appendix "FLUX
 * experimental details") or group128 (Appendix "DiT-XL/2 experimental details", "ELF-B and
 * LLaDA-8B experimental details"); the formula is the reading above.
 *   x_bf16 : bf16 [M, ldx] (the first K columns are used), ldx >= K, ldx*2 % 16 == 0
 *   q      : uint8 [M, K/2] packed codes (output)
 *   s_a    : fp32 [M, K/group] scales (output)
 * Errors: JQ_ERR_INVALID_ARG (null, K/group unsupported, ldx < K), JQ_ERR_MISALIGNED,
 * JQ_ERR_UNSUPPORTED (the current device is not sm_103), JQ_ERR_CUDA (the launch failed).
 */
JQ_API jq_status jq_quantize_act(const void* x_bf16, int64_t M, int64_t K, int64_t ldx, int32_t group,
                          uint8_t* q, float* s_a, void* stream);

/*
 * Weight packer (offline; the same rule per output channel and K-group).  INT4 weights with the
 * activations' group size (the same Appendix tables); packing is one of the kernels the deployed
 * graph needs (Appendix FAQ Q7).
 *   w   : fp32 [N, K] row-major
 *   qw  : uint8 [N, K/2] packed codes (output)
 *   s_w : fp32 [K/group, N] scales (output, group-major)
 * Errors as jq_quantize_act.
 */
JQ_API jq_status jq_pack_weight(const float* w, int64_t N, int64_t K, int32_t group, uint8_t* qw, float* s_w,
                         void* stream);

/*
 * DiT neighbour operations fused with the activation quantiser.  The paper's deployment remark
 * (Sec. 1, the figure on naive W1.58A4 deployment) concerns a 0.6B DiT, DiT-XL/2, where small
 * matrices and non-GEMM time limit the speed-up; its W4A4 / W1.58A4 setting there is group128
 * (Appendix "DiT-XL/2 experimental details").  In a DiT-XL/2 block the inputs of the linears
 * come from the adaLN modulation (before the attention's QKV projection and the MLP's first
 * linear) and from the MLP's tanh GELU (before its second linear); these calls read that
 * operation's input and write the quantised codes of its output, so the bf16 activation between
 * the two never goes to memory.  The paper prints neither operation; the readings:
 *   modulation: token m of sample b = m / tokens_per_sample, channel k:
 *     z = bf16( fl32( fl32( x * fl32(1 + scale[b,k]) ) + shift[b,k] ) )
 *     (IEEE single steps, no fused multiply-add, one rounding to bf16, nearest even);
 *   GELU: z = bf16( 0.5 h (1 + tanh(sqrt(2/pi) (h + 0.044715 h^3))) ), the exact value rounded
 *     once to bf16 (nearest even; +-0 stays +-0);
 * then the activation rule above on z.  Codes and scales are exactly those of
 * jq_quantize_act applied to z.
 *   x_bf16 / h_bf16 : bf16 [M, ldx] (ldx >= K, ldx*2 % 16 == 0)
 *   shift, scale    : fp32 [ceil(M / tokens_per_sample), K], dense rows (modulation)
 *   tokens_per_sample > 0
 *   q, s_a          : outputs as jq_quantize_act
 * Errors as jq_quantize_act (JQ_ERR_INVALID_ARG also for tokens_per_sample <= 0 or a NULL
 * shift / scale).
 * The GELU is read from a table of its value at every bf16 input (65536 entries, in the
 * library's device memory), computed on the device by the first call on each device: outside
 * a stream capture that call runs the filling kernel on `stream` and synchronises `stream` once
 * (later calls on any stream then read the finished table); a first call made while `stream`
 * is being captured puts the filling kernel into the graph ahead of the quantiser instead
 * (each replay rewrites the same values) and leaves the once-per-device filling to the first
 * call made outside a capture.
 */
JQ_API jq_status jq_modulate_quantize_act(const void* x_bf16, int64_t M, int64_t K, int64_t ldx, const float* shift,
                                          const float* scale, int64_t tokens_per_sample, int32_t group, uint8_t* q,
                                          float* s_a, void* stream);
JQ_API jq_status jq_gelu_quantize_act(const void* h_bf16, int64_t M, int64_t K, int64_t ldh, int32_t group,
                                      uint8_t* q, float* s_a, void* stream);

/*
 * Bytes of device scratch the two linear entry points need for this shape
 * (fused != 0: jq_fused_quant_linear, else jq_w4a4_linear).  The caller owns it.  (The paper has
 * no counterpart: the scratch holds the activations in the GEMM's operand layout, the library's
 * own design, so that the library itself never allocates.)
 */
JQ_API size_t jq_workspace_size(int64_t M, int64_t N, int64_t K, int32_t group, int32_t fused);

/*
 * W4A4 linear on pre-quantised activations -- the deployed "naive W4A4" linear layer, a plain
 * low-bit GEMM with no smoothing, rotation or SVD branch (Sec. 1; Appendix FAQ Q7), with group
 * scales (Sec. 4.2; Appendix experimental-detail tables):
 *   y = bf16( sum_g acc[m,n,g] * s_a[m,g] * s_w[g,n] + bias[n] ).
 *   (The weight scales are group-major [K/group, N] so that one group's channel scales are
 *   contiguous for the GEMM's scale loads; the workspace keeps allocation with the caller.)
 *   q         : uint8 [M, K/2] packed activation codes (jq_quantize_act)
 *   s_a       : fp32 [M, K/group]
 *   qw, s_w   : packed weights and scales (jq_pack_weight, or any codes/finite scales in
 *               these layouts, including the code -8)
 *   bias      : fp32 [N] or NULL
 *   y_bf16    : bf16 [M, N] (output)
 *   workspace : >= jq_workspace_size(M, N, K, group, 0) bytes of device memory, 16-byte aligned
 * Errors: JQ_ERR_INVALID_ARG, JQ_ERR_MISALIGNED, JQ_ERR_WORKSPACE, JQ_ERR_UNSUPPORTED, JQ_ERR_CUDA.
 */
JQ_API jq_status jq_w4a4_linear(const uint8_t* q, const float* s_a, const uint8_t* qw, const float* s_w,
                         const float* bias, void* y_bf16, int64_t M, int64_t N, int64_t K, int32_t group,
                         void* workspace, size_t workspace_bytes, void* stream);

/*
 * W4A4 linear straight from bf16 activations (the quantise + low-bit GEMM pair of Appendix FAQ
 * Q7 in one call): quantises x (rule above, per token and K-group) directly into the GEMM's
 * operand layout, then runs the same GEMM.  Results are
 * bit-identical to jq_quantize_act followed by jq_w4a4_linear.
 *   x_bf16    : bf16 [M, ldx]
 *   workspace : >= jq_workspace_size(M, N, K, group, 1) bytes
 * Other arguments and errors as jq_w4a4_linear.
 */
JQ_API jq_status jq_fused_quant_linear(const void* x_bf16, int64_t ldx, const uint8_t* qw, const float* s_w,
                                const float* bias, void* y_bf16, int64_t M, int64_t N, int64_t K,
                                int32_t group, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Verification export of the exact per-group integer partials of the GEMM (no counterpart in the
 * paper; it exposes the exact integer sums of the linear layer above for testing):
 *   acc : int32 [M, N, K/group], acc[m,n,g] = sum_{k in g} qa[m,k] * qw[n,k].
 * Runs the same mainloop as jq_w4a4_linear with the dequantising epilogue replaced by an
 * integer store; meant for small shapes.  workspace as jq_w4a4_linear.
 */
JQ_API jq_status jq_w4a4_group_partials(const uint8_t* q, const uint8_t* qw, int32_t* acc, int64_t M, int64_t N,
                                 int64_t K, int32_t group, void* workspace, size_t workspace_bytes,
                                 void* stream);

/*
 * jq_w4a4_linear for callers that cannot allocate device memory.  (The paper has no
 * counterpart; this is a deployment convenience.)  jq_w4a4_linear needs a caller-provided
 * workspace; code that may not call cudaMalloc at all -- a host callback, a plug-in whose
 * framework owns every allocation, a serving loop that must not allocate after start-up --
 * cannot provide one.  This variant keeps that scratch (the activation operand bytes and their
 * per-group code sums) in a fixed device array inside the library instead,
 * JQ_NOALLOC_MAX_SCRATCH_BYTES large, which every GPU that loads the library holds until the
 * process exits.  It allocates nothing and
 * runs the same kernels, so its output is identical to jq_w4a4_linear's.
 *   Arguments as jq_w4a4_linear, without the workspace.
 *   Limit: ceil(M / 128) * 128 * K + ceil(4 * M * (K/group) / 256) * 256 <=
 *   JQ_NOALLOC_MAX_SCRATCH_BYTES (the operand bytes and one fp32 per token and group), else
 *   JQ_ERR_WORKSPACE (nothing launched); calls that take the few-token kernel need no scratch.
 *   The first call on a device looks up the array's device address (cudaGetSymbolAddress);
 *   make that first call before any stream capture.  All calls on a device share the one
 *   array, so calls whose kernels may overlap on the GPU (different streams without ordering
 *   between them) race and corrupt each other's results; order them on one stream.
 * Errors: JQ_ERR_INVALID_ARG, JQ_ERR_MISALIGNED, JQ_ERR_WORKSPACE, JQ_ERR_UNSUPPORTED, JQ_ERR_CUDA.
 */
#define JQ_NOALLOC_MAX_SCRATCH_BYTES (16u * 1024u * 1024u)
JQ_API jq_status jq_w4a4_linear_noalloc(const uint8_t* q, const float* s_a, const uint8_t* qw, const float* s_w,
                                        const float* bias, void* y_bf16, int64_t M, int64_t N, int64_t K,
                                        int32_t group, void* stream);

/*
 * W1.58A4: ternary weights with INT4 activations (the paper's W1.58A4 setting: "Ternary
 * weights, INT4 activations, group128", Appendix table "DiT-XL/2 experimental details"; the
 * ELF-B table likewise).  The paper prints no ternary rule; the reading is the absmean rule per
 * output channel and K-group:
 *     s = fl32(mean |w|)   (fp64 sum of the group in index order, one division by group)
 *     q = clamp(rint(fl32(w / s)), -1, 1)   (round half to even; s = q = 0 for a zero group)
 * Packed ternary codes: q + 1 in {0, 1, 2}, 2 bits each, a row of K codes is K/4 bytes; every
 * 16 consecutive elements fill one little-endian 32-bit word whose byte j (j = 0..3) holds
 * elements 2j, 2j+1, 8+2j, 9+2j in bits 0-1, 2-3, 4-5, 6-7.
 *
 * Ternary weight packer (offline).
 *   w   : fp32 [N, K] row-major
 *   qw2 : uint8 [N, K/4] packed ternary codes (output)
 *   s_w : fp32 [K/group, N] scales (output, group-major, as jq_pack_weight)
 * Errors as jq_pack_weight.
 */
JQ_API jq_status jq_pack_weight_ternary(const float* w, int64_t N, int64_t K, int32_t group, uint8_t* qw2,
                                        float* s_w, void* stream);

/* Bytes of device scratch jq_w158a4_linear needs for this shape (the caller owns it; as
 * jq_workspace_size, the paper has no counterpart). */
JQ_API size_t jq_w158a4_workspace_size(int64_t M, int64_t N, int64_t K, int32_t group);

/*
 * W1.58A4 linear on pre-quantised activations: the linear layer above with ternary weight codes,
 *   y = bf16( sum_g acc[m,n,g] * s_a[m,g] * s_w[g,n] + bias[n] ),  acc over qa * qw, qw in {-1,0,1}.
 *   q, s_a    : packed INT4 activation codes and scales (jq_quantize_act)
 *   qw2, s_w  : packed ternary weights and scales (jq_pack_weight_ternary, or any ternary codes
 *               and finite scales in these layouts; a 2-bit field of 3 is not a code and gives an
 *               unspecified result)
 *   workspace : >= jq_w158a4_workspace_size(M, N, K, group) bytes, 16-byte aligned (the same
 *               size as jq_workspace_size(M, N, K, group, 0))
 * Both kernels read the 2-bit codes directly (half the weight bytes of INT4): up to 64 tokens the
 * few-token kernel, for more tokens the INT4 GEMM, whose weight-unpack warps convert them.
 * Other arguments, shapes and errors as jq_w4a4_linear.
 */
JQ_API jq_status jq_w158a4_linear(const uint8_t* q, const float* s_a, const uint8_t* qw2, const float* s_w,
                                  const float* bias, void* y_bf16, int64_t M, int64_t N, int64_t K, int32_t group,
                                  void* workspace, size_t workspace_bytes, void* stream);

/*
 * Training side: fake quantisation of bf16 activations (forward of the straight-through
 * estimator).  Stage 1 of Theseus QAD (Sec. 3, Algorithm 1) trains the quantised student blocks
 * by gradient descent, and Sec. 3 ("Why QAT fails") names the straight-through estimator as the
 * gradient rule of 4-bit activations; the paper prints neither rule, and this is the reading:
 *   xhat[m,k] = bf16( q * s )   with q = clamp(rint(fl32(x / s)), -8, 7), the deployed code,
 *   the product formed exactly and rounded once (nearest even); a zero code gives +0;
 *   mask[m,k] = 1 where the unclamped rint(fl32(x / s)) lies in [-8, 7], else 0.
 *   x_bf16    : bf16 [M, K], dense rows (device)
 *   group     : 64, 128 or K (K a multiple of 128, at most 262016)
 *   s_in      : fp32 [M, K/group] positive finite scales with 8*s finite (e.g. learned ones), or
 *               NULL for the quantiser's own rule s = fl32(amax/7) (then s = 0, xhat = 0 and
 *               mask = 1 for an all-zero group, and no code is clamped)
 *   xhat_bf16 : bf16 [M, K] (output);  mask : uint8 [M, K] (output, 0/1)
 *   s_out     : fp32 [M, K/group] (output): the scales used
 * All pointers 16-byte aligned; M = 0 is a no-op.  Errors: JQ_ERR_INVALID_ARG (null, K/group
 * unsupported, M < 0), JQ_ERR_MISALIGNED, JQ_ERR_UNSUPPORTED (not sm_103), JQ_ERR_CUDA.
 */
JQ_API jq_status jq_fake_quant_act(const void* x_bf16, int64_t M, int64_t K, int32_t group, const float* s_in,
                                   void* xhat_bf16, uint8_t* mask, float* s_out, void* stream);

/*
 * Training side: fake quantisation of the student's fp32 weights, the same reading per output
 * channel and K-group: what[n,k] = fl32(q * s) (one rounding of the exact product), with mask and
 * scales as in jq_fake_quant_act.
 *   w         : fp32 [N, K] row-major (device);  s_in : fp32 [N, K/group] or NULL (amax rule)
 *   what      : fp32 [N, K] (output);  mask : uint8 [N, K] (output);  s_out : fp32 [N, K/group]
 *               (output; row-major, unlike jq_pack_weight's group-major scales)
 * Checks and errors as jq_fake_quant_act.
 */
JQ_API jq_status jq_fake_quant_weight(const float* w, int64_t N, int64_t K, int32_t group, const float* s_in,
                                      float* what, uint8_t* mask, float* s_out, void* stream);

/*
 * Training side: the straight-through backward (the reading above):
 *   grad_x[i] = grad[i] where mask[i] != 0, else +0.
 *   grad_bf16, grad_x_bf16 : bf16 [n] (device; grad_x may not overlap grad unless equal)
 *   mask                   : uint8 [n] (jq_fake_quant_act's mask)
 * Any n >= 0 (n = 0 is a no-op); pointers 16-byte aligned.  Errors: JQ_ERR_INVALID_ARG,
 * JQ_ERR_MISALIGNED, JQ_ERR_UNSUPPORTED, JQ_ERR_CUDA.
 */
JQ_API jq_status jq_ste_backward(const void* grad_bf16, const uint8_t* mask, int64_t n, void* grad_x_bf16,
                                 void* stream);

/*
 * NVFP4 W4A4, the format of the paper's LLaDA-8B rows (Appendix table "ELF-B and LLaDA-8B
 * experimental details": "NVFP4 W4A4"; the paper defines nothing more, the reading is the
 * published NVFP4 format): E2M1 elements, one E4M3 scale per 16 consecutive K elements of a row,
 * one fp32 scale g per tensor.  Per block b: s_b = e4m3(fl32(amax_b / fl32(6 g))), S_b =
 * fl32(s_b g), q = e2m1(fl32(x / S_b)), both nearest with ties to the even mantissa and
 * saturating (448, 6); q = 0 where g = 0 or S_b = 0.  Codes: 4-bit E2M1 (bit 3 sign, bits 1-2
 * exponent, bit 0 mantissa), element 2j in the low nibble of byte j; block scales: E4M3 bytes.
 *
 * Activations with the caller's (calibrated) tensor scale g_a >= 0:
 *   x_bf16 : bf16 [M, ldx] (device);  codes : uint8 [M, K/2] (output);  scales : uint8 [M, K/16]
 * K a multiple of 64, at most 262016; x, codes 16-byte aligned, ldx*2 a multiple of 16; M = 0
 * is a no-op.  Errors: JQ_ERR_INVALID_ARG (null, K, M < 0, ldx < K, g_a negative or not finite),
 * JQ_ERR_MISALIGNED, JQ_ERR_UNSUPPORTED, JQ_ERR_CUDA.
 */
JQ_API jq_status jq_nvfp4_quantize_act(const void* x_bf16, int64_t M, int64_t K, int64_t ldx, float g_a,
                                       uint8_t* codes, uint8_t* scales, void* stream);

/*
 * Weights, with their tensor scale computed on the device: g_w = fl32(amax |w| / 2688).
 *   w : fp32 [N, K] (device);  codes : uint8 [N, K/2];  scales : uint8 [N, K/16];
 *   g_w : one fp32 (device, output; the linear layer reads it there)
 * K as above; w, codes and g_w 16-byte aligned.  Errors as jq_nvfp4_quantize_act.
 */
JQ_API jq_status jq_nvfp4_pack_weight(const float* w, int64_t N, int64_t K, uint8_t* codes, uint8_t* scales,
                                      float* g_w, void* stream);

/* Workspace bytes jq_nvfp4_linear needs: two bf16 operand images (activations and weights). */
JQ_API size_t jq_nvfp4_workspace_size(int64_t M, int64_t N, int64_t K);

/*
 * The NVFP4 linear layer:
 *   y[m,n] = bf16( sum_b (sum_{k in b} qa qw) sa_b sw_b * g_a * g_w + bias[n] )
 * Each element's value q * s_b is exact in bf16; the layer multiplies those in the tensor core
 * (exact products) and sums them in fp32 over all of K, then scales by g_a and g_w and adds the
 * bias in fp32.  The fp32 sum is the one step that is not exact: |y - y64| is within one bf16 ulp
 * plus (K + 2) * 2^-24 * (sum_k |term| + |bias|).
 *   codes_a, scales_a : jq_nvfp4_quantize_act's output for [M, K];  g_a as given there
 *   codes_w, scales_w, g_w : jq_nvfp4_pack_weight's output for [N, K]
 *   bias : fp32 [N] or NULL;  y_bf16 : bf16 [M, N] (output)
 * K as above, N % 8 == 0; codes, y and bias 16-byte aligned; workspace >= jq_nvfp4_workspace_size
 * bytes, 16-byte aligned; M = 0 or N = 0 is a no-op.  Errors: JQ_ERR_INVALID_ARG,
 * JQ_ERR_MISALIGNED, JQ_ERR_WORKSPACE, JQ_ERR_UNSUPPORTED, JQ_ERR_CUDA.
 */
JQ_API jq_status jq_nvfp4_linear(const uint8_t* codes_a, const uint8_t* scales_a, float g_a, const uint8_t* codes_w,
                                 const uint8_t* scales_w, const float* g_w, const float* bias, void* y_bf16, int64_t M,
                                 int64_t N, int64_t K, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Verification export for failure handling (computes nothing; no counterpart in the paper):
 * launches one block in which one
 * thread waits, with the bounded wait every kernel of this library uses, on an mbarrier phase
 * that nothing completes.  After about 2^31 SM clock cycles (about a second) the wait gives up
 * and records JQ_ERR_TIMEOUT in the device status word, which jq_device_status() then reports;
 * nothing faults, traps or hangs, and the CUDA context stays usable.  It lets a caller test its
 * handling of a kernel that gave up.  Errors: JQ_ERR_UNSUPPORTED, JQ_ERR_CUDA.
 */
JQ_API jq_status jq_debug_wait_timeout(void* stream);

/*
 * (No counterpart in the paper; the library's failure reporting.)
 * Synchronises `stream` and returns JQ_ERR_TIMEOUT if any kernel of this library on the
 * current device gave up a bounded wait since the last reset (reset != 0 clears the flag),
 * JQ_ERR_UNSUPPORTED if a GEMM launch found its shared-memory window not 1024-byte aligned
 * (it then wrote nothing), JQ_ERR_CUDA if the stream reports an error, JQ_OK otherwise.
 */
JQ_API jq_status jq_device_status(void* stream, int32_t reset);

#ifdef __cplusplus
}
#endif

#endif /* JQ_H */
