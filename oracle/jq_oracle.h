/* jq_oracle.h -- declarations of the CPU oracle (test infrastructure only;
 * see jq_oracle.c for the definitions and the passages they follow). */
#ifndef JQ_ORACLE_H
#define JQ_ORACLE_H
#include <stdint.h>
#ifdef __cplusplus
extern "C" {
#endif
uint16_t oracle_bf16_rne(double v);
void oracle_quantize_bf16(const uint16_t* x, int64_t M, int64_t K, int64_t ldx, int64_t G,
                          int8_t* codes, float* scales);
void oracle_quantize_f32(const float* w, int64_t N, int64_t K, int64_t G, int8_t* codes,
                         float* scales);
void oracle_pack(const int8_t* codes, int64_t rows, int64_t K, uint8_t* packed);
void oracle_unpack(const uint8_t* packed, int64_t rows, int64_t K, int8_t* codes);
void oracle_quantize_ternary_f32(const float* w, int64_t N, int64_t K, int64_t G, int8_t* codes,
                                 float* scales);
void oracle_pack_ternary(const int8_t* codes, int64_t rows, int64_t K, uint8_t* packed);
void oracle_unpack_ternary(const uint8_t* packed, int64_t rows, int64_t K, int8_t* codes);
void oracle_set_threads(int n);
int oracle_max_threads(void);
float oracle_nvfp4_tensor_scale(const float* x, int64_t n);
void oracle_quantize_nvfp4(const float* x, int64_t rows, int64_t K, float g, int8_t* codes2,
                           float* block_scales);
void oracle_pack_nvfp4(const int8_t* codes2, int64_t rows, int64_t K, uint8_t* packed);
void oracle_unpack_nvfp4(const uint8_t* packed, int64_t rows, int64_t K, int8_t* codes2);
void oracle_linear_nvfp4(const int8_t* qa2, const float* sa, float ga, const int8_t* qw2, const float* sw,
                         float gw, const float* bias, int64_t M, int64_t N, int64_t K, double* y64,
                         uint16_t* ybf16);
void oracle_group_partials(const int8_t* qa, const int8_t* qw, int64_t M, int64_t N, int64_t K,
                           int64_t G, int32_t* acc);
void oracle_linear(const int8_t* qa, const float* s_a, const int8_t* qw, const float* s_w,
                   const float* bias, int64_t M, int64_t N, int64_t K, int64_t G, double* y64,
                   uint16_t* ybf16);
void oracle_fake_quant_bf16(const uint16_t* x, int64_t M, int64_t K, int64_t G, const float* s_in,
                            uint16_t* xhat, uint8_t* mask, float* s_out);
void oracle_fake_quant_f32(const float* w, int64_t N, int64_t K, int64_t G, const float* s_in,
                           float* what, uint8_t* mask, float* s_out);
void oracle_ste_backward_bf16(const uint16_t* grad, const uint8_t* mask, int64_t n, uint16_t* grad_x);
float oracle_gelu_tanh_f32(float h);
void oracle_modulate_quantize_bf16(const uint16_t* x, int64_t M, int64_t K, int64_t ldx, const float* shift,
                                   const float* scale, int64_t tokens_per_sample, int64_t G, uint16_t* z,
                                   int8_t* codes, float* scales);
void oracle_gelu_quantize_bf16(const uint16_t* h, int64_t M, int64_t K, int64_t ldh, int64_t G, uint16_t* z,
                               int8_t* codes, float* scales);
#ifdef __cplusplus
}
#endif
#endif
