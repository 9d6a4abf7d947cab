/*
 * orc.h — CPU oracle for the batch-1 decode step of a Llama-2-architecture
 * decoder, as restated in "Bare-Metal Tensor Virtualization" (Kilictas &
 * Alpay, arXiv 2601.03324).
 *
 * TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and the
 * bench's CPU-baseline / reference arms may load this library. The CUDA path
 * in paper_2601_03324_gb300/ never includes this header or links this code,
 * and this code includes nothing from there.
 *
 * Every routine is the plain definition, written as scalar loops in the
 * accumulator type Acc (double: parity truth; float: the "scalar C++"
 * analogue of the paper's Table 1 baseline). Weights are read as float32
 * from the caller's blob, laid out in this oracle's own reading of the
 * packed layout (see orc_layout in orc.cpp).
 */
#ifndef ORC_H
#define ORC_H
#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  int32_t dim, hidden_dim, n_layers, n_heads, n_kv_heads, vocab_size, max_seq;
  double rope_theta; /* RoPE base, 10000 in every workload */
  double norm_eps;   /* RMSNorm epsilon, 1e-5 (paper, RMSNorm listing) */
  int32_t shared_classifier; /* 1 tied, 0 untied, -1 infer from blob size */
} orc_config;

/* Bytes of the packed blob for cfg with the classifier tied (tied=1) or not. */
int64_t orc_blob_bytes(const orc_config* cfg, int tied);
/* Byte offset of tensor `which` (0 E, 1 g_att, 2 Wq, 3 Wk, 4 Wv, 5 Wo,
 * 6 g_ffn, 7 W1, 8 W3, 9 W2, 10 g_final, 11 Wcls) of layer `layer` (ignored
 * for 0, 10, 11); -1 if absent (Wcls when tied). */
int64_t orc_tensor_offset(const orc_config* cfg, int tied, int which, int layer);

/* Model handle: acc_bits 64 (double accumulators and activations) or 32.
 * The blob is borrowed (not copied) and must outlive the handle.
 * Returns NULL and sets *err (1 invalid config, 2 size mismatch, 4 no memory). */
void* orc_model_new(const orc_config* cfg, const void* blob, size_t blob_bytes,
                    int acc_bits, int* err);
/* Same, with every weight matrix replaced by codes and row scales, quantized
 * at construction as orc_quantize_rows_q8 (weight_bits 8) or
 * orc_quantize_rows_q4 (weight_bits 4) defines; 0 keeps float32. */
void* orc_model_new_fmt(const orc_config* cfg, const void* blob, size_t blob_bytes,
                        int acc_bits, int weight_bits, int* err);
/* One decode step (token at position pos); writes vocab_size logits.
 * Returns 0, or 6 when token/pos is out of range. */
int orc_forward(void* model, int32_t token, int32_t pos, double* logits);
int orc_model_tied(const void* model);
void orc_model_free(void* model);

/* Primitives, exposed so that tests can pin each one on its own. */
/* Weight-only 8-bit codes of W [M x K]: s[i] = max_j |W[i][j]| / 127 and
 * q[i][j] = nearest integer (ties to even) to W[i][j] / s[i], all in float32
 * (0 codes and scale for an all-zero row). */
void orc_quantize_rows_q8(const float* W, int64_t M, int64_t K, int8_t* q, float* s);
/* Weight-only 4-bit codes (quantization future work, read as symmetric
 * per-row codes like the 8-bit ones): s[i] = max_j |W[i][j]| / 7 and q[i][j]
 * = nearest integer (ties to even) to W[i][j] / s[i], in [-7, 7], all in
 * float32; one code per int8 (the packing is the GPU format's business). */
void orc_quantize_rows_q4(const float* W, int64_t M, int64_t K, int8_t* q, float* s);
/* y[i] = sum_j (s[i] * q[i][j]) * x[j] in double (8-bit or 4-bit codes). */
void orc_gemv_q8_f64(const int8_t* q, const float* s, const double* x, double* y, int64_t M,
                     int64_t K);
void orc_gemv_f64(const float* W, const double* x, double* y, int64_t M, int64_t K);
void orc_gemv_f32(const float* W, const float* x, float* y, int64_t M, int64_t K);
void orc_rmsnorm_f64(const double* x, const float* g, double* out, int64_t n, double eps);
void orc_rope_f64(double* v, int64_t n, int64_t head_dim, int32_t pos, double theta);
void orc_softmax_f64(double* s, int64_t n);
double orc_silu_f64(double z);
/* One attention head over positions 0..npos-1: q [hd]; K and V rows of hd
 * values, `stride` values apart; out [hd]. */
void orc_attention_head_f64(const double* q, const double* K, const double* V,
                            int64_t npos, int64_t hd, int64_t stride, double* out);

#ifdef __cplusplus
}
#endif
#endif
