// gemm.h — the tensor-core GEMM of gemm.cu for the library's other host files.
#pragma once
#include <cuda_bf16.h>

#include "host_common.h"

namespace tvl {

// The bf16 parts of a float32 value v, hi = bf16(v) and lo = bf16(v - hi),
// stored at index i of hi and lo: the form in which the products below take
// their operands.
__device__ __forceinline__ void store_bf16_parts(__nv_bfloat16* hi, __nv_bfloat16* lo, size_t i,
                                                 float v) {
  const __nv_bfloat16 h = __float2bfloat16_rn(v);
  hi[i] = h;
  lo[i] = __float2bfloat16_rn(v - __bfloat162float(h));
}

// hi = bf16(src), lo = bf16(src - hi), count floats, on stream s.
tvl_status split_bf16(const float* src, void* hi, void* lo, long long count, cudaStream_t s);

// Y[i][m] (row stride ldy) = sum_k W[m][k] X[i][k] for i < n, m < M, in float32
// accuracy from the bf16 parts (w_hi, w_lo: [M x K]; x_hi, x_lo: [n x K];
// 16-byte aligned, K % 8 == 0). err: device word that receives TVL_E_TIMEOUT
// if a bounded wait in the kernel runs out. Queued on s.
tvl_status gemm_bf16x3(const void* w_hi, const void* w_lo, const void* x_hi, const void* x_lo,
                       float* Y, int n, int M, int K, int ldy, int* err, cudaStream_t s);

// Device address of the tensor-core GEMM's error word on the current device
// (the word tvl_gemm_status reads).
tvl_status gemm_error_word(int** out);

}  // namespace tvl
