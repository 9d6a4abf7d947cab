// prefill.cu — multi-token prefill: n prompt tokens of one sequence at
// positions start .. start + n - 1 run through every layer as blocks of rows,
// writing their K/V rows into the cache (slot 0), and the last position's
// logits come out. It is the same computation as n decode steps (paper §2.1
// and §7.1 define the step; here the positions of a prompt share each layer's
// weight reads), so its results equal n tvl_forward calls up to float
// rounding. The products with the weight matrices are plain GEMMs
// ([n x K] times [K x M]) and go to cuBLAS SGEMM in float32; the rest —
// embedding rows, RMSNorm, RoPE and the cache write, causal attention, SwiGLU,
// the residual adds — are the kernels below.
#include <cublas_v2.h>

#include <cmath>
#include <string>

#include "model.h"

using namespace tvl;

namespace {

constexpr int kRowThreads = 256;

__device__ __forceinline__ float warp_sum32(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// x[i] = E[tok[i]] (paper §4.1: a row of the embedding table).
__global__ void embed_rows_kernel(const float* __restrict__ E, const int* __restrict__ tok,
                                  float* __restrict__ x, int d) {
  const float4* src = reinterpret_cast<const float4*>(E + (size_t)tok[blockIdx.x] * d);
  float4* dst = reinterpret_cast<float4*>(x + (size_t)blockIdx.x * d);
  for (int j = threadIdx.x; j < d / 4; j += blockDim.x) dst[j] = src[j];
}

// Row i (one block): x_i += add_i when add is given (the residual update),
// then out_{i - row0} = RMSNorm(x_i, g) = (x_i * g) * 1/sqrt(mean x_i^2 + eps)
// (§11.2); g null: the gain is already in the columns of the next matrix
// (tvl_load folds it there for float32 rows), so out = x_i * r. Rows
// [row0, row0 + gridDim.x); out may be add (each row is read in full before it
// is written).
__global__ void rmsnorm_rows_kernel(float* x, const float* add, const float* __restrict__ g,
                                    float* out, int row0, int d, float eps) {
  __shared__ float red[kRowThreads / 32];
  const int i = row0 + blockIdx.x;
  float* xr = x + (size_t)i * d;
  float ss = 0.f;
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    float v = xr[j];
    if (add) {
      v += add[(size_t)i * d + j];
      xr[j] = v;
    }
    ss = fmaf(v, v, ss);
  }
  ss = warp_sum32(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
  const float r = 1.0f / sqrtf(tot / (float)d + eps);
  float* o = out + (size_t)blockIdx.x * d;
  for (int j = threadIdx.x; j < d; j += blockDim.x) o[j] = (g ? xr[j] * g[j] : xr[j]) * r;
}

// RoPE on q and k of row i (position start + i): pair (2m, 2m+1) of a head
// turns by pos * theta^(-2m/hd) (table `rope`, [S][hd/2] of (cos, sin));
// then k and v go into the cache rows of that position.
__global__ void rope_kv_kernel(float* __restrict__ qkv, const float2* __restrict__ rope,
                               float* __restrict__ kc, float* __restrict__ vc, int start, int d,
                               int kvd, int hd) {
  const int i = blockIdx.x, pos = start + i, half = hd / 2;
  float* row = qkv + (size_t)i * (d + 2 * kvd);
  const float2* rp = rope + (size_t)pos * half;
  const int nq = d / 2, nk = kvd / 2;
  for (int t = threadIdx.x; t < nq + nk; t += blockDim.x) {
    float* v = t < nq ? row + 2 * t : row + d + 2 * (t - nq);
    const int m = (t < nq ? t : t - nq) % half;
    const float2 cs = rp[m];
    const float x0 = v[0], x1 = v[1];
    v[0] = x0 * cs.x - x1 * cs.y;
    v[1] = x0 * cs.y + x1 * cs.x;
  }
  __syncthreads();
  float* kd = kc + (size_t)pos * kvd;
  float* vd = vc + (size_t)pos * kvd;
  for (int j = threadIdx.x; j < kvd; j += blockDim.x) {
    kd[j] = row[d + j];
    vd[j] = row[d + kvd + j];
  }
}

// Causal attention, one warp per (row i, query head h): softmax over the
// positions 0 .. start + i of q . k_t / sqrt(hd), times V (§2.1), with a
// running max and sum (online softmax). Lane l holds elements l, l + 32, ...
// of the head (hd <= 128). Four positions per step, their dot products
// reduced together.
__global__ void attention_rows_kernel(const float* __restrict__ qkv, const float* __restrict__ kc,
                                      const float* __restrict__ vc, float* __restrict__ att,
                                      int n, int start, int d, int kvd, int hd, int H, int Hkv,
                                      float scale) {
  const int gw = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (gw >= n * H) return;
  const int lane = threadIdx.x & 31;
  const int i = gw / H, h = gw - i * H, kvh = h / (H / Hkv);
  const int pos = start + i;
  const float* q = qkv + (size_t)i * (d + 2 * kvd) + h * hd;
  constexpr int kMaxPer = 4;  // hd <= 128
  float qv[kMaxPer], o[kMaxPer];
#pragma unroll
  for (int u = 0; u < kMaxPer; ++u) {
    const int j = lane + 32 * u;
    qv[u] = j < hd ? q[j] : 0.f;
    o[u] = 0.f;
  }
  const float* kb = kc + kvh * hd;
  const float* vb = vc + kvh * hd;
  float m = -INFINITY, l = 0.f;
  for (int t0 = 0; t0 <= pos; t0 += 4) {
    float s[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int t = t0 + r;
      float acc = 0.f;
      if (t <= pos) {
        const float* k = kb + (size_t)t * kvd;
#pragma unroll
        for (int u = 0; u < kMaxPer; ++u) {
          const int j = lane + 32 * u;
          if (j < hd) acc = fmaf(qv[u], k[j], acc);
        }
      }
      s[r] = acc;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
      for (int r = 0; r < 4; ++r) s[r] += __shfl_xor_sync(0xffffffffu, s[r], off);
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int t = t0 + r;
      if (t > pos) break;
      const float sc = s[r] * scale;
      const float mn = fmaxf(m, sc);
      const float c = expf(m - mn), e = expf(sc - mn);
      l = l * c + e;
      const float* v = vb + (size_t)t * kvd;
#pragma unroll
      for (int u = 0; u < kMaxPer; ++u) {
        const int j = lane + 32 * u;
        if (j < hd) o[u] = fmaf(e, v[j], o[u] * c);
      }
      m = mn;
    }
  }
  float* out = att + (size_t)i * d + h * hd;
#pragma unroll
  for (int u = 0; u < kMaxPer; ++u) {
    const int j = lane + 32 * u;
    if (j < hd) out[j] = o[u] / l;
  }
}

// h[i][j] = silu(a) * b with (a, b) = rows (2j, 2j + 1) of the interleaved
// W1/W3 output (§2.1, SwiGLU).
__global__ void swiglu_rows_kernel(const float* __restrict__ h13, float* __restrict__ h,
                                   long long total) {
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const float a = h13[2 * t], b = h13[2 * t + 1];
    h[t] = (a / (1.0f + expf(-a))) * b;
  }
}

tvl_status blas_fail(cublasStatus_t s, const char* what) {
  set_error(std::string(what) + " failed (cuBLAS status " + std::to_string((int)s) + ")");
  return TVL_E_CUDA;
}

#define TVL_BLAS(call)                                  \
  do {                                                  \
    cublasStatus_t s_ = (call);                         \
    if (s_ != CUBLAS_STATUS_SUCCESS) return blas_fail(s_, #call); \
  } while (0)

// Y[rows x M] = X[rows x K] W^T, W row-major [M x K], everything row-major.
tvl_status gemm_rows(cublasHandle_t h, const float* W, const float* X, float* Y, int rows, int M,
                     int K) {
  const float one = 1.f, zero = 0.f;
  TVL_BLAS(cublasSgemm(h, CUBLAS_OP_T, CUBLAS_OP_N, M, rows, K, &one, W, K, X, K, &zero, Y, M));
  return TVL_OK;
}

bool on_device(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

}  // namespace

void prefill_release(tvl_model* m) {
  if (m->blas) cublasDestroy(static_cast<cublasHandle_t>(m->blas));
  lib_free(m->pf);
  m->blas = nullptr;
  m->pf = nullptr;
  m->pf_bytes = 0;
}

extern "C" tvl_status tvl_prefill(tvl_model* m, const int32_t* tokens, int32_t n,
                                  int32_t start_pos, float* logits_out) {
  if (!m || !tokens) {
    set_error("tvl_prefill: null argument");
    return TVL_E_INVAL;
  }
  if (m->sticky != TVL_OK) return m->sticky;
  if (m->cfg.weight_bits != 0) {
    set_error("tvl_prefill: needs float32 weights (weight_bits 0)");
    return TVL_E_UNSUPPORTED;
  }
  const tvl_config& c = m->cfg;
  if (n < 1 || start_pos < 0 || (int64_t)start_pos + n > c.max_seq) {
    set_error("tvl_prefill: n or start_pos out of range");
    return TVL_E_RANGE;
  }
  for (int i = 0; i < n; ++i)
    if (tokens[i] < 0 || tokens[i] >= c.vocab_size) {
      set_error("tvl_prefill: token out of range");
      return TVL_E_RANGE;
    }
  const DecodeArgs& a = m->args;
  const int d = a.d, F = a.F, kvd = a.kvd, hd = a.hd, S = a.S, L = a.L, V = a.V;
  cudaStream_t st = m->stream;
  // activations of up to S rows: x, x_b, qkv, att, h13, h; the last row's
  // normalised vector; the tokens
  const size_t fx = (size_t)S * d, fqkv = (size_t)S * (d + 2 * kvd), fh13 = (size_t)S * 2 * F,
               fh = (size_t)S * F;
  const size_t need = 4 * (3 * fx + fqkv + fh13 + fh + d) + 4 * (size_t)S + 256;
  if (!m->pf) {
    TVL_CK(lib_malloc((void**)&m->pf, need));
    m->pf_bytes = need;
  }
  if (!m->blas) {
    cublasHandle_t h = nullptr;
    TVL_BLAS(cublasCreate(&h));
    m->blas = h;
    TVL_BLAS(cublasSetMathMode(h, CUBLAS_DEFAULT_MATH));  // float32 products and sums
  }
  cublasHandle_t bh = static_cast<cublasHandle_t>(m->blas);
  TVL_BLAS(cublasSetStream(bh, st));
  float* X = m->pf;
  float* XB = X + fx;
  float* QKV = XB + fx;
  float* ATT = QKV + fqkv;
  float* H13 = ATT + fx;
  float* Hh = H13 + fh13;
  float* XN = Hh + fh;
  int* tok = reinterpret_cast<int*>(XN + d);
  TVL_CK(cudaMemcpyAsync(tok, tokens, 4ull * n, cudaMemcpyHostToDevice, st));

  embed_rows_kernel<<<n, kRowThreads, 0, st>>>(a.E, tok, X, d);
  TVL_CK(cudaGetLastError());
  const float* pending = nullptr;  // residual update not yet added into X
  for (int l = 0; l < L; ++l) {
    const unsigned char* lw = a.layer0 + (size_t)l * a.layer_stride;
    const float* g_att = a.gains_folded ? nullptr : reinterpret_cast<const float*>(lw + a.o_gatt);
    const float* g_ffn = a.gains_folded ? nullptr : reinterpret_cast<const float*>(lw + a.o_gffn);
    const float* Wqkv = reinterpret_cast<const float*>(lw + a.o_wqkv);
    const float* Wo = reinterpret_cast<const float*>(lw + a.o_wo);
    const float* W13 = reinterpret_cast<const float*>(lw + a.o_w13);  // interleaved rows
    const float* W2 = reinterpret_cast<const float*>(lw + a.o_w2);
    float* kc = a.kc + (size_t)l * S * kvd;
    float* vc = a.vc + (size_t)l * S * kvd;
    rmsnorm_rows_kernel<<<n, kRowThreads, 0, st>>>(X, pending, g_att, XB, 0, d, a.eps);
    TVL_CK(cudaGetLastError());
    tvl_status s;
    if ((s = gemm_rows(bh, Wqkv, XB, QKV, n, d + 2 * kvd, d)) != TVL_OK) return s;
    rope_kv_kernel<<<n, kRowThreads, 0, st>>>(QKV, a.rope, kc, vc, start_pos, d, kvd, hd);
    TVL_CK(cudaGetLastError());
    const int warps = n * a.H, wpb = kRowThreads / 32;
    attention_rows_kernel<<<(warps + wpb - 1) / wpb, kRowThreads, 0, st>>>(
        QKV, kc, vc, ATT, n, start_pos, d, kvd, hd, a.H, a.Hkv, a.att_scale);
    TVL_CK(cudaGetLastError());
    if ((s = gemm_rows(bh, Wo, ATT, XB, n, d, d)) != TVL_OK) return s;  // XB = Wo o
    rmsnorm_rows_kernel<<<n, kRowThreads, 0, st>>>(X, XB, g_ffn, ATT, 0, d, a.eps);  // ATT = x_b
    TVL_CK(cudaGetLastError());
    if ((s = gemm_rows(bh, W13, ATT, H13, n, 2 * F, d)) != TVL_OK) return s;
    const long long tot = (long long)n * F;
    swiglu_rows_kernel<<<(int)std::min<long long>((tot + 255) / 256, 4096), 256, 0, st>>>(H13, Hh,
                                                                                        tot);
    TVL_CK(cudaGetLastError());
    if ((s = gemm_rows(bh, W2, Hh, XB, n, d, F)) != TVL_OK) return s;  // XB = W2 h
    pending = XB;
  }
  // the last position: x += (last update), x_b = RMSNorm(x, g_final), logits = Wcls x_b
  rmsnorm_rows_kernel<<<1, kRowThreads, 0, st>>>(X, pending, a.final_gain_folded ? nullptr : a.g_final,
                                                  XN, n - 1, d, a.eps);
  TVL_CK(cudaGetLastError());
  {
    const float one = 1.f, zero = 0.f;
    TVL_BLAS(cublasSgemv(bh, CUBLAS_OP_T, d, V, &one, a.Wcls, d, XN, 1, &zero, a.logits, 1));
  }
  if (!logits_out) return TVL_OK;
  const size_t bytes = (size_t)V * 4;
  if (on_device(logits_out)) {
    TVL_CK(cudaMemcpyAsync(logits_out, a.logits, bytes, cudaMemcpyDeviceToDevice, st));
    return TVL_OK;
  }
  TVL_CK(cudaMemcpyAsync(logits_out, a.logits, bytes, cudaMemcpyDeviceToHost, st));
  TVL_CK(cudaStreamSynchronize(st));
  return TVL_OK;
}
