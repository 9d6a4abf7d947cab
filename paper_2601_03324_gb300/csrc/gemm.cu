// gemm.cu — Y = X W^T in float32 accuracy on the tensor cores (tcgen05), for
// products of a block of positions with the weight matrices (multi-token
// prefill: the computation of n decode steps, paper §2.1 and §7.1, with each
// weight read once for all n positions).
//
// Float32 accuracy from bf16 tensor-core products: every float a is split
// into a_hi = bf16(a) and a_lo = bf16(a - a_hi), and
//   sum_k w x  ~  sum_k (w_hi x_hi + w_hi x_lo + w_lo x_hi)
// accumulated in fp32 in tensor memory. The dropped w_lo x_lo term and the
// representation error of the split are about 2^-16 of each product, far
// below the float32 decode tolerances (the rounding of plain float32 sums of
// K = 4096 terms is of the same order).
//
// One CTA computes a 128 x 128 tile D[m][n] = sum_k W[m][k] X[n][k] (W rows on
// the MMA's M side, positions on its N side; both operands K-major):
//   warp 4 (one thread): TMA loads of W_hi, W_lo, X_hi, X_lo k-blocks of 64
//     into a ring of stages (128-byte swizzle), completing on mbarriers;
//   warp 5 (one thread): per k-block 4 K-steps x 3 tcgen05.mma into one TMEM
//     accumulator, then tcgen05.commit frees the stage;
//   warps 0-3: wait for the last commit, read the accumulator with tcgen05.ld
//     (warp w holds rows 32w..32w+31) and store Y[n][m] (coalesced along m).
// Every wait is bounded (one second); a CTA that gives up raises TVL_E_TIMEOUT
// in the error word and stores nothing.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <map>
#include <mutex>
#include <string>
#include <utility>

#include "gemm.h"
#include "tc.cuh"

namespace tvl {

constexpr int kGemmBM = 128;   // W rows per tile (MMA M)
constexpr int kGemmBN = 128;   // positions per tile (MMA N; TMEM columns)
constexpr int kGemmBK = 64;    // K per stage: 64 bf16, one 128-byte swizzle row
constexpr int kGemmStages = 3;
constexpr int kGemmThreads = 192;
constexpr int kTileW = kGemmBM * kGemmBK * 2;  // 16 KB
constexpr int kTileX = kGemmBN * kGemmBK * 2;  // 16 KB
constexpr int kGemmStage = 2 * kTileW + 2 * kTileX;
constexpr int kGemmSmem = kGemmStages * kGemmStage + 1024 + 256;
constexpr unsigned long long kGemmWaitNs = 1000000000ull;

struct GemmArgs {
  float* Y;
  int n, M, K, ldy;
  int* err;
};

// Bounded wait on an mbarrier phase; gives up on the CTA's abort flag.
__device__ inline bool gemm_wait(uint64_t* bar, uint32_t par, volatile int* s_abort) {
  if (mbar_try_wait(bar, par)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, par)) return true;
    if ((it & 15u) == 0) {
      if (*s_abort) return false;
      if (globaltimer_ns() - t0 > kGemmWaitNs || it > (1u << 26)) return false;
    }
  }
}

__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_bf16x3_kernel(const __grid_constant__ CUtensorMap tWh,
                       const __grid_constant__ CUtensorMap tWl,
                       const __grid_constant__ CUtensorMap tXh,
                       const __grid_constant__ CUtensorMap tXl, const __grid_constant__ GemmArgs a) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kGemmStages * kGemmStage);
  uint64_t* empty = full + kGemmStages;
  uint64_t* done = empty + kGemmStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * kGemmBM, n0 = blockIdx.y * kGemmBN;
  const int nkb = (a.K + kGemmBK - 1) / kGemmBK;
  auto tile_wh = [&](int s) { return smem + s * kGemmStage; };
  auto tile_wl = [&](int s) { return smem + s * kGemmStage + kTileW; };
  auto tile_xh = [&](int s) { return smem + s * kGemmStage + 2 * kTileW; };
  auto tile_xl = [&](int s) { return smem + s * kGemmStage + 2 * kTileW + kTileX; };
  if (threadIdx.x == 0) {
    for (int s = 0; s < kGemmStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    *s_abort = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, kGemmBN);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 4) {
    if (lane == 0) {  // TMA producer
      int kb = 0;
      for (; kb < nkb; ++kb) {
        const int s = kb % kGemmStages;
        if (kb >= kGemmStages && !gemm_wait(&empty[s], ((kb / kGemmStages) - 1) & 1, s_abort)) {
          *s_abort = 1;
          break;
        }
        mbar_arrive_expect_tx(&full[s], kGemmStage);
        const int k = kb * kGemmBK;
        tma_load_2d(tile_wh(s), &tWh, k, m0, &full[s]);
        tma_load_2d(tile_wl(s), &tWl, k, m0, &full[s]);
        tma_load_2d(tile_xh(s), &tXh, k, n0, &full[s]);
        tma_load_2d(tile_xl(s), &tXl, k, n0, &full[s]);
      }
      // every load issued has landed before the CTA may exit
      for (int j = kb - kGemmStages > 0 ? kb - kGemmStages : 0; j < kb; ++j) {
        const int s = j % kGemmStages;
        if (!mbar_try_wait(&full[s], (j / kGemmStages) & 1)) {
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(&full[s], (j / kGemmStages) & 1) &&
                 globaltimer_ns() - t0 < kGemmWaitNs) {
          }
        }
      }
    }
  } else if (warp == 5) {
    if (lane == 0) {  // MMA issuer
      constexpr uint32_t idesc = umma_idesc_bf16_f32(kGemmBM, kGemmBN);
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % kGemmStages;
        if (!gemm_wait(&full[s], (kb / kGemmStages) & 1, s_abort)) {
          *s_abort = 1;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kGemmBK / 16; ++kk) {
          const uint64_t wh = umma_desc_sw128(tile_wh(s) + 32 * kk);
          const uint64_t wl = umma_desc_sw128(tile_wl(s) + 32 * kk);
          const uint64_t xh = umma_desc_sw128(tile_xh(s) + 32 * kk);
          const uint64_t xl = umma_desc_sw128(tile_xl(s) + 32 * kk);
          tc_mma_bf16(tmem, wl, xh, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          tc_mma_bf16(tmem, wh, xl, idesc, 1u);
          tc_mma_bf16(tmem, wh, xh, idesc, 1u);
        }
        tc_commit(&empty[s]);  // the stage is free once these products are done
      }
      tc_commit(done);  // every product issued above has completed
    }
  } else {  // epilogue: warps 0-3 hold TMEM lanes 32w .. 32w + 31 (rows of the tile)
    bool ok = true;
    if (lane == 0) ok = gemm_wait(done, 0, s_abort);
    ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    tc_fence_after();
    if (!ok || *s_abort) {
      if (lane == 0) {
        atomicCAS(a.err, 0, 7);
        *s_abort = 1;
      }
    } else {
      const int m = m0 + warp * 32 + lane;
      const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
      for (int c = 0; c < kGemmBN; c += 16) {
        float v[16];
        tc_ld16(trow + (uint32_t)c, v);
        if (m < a.M) {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int n = n0 + c + j;
            if (n < a.n) a.Y[(size_t)n * a.ldy + m] = v[j];
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kGemmBN);
  }
}

// hi = bf16(v), lo = bf16(v - hi) for count floats (round to nearest).
__global__ void split_bf16_kernel(const float* __restrict__ src, __nv_bfloat16* __restrict__ hi,
                                  __nv_bfloat16* __restrict__ lo, long long count) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < count;
       i += (long long)gridDim.x * blockDim.x) {
    store_bf16_parts(hi, lo, (size_t)i, src[i]);
  }
}

}  // namespace tvl

using namespace tvl;

namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::mutex g_encode_mu;

tvl_status encoder(PFN_cuTensorMapEncodeTiled_v12000* out) {
  std::lock_guard<std::mutex> lk(g_encode_mu);
  if (!g_encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q{};
    TVL_CK(cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                            cudaEnableDefault, &q));
    if (q != cudaDriverEntryPointSuccess || !fn) {
      set_error("cuTensorMapEncodeTiled is not available from the driver");
      return TVL_E_CUDA;
    }
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  *out = g_encode;
  return TVL_OK;
}

// 2-D map of a row-major bf16 matrix [rows x cols], box [box_rows x 64],
// 128-byte swizzle, zeros outside the matrix.
tvl_status bf16_map(CUtensorMap* map, const void* base, long long rows, long long cols,
                    int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = nullptr;
  tvl_status st = encoder(&enc);
  if (st != TVL_OK) return st;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kGemmBK, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                         strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
    return TVL_E_CUDA;
  }
  return TVL_OK;
}

}  // namespace

namespace tvl {

tvl_status split_bf16(const float* src, void* hi, void* lo, long long count, cudaStream_t s) {
  const int blocks = (int)std::min<long long>((count + 255) / 256, 8192);
  split_bf16_kernel<<<blocks, 256, 0, s>>>(src, reinterpret_cast<__nv_bfloat16*>(hi),
                                           reinterpret_cast<__nv_bfloat16*>(lo), count);
  TVL_CK(cudaGetLastError());
  return TVL_OK;
}

tvl_status gemm_bf16x3(const void* w_hi, const void* w_lo, const void* x_hi, const void* x_lo,
                       float* Y, int n, int M, int K, int ldy, int* err, cudaStream_t s) {
  if (n < 1 || M < 1 || K < 1 || K % 8 != 0 || ldy < M) {
    set_error("gemm: n, M, K >= 1, K % 8 == 0 and ldy >= M are required");
    return TVL_E_INVAL;
  }
  static std::mutex mu;
  static bool attr_set[64] = {};
  int dev = 0;
  TVL_CK(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 64) {
    set_error("gemm: device ordinal beyond the 64-entry table");
    return TVL_E_UNSUPPORTED;
  }
  {
    std::lock_guard<std::mutex> lk(mu);
    if (!attr_set[dev]) {
      TVL_CK(cudaFuncSetAttribute((const void*)gemm_bf16x3_kernel,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, kGemmSmem));
      attr_set[dev] = true;
    }
  }
  CUtensorMap mwh, mwl, mxh, mxl;
  tvl_status st;
  if ((st = bf16_map(&mwh, w_hi, M, K, kGemmBM)) != TVL_OK) return st;
  if ((st = bf16_map(&mwl, w_lo, M, K, kGemmBM)) != TVL_OK) return st;
  if ((st = bf16_map(&mxh, x_hi, n, K, kGemmBN)) != TVL_OK) return st;
  if ((st = bf16_map(&mxl, x_lo, n, K, kGemmBN)) != TVL_OK) return st;
  GemmArgs a{Y, n, M, K, ldy, err};
  const dim3 grid((M + kGemmBM - 1) / kGemmBM, (n + kGemmBN - 1) / kGemmBN);
  gemm_bf16x3_kernel<<<grid, kGemmThreads, kGemmSmem, s>>>(mwh, mwl, mxh, mxl, a);
  TVL_CK(cudaGetLastError());
  return TVL_OK;
}

}  // namespace tvl

// ---- tvl_gemm: the standalone entry point ------------------------------------------

namespace {

static __device__ int g_gemm_err;

struct GemmScratch {
  void* buf = nullptr;  // W_hi | W_lo | X_hi | X_lo
  size_t bytes = 0;
};
std::mutex g_gemm_mu;
std::map<std::pair<int, cudaStream_t>, GemmScratch> g_gemm_ws;

}  // namespace

namespace tvl {

tvl_status gemm_error_word(int** out) {
  void* e = nullptr;
  TVL_CK(cudaGetSymbolAddress(&e, g_gemm_err));
  *out = reinterpret_cast<int*>(e);
  return TVL_OK;
}

}  // namespace tvl

extern "C" tvl_status tvl_gemm(const float* W, const float* X, float* Y, int32_t n, int32_t M,
                               int32_t K, void* stream) {
  if (!W || !X || !Y || n < 1 || M < 1 || K < 1) {
    set_error("tvl_gemm: null pointer or non-positive size");
    return TVL_E_INVAL;
  }
  if (K % 8 != 0) {
    set_error("tvl_gemm: K must be a multiple of 8 (16-byte rows of bf16 parts)");
    return TVL_E_UNSUPPORTED;
  }
  cudaStream_t s = (cudaStream_t)stream;
  int dev = 0;
  TVL_CK(cudaGetDevice(&dev));
  // every part 256-byte aligned (TMA needs 16)
  auto al = [](size_t b) { return (b + 255) / 256 * 256; };
  const size_t wpart = al((size_t)M * K * 2), xpart = al((size_t)n * K * 2);
  const size_t need = 2 * (wpart + xpart);
  unsigned char* buf = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_gemm_mu);
    GemmScratch& ws = g_gemm_ws[{dev, s}];
    if (ws.bytes < need) {
      if (ws.buf) {  // earlier kernels on this stream may still read the old buffer
        TVL_CK(cudaStreamSynchronize(s));
        lib_free(ws.buf);
        ws.buf = nullptr;
        ws.bytes = 0;
      }
      const cudaError_t e = lib_malloc(&ws.buf, need);
      if (e != cudaSuccess) return cuda_fail(e, "tvl_gemm: scratch");
      ws.bytes = need;
    }
    buf = static_cast<unsigned char*>(ws.buf);
  }
  unsigned char* wh = buf;
  unsigned char* wl = wh + wpart;
  unsigned char* xh = wl + wpart;
  unsigned char* xl = xh + xpart;
  tvl_status st = split_bf16(W, wh, wl, (long long)M * K, s);
  if (st == TVL_OK) st = split_bf16(X, xh, xl, (long long)n * K, s);
  int* err = nullptr;
  if (st == TVL_OK) st = gemm_error_word(&err);
  if (st == TVL_OK) st = gemm_bf16x3(wh, wl, xh, xl, Y, n, M, K, M, err, s);
  return st;
}

extern "C" tvl_status tvl_gemm_status(void* stream) {
  TVL_CK(cudaStreamSynchronize((cudaStream_t)stream));
  int code = 0;
  TVL_CK(cudaMemcpyFromSymbol(&code, g_gemm_err, sizeof(int)));
  if (code == 0) return TVL_OK;
  const int zero = 0;
  TVL_CK(cudaMemcpyToSymbol(g_gemm_err, &zero, sizeof(int)));
  set_error("a bounded wait in the tensor-core GEMM expired; that call's Y is incomplete");
  return (tvl_status)code;
}
