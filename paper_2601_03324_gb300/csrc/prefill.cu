// prefill.cu — multi-token prefill: n prompt tokens of one sequence at
// positions start .. start + n - 1 run through every layer as blocks of rows,
// writing their K/V rows into the cache (slot 0), and the last position's
// logits come out. It is the same computation as n decode steps (paper §2.1
// and §7.1 define the step; here the positions of a prompt share each layer's
// weight reads), so its results equal n tvl_forward calls up to float
// rounding. The products with the weight matrices ([n x K] times [K x M])
// run on the tensor cores (gemm.cu: tcgen05, bf16 parts of every float, fp32
// accumulation, float32 accuracy); the bf16 parts of the weights are made
// once, at the first call. The rest — embedding rows, RMSNorm, RoPE and the
// cache write, causal attention, SwiGLU, the residual adds — are the kernels
// below, and the classifier row of the last position is the library's
// streaming GEMV.
#include <cmath>
#include <string>

#include "gemm.h"
#include "model.h"

using namespace tvl;

namespace {

constexpr int kRowThreads = 256;

// Where a kernel puts rows that a weight product reads next: the bf16 parts
// (hi, lo) that the tensor-core GEMM takes, written here so that no separate
// split pass runs; or plain floats (f) when hi is null.
struct RowOut {
  float* f;
  __nv_bfloat16* hi;
  __nv_bfloat16* lo;
  __device__ __forceinline__ void put(size_t i, float v) const {
    if (hi) store_bf16_parts(hi, lo, i, v);
    else f[i] = v;
  }
  // four values at i, a multiple of 4: one 16-byte or two 8-byte stores
  __device__ __forceinline__ void put4(size_t i, float4 v) const {
    if (hi) {
      const __nv_bfloat162 h01 = __floats2bfloat162_rn(v.x, v.y), h23 = __floats2bfloat162_rn(v.z, v.w);
      const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
      const __nv_bfloat162 l01 = __floats2bfloat162_rn(v.x - f01.x, v.y - f01.y);
      const __nv_bfloat162 l23 = __floats2bfloat162_rn(v.z - f23.x, v.w - f23.y);
      uint2 hv, lv;
      hv.x = *reinterpret_cast<const unsigned*>(&h01);
      hv.y = *reinterpret_cast<const unsigned*>(&h23);
      lv.x = *reinterpret_cast<const unsigned*>(&l01);
      lv.y = *reinterpret_cast<const unsigned*>(&l23);
      *reinterpret_cast<uint2*>(hi + i) = hv;
      *reinterpret_cast<uint2*>(lo + i) = lv;
    } else {
      *reinterpret_cast<float4*>(f + i) = v;
    }
  }
};

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
// [row0, row0 + gridDim.x); out's floats may be add (each row is read in full
// before it is written).
__global__ void rmsnorm_rows_kernel(float* x, const float* add, const float* __restrict__ g,
                                    RowOut out, int row0, int d, float eps) {
  __shared__ float red[kRowThreads / 32];
  const int i = row0 + blockIdx.x;
  float4* xr = reinterpret_cast<float4*>(x + (size_t)i * d);  // d % 32 == 0
  const float4* ar = add ? reinterpret_cast<const float4*>(add + (size_t)i * d) : nullptr;
  const float4* g4 = reinterpret_cast<const float4*>(g);
  const int d4 = d >> 2;
  float ss = 0.f;
  for (int j = threadIdx.x; j < d4; j += blockDim.x) {
    float4 v = xr[j];
    if (ar) {
      const float4 u = ar[j];
      v = make_float4(v.x + u.x, v.y + u.y, v.z + u.z, v.w + u.w);
      xr[j] = v;
    }
    ss = fmaf(v.x, v.x, fmaf(v.y, v.y, fmaf(v.z, v.z, fmaf(v.w, v.w, ss))));
  }
  ss = warp_sum32(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
  const float r = 1.0f / sqrtf(tot / (float)d + eps);
  const size_t o = (size_t)blockIdx.x * d;
  for (int j = threadIdx.x; j < d4; j += blockDim.x) {
    float4 v = xr[j];
    if (g4) {
      const float4 gg = g4[j];
      v = make_float4(v.x * gg.x, v.y * gg.y, v.z * gg.z, v.w * gg.w);
    }
    out.put4(o + 4 * j, make_float4(v.x * r, v.y * r, v.z * r, v.w * r));
  }
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
                                      const float* __restrict__ vc, RowOut att,
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
  const size_t out = (size_t)i * d + h * hd;
#pragma unroll
  for (int u = 0; u < kMaxPer; ++u) {
    const int j = lane + 32 * u;
    if (j < hd) att.put(out + j, o[u] / l);
  }
}

// Causal attention of a block of queries, tiled (§2.1; the same arithmetic as
// the per-row kernel above, in another order): one CTA of 128 threads takes 32
// consecutive query rows of one head and walks its share of the keys
// 0 .. (its last position) in tiles of 32 (split z of the key range:
// tiles [z T, (z + 1) T); with more than one split each CTA writes its rows'
// unnormalised partials (o, max, sum) to `part` and attention_merge_kernel
// combines them), with the Q, K and V tiles in shared memory (rows
// padded by 4 floats, so that the float4 reads below hit distinct banks).
// Thread (q, sub) = (tid / 4, tid % 4) scores keys sub, sub + 4, ..., sub + 28
// of each tile for query q, the four threads of a query share an online
// softmax (running max and sum, shuffles), and each accumulates its quarter of
// the output row: float4 chunks sub, sub + 4, ... of the head's dims. kDpt =
// head_dim / 4 (4 to 32, a multiple of 4).
constexpr int kAttBQ = 32, kAttBK = 32, kAttThreads = 128;
constexpr int kAttSplits = 8;  // key splits of the longest rows, at most

template <int kDpt>
__global__ void __launch_bounds__(kAttThreads)
    attention_tiles_kernel(const float* __restrict__ qkv, const float* __restrict__ kc,
                           const float* __restrict__ vc, RowOut att, int n, int start,
                           int d, int kvd, int H, int Hkv, float scale, int tiles_per_split,
                           float* __restrict__ part) {
  constexpr int hd = 4 * kDpt, hp = hd + 4, hd4 = kDpt, nc = kDpt / 4;
  extern __shared__ float sm[];
  float* Qs = sm;                  // [BQ][hp], scaled by 1/sqrt(hd)
  float* Ks = Qs + kAttBQ * hp;    // [BK][hp]
  float* Vs = Ks + kAttBK * hp;    // [BK][hp]
  float* Ps = Vs + kAttBK * hp;    // [BQ][BK + 1]
  const int h = blockIdx.y, kvh = h / (H / Hkv);
  const int i0 = blockIdx.x * kAttBQ;
  const int tid = threadIdx.x, q = tid >> 2, sub = tid & 3;
  const size_t rowlen = (size_t)d + 2 * kvd;
  const int last = min(start + i0 + kAttBQ - 1, start + n - 1);  // the tile's last position
  const int k_begin = blockIdx.z * tiles_per_split * kAttBK;
  if (k_begin > last) return;  // this split holds no key of these rows (uniform in the CTA)
  const int k_end = min(last, k_begin + tiles_per_split * kAttBK - 1);
  for (int e = tid; e < kAttBQ * hd4; e += kAttThreads) {
    const int r = e / hd4, c = e - r * hd4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i0 + r < n) v = reinterpret_cast<const float4*>(qkv + (size_t)(i0 + r) * rowlen + h * hd)[c];
    v.x *= scale;
    v.y *= scale;
    v.z *= scale;
    v.w *= scale;
    reinterpret_cast<float4*>(Qs + r * hp)[c] = v;
  }
  const int qpos = start + i0 + q;
  float m = -INFINITY, l = 0.f;
  float4 o[nc];
#pragma unroll
  for (int c = 0; c < nc; ++c) o[c] = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int t0 = k_begin; t0 <= k_end; t0 += kAttBK) {
    __syncthreads();  // the previous tile's K, V and P are read
    for (int e = tid; e < kAttBK * hd4; e += kAttThreads) {
      const int r = e / hd4, c = e - r * hd4, t = t0 + r;
      float4 kv = make_float4(0.f, 0.f, 0.f, 0.f), vv = kv;
      if (t <= k_end) {
        kv = reinterpret_cast<const float4*>(kc + (size_t)t * kvd + kvh * hd)[c];
        vv = reinterpret_cast<const float4*>(vc + (size_t)t * kvd + kvh * hd)[c];
      }
      reinterpret_cast<float4*>(Ks + r * hp)[c] = kv;
      reinterpret_cast<float4*>(Vs + r * hp)[c] = vv;
    }
    __syncthreads();
    float s[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) s[j] = 0.f;
#pragma unroll 4
    for (int c = 0; c < hd4; ++c) {
      const float4 qv = reinterpret_cast<const float4*>(Qs + q * hp)[c];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float4 kv = reinterpret_cast<const float4*>(Ks + (sub + 4 * j) * hp)[c];
        s[j] = fmaf(qv.x, kv.x, fmaf(qv.y, kv.y, fmaf(qv.z, kv.z, fmaf(qv.w, kv.w, s[j]))));
      }
    }
    float mt = -INFINITY;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (t0 + sub + 4 * j > qpos) s[j] = -INFINITY;  // causal: keys after the query
      mt = fmaxf(mt, s[j]);
    }
    mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 1));
    mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 2));
    // a query whose keys so far in this split are all after it has no
    // maximum yet (mn = -inf): nothing to add and nothing to rescale
    const float mn = fmaxf(m, mt);
    const bool none = mn == -INFINITY;
    const float corr = none ? 1.f : expf(m - mn);
    float ps = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      s[j] = none ? 0.f : expf(s[j] - mn);
      ps += s[j];
    }
    ps += __shfl_xor_sync(0xffffffffu, ps, 1);
    ps += __shfl_xor_sync(0xffffffffu, ps, 2);
    l = l * corr + ps;
    m = mn;
#pragma unroll
    for (int c = 0; c < nc; ++c) {
      o[c].x *= corr;
      o[c].y *= corr;
      o[c].z *= corr;
      o[c].w *= corr;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) Ps[q * (kAttBK + 1) + sub + 4 * j] = s[j];
    __syncwarp();  // the four threads of a query are lanes of one warp
#pragma unroll 4
    for (int k = 0; k < kAttBK; ++k) {
      const float p = Ps[q * (kAttBK + 1) + k];
      const float4* vr = reinterpret_cast<const float4*>(Vs + k * hp);
#pragma unroll
      for (int c = 0; c < nc; ++c) {
        const float4 v = vr[4 * c + sub];
        o[c].x = fmaf(p, v.x, o[c].x);
        o[c].y = fmaf(p, v.y, o[c].y);
        o[c].z = fmaf(p, v.z, o[c].z);
        o[c].w = fmaf(p, v.w, o[c].w);
      }
    }
  }
  if (i0 + q < n) {
    if (part) {  // partial of split z: o (unnormalised), then max and sum
      float* pr = part + (((size_t)blockIdx.z * n + i0 + q) * H + h) * (hd + 4);
      float4* out = reinterpret_cast<float4*>(pr);
#pragma unroll
      for (int c = 0; c < nc; ++c) out[4 * c + sub] = o[c];
      if (sub == 0) {
        pr[hd] = m;
        pr[hd + 1] = l;
      }
    } else {
      const float inv = 1.0f / l;
      const size_t out = (size_t)(i0 + q) * d + h * hd;
#pragma unroll
      for (int c = 0; c < nc; ++c) {
        const size_t e = out + 4 * (4 * c + sub);
        att.put(e, o[c].x * inv);
        att.put(e + 1, o[c].y * inv);
        att.put(e + 2, o[c].z * inv);
        att.put(e + 3, o[c].w * inv);
      }
    }
  }
}

// The same causal attention with more work per thread, for head dims that
// are multiples of 32 (kDpt = head_dim / 4 a multiple of 8): a CTA of 128
// threads takes 64 query rows of one head and walks its share of the keys in
// tiles of 32. The tile kernel above reads about one shared-memory value per
// multiply-add and is bound by the shared-memory port; here each thread keeps
// a 4 x 4 block of scores (queries 4g .. 4g + 3 of its group g = tid / 8,
// keys j, j + 8, j + 16, j + 24 of the tile for j = tid % 8) and a 4-query
// block of the output (float4 chunks j, j + 8, ... of the head's dims), so
// every value read from shared memory meets four others. The eight threads of
// a group are lanes of one warp: the scores' row maxima and sums are shuffles
// among them, and the softmax weights go through shared memory within the
// warp. Key splits and partials as above.
constexpr int kAtt2BQ = 64;

template <int kDpt>
__global__ void __launch_bounds__(kAttThreads)
    attention_tiles64_kernel(const float* __restrict__ qkv, const float* __restrict__ kc,
                             const float* __restrict__ vc, RowOut att, int n, int start,
                             int d, int kvd, int H, int Hkv, float scale, int tiles_per_split,
                             float* __restrict__ part) {
  constexpr int hd = 4 * kDpt, hp = hd + 4, hd4 = kDpt, nv = kDpt / 8;
  static_assert(kDpt % 8 == 0, "head_dim must be a multiple of 32");
  extern __shared__ __align__(16) float sm[];
  float* Qs = sm;                       // [64][hp], q * scale
  float* Ks = Qs + kAtt2BQ * hp;        // [32][hp]
  float* Vs = Ks + kAttBK * hp;         // [32][hp]
  float* Ps = Vs + kAttBK * hp;         // [64][33] softmax weights of the tile
  const int h = blockIdx.y, kvh = h / (H / Hkv);
  const int i0 = blockIdx.x * kAtt2BQ;
  const int tid = threadIdx.x, g = tid >> 3, j = tid & 7;
  const size_t rowlen = (size_t)d + 2 * kvd;
  const int last = min(start + i0 + kAtt2BQ - 1, start + n - 1);  // the block's last position
  const int k_begin = blockIdx.z * tiles_per_split * kAttBK;
  if (k_begin > last) return;  // this split holds no key of these rows (uniform in the CTA)
  const int k_end = min(last, k_begin + tiles_per_split * kAttBK - 1);
  for (int e = tid; e < kAtt2BQ * hd4; e += kAttThreads) {
    const int r = e / hd4, c = e - r * hd4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i0 + r < n) v = reinterpret_cast<const float4*>(qkv + (size_t)(i0 + r) * rowlen + h * hd)[c];
    reinterpret_cast<float4*>(Qs + r * hp)[c] =
        make_float4(v.x * scale, v.y * scale, v.z * scale, v.w * scale);
  }
  float m[4], l[4];
  float4 o[4][nv];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    m[i] = -INFINITY;
    l[i] = 0.f;
#pragma unroll
    for (int u = 0; u < nv; ++u) o[i][u] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  for (int t0 = k_begin; t0 <= k_end; t0 += kAttBK) {
    __syncthreads();  // the previous tile's K and V are read (and Q written, the first time)
    for (int e = tid; e < kAttBK * hd4; e += kAttThreads) {
      const int r = e / hd4, c = e - r * hd4, t = t0 + r;
      float4 kv = make_float4(0.f, 0.f, 0.f, 0.f), vv = kv;
      if (t <= k_end) {
        kv = reinterpret_cast<const float4*>(kc + (size_t)t * kvd + kvh * hd)[c];
        vv = reinterpret_cast<const float4*>(vc + (size_t)t * kvd + kvh * hd)[c];
      }
      reinterpret_cast<float4*>(Ks + r * hp)[c] = kv;
      reinterpret_cast<float4*>(Vs + r * hp)[c] = vv;
    }
    __syncthreads();
    float s[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) s[i][jj] = 0.f;
#pragma unroll 2
    for (int c = 0; c < hd4; ++c) {
      float4 qv[4], kv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) qv[i] = reinterpret_cast<const float4*>(Qs + (4 * g + i) * hp)[c];
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) kv[jj] = reinterpret_cast<const float4*>(Ks + (j + 8 * jj) * hp)[c];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int jj = 0; jj < 4; ++jj)
          s[i][jj] = fmaf(qv[i].x, kv[jj].x, fmaf(qv[i].y, kv[jj].y,
                     fmaf(qv[i].z, kv[jj].z, fmaf(qv[i].w, kv[jj].w, s[i][jj]))));
    }
    // online softmax per query over the eight lanes of the group
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int qpos = start + i0 + 4 * g + i;
      float mt = -INFINITY;
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        if (t0 + j + 8 * jj > qpos) s[i][jj] = -INFINITY;  // causal: keys after the query
        mt = fmaxf(mt, s[i][jj]);
      }
      mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 1));
      mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 2));
      mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 4));
      // a query whose keys so far in this split are all after it has no
      // maximum yet (mn = -inf): nothing to add and nothing to rescale
      const float mn = fmaxf(m[i], mt);
      const bool none = mn == -INFINITY;
      const float corr = none ? 1.f : expf(m[i] - mn);
      float ps = 0.f;
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        const float e = none ? 0.f : expf(s[i][jj] - mn);
        Ps[(4 * g + i) * (kAttBK + 1) + j + 8 * jj] = e;
        ps += e;
      }
      ps += __shfl_xor_sync(0xffffffffu, ps, 1);
      ps += __shfl_xor_sync(0xffffffffu, ps, 2);
      ps += __shfl_xor_sync(0xffffffffu, ps, 4);
      l[i] = l[i] * corr + ps;
      m[i] = mn;
#pragma unroll
      for (int u = 0; u < nv; ++u) {
        o[i][u].x *= corr;
        o[i][u].y *= corr;
        o[i][u].z *= corr;
        o[i][u].w *= corr;
      }
    }
    __syncwarp();  // the group's weights are written by lanes of this warp
#pragma unroll 2
    for (int k = 0; k < kAttBK; ++k) {
      float p[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) p[i] = Ps[(4 * g + i) * (kAttBK + 1) + k];
      const float4* vr = reinterpret_cast<const float4*>(Vs + k * hp);
#pragma unroll
      for (int u = 0; u < nv; ++u) {
        const float4 v = vr[j + 8 * u];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          o[i][u].x = fmaf(p[i], v.x, o[i][u].x);
          o[i][u].y = fmaf(p[i], v.y, o[i][u].y);
          o[i][u].z = fmaf(p[i], v.z, o[i][u].z);
          o[i][u].w = fmaf(p[i], v.w, o[i][u].w);
        }
      }
    }
    __syncwarp();  // the weights are read before the next tile writes them
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = i0 + 4 * g + i;
    if (row >= n) continue;
    if (part) {  // partial of split z: o (unnormalised), then max and sum
      float* pr = part + (((size_t)blockIdx.z * n + row) * H + h) * (hd + 4);
#pragma unroll
      for (int u = 0; u < nv; ++u) reinterpret_cast<float4*>(pr)[j + 8 * u] = o[i][u];
      if (j == 0) {
        pr[hd] = m[i];
        pr[hd + 1] = l[i];
      }
    } else {
      const float inv = 1.0f / l[i];
      const size_t out = (size_t)row * d + h * hd;
#pragma unroll
      for (int u = 0; u < nv; ++u) {
        const size_t e = out + 4 * (j + 8 * u);
        att.put(e, o[i][u].x * inv);
        att.put(e + 1, o[i][u].y * inv);
        att.put(e + 2, o[i][u].z * inv);
        att.put(e + 3, o[i][u].w * inv);
      }
    }
  }
}

// Combines the key splits of attention_tiles_kernel, one warp per (row, head):
// o = sum_z e^(m_z - M) o_z / sum_z e^(m_z - M) l_z, M = max_z m_z, over the
// splits that hold keys of the row's 32-row block (split 0 holds key 0 of every
// row, so M is finite; a split with no key up to the row has m = -inf and
// weight 0).
__global__ void attention_merge_kernel(const float* __restrict__ part, RowOut att,
                                       int n, int start, int d, int H, int hd,
                                       int tiles_per_split) {
  const int gw = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (gw >= n * H) return;
  const int lane = threadIdx.x & 31, i = gw / H, h = gw - i * H;
  const int last = min(start + (i / kAttBQ) * kAttBQ + kAttBQ - 1, start + n - 1);
  const int nz = last / (tiles_per_split * kAttBK) + 1;  // at most kAttSplits
  const size_t stride = (size_t)n * H * (hd + 4);
  const float* p0 = part + ((size_t)i * H + h) * (hd + 4);
  // lane z < nz holds split z's max and sum; every load below is issued at once
  const float mz = lane < nz ? p0[lane * stride + hd] : -INFINITY;
  const float lz = lane < nz ? p0[lane * stride + hd + 1] : 0.f;
  float M = mz;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  const float wz = mz == -INFINITY ? 0.f : expf(mz - M);
  const float inv = 1.0f / warp_sum32(wz * lz);
  for (int jj = lane; jj < hd; jj += 32) {
    float v[kAttSplits];
#pragma unroll
    for (int z = 0; z < kAttSplits; ++z) v[z] = z < nz ? p0[z * stride + jj] : 0.f;
    float o = 0.f;
#pragma unroll
    for (int z = 0; z < kAttSplits; ++z) o = fmaf(__shfl_sync(0xffffffffu, wz, z), v[z], o);
    att.put((size_t)i * d + h * hd + jj, o * inv);
  }
}

template <int kDpt>
tvl_status launch_attention_tiles(const float* qkv, const float* kc, const float* vc, RowOut att,
                                  int n, int start, int d, int kvd, int H, int Hkv, float scale,
                                  float* part, cudaStream_t st) {
  constexpr int hp = 4 * kDpt + 4;
  const int smem = (int)(sizeof(float) * ((kAttBQ + 2 * kAttBK) * hp + kAttBQ * (kAttBK + 1)));
  TVL_CK(cudaFuncSetAttribute((const void*)attention_tiles_kernel<kDpt>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  // split the key range of the longest rows over up to kAttSplits CTAs of at
  // least four tiles each
  const int ntiles = (start + n + kAttBK - 1) / kAttBK;
  int tps = (ntiles + kAttSplits - 1) / kAttSplits;
  if (tps < 4) tps = 4;
  const int nsplit = (ntiles + tps - 1) / tps;
  const dim3 grid((n + kAttBQ - 1) / kAttBQ, H, nsplit);
  attention_tiles_kernel<kDpt><<<grid, kAttThreads, smem, st>>>(
      qkv, kc, vc, att, n, start, d, kvd, H, Hkv, scale, tps, nsplit > 1 ? part : nullptr);
  TVL_CK(cudaGetLastError());
  if (nsplit > 1) {
    const int warps = n * H, wpb = kRowThreads / 32;
    attention_merge_kernel<<<(warps + wpb - 1) / wpb, kRowThreads, 0, st>>>(part, att, n, start, d,
                                                                           H, 4 * kDpt, tps);
    TVL_CK(cudaGetLastError());
  }
  return TVL_OK;
}

template <int kDpt>
tvl_status launch_attention_tiles64(const float* qkv, const float* kc, const float* vc,
                                    RowOut att, int n, int start, int d, int kvd, int H, int Hkv,
                                    float scale, float* part, cudaStream_t st) {
  constexpr int hp = 4 * kDpt + 4;
  const int smem =
      (int)(sizeof(float) * ((kAtt2BQ + 2 * kAttBK) * hp + kAtt2BQ * (kAttBK + 1)));
  TVL_CK(cudaFuncSetAttribute((const void*)attention_tiles64_kernel<kDpt>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  const int ntiles = (start + n + kAttBK - 1) / kAttBK;
  int tps = (ntiles + kAttSplits - 1) / kAttSplits;
  if (tps < 4) tps = 4;
  const int nsplit = (ntiles + tps - 1) / tps;
  const dim3 grid((n + kAtt2BQ - 1) / kAtt2BQ, H, nsplit);
  attention_tiles64_kernel<kDpt><<<grid, kAttThreads, smem, st>>>(
      qkv, kc, vc, att, n, start, d, kvd, H, Hkv, scale, tps, nsplit > 1 ? part : nullptr);
  TVL_CK(cudaGetLastError());
  if (nsplit > 1) {
    const int warps = n * H, wpb = kRowThreads / 32;
    attention_merge_kernel<<<(warps + wpb - 1) / wpb, kRowThreads, 0, st>>>(part, att, n, start, d,
                                                                           H, 4 * kDpt, tps);
    TVL_CK(cudaGetLastError());
  }
  return TVL_OK;
}

// h[i][j] = silu(a) * b with (a, b) = rows (2j, 2j + 1) of the interleaved
// W1/W3 output (§2.1, SwiGLU).
__global__ void swiglu_rows_kernel(const float* __restrict__ h13, RowOut h, long long total) {
  auto silu_mul = [](float a, float b) { return (a / (1.0f + expf(-a))) * b; };
  const long long t4 = total >> 2;  // four outputs from eight inputs at a time
  const float4* in = reinterpret_cast<const float4*>(h13);
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < t4;
       t += (long long)gridDim.x * blockDim.x) {
    const float4 p = in[2 * t], q = in[2 * t + 1];
    h.put4((size_t)(4 * t), make_float4(silu_mul(p.x, p.y), silu_mul(p.z, p.w),
                                         silu_mul(q.x, q.y), silu_mul(q.z, q.w)));
  }
  for (long long t = 4 * t4 + blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x)
    h.put((size_t)t, silu_mul(h13[2 * t], h13[2 * t + 1]));
}

// The bf16 parts (hi then lo) of one weight matrix [M x K] in the prefill's
// weight copy.
struct Parts {
  const unsigned char* hi;
  const unsigned char* lo;
};

// Y[rows x M] = X[rows x K] W^T (everything row-major) on the tensor cores,
// X given as its bf16 parts (xh, xl), which the kernel before wrote.
tvl_status gemm_rows(const Parts& w, const void* xh, const void* xl, float* Y, int rows, int M,
                     int K, int* err, cudaStream_t st) {
  return gemm_bf16x3(w.hi, w.lo, xh, xl, Y, rows, M, K, M, err, st);
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
  lib_free(m->pf);
  lib_free(m->pf_w);
  m->pf = nullptr;
  m->pf_w = nullptr;
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
  auto al = [](size_t b) { return (b + 255) / 256 * 256; };
  // bf16 parts (hi, lo) of every layer's [Wq|Wk|Wv], Wo, W1/W3 (rows
  // interleaved as in the arena, gains folded in) and W2, made at the first call
  const size_t pq = al(2ull * (d + 2 * kvd) * d), po = al(2ull * d * d), p13 = al(4ull * F * d),
               p2 = al(2ull * d * F);
  const size_t per_layer = 2 * (pq + po + p13 + p2);
  auto wsrc = [&](int l, int k) {  // the float32 matrix k of layer l in the arena
    const unsigned char* lw = a.layer0 + (size_t)l * a.layer_stride;
    return reinterpret_cast<const float*>(
        lw + (k == 0 ? a.o_wqkv : k == 1 ? a.o_wo : k == 2 ? a.o_w13 : a.o_w2));
  };
  const size_t part_off[4] = {0, 2 * pq, 2 * pq + 2 * po, 2 * pq + 2 * po + 2 * p13};
  const size_t part_len[4] = {pq, po, p13, p2};
  const long long part_count[4] = {(long long)(d + 2 * kvd) * d, (long long)d * d,
                                   2LL * F * d, (long long)d * F};
  auto wparts = [&](int l, int k) {
    const unsigned char* base = m->pf_w + (size_t)l * per_layer + part_off[k];
    return Parts{base, base + part_len[k]};
  };
  if (!m->pf_w && L > 0) {
    TVL_CK(lib_malloc((void**)&m->pf_w, per_layer * L));
    for (int l = 0; l < L; ++l)
      for (int k = 0; k < 4; ++k) {
        const Parts p = wparts(l, k);
        tvl_status s2 = split_bf16(wsrc(l, k), const_cast<unsigned char*>(p.hi),
                                   const_cast<unsigned char*>(p.lo), part_count[k], st);
        if (s2 != TVL_OK) return s2;
      }
  }
  // activations of up to S rows: x, the products' outputs (Wo and W2: y;
  // [Wq|Wk|Wv]: qkv; W1/W3: h13); the last row's normalised vector; the
  // tokens; the bf16 parts of the next product's input (the normalised rows,
  // the attention output or h), written by the kernel that makes them
  const size_t fx = (size_t)S * d, fqkv = (size_t)S * (d + 2 * kvd), fh13 = (size_t)S * 2 * F;
  const size_t xpart = al(2ull * S * (d > F ? d : F));
  // partials (o, max, sum) of the attention's key splits
  const size_t fpart = (size_t)kAttSplits * S * a.H * (hd + 4);
  const size_t fbytes = al(4 * (2 * fx + fqkv + fh13 + d) + 4 * (size_t)S);
  const size_t need = fbytes + 2 * xpart + al(4 * fpart);
  if (!m->pf) {
    TVL_CK(lib_malloc((void**)&m->pf, need));
    m->pf_bytes = need;
  }
  float* X = m->pf;
  float* Y = X + fx;
  float* QKV = Y + fx;
  float* H13 = QKV + fqkv;
  float* XN = H13 + fh13;
  int* tok = reinterpret_cast<int*>(XN + d);
  unsigned char* xh = reinterpret_cast<unsigned char*>(m->pf) + fbytes;
  unsigned char* xl = xh + xpart;
  const RowOut parts{nullptr, reinterpret_cast<__nv_bfloat16*>(xh),
                     reinterpret_cast<__nv_bfloat16*>(xl)};
  float* PART = reinterpret_cast<float*>(xl + xpart);
  int* err = nullptr;
  tvl_status s = gemm_error_word(&err);
  if (s != TVL_OK) return s;
  TVL_CK(cudaMemcpyAsync(tok, tokens, 4ull * n, cudaMemcpyHostToDevice, st));

  embed_rows_kernel<<<n, kRowThreads, 0, st>>>(a.E, tok, X, d);
  TVL_CK(cudaGetLastError());
  const float* pending = nullptr;  // residual update not yet added into X
  for (int l = 0; l < L; ++l) {
    const unsigned char* lw = a.layer0 + (size_t)l * a.layer_stride;
    const float* g_att = a.gains_folded ? nullptr : reinterpret_cast<const float*>(lw + a.o_gatt);
    const float* g_ffn = a.gains_folded ? nullptr : reinterpret_cast<const float*>(lw + a.o_gffn);
    float* kc = a.kc + (size_t)l * S * kvd;
    float* vc = a.vc + (size_t)l * S * kvd;
    rmsnorm_rows_kernel<<<n, kRowThreads, 0, st>>>(X, pending, g_att, parts, 0, d, a.eps);
    TVL_CK(cudaGetLastError());
    if ((s = gemm_rows(wparts(l, 0), xh, xl, QKV, n, d + 2 * kvd, d, err, st)) != TVL_OK)
      return s;
    rope_kv_kernel<<<n, kRowThreads, 0, st>>>(QKV, a.rope, kc, vc, start_pos, d, kvd, hd);
    TVL_CK(cudaGetLastError());
    {  // head dims of 16 to 128 in steps of 16 take a tiled kernel (multiples of 32:
       // 64 queries per CTA, register blocks; the others: 32 queries per CTA)
      const float sc = a.att_scale;
      s = TVL_OK;
      switch (hd) {
        case 16: s = launch_attention_tiles<4>(QKV, kc, vc, parts, n, start_pos, d, kvd, a.H, a.Hkv, sc, PART, st); break;
        case 32: s = launch_attention_tiles64<8>(QKV, kc, vc, parts, n, start_pos, d, kvd, a.H, a.Hkv, sc, PART, st); break;
        case 48: s = launch_attention_tiles<12>(QKV, kc, vc, parts, n, start_pos, d, kvd, a.H, a.Hkv, sc, PART, st); break;
        case 64: s = launch_attention_tiles64<16>(QKV, kc, vc, parts, n, start_pos, d, kvd, a.H, a.Hkv, sc, PART, st); break;
        case 80: s = launch_attention_tiles<20>(QKV, kc, vc, parts, n, start_pos, d, kvd, a.H, a.Hkv, sc, PART, st); break;
        case 96: s = launch_attention_tiles64<24>(QKV, kc, vc, parts, n, start_pos, d, kvd, a.H, a.Hkv, sc, PART, st); break;
        case 112: s = launch_attention_tiles<28>(QKV, kc, vc, parts, n, start_pos, d, kvd, a.H, a.Hkv, sc, PART, st); break;
        case 128: s = launch_attention_tiles64<32>(QKV, kc, vc, parts, n, start_pos, d, kvd, a.H, a.Hkv, sc, PART, st); break;
        default: {
          const int warps = n * a.H, wpb = kRowThreads / 32;
          attention_rows_kernel<<<(warps + wpb - 1) / wpb, kRowThreads, 0, st>>>(
              QKV, kc, vc, parts, n, start_pos, d, kvd, hd, a.H, a.Hkv, a.att_scale);
          TVL_CK(cudaGetLastError());
        }
      }
      if (s != TVL_OK) return s;
    }
    // Y = Wo o; x += Y and the parts of x_b = RMSNorm(x)
    if ((s = gemm_rows(wparts(l, 1), xh, xl, Y, n, d, d, err, st)) != TVL_OK) return s;
    rmsnorm_rows_kernel<<<n, kRowThreads, 0, st>>>(X, Y, g_ffn, parts, 0, d, a.eps);
    TVL_CK(cudaGetLastError());
    if ((s = gemm_rows(wparts(l, 2), xh, xl, H13, n, 2 * F, d, err, st)) != TVL_OK) return s;
    const long long tot = (long long)n * F;
    swiglu_rows_kernel<<<(int)std::min<long long>((tot / 4 + 255) / 256 + 1, 4096), 256, 0, st>>>(
        H13, parts, tot);
    TVL_CK(cudaGetLastError());
    // Y = W2 h
    if ((s = gemm_rows(wparts(l, 3), xh, xl, Y, n, d, F, err, st)) != TVL_OK) return s;
    pending = Y;
  }
  // the last position: x += (last update), x_b = RMSNorm(x, g_final), logits = Wcls x_b
  rmsnorm_rows_kernel<<<1, kRowThreads, 0, st>>>(X, pending, a.final_gain_folded ? nullptr : a.g_final,
                                                  RowOut{XN, nullptr, nullptr}, n - 1, d, a.eps);
  TVL_CK(cudaGetLastError());
  if ((s = tvl_gemv(a.Wcls, XN, a.logits, V, d, st)) != TVL_OK) return s;
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
