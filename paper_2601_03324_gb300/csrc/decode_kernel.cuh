// decode_kernel.cuh — one persistent kernel runs whole decode steps of a
// Llama-2-architecture decoder (paper §2.1, §7.1), one CTA per SM.
//
// Per step and layer the consumer warps of every CTA run five phases, each
// ended by a grid-wide barrier (every phase needs all outputs of the one
// before):
//   1. x_b = RMSNorm(x, g_att); [q|k|v] = Wqkv x_b         (rows split over CTAs)
//   2. RoPE on q, k; k, v into the cache; attention partials per
//      (head, position chunk)                              (items split over CTAs)
//   3. o = merge of the partials; y = Wo o
//   4. x += y; x_b = RMSNorm(x, g_ffn); [a|b] = W13 x_b
//   5. h = silu(a) * b; y = W2 h; then x += y
// and after the last layer: x_b = RMSNorm(x, g_final); logits = Wcls x_b with
// a per-CTA argmax. The residual stream x is held, identically, in every
// CTA's shared memory: each CTA adds the same values in the same order.
//
// Weights never depend on activations, so the producer warp of each CTA
// streams its rows of every phase, in order, through the stage ring without
// waiting for the barriers: while the consumers wait at a barrier, the next
// phases' weights are already landing. HBM stays busy across the barriers.
#pragma once
#include "stream_gemv.cuh"

namespace tvl {

constexpr int kAttMinChunk = 32;    // positions per attention work item, at least
constexpr int kAttMaxChunk = 1024;  // and at most

struct DecodeArgs {
  // weights (inside the arena)
  const float* E;
  const float* g_final;
  const float* Wcls;
  const unsigned char* layer0;
  long long layer_stride;  // bytes between consecutive layers
  long long o_gatt, o_wqkv, o_wo, o_gffn, o_w13, o_w2;  // byte offsets in a layer
  const float2* rope;  // [S][hd/2] (cos, sin)
  float* kc;           // [L][S][kvd]
  float* vc;
  // scratch
  float* qkv;     // [d + 2 kvd]
  float* o_out;   // [d]
  float* h13;     // [2F]
  float* f_out;   // [d]
  float* logits;  // [V]
  float* att;     // [H][nch_cap][att_stride]: m, l, -, -, o[hd]
  float* cand_val;
  int* cand_idx;  // [G]
  int* tokens;    // [S]
  unsigned long long* ts;   // [S]
  unsigned long long* bar;  // grid barrier counter (monotonic)
  int* err;
  int* err_host;  // mapped pinned host word (may be null)
  // shape
  int d, F, V, L, H, Hkv, hd, kvd, S, G;
  int att_stride, nch_cap;
  float eps, att_scale;
  // this launch
  int start_token, start_pos, n_steps, final_token;
  int nst;
  int sm_ring, sm_bars, sm_xs, sm_vec, sm_pdot, sm_att, sm_misc;  // byte offsets
  unsigned long long barrier_limit_ns;
};

__host__ __device__ inline int ceil_div_i(int a, int b) { return (a + b - 1) / b; }

// Attention work split for position pos: chunks per head (all non-empty).
__host__ __device__ inline void att_split(int pos, int H, int G, int* nch, int* clen) {
  const int n = pos + 1;
  int per_head = G / H;
  if (per_head < 1) per_head = 1;
  int want = ceil_div_i(n, kAttMinChunk);
  int c0 = want < per_head ? want : per_head;
  const int need = ceil_div_i(n, kAttMaxChunk);
  if (c0 < need) c0 = need;
  *clen = ceil_div_i(n, c0);
  *nch = ceil_div_i(n, *clen);
}

// ---- grid barrier ------------------------------------------------------------

// Thread 0 of each CTA arrives on a monotonic 64-bit counter and spins until
// it reaches base + n*G. The spin is bounded in time; on expiry the kernel
// raises TVL_E_TIMEOUT and every CTA leaves at its next barrier or wait.
struct GridBar {
  unsigned long long base = 0, n = 0;

  __device__ void init(const DecodeArgs& a) {
    if (threadIdx.x == 0) {
      // No CTA of this launch can pass the first barrier before this one
      // arrives, so the counter holds k*G + (arrivals so far < G).
      const unsigned long long v = ld_acquire_u64(a.bar);
      base = v - v % (unsigned long long)a.G;
    }
  }

  __device__ bool sync(const DecodeArgs& a, volatile int* s_abort) {
    named_bar_sync(kBarConsumers, kConsumerThreads);
    bool give_up = false;
    if (threadIdx.x == 0) {
      n += 1;
      const unsigned long long target = base + n * (unsigned long long)a.G;
      __threadfence();
      red_release_add_u64(a.bar, 1ull);
      if (!*s_abort) {
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t it = 0;; ++it) {
          if (ld_acquire_u64(a.bar) >= target) break;
          if ((it & 31u) == 31u) {
            if (ld_volatile_s32(a.err)) {
              *s_abort = 1;
              break;
            }
            if (globaltimer_ns() - t0 > a.barrier_limit_ns || it > (1u << 22)) {
              raise_error(a.err, a.err_host, kErrTimeout);
              *s_abort = 1;
              break;
            }
          }
        }
      }
      give_up = *s_abort != 0;
    }
    // thread 0's verdict, given to every consumer thread by a barrier vote
    return !named_bar_or(kBarConsumers, kConsumerThreads, give_up);
  }
};

// ---- small block-level pieces (consumer threads only) --------------------------

// Sum over the consumer threads in a fixed order; every thread gets the result.
__device__ inline float block_sum(float v, float* red) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  v = warp_sum(v);
  if (lane == 0) red[warp] = v;
  named_bar_sync(kBarConsumers, kConsumerThreads);
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < kConsumerWarps; ++w) t += red[w];
  named_bar_sync(kBarConsumers, kConsumerThreads);
  return t;
}

__device__ inline float block_max(float v, float* red) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  v = warp_max(v);
  if (lane == 0) red[warp] = v;
  named_bar_sync(kBarConsumers, kConsumerThreads);
  float t = red[0];
#pragma unroll
  for (int w = 1; w < kConsumerWarps; ++w) t = fmaxf(t, red[w]);
  named_bar_sync(kBarConsumers, kConsumerThreads);
  return t;
}

__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

// Argmax over the consumer threads: largest value, lowest index on ties.
__device__ inline void block_argmax(float& v, int& idx, float* redv, int* redi) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
    if (better(ov, oi, v, idx)) { v = ov; idx = oi; }
  }
  if (lane == 0) { redv[warp] = v; redi[warp] = idx; }
  named_bar_sync(kBarConsumers, kConsumerThreads);
  v = redv[0];
  idx = redi[0];
  for (int w = 1; w < kConsumerWarps; ++w)
    if (better(redv[w], redi[w], v, idx)) { v = redv[w]; idx = redi[w]; }
  named_bar_sync(kBarConsumers, kConsumerThreads);
}

// out = RMSNorm(x, g) (paper §11.2: ss/n + eps, 1/sqrt, then (x*g)*r).
__device__ inline void rmsnorm_to(float* out, const float* x, const float* g, int n, float eps,
                                  float* red) {
  float ss = 0.f;
  for (int j = threadIdx.x; j < n; j += kConsumerThreads) ss = fmaf(x[j], x[j], ss);
  const float tot = block_sum(ss, red);
  const float r = 1.0f / sqrtf(tot / (float)n + eps);
  for (int j = threadIdx.x; j < n; j += kConsumerThreads) out[j] = (x[j] * __ldg(g + j)) * r;
  named_bar_sync(kBarConsumers, kConsumerThreads);
}

__device__ inline void residual_add(float* x, const float* y, int n) {
  for (int j = threadIdx.x; j < n; j += kConsumerThreads) x[j] += ldcg(y + j);
  named_bar_sync(kBarConsumers, kConsumerThreads);
}

// h = silu(W1 x_b) * (W3 x_b) (paper §2.1, SwiGLU).
__device__ inline void swiglu_to(float* h, const float* ab, int F) {
  for (int k = threadIdx.x; k < F; k += kConsumerThreads) {
    const float a = ldcg(ab + k), b = ldcg(ab + F + k);
    h[k] = (a / (1.0f + expf(-a))) * b;
  }
  named_bar_sync(kBarConsumers, kConsumerThreads);
}

struct EpiArgmax {
  float* out;
  float bv;
  int bi;
  __device__ __forceinline__ void store(int row, float v) {
    out[row] = v;
    if (better(v, row, bv, bi)) { bv = v; bi = row; }
  }
};

// ---- attention -------------------------------------------------------------------

// Attention partials of this CTA's items for layer l at position pos. Item
// (h, c): query head h over the positions of chunk c; writes the chunk's
// max score m, sum of exp(s - m), and sum of exp(s - m) * v.
__device__ inline void attention_phase(const DecodeArgs& a, int l, int pos, float* sm, float* red) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int hd = a.hd, hd4 = hd >> 2, half = hd >> 1;
  int nch, clen;
  att_split(pos, a.H, a.G, &nch, &clen);
  const int group = a.H / a.Hkv;
  float* q = sm;             // hd
  float* kp = q + hd;        // hd: key of this position (after RoPE)
  float* vp = kp + hd;       // hd
  float* sc = vp + hd;       // clen <= kAttMaxChunk scores
  float* part = sc + kAttMaxChunk;  // 4 * kConsumerThreads
  const float2* rp = a.rope + (size_t)pos * half;
  const size_t lay = (size_t)l * a.S * a.kvd;
  // lanes per position for the score dot products
  int lpp = 1;
  while (lpp < hd4 && lpp < 32) lpp <<= 1;
  const int ppw = 32 / lpp;
  const int sub = lane / lpp, li = lane - sub * lpp;

  for (int it = blockIdx.x; it < a.H * nch; it += a.G) {
    const int h = it / nch, c = it - h * nch;
    const int kvh = h / group;
    const int t0 = c * clen;
    const int t1 = (t0 + clen < pos + 1) ? t0 + clen : pos + 1;
    const bool has_new = (t1 == pos + 1);
    // q (and the new k, v) with RoPE: pair i turns by pos * theta^(-2i/hd)
    for (int i = tid; i < half; i += kConsumerThreads) {
      const float2 cs = rp[i];
      const float qa = ldcg(a.qkv + h * hd + 2 * i), qb = ldcg(a.qkv + h * hd + 2 * i + 1);
      q[2 * i] = qa * cs.x - qb * cs.y;
      q[2 * i + 1] = qa * cs.y + qb * cs.x;
      if (has_new) {
        const float* kk = a.qkv + a.d + kvh * hd;
        const float ka = ldcg(kk + 2 * i), kb = ldcg(kk + 2 * i + 1);
        kp[2 * i] = ka * cs.x - kb * cs.y;
        kp[2 * i + 1] = ka * cs.y + kb * cs.x;
        const float* vv = a.qkv + a.d + a.kvd + kvh * hd;
        vp[2 * i] = ldcg(vv + 2 * i);
        vp[2 * i + 1] = ldcg(vv + 2 * i + 1);
      }
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
    if (has_new && (h % group) == 0) {  // one writer per kv head
      float* kd = a.kc + lay + (size_t)pos * a.kvd + kvh * hd;
      float* vd = a.vc + lay + (size_t)pos * a.kvd + kvh * hd;
      for (int j = tid; j < hd; j += kConsumerThreads) {
        kd[j] = kp[j];
        vd[j] = vp[j];
      }
    }
    // scores s_t = (q . k_t) * scale for t in [t0, t1)
    const float4* q4 = reinterpret_cast<const float4*>(q);
    for (int tb = t0 + warp * ppw; tb < t1; tb += kConsumerWarps * ppw) {
      const int t = tb + sub;
      float acc = 0.f;
      if (t < t1) {
        const float4* k4 = (t == pos)
                               ? reinterpret_cast<const float4*>(kp)
                               : reinterpret_cast<const float4*>(a.kc + lay + (size_t)t * a.kvd +
                                                                 kvh * hd);
        for (int f = li; f < hd4; f += lpp) {
          const float4 kv = (t == pos) ? k4[f] : ldcg4(k4 + f);
          const float4 qv = q4[f];
          acc = fmaf(qv.x, kv.x, acc);
          acc = fmaf(qv.y, kv.y, acc);
          acc = fmaf(qv.z, kv.z, acc);
          acc = fmaf(qv.w, kv.w, acc);
        }
      }
      for (int o = lpp >> 1; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (t < t1 && li == 0) sc[t - t0] = acc * a.att_scale;
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
    const int n = t1 - t0;
    float m = -INFINITY;
    for (int i = tid; i < n; i += kConsumerThreads) m = fmaxf(m, sc[i]);
    m = block_max(m, red);
    float ls = 0.f;
    for (int i = tid; i < n; i += kConsumerThreads) {
      const float e = expf(sc[i] - m);
      sc[i] = e;
      ls += e;
    }
    ls = block_sum(ls, red);  // its barriers also publish sc
    // o = sum_t e_t v_t: thread (g, f) sums float4 column f over t = g, g+ng, ...
    const int ng = kConsumerThreads / hd4;
    const int gi = tid / hd4, f = tid - gi * hd4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (gi < ng) {
      for (int i = gi; i < n; i += ng) {
        const int t = t0 + i;
        const float e = sc[i];
        const float4 vv =
            (t == pos) ? reinterpret_cast<const float4*>(vp)[f]
                       : ldcg4(reinterpret_cast<const float4*>(a.vc + lay + (size_t)t * a.kvd +
                                                               kvh * hd) + f);
        acc.x = fmaf(e, vv.x, acc.x);
        acc.y = fmaf(e, vv.y, acc.y);
        acc.z = fmaf(e, vv.z, acc.z);
        acc.w = fmaf(e, vv.w, acc.w);
      }
      reinterpret_cast<float4*>(part)[gi * hd4 + f] = acc;
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
    float* rec = a.att + ((size_t)h * a.nch_cap + c) * a.att_stride;
    for (int j = tid; j < hd; j += kConsumerThreads) {
      float o = 0.f;
      for (int g2 = 0; g2 < ng; ++g2) o += part[g2 * hd + j];
      rec[4 + j] = o;
    }
    if (tid == 0) {
      rec[0] = m;
      rec[1] = ls;
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
  }
}

// o[h*hd + j] = sum_c w_c o_c[j] / sum_c w_c l_c with w_c = exp(m_c - max m).
__device__ inline void merge_attention(const DecodeArgs& a, int pos, float* o, float* sm) {
  const int tid = threadIdx.x;
  int nch, clen;
  att_split(pos, a.H, a.G, &nch, &clen);
  const int nrec = a.H * nch;
  float* mv = sm;         // [H * nch]
  float* wv = sm + nrec;  // [H * nch]
  for (int i = tid; i < nrec; i += kConsumerThreads) {
    const int h = i / nch, c = i - h * nch;
    mv[i] = ldcg(a.att + ((size_t)h * a.nch_cap + c) * a.att_stride);
    wv[i] = ldcg(a.att + ((size_t)h * a.nch_cap + c) * a.att_stride + 1);
  }
  named_bar_sync(kBarConsumers, kConsumerThreads);
  for (int h = tid; h < a.H; h += kConsumerThreads) {
    float M = -INFINITY;
    for (int c = 0; c < nch; ++c) M = fmaxf(M, mv[h * nch + c]);
    float Lsum = 0.f;
    for (int c = 0; c < nch; ++c) Lsum += expf(mv[h * nch + c] - M) * wv[h * nch + c];
    for (int c = 0; c < nch; ++c) wv[h * nch + c] = expf(mv[h * nch + c] - M) / Lsum;
  }
  named_bar_sync(kBarConsumers, kConsumerThreads);
  for (int e = tid; e < a.d; e += kConsumerThreads) {
    const int h = e / a.hd, j = e - h * a.hd;
    float acc = 0.f;
    for (int c = 0; c < nch; ++c)
      acc = fmaf(wv[h * nch + c], ldcg(a.att + ((size_t)h * a.nch_cap + c) * a.att_stride + 4 + j),
                 acc);
    o[e] = acc;
  }
  named_bar_sync(kBarConsumers, kConsumerThreads);
}

// Next token: argmax over the per-CTA candidates (identical in every CTA).
__device__ inline int reduce_candidates(const DecodeArgs& a, float* redv, int* redi) {
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  for (int c = threadIdx.x; c < a.G; c += kConsumerThreads) {
    const float v = ldcg(a.cand_val + c);
    const int i = __ldcg(a.cand_idx + c);
    if (better(v, i, bv, bi)) { bv = v; bi = i; }
  }
  block_argmax(bv, bi, redv, redi);
  return bi;
}

// ---- the kernel --------------------------------------------------------------------

__device__ inline void decode_producer(const DecodeArgs& a, const Ring& r, volatile int* s_abort) {
  const uint64_t pol = l2_evict_first();
  const int c = blockIdx.x;
  uint32_t g = 0;
  bool ok = true;
  for (int s = 0; s < a.n_steps && ok; ++s) {
    for (int l = 0; l < a.L && ok; ++l) {
      const unsigned char* lw = a.layer0 + (size_t)l * a.layer_stride;
      ok = produce_phase(r, g, reinterpret_cast<const float*>(lw + a.o_wqkv),
                         plan_stages(a.d + 2 * a.kvd, a.d, a.G, c), pol, a.err, a.err_host,
                         s_abort) &&
           produce_phase(r, g, reinterpret_cast<const float*>(lw + a.o_wo),
                         plan_stages(a.d, a.d, a.G, c), pol, a.err, a.err_host, s_abort) &&
           produce_phase(r, g, reinterpret_cast<const float*>(lw + a.o_w13),
                         plan_stages(2 * a.F, a.d, a.G, c), pol, a.err, a.err_host, s_abort) &&
           produce_phase(r, g, reinterpret_cast<const float*>(lw + a.o_w2),
                         plan_stages(a.d, a.F, a.G, c), pol, a.err, a.err_host, s_abort);
    }
    ok = ok && produce_phase(r, g, a.Wcls, plan_stages(a.V, a.d, a.G, c), pol, a.err, a.err_host,
                             s_abort);
  }
  drain_ring(r, g);
}

__device__ inline void decode_consumer(const DecodeArgs& a, const Ring& r, unsigned char* smem,
                                       volatile int* s_abort) {
  float* xs = reinterpret_cast<float*>(smem + a.sm_xs);
  float* vec = reinterpret_cast<float*>(smem + a.sm_vec);
  float* pdot = reinterpret_cast<float*>(smem + a.sm_pdot);
  float* asm_ = reinterpret_cast<float*>(smem + a.sm_att);
  float* red = reinterpret_cast<float*>(smem + a.sm_misc) + 8;
  int* redi = reinterpret_cast<int*>(smem + a.sm_misc) + 24;
  const int tid = threadIdx.x, c = blockIdx.x;
  uint32_t g = 0;
  GridBar gb;
  gb.init(a);
  int token = a.start_token;
  for (int s = 0; s < a.n_steps; ++s) {
    const int pos = a.start_pos + s;
    if (s > 0) {
      token = reduce_candidates(a, red, redi);
      if (token < 0 || token >= a.V) token = 0;  // only if every logit was NaN
      if (c == 0 && tid == 0) {
        a.tokens[s - 1] = token;
        a.ts[s - 1] = globaltimer_ns();
      }
    }
    // x = E[token] (paper §4.1: weights are rows at offsets in the blob)
    const float4* e4 = reinterpret_cast<const float4*>(a.E + (size_t)token * a.d);
    for (int j = tid; j < (a.d >> 2); j += kConsumerThreads)
      reinterpret_cast<float4*>(xs)[j] = __ldg(e4 + j);
    named_bar_sync(kBarConsumers, kConsumerThreads);
    for (int l = 0; l < a.L; ++l) {
      const unsigned char* lw = a.layer0 + (size_t)l * a.layer_stride;
      rmsnorm_to(vec, xs, reinterpret_cast<const float*>(lw + a.o_gatt), a.d, a.eps, red);
      EpiStore e_qkv{a.qkv};
      if (!consume_phase(r, g, plan_stages(a.d + 2 * a.kvd, a.d, a.G, c), vec, 1, a.d, pdot,
                         e_qkv, a.err, a.err_host, s_abort))
        return;
      if (!gb.sync(a, s_abort)) return;
      attention_phase(a, l, pos, asm_, red);
      if (!gb.sync(a, s_abort)) return;
      merge_attention(a, pos, vec, asm_);
      EpiStore e_o{a.o_out};
      if (!consume_phase(r, g, plan_stages(a.d, a.d, a.G, c), vec, 1, a.d, pdot, e_o, a.err,
                         a.err_host, s_abort))
        return;
      if (!gb.sync(a, s_abort)) return;
      residual_add(xs, a.o_out, a.d);
      rmsnorm_to(vec, xs, reinterpret_cast<const float*>(lw + a.o_gffn), a.d, a.eps, red);
      EpiStore e_13{a.h13};
      if (!consume_phase(r, g, plan_stages(2 * a.F, a.d, a.G, c), vec, 1, a.d, pdot, e_13, a.err,
                         a.err_host, s_abort))
        return;
      if (!gb.sync(a, s_abort)) return;
      swiglu_to(vec, a.h13, a.F);
      EpiStore e_2{a.f_out};
      if (!consume_phase(r, g, plan_stages(a.d, a.F, a.G, c), vec, 1, a.F, pdot, e_2, a.err,
                         a.err_host, s_abort))
        return;
      if (!gb.sync(a, s_abort)) return;
      residual_add(xs, a.f_out, a.d);
    }
    rmsnorm_to(vec, xs, a.g_final, a.d, a.eps, red);
    EpiArgmax ea{a.logits, -INFINITY, 0x7fffffff};
    if (!consume_phase(r, g, plan_stages(a.V, a.d, a.G, c), vec, 1, a.d, pdot, ea, a.err,
                       a.err_host, s_abort))
      return;
    float bv = ea.bv;
    int bi = ea.bi;
    block_argmax(bv, bi, red, redi);
    if (tid == 0) {
      a.cand_val[c] = bv;
      a.cand_idx[c] = bi;
    }
    if (s + 1 < a.n_steps || a.final_token) {
      if (!gb.sync(a, s_abort)) return;
    }
  }
  if (a.final_token && c == 0) {
    token = reduce_candidates(a, red, redi);
    if (tid == 0) {
      a.tokens[a.n_steps - 1] = token;
      a.ts[a.n_steps - 1] = globaltimer_ns();
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const DecodeArgs a) {
  extern __shared__ __align__(128) unsigned char smem[];
  Ring r;
  r.buf = smem + a.sm_ring;
  r.full = reinterpret_cast<uint64_t*>(smem + a.sm_bars);
  r.empty = r.full + a.nst;
  r.nst = a.nst;
  volatile int* s_abort = reinterpret_cast<volatile int*>(smem + a.sm_misc);
  if (threadIdx.x == 0) {
    for (int i = 0; i < a.nst; ++i) {
      mbar_init(&r.full[i], 1);
      mbar_init(&r.empty[i], 1);
    }
    *s_abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x >= kConsumerThreads) {
    if (threadIdx.x == kConsumerThreads) decode_producer(a, r, s_abort);
    return;
  }
  decode_consumer(a, r, smem, s_abort);
}

// Failure-detection self-test: one barrier whose count nothing will reach.
__global__ void barrier_selftest_kernel(DecodeArgs a) {
  __shared__ int s_abort;
  if (threadIdx.x == 0) s_abort = 0;
  __syncthreads();
  if (threadIdx.x >= kConsumerThreads) return;
  GridBar gb;
  gb.init(a);
  if (threadIdx.x == 0) gb.n = 1;  // expect one more full round than will ever arrive
  gb.sync(a, reinterpret_cast<volatile int*>(&s_abort));
}

}  // namespace tvl
