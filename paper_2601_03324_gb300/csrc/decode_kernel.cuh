// decode_kernel.cuh — one persistent kernel runs whole decode steps of a
// Llama-2-architecture decoder (paper §2.1, §7.1), one CTA per SM.
//
// Per step and layer the consumer warps of every CTA run five phases; each
// needs all outputs of the phase before:
//   1. x_b = RMSNorm(x, g_att); [q|k|v] = Wqkv x_b         (rows split over CTAs)
//   2. RoPE on q, k; k, v into the cache; attention partials per
//      (head, position chunk)                              (items split over CTAs)
//   3. o = merge of the partials; y = Wo o
//   4. x += y; x_b = RMSNorm(x, g_ffn); a = W1 x_b, b = W3 x_b, and
//      h = silu(a) * b where a_i and b_i are computed (the device copy of
//      W1 and W3 interleaves their rows: row 2i is W1's row i, row 2i + 1
//      W3's)                                                (row pairs split over CTAs)
//   5. y = W2 h; then x += y
// and after the last layer: x_b = RMSNorm(x, g_final); logits = Wcls x_b with
// a per-CTA argmax. The residual stream x is held, identically, in every
// CTA's shared memory: each CTA adds the same values in the same order.
//
// Exchange between phases: every value a phase publishes is one 64-bit word,
// (epoch tag << 32) | float bits, written once (an unsigned-max reduction:
// tags only grow, so the new word wins). A reader polls the words it
// needs until each carries the epoch of the current (step, layer, phase); the
// wait and the read are the same L2 round trip, and no grid-wide barrier is
// needed. A buffer is rewritten only one layer later, after an exchange that
// every reader of the old contents had to join first, so no reader can miss
// its data (the per-step argmax candidates, which can lack such an exchange
// when there are no layers, are double-buffered by step parity).
//
// Weights never depend on activations, so the producer warp of each CTA
// streams its rows of every phase, in order, through the stage ring without
// waiting for the exchanges: while consumers wait on one, the next phases'
// weights are already landing. HBM stays busy across the waits.
#pragma once
#include "stream_gemv.cuh"

namespace tvl {

constexpr int kAttMinChunk = 32;    // positions per attention work item, at least
constexpr int kAttMaxChunk = 1024;  // and at most
constexpr int kPhasesPerLayer = 5;  // exchanges per layer: qkv, att, o, h13, f
constexpr int kMaxBatch = 4;        // sequences one launch can decode together
// The small shared region of the decode kernel: the abort flag (word 0),
// reduction scratch (floats 8..39, ints 80..87), the five stage plans.
constexpr int kPlansOffset = 512;
constexpr int kMiscBytes = 1024;
constexpr uint32_t kRefillDelayNs = 0;  // producer pause before refilling freed stages (measured best: 0, with the L2 prefetch)

struct DecodeArgs {
  // weights (inside the arena)
  const float* E;
  const float* g_final;
  const float* Wcls;
  const unsigned char* layer0;
  // 8-bit rows (models loaded with weight_bits 8): per layer [Wq|Wk|Wv], Wo,
  // [W1|W3], W2 at these byte offsets; the embedding table; the classifier
  const unsigned char* q_layer0;
  long long q_stride, q_wqkv, q_wo, q_w13, q_w2;
  const unsigned char* q_E;
  const unsigned char* q_cls;
  long long layer_stride;  // bytes between consecutive layers
  long long o_gatt, o_wqkv, o_wo, o_gffn, o_w13, o_w2;  // byte offsets in a layer
  const float2* rope;  // [S][hd/2] (cos, sin)
  float* kc;           // [L][S][kvd]
  float* vc;
  // tagged exchange buffers (64-bit words: tag << 32 | float bits)
  unsigned long long* x_qkv;   // [d + 2 kvd]
  unsigned long long* x_att;   // [H][nch_cap][att_stride]: m, l, -, -, sum[hd] of chunks > 0
  unsigned long long* x_attn;  // [d]: attention output, merged per head
  unsigned long long* x_o;     // [d]
  unsigned long long* x_h13;   // [F]: h = silu(W1 x_b) * (W3 x_b)
  unsigned long long* x_f;     // [d]
  unsigned long long* x_cand;  // [2][G][2]: per step parity, per CTA (value, index)
  float* logits;               // [V]
  int* tokens;                 // [S]
  unsigned long long* ts;      // [S]
  int* err;
  int* err_host;  // mapped pinned host word (may be null)
  // shape
  int d, F, V, L, H, Hkv, hd, kvd, S, G;
  int att_stride, nch_cap;
  float eps, att_scale;
  // RMSNorm gains already multiplied into the columns of the matrices that
  // read the normalised vector (the layers' [Wq|Wk|Wv] and W1/W3; the
  // classifier when it is not the embedding table): the phase input is then x
  // itself, and no gain is loaded on the way from an exchange to a GEMV
  bool gains_folded, final_gain_folded;
  // this launch
  int start_pos, n_steps, final_token;
  // B sequences decode in lockstep at the same positions: sequence b's words
  // in an exchange buffer sit b vector lengths in, its K/V cache b * kv_seq
  // floats in, its logits b * V floats in; tokens are [step][B]
  int start_tokens[kMaxBatch];
  long long kv_seq;
  int vs;  // floats between two sequences' phase inputs in shared memory
  unsigned epoch0;  // tag of the first exchange of this launch
  int nst;
  int sm_ring, sm_bars, sm_xs, sm_vec, sm_seg, sm_att, sm_misc;  // byte offsets
  unsigned long long wait_limit_ns;
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

// ---- tagged exchange -------------------------------------------------------------

// Publishes one tagged word. A word's tag only grows (the exchange words are
// cleared before the tag would wrap), so an unsigned max leaves exactly the new
// word; the reduction reaches the pollers sooner than a plain store when many
// CTAs poll the same lines (fire and forget, like a store).
__device__ __forceinline__ void st_tag(unsigned long long* p, unsigned tag, float v) {
  const unsigned long long w =
      ((unsigned long long)tag << 32) | (unsigned long long)__float_as_uint(v);
  asm volatile("red.relaxed.gpu.global.max.u64 [%0], %1;" ::"l"(p), "l"(w) : "memory");
}

__device__ __forceinline__ ulonglong2 ld_tag2(const unsigned long long* p) {
  ulonglong2 v;
  asm volatile("ld.global.cg.v2.u64 {%0, %1}, [%2];" : "=l"(v.x), "=l"(v.y) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ bool tags_are(const ulonglong2& v, unsigned tag) {
  return (unsigned)(v.x >> 32) == tag && (unsigned)(v.y >> 32) == tag;
}

__device__ __forceinline__ float lo_f(unsigned long long w) { return __uint_as_float((unsigned)w); }

struct Poll {
  int* err;
  int* err_host;
  volatile int* s_abort;
  unsigned long long limit_ns;
};

// Bounded-wait bookkeeping of one polling thread: gives up on abort, on an
// error raised elsewhere, or after the limit (raising TVL_E_TIMEOUT).
struct PollClock {
  uint64_t t0 = 0;
  uint32_t it = 0;
  __device__ __forceinline__ bool keep_waiting(const Poll& c) {
    if ((++it & 15u) != 0) return true;
    if (*c.s_abort || ld_volatile_s32(c.err)) return false;
    const uint64_t now = globaltimer_ns();
    if (t0 == 0) t0 = now;
    if (now - t0 > c.limit_ns || it > (1u << 24)) {
      raise_error(c.err, c.err_host, kErrTimeout);
      *c.s_abort = 1;
      return false;
    }
    return true;
  }
};

// Poll pairs p = tid, tid + 256, ... of a tagged vector (npairs pairs), up to
// four 16-byte loads in flight per thread; every not-yet-current pair of a
// batch is re-read together, so waiting costs one round trip after the last
// producer's store. fn(p, v0, v1) takes each ready pair. Returns false if this
// thread gave up (the caller votes).
template <int D = 4, class Fn>
__device__ inline bool poll_pairs(const unsigned long long* src, int npairs, unsigned tag,
                                  const Poll& c, Fn fn) {
  for (int base = threadIdx.x; base < npairs; base += kConsumerThreads * D) {
    ulonglong2 v[D];
    unsigned pending = 0;
#pragma unroll
    for (int b = 0; b < D; ++b) {
      const int p = base + b * kConsumerThreads;
      if (p < npairs) {
        v[b] = ld_tag2(src + 2 * p);
        pending |= 1u << b;
      }
    }
    PollClock clk;
    while (true) {
#pragma unroll
      for (int b = 0; b < D; ++b) {
        if ((pending >> b) & 1u) {
          if (tags_are(v[b], tag)) {
            fn(base + b * kConsumerThreads, lo_f(v[b].x), lo_f(v[b].y));
            pending &= ~(1u << b);
          }
        }
      }
      if (!pending) break;
      if (!clk.keep_waiting(c)) return false;
#pragma unroll
      for (int b = 0; b < D; ++b)
        if ((pending >> b) & 1u) v[b] = ld_tag2(src + 2 * (base + b * kConsumerThreads));
    }
  }
  return true;
}

// Poll pairs p = tid, tid + 224, ... (npairs pairs) at addresses addr(p), up
// to four 16-byte loads in flight per thread; fn(p, v0, v1) takes each ready
// pair. Returns false if this thread gave up (the caller votes).
template <class Addr, class Fn>
__device__ inline bool poll_pairs_at(int npairs, Addr addr, unsigned tag, const Poll& c, Fn fn) {
  for (int base = threadIdx.x; base < npairs; base += kConsumerThreads * 4) {
    ulonglong2 v[4];
    unsigned pending = 0;
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int p = base + b * kConsumerThreads;
      if (p < npairs) {
        v[b] = ld_tag2(addr(p));
        pending |= 1u << b;
      }
    }
    PollClock clk;
    while (true) {
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        if (((pending >> b) & 1u) && tags_are(v[b], tag)) {
          fn(base + b * kConsumerThreads, lo_f(v[b].x), lo_f(v[b].y));
          pending &= ~(1u << b);
        }
      }
      if (!pending) break;
      if (!clk.keep_waiting(c)) return false;
#pragma unroll
      for (int b = 0; b < 4; ++b)
        if ((pending >> b) & 1u) v[b] = ld_tag2(addr(base + b * kConsumerThreads));
    }
  }
  return true;
}

// Poll quads j = tid, tid + 224, ... (nquads quads of four consecutive words),
// Q quads (2 Q 16-byte loads) in flight per thread, and load quad j mod n4 of
// aux (the RMSNorm gains; null: all ones) for each while the polls are out;
// fn(j, v, aux quad) takes each ready quad. Returns false if this thread gave up.
template <int Q, class Fn>
__device__ inline bool poll_quads(const unsigned long long* src, int nquads, unsigned tag,
                                  const float4* aux, int n4, const Poll& c, Fn fn) {
  for (int base = threadIdx.x; base < nquads; base += kConsumerThreads * Q) {
    ulonglong2 lo[Q], hi[Q];
    float4 ax[Q];
    unsigned pending = 0;
#pragma unroll
    for (int b = 0; b < Q; ++b) {
      const int j = base + b * kConsumerThreads;
      if (j < nquads) {
        lo[b] = ld_tag2(src + 4 * j);
        hi[b] = ld_tag2(src + 4 * j + 2);
        pending |= 1u << b;
      }
    }
#pragma unroll
    for (int b = 0; b < Q; ++b) {
      const int j = base + b * kConsumerThreads;
      if (j < nquads) ax[b] = aux ? __ldg(aux + j % n4) : make_float4(1.f, 1.f, 1.f, 1.f);
    }
    PollClock clk;
    while (true) {
#pragma unroll
      for (int b = 0; b < Q; ++b) {
        if (((pending >> b) & 1u) && tags_are(lo[b], tag) && tags_are(hi[b], tag)) {
          fn(base + b * kConsumerThreads,
             make_float4(lo_f(lo[b].x), lo_f(lo[b].y), lo_f(hi[b].x), lo_f(hi[b].y)), ax[b]);
          pending &= ~(1u << b);
        }
      }
      if (!pending) break;
      if (!clk.keep_waiting(c)) return false;
#pragma unroll
      for (int b = 0; b < Q; ++b) {
        if ((pending >> b) & 1u) {
          const int j = base + b * kConsumerThreads;
          lo[b] = ld_tag2(src + 4 * j);
          hi[b] = ld_tag2(src + 4 * j + 2);
        }
      }
    }
  }
  return true;
}

// One pair, re-read until current (used where a thread needs a single pair).
__device__ inline bool poll_one(const unsigned long long* p, unsigned tag, const Poll& c,
                                ulonglong2& v) {
  v = ld_tag2(p);
  PollClock clk;
  while (!tags_are(v, tag)) {
    if (!clk.keep_waiting(c)) return false;
    v = ld_tag2(p);
  }
  return true;
}

// Leaves the consumer warps together if any of them gave up.
__device__ __forceinline__ bool vote_ok(bool ok, volatile int* s_abort) {
  if (named_bar_or(kBarConsumers, kConsumerThreads, !ok)) {
    if (threadIdx.x == 0) *s_abort = 1;
    return false;
  }
  return true;
}

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

// The input of a phase that follows an RMSNorm is x * g without the factor
// r = 1/sqrt(mean x^2 + eps); each row's dot product is multiplied by r here
// (W ((x * g) r) = r W (x * g)). scale[b] is sequence b's factor, 1 for the
// phases without a norm.
__device__ __forceinline__ float pick_scale(const float (&sc)[kMaxBatch], int b) {
  float v = sc[0];
#pragma unroll
  for (int i = 1; i < kMaxBatch; ++i)
    if (b == i) v = sc[i];
  return v;
}

// Publishes GEMV rows as tagged words (M words per sequence). With swiglu
// the rows are interleaved pairs (W1 row i, W3 row i) and the pair publishes
// h_i = silu(a_i) * b_i at word i instead (paper §2.1, SwiGLU).
struct EpiTag {
  unsigned long long* out;
  unsigned tag;
  int M;
  bool swiglu;
  float scale[kMaxBatch];
  __device__ __forceinline__ void store(int row, float v) { store_b(row, 0, v); }
  __device__ __forceinline__ void store_b(int row, int b, float v) {
    st_tag(out + (size_t)b * M + row, tag, v * pick_scale(scale, b));
  }
  __device__ __forceinline__ void store_pair(int row, float v0, float v1) {
    store_pair_b(row, 0, v0, v1);
  }
  __device__ __forceinline__ void store_pair_b(int row, int b, float v0, float v1) {
    const float sc = pick_scale(scale, b);
    v0 *= sc;
    v1 *= sc;
    if (swiglu) {
      st_tag(out + (size_t)b * M + (row >> 1), tag, (v0 / (1.0f + expf(-v0))) * v1);
    } else {
      st_tag(out + (size_t)b * M + row, tag, v0);
      st_tag(out + (size_t)b * M + row + 1, tag, v1);
    }
  }
};

// Logits of every sequence (V apart) and each thread's best (value, index)
// per sequence so far.
template <int kB>
struct EpiArgmax {
  float* out;
  int V;
  float scale[kMaxBatch];  // RMSNorm factor of sequence b's input
  float bv[kB];
  int bi[kB];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int b = 0; b < kB; ++b) { bv[b] = -INFINITY; bi[b] = 0x7fffffff; }
  }
  __device__ __forceinline__ void store(int row, float v) { store_b(row, 0, v); }
  __device__ __forceinline__ void store_pair(int row, float v0, float v1) {
    store_b(row, 0, v0);
    store_b(row + 1, 0, v1);
  }
  __device__ __forceinline__ void store_pair_b(int row, int b, float v0, float v1) {
    store_b(row, b, v0);
    store_b(row + 1, b, v1);
  }
  __device__ __forceinline__ void store_b(int row, int b, float v) {
    v *= pick_scale(scale, b);
    out[(size_t)b * V + row] = v;
#pragma unroll
    for (int bb = 0; bb < kB; ++bb)
      if (bb == b && better(v, row, bv[bb], bi[bb])) { bv[bb] = v; bi[bb] = row; }
  }
};

// ---- attention -------------------------------------------------------------------

// Ask L2 for the K/V rows (positions before pos) that this CTA's attention
// items of layer l will read: the cache lines are usually no longer in L2
// (the weight stream has gone through it since), and the request is issued a
// phase ahead so that the items' own loads find them there.
template <int kB>
__device__ inline void att_prefetch_l2(const DecodeArgs& a, int l, int pos) {
  int nch, clen;
  att_split(pos, a.H * kB, a.G, &nch, &clen);
  const int group = a.H / a.Hkv, hd = a.hd;
  const int lpr = (hd * 4 + 127) / 128;  // 128-byte lines per row
  for (int it = blockIdx.x; it < kB * a.H * nch; it += a.G) {
    const int b = kB == 1 ? 0 : it / (a.H * nch), hc = it - b * a.H * nch;
    const int h = hc / nch, c = hc - h * nch, kvh = h / group;
    const size_t lay = (size_t)b * a.kv_seq + (size_t)l * a.S * a.kvd;
    const int t0 = c * clen, te = (t0 + clen < pos) ? t0 + clen : pos;
    const int per = (te - t0) * lpr;
    for (int i = threadIdx.x; i < 2 * per; i += kConsumerThreads) {
      const int which = i >= per, rem = i - which * per;
      const int t = t0 + rem / lpr, ln = rem - (rem / lpr) * lpr;
      const float* q = (which ? a.vc : a.kc) + lay + (size_t)t * a.kvd + kvh * hd + ln * 32;
      asm volatile("prefetch.global.L2 [%0];" ::"l"(q));
    }
  }
}

// Attention partials of this CTA's items for layer l at position pos. Item
// (h, c): query head h over the positions of chunk c; publishes the chunk's
// max score m, sum of exp(s - m), and sum of exp(s - m) * v.
// With kB sequences the items are (sequence, head, chunk); sequence b has
// its own q/k/v words, K/V cache, records and output.
template <int kB>
__device__ inline bool attention_phase(const DecodeArgs& a, int l, int pos, unsigned tag_qkv,
                                       unsigned tag_att, float* sm, float* red, const Poll& pc,
                                       bool& wrote_kv) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int hd = a.hd, hd4 = hd >> 2, half = hd >> 1;
  int nch, clen;
  att_split(pos, a.H * kB, a.G, &nch, &clen);
  const int group = a.H / a.Hkv;
  float* q = sm;             // hd
  float* kp = q + hd;        // hd: key of this position (after RoPE)
  float* vp = kp + hd;       // hd
  float* sc = vp + hd;       // clen <= kAttMaxChunk scores
  float* part = sc + kAttMaxChunk;  // 4 * kConsumerThreads
  const float2* rp = a.rope + (size_t)pos * half;
  // lanes per position for the score dot products
  int lpp = 1;
  while (lpp < hd4 && lpp < 32) lpp <<= 1;
  const int ppw = 32 / lpp;
  const int sub = lane / lpp, li = lane - sub * lpp;

  // the items of chunk 0 (the heads' mergers) come after the other items of
  // the same CTA, which they wait for
  for (int pass = 0; pass < 2; ++pass)
  for (int it = blockIdx.x; it < kB * a.H * nch; it += a.G) {
    const int b = kB == 1 ? 0 : it / (a.H * nch), hc = it - b * a.H * nch;
    const int h = hc / nch, c = hc - h * nch;
    if ((c == 0) != (pass == 1)) continue;
    const int kvh = h / group;
    const size_t lay = (size_t)b * a.kv_seq + (size_t)l * a.S * a.kvd;
    const unsigned long long* xq = a.x_qkv + (size_t)b * (a.d + 2 * a.kvd);
    const int hb = b * a.H + h;  // record and output index of (sequence, head)
    const int t0 = c * clen;
    const int t1 = (t0 + clen < pos + 1) ? t0 + clen : pos + 1;
    const bool has_new = (t1 == pos + 1);
    const float* kbase = a.kc + lay + kvh * hd;
    const float* vbase = a.vc + lay + kvh * hd;
    const int pstride = kConsumerWarps * ppw;
    const int ng = kConsumerThreads / hd4;
    const int gi = tid / hd4, f = tid - gi * hd4;
    const int n = t1 - t0;
    const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
    // this thread's q/k/v pair (at most one: nget <= 3 hd / 2 <= 192 < 224
    // threads) is asked for first, so that its poll is not queued behind the
    // row loads below
    const int nget = has_new ? 3 * half : half;
    const int tq = tid < nget ? tid : 0;  // head_dim <= 128 keeps nget below 224
    const int which0 = tq / half, i0 = tq - which0 * half;
    const unsigned long long* src0 =
        xq + (which0 == 0 ? h * hd : a.d + (which0 - 1) * a.kvd + kvh * hd) + 2 * i0;
    ulonglong2 qv = make_ulonglong2(0ull, 0ull);
    if (tid < nget) qv = ld_tag2(src0);
    // the first three K and V rows of each thread, loaded before q is ready
    float4 kr0 = z4, kr1 = z4, kr2 = z4, v0 = z4, v1 = z4, v2 = z4;
    {
      const int tk = t0 + warp * ppw + sub;
      if (li < hd4 && tk < t1 && tk != pos)
        kr0 = ldcg4(reinterpret_cast<const float4*>(kbase + (size_t)tk * a.kvd) + li);
      if (li < hd4 && tk + pstride < t1 && tk + pstride != pos)
        kr1 = ldcg4(reinterpret_cast<const float4*>(kbase + (size_t)(tk + pstride) * a.kvd) + li);
      if (li < hd4 && tk + 2 * pstride < t1 && tk + 2 * pstride != pos)
        kr2 = ldcg4(reinterpret_cast<const float4*>(kbase + (size_t)(tk + 2 * pstride) * a.kvd) +
                    li);
      if (gi < ng && gi < n && t0 + gi != pos)
        v0 = ldcg4(reinterpret_cast<const float4*>(vbase + (size_t)(t0 + gi) * a.kvd) + f);
      if (gi < ng && gi + ng < n && t0 + gi + ng != pos)
        v1 = ldcg4(reinterpret_cast<const float4*>(vbase + (size_t)(t0 + gi + ng) * a.kvd) + f);
      if (gi < ng && gi + 2 * ng < n && t0 + gi + 2 * ng != pos)
        v2 = ldcg4(reinterpret_cast<const float4*>(vbase + (size_t)(t0 + gi + 2 * ng) * a.kvd) + f);
    }
    // q (and the new k, v) with RoPE: pair i turns by pos * theta^(-2i/hd).
    // Pair i of a head is one 16-byte tagged load.
    bool ok = true;
    if (tid < nget) {
      const int which = which0, i = i0;
      ulonglong2 v = qv;
      {
        PollClock clk;
        while (!tags_are(v, tag_qkv)) {
          if (!clk.keep_waiting(pc)) {
            ok = false;
            break;
          }
          v = ld_tag2(src0);
        }
      }
      const float x0 = lo_f(v.x), x1 = lo_f(v.y);
      if (which == 2) {
        vp[2 * i] = x0;
        vp[2 * i + 1] = x1;
      } else {
        const float2 cs = rp[i];
        float* dst = which == 0 ? q : kp;
        dst[2 * i] = x0 * cs.x - x1 * cs.y;
        dst[2 * i + 1] = x0 * cs.y + x1 * cs.x;
      }
    }
    if (!vote_ok(ok, pc.s_abort)) return false;
    const bool kv_writer = has_new && (h % group) == 0;  // one writer per kv head
    if (kv_writer) {  // thread j < hd writes element j of the new K and V rows
      wrote_kv = true;
      float* kd = a.kc + lay + (size_t)pos * a.kvd + kvh * hd;
      float* vd = a.vc + lay + (size_t)pos * a.kvd + kvh * hd;
      if (tid < hd) {
        kd[tid] = kp[tid];
        vd[tid] = vp[tid];
      }
    }
    if (gi < ng && t0 + gi == pos) v0 = reinterpret_cast<const float4*>(vp)[f];
    if (gi < ng && t0 + gi + ng == pos) v1 = reinterpret_cast<const float4*>(vp)[f];
    if (gi < ng && t0 + gi + 2 * ng == pos) v2 = reinterpret_cast<const float4*>(vp)[f];
    // scores s_t = (q . k_t) * scale for t in [t0, t1); the first pass uses the rows loaded above
    const float4* q4 = reinterpret_cast<const float4*>(q);
    {
      // positions in groups of three rows per lane: row rr of group j is
      // position t0 + j * 3 * pstride + warp * ppw + sub + rr * pstride; the
      // first group is the rows loaded above, each later one three loads at once
      const float4 qv = li < hd4 ? q4[li] : z4;
      const float4 kn = li < hd4 ? reinterpret_cast<const float4*>(kp)[li] : z4;
      for (int tg = t0 + warp * ppw + sub; tg - sub < t1; tg += 3 * pstride) {
        float4 kv[3];
        if (tg - sub == t0 + warp * ppw) {
          kv[0] = kr0;
          kv[1] = kr1;
          kv[2] = kr2;
        } else {
#pragma unroll
          for (int rr = 0; rr < 3; ++rr) {
            const int t = tg + rr * pstride;
            kv[rr] = (li < hd4 && t < t1 && t != pos)
                         ? ldcg4(reinterpret_cast<const float4*>(kbase + (size_t)t * a.kvd) + li)
                         : z4;
          }
        }
        float s3[3];
#pragma unroll
        for (int rr = 0; rr < 3; ++rr) {
          const float4 k = tg + rr * pstride == pos ? kn : kv[rr];
          float acc = 0.f;
          acc = fmaf(qv.x, k.x, acc);
          acc = fmaf(qv.y, k.y, acc);
          acc = fmaf(qv.z, k.z, acc);
          acc = fmaf(qv.w, k.w, acc);
          s3[rr] = acc;
        }
        for (int o = lpp >> 1; o > 0; o >>= 1) {
#pragma unroll
          for (int rr = 0; rr < 3; ++rr) s3[rr] += __shfl_xor_sync(0xffffffffu, s3[rr], o);
        }
#pragma unroll
        for (int rr = 0; rr < 3; ++rr) {
          const int t = tg + rr * pstride;
          if (t < t1 && li == 0) sc[t - t0] = s3[rr] * a.att_scale;
        }
      }
    }
    auto vrow = [&](int t) -> float4 {
      return (t == pos) ? reinterpret_cast<const float4*>(vp)[f]
                        : ldcg4(reinterpret_cast<const float4*>(a.vc + lay + (size_t)t * a.kvd +
                                                                kvh * hd) + f);
    };
    named_bar_sync(kBarConsumers, kConsumerThreads);
    // softmax weights e_t = exp(s_t - m), m = max s_t, and l = sum e_t. A chunk
    // of at most 64 positions is reduced by every warp on its own (the same
    // values in every warp, no barrier); a longer one by the whole block,
    // which leaves e_t in sc.
    const bool warp_softmax = n <= 64;
    float m, ls;
    if (warp_softmax) {
      const float s0 = lane < n ? sc[lane] : -INFINITY;
      const float s1 = lane + 32 < n ? sc[lane + 32] : -INFINITY;
      m = warp_max(fmaxf(s0, s1));
      const float e0 = lane < n ? expf(s0 - m) : 0.f;
      const float e1 = lane + 32 < n ? expf(s1 - m) : 0.f;
      ls = warp_sum(e0 + e1);
    } else {
      m = -INFINITY;
      for (int i = tid; i < n; i += kConsumerThreads) m = fmaxf(m, sc[i]);
      m = block_max(m, red);
      ls = 0.f;
      for (int i = tid; i < n; i += kConsumerThreads) {
        const float e = expf(sc[i] - m);
        sc[i] = e;
        ls += e;
      }
      ls = block_sum(ls, red);  // its barriers also publish sc
    }
    auto weight = [&](int i) { return warp_softmax ? expf(sc[i] - m) : sc[i]; };
    // o = sum_t e_t v_t: thread (gi, f) sums float4 column f over t = gi, gi+ng, ...
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (gi < ng) {
      auto fma4 = [&](float e, const float4& vv) {
        acc.x = fmaf(e, vv.x, acc.x);
        acc.y = fmaf(e, vv.y, acc.y);
        acc.z = fmaf(e, vv.z, acc.z);
        acc.w = fmaf(e, vv.w, acc.w);
      };
      if (gi < n) fma4(weight(gi), v0);
      if (gi + ng < n) fma4(weight(gi + ng), v1);
      if (gi + 2 * ng < n) fma4(weight(gi + 2 * ng), v2);
      for (int i = gi + 3 * ng; i < n; i += ng) fma4(weight(i), vrow(t0 + i));
      reinterpret_cast<float4*>(part)[gi * hd4 + f] = acc;
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
    float own = 0.f;  // this chunk's sum of e_t v_t, element tid (tid < hd)
    if (tid < hd)
      for (int g2 = 0; g2 < ng; ++g2) own += part[g2 * hd + tid];
    // the chunk's record (the new cache row is released later, off this
    // path: see wrote_kv)
    if (c != 0) {
      unsigned long long* rec = a.x_att + ((size_t)hb * a.nch_cap + c) * a.att_stride;
      if (tid < hd) st_tag(rec + 4 + tid, tag_att, own);
      if (tid == 0) {
        st_tag(rec, tag_att, m);
        st_tag(rec + 1, tag_att, ls);
      }
    } else {
      // the head's merger: records of chunks 1..nch-1 as pairs (m, l), (sum[2i], sum[2i+1]);
      // o_h[j] = sum_c w_c sum_c[j], w_c = exp(m_c - M) / sum_c' exp(m_c' - M) l_c', chunk order
      float* mrg = part + 4 * kConsumerThreads;  // [nch - 1][hd + 2]
      const int ppr = 1 + half;
      const bool ok2 = poll_pairs_at(
          (nch - 1) * ppr,
          [&](int p) {
            const int cc = 1 + p / ppr, k = p - (cc - 1) * ppr;
            const unsigned long long* r0 = a.x_att + ((size_t)hb * a.nch_cap + cc) * a.att_stride;
            return k == 0 ? r0 : r0 + 4 + 2 * (k - 1);
          },
          tag_att, pc, [&](int p, float x0, float x1) {
            const int cc = p / ppr, k = p - cc * ppr;
            float* rr = mrg + cc * (hd + 2);
            rr[k == 0 ? 0 : 2 * k] = x0;
            rr[k == 0 ? 1 : 2 * k + 1] = x1;
          });
      if (!vote_ok(ok2, pc.s_abort)) return false;
      if (tid < hd) {  // one exponential per chunk, one division
        float M = m;
        for (int cc = 0; cc < nch - 1; ++cc) M = fmaxf(M, mrg[cc * (hd + 2)]);
        const float e0 = expf(m - M);
        float Lsum = e0 * ls, o = e0 * own;
        for (int cc = 0; cc < nch - 1; ++cc) {
          const float e = expf(mrg[cc * (hd + 2)] - M);
          Lsum = fmaf(e, mrg[cc * (hd + 2) + 1], Lsum);
          o = fmaf(e, mrg[cc * (hd + 2) + 2 + tid], o);
        }
        st_tag(a.x_attn + (size_t)hb * hd + tid, tag_att, o / Lsum);
      }
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
  }
  return true;
}

// Next token of each sequence: argmax over the per-CTA candidates
// ([kB][G] pairs; identical in every CTA).
template <int kB>
__device__ inline bool reduce_candidates(const DecodeArgs& a, int parity, unsigned tag,
                                         float* redv, int* redi, const Poll& pc,
                                         int (&token)[kB]) {
  float bv[kB];
  int bi[kB];
#pragma unroll
  for (int b = 0; b < kB; ++b) { bv[b] = -INFINITY; bi[b] = 0x7fffffff; }
  const unsigned long long* base = a.x_cand + (size_t)parity * kB * a.G * 2;
  const bool ok = poll_pairs(base, kB * a.G, tag, pc, [&](int p, float v, float idx) {
    const int i = (int)__float_as_uint(idx), pb = kB == 1 ? 0 : p / a.G;
#pragma unroll
    for (int b = 0; b < kB; ++b)
      if (b == pb && better(v, i, bv[b], bi[b])) { bv[b] = v; bi[b] = i; }
  });
  if (!vote_ok(ok, pc.s_abort)) return false;
#pragma unroll
  for (int b = 0; b < kB; ++b) {
    block_argmax(bv[b], bi[b], redv, redi);
    token[b] = (bi[b] >= 0 && bi[b] < a.V) ? bi[b] : 0;  // 0 only if every logit was NaN
  }
  return true;
}

// ---- the kernel --------------------------------------------------------------------

static_assert(kPlansOffset + 5 * sizeof(StagePlan) <= kMiscBytes, "stage plans overflow");

// This CTA's stage plans of the five GEMV kinds — [Wq|Wk|Wv], Wo, W1/W3
// (interleaved row pairs), W2, the classifier — the same in every layer and
// step, so they are worked out once per launch (8-bit rows are 4 + K/4 words,
// 4-bit rows 4 + K/8).
template <bool kQ8, bool kQ4 = false>
__device__ inline void phase_plans(const DecodeArgs& a, int c, StagePlan* plans) {
  const int kd = kQ4 ? 4 + a.d / 8 : kQ8 ? 4 + a.d / 4 : a.d;
  const int kf = kQ4 ? 4 + a.F / 8 : kQ8 ? 4 + a.F / 4 : a.F;
  plans[0] = plan_stages(a.d + 2 * a.kvd, kd, a.G, c);
  plans[1] = plan_stages(a.d, kd, a.G, c);
  plans[2] = plan_stages(2 * a.F, kd, a.G, c, 2);
  plans[3] = plan_stages(a.d, kf, a.G, c);
  plans[4] = plan_stages(a.V, kd, a.G, c);
}

// The weight stream of one launch, in consumption order: per step, each
// layer's [Wq|Wk|Wv], Wo, W1/W3, W2, then the classifier; this CTA's rows.
template <bool kQ8>
struct DecodeSched {
  const DecodeArgs* a;
  const StagePlan* plans;
  uint32_t refill_delay_ns = kRefillDelayNs;
  int s = 0, l = 0, k = 0;
  int prefetch_ahead = kPrefetchAhead;  // stages prefetched into L2 ahead of the copies
  __device__ void before_copies() {}  // launched without a programmatic dependency
  __device__ bool next(const float*& W, StagePlan& p) {
    if (s >= a->n_steps) return false;
    if (l < a->L) {
      const unsigned char* lw = a->layer0 + (size_t)l * a->layer_stride;
      const unsigned char* ql = kQ8 ? a->q_layer0 + (size_t)l * a->q_stride : nullptr;
      const long long off = k == 0 ? (kQ8 ? a->q_wqkv : a->o_wqkv)
                            : k == 1 ? (kQ8 ? a->q_wo : a->o_wo)
                            : k == 2 ? (kQ8 ? a->q_w13 : a->o_w13)
                                     : (kQ8 ? a->q_w2 : a->o_w2);
      W = reinterpret_cast<const float*>((kQ8 ? ql : lw) + off);
      p = plans[k];
      if (++k == 4) {
        k = 0;
        ++l;
      }
      return true;
    }
    W = kQ8 ? reinterpret_cast<const float*>(a->q_cls) : a->Wcls;
    p = plans[4];
    l = 0;
    k = 0;
    ++s;
    return true;
  }
};

// kB sequences decode in lockstep: sequence b's residual at xs + b d, its
// phase input at vec + b vs, its words in every exchange buffer one vector
// length after sequence b - 1's. The weights stream once for all of them.
// kQ8: quantized rows (8-bit, or 4-bit with kQ4).
template <bool kQ8, int kB, bool kQ4 = false>
__device__ inline bool decode_steps(const DecodeArgs& a, const Ring& r, unsigned char* smem,
                                    volatile int* s_abort) {
  float* xs = reinterpret_cast<float*>(smem + a.sm_xs);
  float* vec = reinterpret_cast<float*>(smem + a.sm_vec);
  float* seg = reinterpret_cast<float*>(smem + a.sm_seg);
  float* asm_ = reinterpret_cast<float*>(smem + a.sm_att);
  float* red = reinterpret_cast<float*>(smem + a.sm_misc) + 8;
  int* redi = reinterpret_cast<int*>(smem + a.sm_misc) + 80;
  const StagePlan* plans = reinterpret_cast<const StagePlan*>(smem + a.sm_misc + kPlansOffset);
  const int tid = threadIdx.x, c = blockIdx.x;
  const int vs = kB == 1 ? 0 : a.vs;
  // 16-byte polls in flight per thread: one batch covers a 768-wide vector,
  // and the 1024 pairs of h at hidden width 2048
  constexpr int kPollDepth = 4;
  constexpr int kPollDepthH = kB == 1 ? 5 : 8;
  const Poll pc{a.err, a.err_host, s_abort, a.wait_limit_ns};
  const unsigned per_step = (unsigned)(kPhasesPerLayer * a.L + 1);
  StageCursor cur;
  bool wrote_kv = false;  // this CTA wrote K/V rows in the current layer's attention
  int token[kB];
#pragma unroll
  for (int b = 0; b < kB; ++b) token[b] = a.start_tokens[b];
  const int n4 = a.d >> 2;  // quads of a residual vector
  // The RMSNorm of a phase input, paper §11.2: x_b = (x * g) * r with r =
  // 1/sqrt(ss/n + eps). The thread that owns quad j of x (j = tid + 224 k over
  // the kB stacked vectors) writes vec = x * g for it and adds x^2 to its share
  // ss[b]; r goes to the GEMV epilogue (EpiTag, EpiArgmax scale), so no pass
  // over the vector and no block reduction stand between the exchange and the
  // GEMV.
  auto norm_quad = [&](int j, const float4& x, const float4& g, float(&ss)[kB]) {
    const int pb = kB == 1 ? 0 : j / n4, jj = j - pb * n4;
    reinterpret_cast<float4*>(vec + (size_t)pb * vs)[jj] =
        make_float4(x.x * g.x, x.y * g.y, x.z * g.z, x.w * g.w);
#pragma unroll
    for (int b = 0; b < kB; ++b)
      if (b == pb) ss[b] = fmaf(x.w, x.w, fmaf(x.z, x.z, fmaf(x.y, x.y, fmaf(x.x, x.x, ss[b]))));
  };
  // x += (published vector), identically in every CTA, and the norm input
  auto add_published = [&](const unsigned long long* src, unsigned tag, const float* gain,
                           float(&ss)[kB]) {
    const float4* g4 = reinterpret_cast<const float4*>(gain);
    return poll_quads<2>(src, kB * n4, tag, g4, n4, pc, [&](int j, float4 v, const float4& g) {
      float4* x4 = reinterpret_cast<float4*>(xs) + j;
      float4 x = *x4;
      x.x += v.x;
      x.y += v.y;
      x.z += v.z;
      x.w += v.w;
      *x4 = x;
      norm_quad(j, x, g, ss);
    });
  };
  // the norm input when no exchange delivered x (the embedding row)
  auto norm_local = [&](const float* gain, float(&ss)[kB]) {
    const float4* g4 = reinterpret_cast<const float4*>(gain);
    for (int j = tid; j < kB * n4; j += kConsumerThreads)
      norm_quad(j, reinterpret_cast<const float4*>(xs)[j],
                g4 ? __ldg(g4 + j % n4) : make_float4(1.f, 1.f, 1.f, 1.f), ss);
  };
  // r_b from every thread's share of ss_b: warp sums go to red, and the block
  // vote that follows the exchange publishes them (and x, vec)
  auto norm_scales = [&](bool ok, float(&ss)[kB], float(&rs)[kMaxBatch]) {
    const int warp = tid >> 5, lane = tid & 31;
#pragma unroll
    for (int b = 0; b < kB; ++b) {
      const float t = warp_sum(ss[b]);
      if (lane == 0) red[warp * kB + b] = t;
    }
    if (!vote_ok(ok, s_abort)) return false;
#pragma unroll
    for (int b = 0; b < kMaxBatch; ++b) {
      float t = 0.f;
      if (b < kB) {
#pragma unroll
        for (int w = 0; w < kConsumerWarps; ++w) t += red[w * kB + b];
      }
      rs[b] = b < kB ? 1.0f / sqrtf(t / (float)a.d + a.eps) : 1.0f;
    }
    return true;
  };
  for (int s = 0; s < a.n_steps; ++s) {
    const int pos = a.start_pos + s;
    const unsigned es = a.epoch0 + (unsigned)s * per_step;
    if (s > 0) {
      if (!reduce_candidates<kB>(a, (s - 1) & 1, es - 1, red, redi, pc, token)) return false;
      if (c == 0 && tid == 0) {
#pragma unroll
        for (int b = 0; b < kB; ++b) a.tokens[(size_t)(s - 1) * kB + b] = token[b];
        a.ts[s - 1] = globaltimer_ns();
      }
    }
    // Acquire: K/V rows written in earlier steps were released (fence, then a
    // published record) before this CTA read those records; this fence and the
    // barrier below order every later row load of the CTA after them.
    if (tid == 0) __threadfence();
    // x = E[token] (paper §4.1: weights are rows at offsets in the blob)
#pragma unroll
    for (int b = 0; b < kB; ++b) {
      float* xb = xs + (size_t)b * a.d;
      if (kQ4) {  // the row the 4-bit codes stand for: scale * code
        const unsigned char* er = a.q_E + (size_t)token[b] * (16 + a.d / 2);
        const float sc = __ldg(reinterpret_cast<const float*>(er));
        const unsigned* cw = reinterpret_cast<const unsigned*>(er + 16);
        for (int j = tid; j < (a.d >> 3); j += kConsumerThreads) {
          const unsigned w = __ldg(cw + j);
          float v[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int c4 = (int)((w >> (4 * k)) & 0xFu);
            v[k] = sc * (float)(c4 >= 8 ? c4 - 16 : c4);
          }
          reinterpret_cast<float4*>(xb)[2 * j] = make_float4(v[0], v[1], v[2], v[3]);
          reinterpret_cast<float4*>(xb)[2 * j + 1] = make_float4(v[4], v[5], v[6], v[7]);
        }
      } else if (kQ8) {  // the row the codes stand for: scale * code
        const unsigned char* er = a.q_E + (size_t)token[b] * (16 + a.d);
        const float sc = __ldg(reinterpret_cast<const float*>(er));
        const int* cw = reinterpret_cast<const int*>(er + 16);
        for (int j = tid; j < (a.d >> 2); j += kConsumerThreads) {
          const int w = __ldg(cw + j);
          reinterpret_cast<float4*>(xb)[j] =
              make_float4(sc * (float)(int)(signed char)(w & 0xff),
                          sc * (float)(int)(signed char)((w >> 8) & 0xff),
                          sc * (float)(int)(signed char)((w >> 16) & 0xff), sc * (float)(w >> 24));
        }
      } else {
        const float4* e4 = reinterpret_cast<const float4*>(a.E + (size_t)token[b] * a.d);
        for (int j = tid; j < (a.d >> 2); j += kConsumerThreads)
          reinterpret_cast<float4*>(xb)[j] = __ldg(e4 + j);
      }
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
    // The four GEMV phases of a layer run one copy of the phase code, in a
    // loop that is not unrolled, so the code stays in the instruction cache
    // from one phase to the next. Phase k's prologue leaves its input in vec.
    for (int l = 0; l < a.L; ++l) {
      const unsigned char* lw = a.layer0 + (size_t)l * a.layer_stride;
      const unsigned el = es + (unsigned)(kPhasesPerLayer * l);
#pragma unroll 1
      for (int k = 0; k < 4; ++k) {
        if (k == 0) att_prefetch_l2<kB>(a, l, pos);
        if (k == 1 && !attention_phase<kB>(a, l, pos, el, el + 1, asm_, red, pc, wrote_kv))
          return false;
        const StagePlan plan = plans[k];
        float rs[kMaxBatch];
#pragma unroll
        for (int b = 0; b < kMaxBatch; ++b) rs[b] = 1.0f;
        if (k == 0 || k == 2) {
          // x += (the previous phase's published output); the input is x * g,
          // scaled by r in the epilogue
          const float* gain =
              a.gains_folded ? nullptr
                             : reinterpret_cast<const float*>(lw + (k == 0 ? a.o_gatt : a.o_gffn));
          float ss[kB];
#pragma unroll
          for (int b = 0; b < kB; ++b) ss[b] = 0.f;
          bool ok = true;
          if (k == 2 || l > 0) ok = add_published(k == 0 ? a.x_f : a.x_o, k == 0 ? el - 1 : el + 2,
                                                  gain, ss);
          else norm_local(gain, ss);
          if (!norm_scales(ok, ss, rs)) return false;
        } else if (k == 1) {
          // o, published by the heads' mergers
          const int hp = a.d >> 1;
          const bool ok = poll_pairs<kPollDepth>(a.x_attn, kB * hp, el + 1, pc,
                                                 [&](int p, float v0, float v1) {
            const int pb = kB == 1 ? 0 : p / hp;
            float* dst = vec + (size_t)pb * vs + 2 * (p - pb * hp);
            dst[0] = v0;
            dst[1] = v1;
          });
          if (!vote_ok(ok, s_abort)) return false;
          // Release the K/V rows this CTA wrote in the attention phase: every
          // result it publishes from here on (at the latest its argmax
          // candidate, which every CTA reads before its next step's attention)
          // orders them before the reads of later steps.
          if (wrote_kv && tid == 0) __threadfence();
          wrote_kv = false;
        } else {  // h, published by the W1/W3 phase
          const int hp = a.F >> 1;
          const bool ok = poll_pairs<kPollDepthH>(a.x_h13, kB * hp, el + 3, pc,
                                                  [&](int p, float v0, float v1) {
            const int pb = kB == 1 ? 0 : p / hp;
            float* dst = vec + (size_t)pb * vs + 2 * (p - pb * hp);
            dst[0] = v0;
            dst[1] = v1;
          });
          if (!vote_ok(ok, s_abort)) return false;
        }
        // [Wq|Wk|Wv] x_b, Wo o, W1/W3 x_b (row pairs: h), W2 h: M rows of K
        // columns, published with the exchange tag of phase k (the attention
        // partials take el + 1)
        const int M = k == 0 ? a.d + 2 * a.kvd : k == 2 ? 2 * a.F : a.d;
        const int K = k == 3 ? a.F : a.d;
        unsigned long long* out = k == 0 ? a.x_qkv : k == 1 ? a.x_o : k == 2 ? a.x_h13 : a.x_f;
        EpiTag e{out, el + (k == 0 ? 0u : (unsigned)k + 1u), k == 2 ? a.F : M, k == 2,
                 {rs[0], rs[1], rs[2], rs[3]}};
        if constexpr (kQ8) {
          uint32_t g = cur.g;
          if (!consume_phase<false, kQ8, kQ4>(r, g, plan, vec, 1, K, seg, e, a.err, a.err_host,
                                              s_abort))
            return false;
          cur.advance(plan.nstages, r.nst);
        } else {
          if (!consume_phase_b<kB>(r, cur, plan, vec, vs, seg, e, a.err, a.err_host, s_abort))
            return false;
        }
      }
    }
    float rs[kMaxBatch];
    {
      float ss[kB];
#pragma unroll
      for (int b = 0; b < kB; ++b) ss[b] = 0.f;
      bool ok = true;
      const float* gf = a.final_gain_folded ? nullptr : a.g_final;
      if (a.L > 0) ok = add_published(a.x_f, es + per_step - 2, gf, ss);
      else norm_local(gf, ss);
      if (!norm_scales(ok, ss, rs)) return false;
    }
    EpiArgmax<kB> ea{a.logits, a.V, {rs[0], rs[1], rs[2], rs[3]}};
    ea.init();
    if constexpr (kQ8) {
      uint32_t g = cur.g;
      if (!consume_phase<false, kQ8, kQ4>(r, g, plans[4], vec, 1, a.d, seg, ea, a.err,
                                          a.err_host, s_abort))
        return false;
      cur.advance(plans[4].nstages, r.nst);
    } else {
      if (!consume_phase_b<kB>(r, cur, plans[4], vec, vs, seg, ea, a.err, a.err_host, s_abort))
        return false;
    }
#pragma unroll
    for (int b = 0; b < kB; ++b) {
      float bv = ea.bv[b];
      int bi = ea.bi[b];
      block_argmax(bv, bi, red, redi);
      if (tid == 0) {
        unsigned long long* dst = a.x_cand + (((size_t)(s & 1) * kB + b) * a.G + c) * 2;
        st_tag(dst, es + per_step - 1, bv);
        st_tag(dst + 1, es + per_step - 1, __uint_as_float((unsigned)bi));
      }
    }
  }
  if (a.final_token && c == 0) {
    const int s = a.n_steps - 1;
    if (!reduce_candidates<kB>(a, s & 1, a.epoch0 + (unsigned)a.n_steps * per_step - 1, red,
                               redi, pc, token))
      return false;
    if (tid == 0) {
#pragma unroll
      for (int b = 0; b < kB; ++b) a.tokens[(size_t)s * kB + b] = token[b];
      a.ts[s] = globaltimer_ns();
    }
  }
  return true;
}

template <bool kQ8, int kB, bool kQ4 = false>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const __grid_constant__ DecodeArgs a) {
  extern __shared__ __align__(128) unsigned char smem[];
  Ring r;
  r.buf = smem + a.sm_ring;
  r.full = reinterpret_cast<uint64_t*>(smem + a.sm_bars);
  r.empty = r.full + a.nst;
  r.seq = reinterpret_cast<volatile int*>(r.empty + a.nst);
  r.nst = a.nst;
  volatile int* s_abort = reinterpret_cast<volatile int*>(smem + a.sm_misc);
  if (threadIdx.x == 0) {
    for (int i = 0; i < a.nst; ++i) {
      mbar_init(&r.full[i], 1);
      mbar_init(&r.empty[i], 1);
      r.seq[i] = 0;
    }
    *s_abort = 0;
    phase_plans<kQ8, kQ4>(a, blockIdx.x,
                          reinterpret_cast<StagePlan*>(smem + a.sm_misc + kPlansOffset));
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x >= kConsumerThreads) {
    if (threadIdx.x == kConsumerThreads) {
      DecodeSched<kQ8> sched;
      sched.a = &a;
      sched.plans = reinterpret_cast<const StagePlan*>(smem + a.sm_misc + kPlansOffset);
      run_producer(r, sched, a.err, a.err_host, s_abort);
    }
    return;
  }
  decode_steps<kQ8, kB, kQ4>(a, r, smem, s_abort);
}

// decode_kernel<false, B> for B = 2..kMaxBatch (defined in decode_batch.cu).
const void* decode_kernel_for_batch(int B);

}  // namespace tvl
