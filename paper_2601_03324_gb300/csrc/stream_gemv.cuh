// stream_gemv.cuh — the weight-streaming GEMV engine shared by the decode
// kernel and the standalone GEMV (paper §3.1: y = W x reads every weight once,
// so the work is bound by memory; §6.1: one dot product per output row).
//
// Per CTA: a producer warp fills a ring of shared-memory stages with bulk
// asynchronous copies (the TMA engine) of a contiguous range of weight rows,
// each stage completing on an mbarrier; seven consumer warps multiply each
// landed stage by the input vector held in shared memory and hand the stage
// back through a second mbarrier. The producer walks a static schedule of
// phases that does not depend on activations, so the copies run ahead of
// whatever the consumers are waiting for. (Eight warps in all: two per SM
// sub-partition, which leaves each thread up to 255 registers; a ninth warp
// would put three warps on one sub-partition and cap them at 168.) The
// producer is a warp of its own because issuing a bulk copy can stall when
// the copy engine's queue is full, and that stall must not hold up the math. This is the GPU form of the paper's two memory ideas: the
// weights flow as one aligned stream (§3.2, §4.1) and several independent
// loads are always in flight (§11.1's four accumulators become several
// 32 KB stages in flight per SM).
//
// Work split: CTA c owns rows [M*c/G, M*(c+1)/G) of an [M x K] matrix, which
// is one contiguous byte range. A stage (16 KB) holds whole rows, or one
// segment of a row longer than a stage. Stage g of the CTA belongs to consumer
// warp g mod 7, which waits for it, computes its rows (two at a time, one
// float4 stream per lane and one shuffle tree per row), stores the results and
// hands the stage back: the warps work on different stages at once and meet
// only at the end of a phase. Segment partial sums of long rows are added in
// segment order at that point, so every result is bit-reproducible.
#pragma once
#include "ptx.cuh"

namespace tvl {

constexpr int kConsumerWarps = 7;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kThreads = kConsumerThreads + 32;  // + the producer warp
constexpr int kStageBytes = 16384;
constexpr int kStageFloats = kStageBytes / 4;
constexpr int kMaxRowsPerStage = 256;
constexpr int kMaxSegParts = 2048;    // segment partials of one phase (rows x segments)
constexpr int kMaxStages = 12;        // ring slots
constexpr uint32_t kBarConsumers = 1; // named barrier of the consumer warps
constexpr unsigned long long kWaitLimitNs = 1000000000ull;  // 1 s per wait

// Error codes written by kernels (same values as tvl_status).
constexpr int kErrTimeout = 7;

// Stage plan of one CTA over rows [r0, r1) of an [M x K] row-major matrix.
struct StagePlan {
  int r0, r1, K;
  int rps;  // rows per stage when a row fits in a stage
  int spr;  // stages per row when it does not (else 1)
  int seg;  // floats per segment when spr > 1 (multiple of 32)
  int nstages;
  int gran;    // 2: rows come in pairs (2i, 2i+1) whose results meet in one epilogue call
  bool defer;  // results wait in the segment scratch and are stored at the end of the phase
};

struct StageDesc {
  int row, nrows, c0, c1;  // rows [row, row+nrows), columns [c0, c1)
};

// Requires K % 4 == 0 (16-byte rows) and kStageFloats % 32 == 0. A stage has
// at most kMaxRowsPerStage rows, or one segment of at most kStageFloats. With
// gran 2 (M even) a CTA owns whole pairs of rows and a stage holds whole
// pairs, unless a pair does not fit a stage: then the rows' results are
// deferred to the end of the phase, like the segments of rows longer than a
// stage.
__host__ __device__ inline StagePlan plan_stages(long long M, int K, int G, int c,
                                                 int gran = 1) {
  StagePlan p;
  p.gran = gran;
  p.r0 = gran * (int)((M / gran) * c / G);
  p.r1 = gran * (int)((M / gran) * (c + 1) / G);
  p.K = K;
  p.defer = false;
  const int nrows = p.r1 - p.r0;
  if (K <= kStageFloats) {
    // rows per stage: as many as fit, but few enough that the CTA's rows of
    // this phase spread over all consumer warps (a phase's latency is that of
    // its busiest warp)
    int cap = kStageFloats / K;
    if (cap > kMaxRowsPerStage) cap = kMaxRowsPerStage;
    int spread = (nrows + kConsumerWarps - 1) / kConsumerWarps;
    if (spread < 1) spread = 1;
    if (gran == 2) spread += spread & 1;
    p.rps = spread < cap ? spread : cap;
    // more than four rows: whole passes of four (the row routine takes up to
    // four rows at once, and a pass of one row costs a full warp reduction)
    if (p.rps > 4) p.rps &= ~3;
    if (gran == 2 && p.rps >= 2) p.rps &= ~1;
    p.defer = gran == 2 && p.rps < 2;
    p.spr = 1;
    p.seg = K;
    p.nstages = (nrows + p.rps - 1) / p.rps;
  } else {
    p.rps = 1;
    p.spr = (K + kStageFloats - 1) / kStageFloats;
    p.seg = ((K + p.spr - 1) / p.spr + 31) / 32 * 32;
    p.nstages = nrows * p.spr;
    p.defer = true;
  }
  return p;
}

__host__ __device__ inline StageDesc stage_desc(const StagePlan& p, int j) {
  StageDesc s;
  if (p.spr == 1) {
    s.row = p.r0 + j * p.rps;
    s.nrows = (p.r1 - s.row < p.rps) ? (p.r1 - s.row) : p.rps;
    s.c0 = 0;
    s.c1 = p.K;
  } else {
    s.row = p.r0 + j / p.spr;
    s.nrows = 1;
    const int k = j % p.spr;
    s.c0 = k * p.seg;
    s.c1 = (s.c0 + p.seg < p.K) ? (s.c0 + p.seg) : p.K;
  }
  return s;
}

struct Ring {
  unsigned char* buf;
  uint64_t* full;     // [nst] stage landed
  uint64_t* empty;    // [nst] stage consumed
  volatile int* seq;  // [nst] 1 + number of the stage last queued into the slot
  int nst;
};

// Shared-memory bytes of a ring's barriers and sequence numbers.
constexpr int kRingBarBytes = 3 * kMaxStages * 8;

__device__ __forceinline__ void raise_error(int* err, int* err_host, int code) {
  if (err) atomicCAS(err, 0, code);
  if (err_host) *reinterpret_cast<volatile int*>(err_host) = code;
}

// Single-thread bounded wait. Gives up on abort (when honoured), on an error
// raised elsewhere, or after kWaitLimitNs; returns false then.
__device__ inline bool wait_bounded(uint64_t* bar, uint32_t par, const int* err,
                                    volatile int* s_abort, bool honour_abort, bool* timed_out) {
  if (mbar_try_wait(bar, par)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, par)) return true;
    if ((it & 15u) == 0) {
      if (honour_abort && (*s_abort || (err && ld_volatile_s32(err)))) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs || it > (1u << 26)) {
        if (timed_out) *timed_out = true;
        return false;
      }
    }
  }
}

// Producer: queue the stages of a static schedule of GEMV phases into the
// ring, in order. Sched::next(W, plan) yields the next phase's matrix and this
// CTA's stage plan, false at the end. Before reusing a slot it waits for the
// consumers to release it; before returning it waits for every copy it queued
// (a CTA must not exit with copies into its shared memory in flight).
// A second walk over the same schedule, kPrefetchAhead stages ahead of the
// copies: each of its stages is prefetched into L2, so that the HBM reads of
// a stage are done well before its copy into shared memory is issued.
constexpr int kPrefetchAhead = 12;
template <class Sched>
struct PrefetchCursor {
  Sched sched;
  const float* W = nullptr;
  StagePlan p;
  int j = 0;
  bool valid = false;
  __device__ void start() {
    valid = sched.next(W, p);
    j = 0;
  }
  __device__ void step() {  // prefetch the next stage of the schedule, if any
    while (valid && j >= p.nstages) {
      valid = sched.next(W, p);
      j = 0;
    }
    if (!valid) return;
    const StageDesc s = stage_desc(p, j++);
    bulk_prefetch_l2(W + (size_t)s.row * p.K + s.c0, (uint32_t)(s.nrows * (s.c1 - s.c0)) * 4u);
  }
};

template <class Sched>
__device__ inline void run_producer(const Ring& r, Sched& sched, int* err, int* err_host,
                                    volatile int* s_abort) {
  const uint64_t pol = l2_evict_first();
  uint32_t g = 0;
  const float* W = nullptr;
  StagePlan p;
  bool ok = true;
  PrefetchCursor<Sched> ahead;
  ahead.sched = sched;
  ahead.start();
  for (int i = 0; i < sched.prefetch_ahead; ++i) ahead.step();
  // the first copies may need the grids this one depends on to have finished
  // (the L2 prefetches above only warm the cache)
  sched.before_copies();
  while (ok && sched.next(W, p)) {
    for (int j = 0; j < p.nstages; ++j, ++g) {
      if (sched.prefetch_ahead > 0) ahead.step();
      const int slot = (int)(g % (uint32_t)r.nst);
      if (g >= (uint32_t)r.nst) {
        bool to = false;
        const uint32_t par = ((g / (uint32_t)r.nst) - 1u) & 1u;
        const bool was_free = mbar_try_wait(&r.empty[slot], par);
        if (!was_free && !wait_bounded(&r.empty[slot], par, err, s_abort, true, &to)) {
          if (to) raise_error(err, err_host, kErrTimeout);
          *s_abort = 1;
          ok = false;
          break;
        }
        // Slots come back in bursts, at the end of a phase, just when the
        // consumers start polling for that phase's exchange; refilling them
        // at once would put a burst of HBM misses in front of those polls.
        if (!was_free && sched.refill_delay_ns) {
          const uint64_t t0 = globaltimer_ns();
          while (globaltimer_ns() - t0 < sched.refill_delay_ns) {}
        }
      }
      const StageDesc s = stage_desc(p, j);
      const uint32_t bytes = (uint32_t)(s.nrows * (s.c1 - s.c0)) * 4u;
      mbar_arrive_expect_tx(&r.full[slot], bytes);
      bulk_g2s(r.buf + (size_t)slot * kStageBytes, W + (size_t)s.row * p.K + s.c0, bytes,
               &r.full[slot], pol);
      // The slot's barrier is now in this stage's phase: say so. Consumers
      // take stages out of order, and a parity wait is only meaningful once
      // the barrier has reached the awaited phase.
      __threadfence_block();
      r.seq[slot] = (int)(g + 1u);
    }
  }
  const uint32_t from = g > (uint32_t)r.nst ? g - (uint32_t)r.nst : 0u;
  for (uint32_t k = from; k < g; ++k)
    wait_bounded(&r.full[k % (uint32_t)r.nst], (k / (uint32_t)r.nst) & 1u, nullptr, nullptr,
                 false, nullptr);
}

// All consumer threads poll; thread 0 alone applies the limit and raises the
// abort flag, which the others observe (the producer may raise it too).
// Returns true if the stage landed. The flag is only a hint to stop waiting:
// the decision to leave is taken by a vote at the next barrier.
__device__ inline bool consumer_wait_full(uint64_t* bar, uint32_t par, int* err, int* err_host,
                                          volatile int* s_abort) {
  if (mbar_try_wait(bar, par)) return true;
  const bool leader = threadIdx.x == 0;
  const uint64_t t0 = leader ? globaltimer_ns() : 0;
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, par)) return true;
    if (*s_abort) return false;
    if (leader && (it & 15u) == 0) {
      if (err && ld_volatile_s32(err)) {
        *s_abort = 1;
        return false;
      }
      if (globaltimer_ns() - t0 > kWaitLimitNs || it > (1u << 26)) {
        raise_error(err, err_host, kErrTimeout);
        *s_abort = 1;
        return false;
      }
    }
  }
}

// Lane part of one row's dot product: n4 float4 of weights (shared memory)
// and input; lane takes float4 lane, lane + 32, ...
__device__ __forceinline__ float row_partial(const float4* w4, const float4* x4, int n4,
                                             int lane) {
  float4 c0 = make_float4(0.f, 0.f, 0.f, 0.f), c1 = c0;
  int e = lane;
#pragma unroll 2
  for (; e + 32 < n4; e += 64) {
    const float4 w0 = w4[e], x0 = x4[e], w1 = w4[e + 32], x1 = x4[e + 32];
    c0.x = fmaf(w0.x, x0.x, c0.x);
    c0.y = fmaf(w0.y, x0.y, c0.y);
    c0.z = fmaf(w0.z, x0.z, c0.z);
    c0.w = fmaf(w0.w, x0.w, c0.w);
    c1.x = fmaf(w1.x, x1.x, c1.x);
    c1.y = fmaf(w1.y, x1.y, c1.y);
    c1.z = fmaf(w1.z, x1.z, c1.z);
    c1.w = fmaf(w1.w, x1.w, c1.w);
  }
  if (e < n4) {
    const float4 w0 = w4[e], x0 = x4[e];
    c0.x = fmaf(w0.x, x0.x, c0.x);
    c0.y = fmaf(w0.y, x0.y, c0.y);
    c0.z = fmaf(w0.z, x0.z, c0.z);
    c0.w = fmaf(w0.w, x0.w, c0.w);
  }
  return ((c0.x + c0.y) + (c0.z + c0.w)) + ((c1.x + c1.y) + (c1.z + c1.w));
}

// Two rows with the same columns in one pass: each x float4 is read once
// for both (half the shared-memory traffic of two separate passes).
__device__ __forceinline__ float2 row2_partial(const float4* w0, const float4* w1, const float4* x4,
                                               int n4, int lane) {
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
#pragma unroll 2
  for (int e = lane; e < n4; e += 32) {
    const float4 x = x4[e], u = w0[e], v = w1[e];
    a.x = fmaf(u.x, x.x, a.x);
    a.y = fmaf(u.y, x.y, a.y);
    a.z = fmaf(u.z, x.z, a.z);
    a.w = fmaf(u.w, x.w, a.w);
    b.x = fmaf(v.x, x.x, b.x);
    b.y = fmaf(v.y, x.y, b.y);
    b.z = fmaf(v.z, x.z, b.z);
    b.w = fmaf(v.w, x.w, b.w);
  }
  return make_float2((a.x + a.y) + (a.z + a.w), (b.x + b.y) + (b.z + b.w));
}

// Same for rows of at most 1024 floats with the lane's slice of x already in
// registers: xr[k] holds x float4 lane + 32k.
__device__ __forceinline__ float row_partial_xr(const float4* w4, const float4 (&xr)[8], int n4,
                                                int lane) {
  float4 c0 = make_float4(0.f, 0.f, 0.f, 0.f), c1 = c0;
#pragma unroll
  for (int k = 0; k < 8; k += 2) {
    if (lane + 32 * k < n4) {
      const float4 w = w4[lane + 32 * k];
      c0.x = fmaf(w.x, xr[k].x, c0.x);
      c0.y = fmaf(w.y, xr[k].y, c0.y);
      c0.z = fmaf(w.z, xr[k].z, c0.z);
      c0.w = fmaf(w.w, xr[k].w, c0.w);
    }
    if (lane + 32 * (k + 1) < n4) {
      const float4 w = w4[lane + 32 * (k + 1)];
      c1.x = fmaf(w.x, xr[k + 1].x, c1.x);
      c1.y = fmaf(w.y, xr[k + 1].y, c1.y);
      c1.z = fmaf(w.z, xr[k + 1].z, c1.z);
      c1.w = fmaf(w.w, xr[k + 1].w, c1.w);
    }
  }
  return ((c0.x + c0.y) + (c0.z + c0.w)) + ((c1.x + c1.y) + (c1.z + c1.w));
}

// 8-bit weight rows (weight-only codes, one scale per row). A packed row is
// 16 + K bytes: the float32 scale, 12 zero bytes, then K int8 codes; in a
// stage a row is Kw = 4 + K/4 words. Code word e holds codes 4e..4e+3 and
// meets x float4 e.
__device__ __forceinline__ void fma_codes(float4& acc, int w, const float4& x) {
  // code + 128 as the low byte of the float 2^23 + (code + 128): one byte
  // permute and one exact subtraction per code, on full-rate pipes (an
  // integer-to-float conversion is a quarter-rate instruction)
  const unsigned u = (unsigned)w ^ 0x80808080u;
  const float c0 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7540)) - 8388736.0f;
  const float c1 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7541)) - 8388736.0f;
  const float c2 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7542)) - 8388736.0f;
  const float c3 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7543)) - 8388736.0f;
  acc.x = fmaf(c0, x.x, acc.x);
  acc.y = fmaf(c1, x.y, acc.y);
  acc.z = fmaf(c2, x.z, acc.z);
  acc.w = fmaf(c3, x.w, acc.w);
}

// Lane partials of sum_j q_j x_j for two 8-bit rows sharing x (nw code words).
__device__ __forceinline__ float2 row2_partial_q8(const int* c0, const int* c1, const float4* x4,
                                                  int nw, int lane) {
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
#pragma unroll 8
  for (int e = lane; e < nw; e += 32) {
    const float4 x = x4[e];
    fma_codes(a, c0[e], x);
    fma_codes(b, c1[e], x);
  }
  return make_float2((a.x + a.y) + (a.z + a.w), (b.x + b.y) + (b.z + b.w));
}

__device__ __forceinline__ float row_partial_q8(const int* c0, const float4* x4, int nw, int lane) {
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
  for (int e = lane; e < nw; e += 32) fma_codes(a, c0[e], x4[e]);
  return (a.x + a.y) + (a.z + a.w);
}

// 4-bit weight rows: a packed row is 16 + K/2 bytes (the float32 scale, 12
// zero bytes, then two codes per byte, low nibble first, each a 4-bit two's
// complement integer in [-7, 7]); in a stage a row is 4 + K/8 words. Code
// word e holds codes 8e..8e+7 and meets x float4 2e and 2e + 1.
__device__ __forceinline__ void fma_nibbles(float4& acc, int w, const float4& xa,
                                            const float4& xb) {
  // code + 8 (in [1, 15]) as the low bits of the float 2^23 + (code + 8):
  // a shift, a mask and an OR per code, then one exact subtraction
  // even columns (low nibbles) and odd columns (high nibbles) as bytes, then
  // each byte into the float 2^23 + (code + 8) by one byte permute
  const unsigned u = (unsigned)w ^ 0x88888888u;
  const unsigned ev = u & 0x0F0F0F0Fu, od = (u >> 4) & 0x0F0F0F0Fu;
  auto c = [](unsigned v, unsigned sel) {
    return __uint_as_float(__byte_perm(v, 0x4B000000u, sel)) - 8388616.0f;
  };
  acc.x = fmaf(c(ev, 0x7540), xa.x, acc.x);  // column 0
  acc.y = fmaf(c(od, 0x7540), xa.y, acc.y);  // column 1
  acc.z = fmaf(c(ev, 0x7541), xa.z, acc.z);  // column 2
  acc.w = fmaf(c(od, 0x7541), xa.w, acc.w);  // column 3
  acc.x = fmaf(c(ev, 0x7542), xb.x, acc.x);  // column 4
  acc.y = fmaf(c(od, 0x7542), xb.y, acc.y);  // column 5
  acc.z = fmaf(c(ev, 0x7543), xb.z, acc.z);  // column 6
  acc.w = fmaf(c(od, 0x7543), xb.w, acc.w);  // column 7
}

// Lane partials of sum_j q_j x_j for two 4-bit rows sharing x (nw code words).
__device__ __forceinline__ float2 row2_partial_q4(const int* c0, const int* c1, const float4* x4,
                                                  int nw, int lane) {
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b = a;
#pragma unroll 4
  for (int e = lane; e < nw; e += 32) {
    const float4 xa = x4[2 * e], xb = x4[2 * e + 1];
    fma_nibbles(a, c0[e], xa, xb);
    fma_nibbles(b, c1[e], xa, xb);
  }
  return make_float2((a.x + a.y) + (a.z + a.w), (b.x + b.y) + (b.z + b.w));
}

__device__ __forceinline__ float row_partial_q4(const int* c0, const float4* x4, int nw, int lane) {
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
  for (int e = lane; e < nw; e += 32) fma_nibbles(a, c0[e], x4[2 * e], x4[2 * e + 1]);
  return (a.x + a.y) + (a.z + a.w);
}

// Warp-level bounded wait for stage gs in `slot` (all lanes poll, lane 0
// applies the limit): first until the producer has queued that stage into the
// slot, then until its bytes have landed. Returns the same answer in every
// lane of the warp.
__device__ inline bool warp_wait_full_at(const Ring& r, int slot, uint32_t par, uint32_t gs,
                                         bool need_seq, int* err, int* err_host,
                                         volatile int* s_abort);

__device__ inline bool warp_wait_full(const Ring& r, int slot, uint32_t gs, int* err,
                                      int* err_host, volatile int* s_abort) {
  return warp_wait_full_at(r, slot, (gs / (uint32_t)r.nst) & 1u, gs, true, err, err_host,
                           s_abort);
}

// The same wait with the slot's parity given (gs / nst, odd or even).
// need_seq: the stage that used the slot before (gs - nst) may still be on its
// way (it belongs to the same phase), so the barrier may be a whole lap behind
// and its parity alone cannot tell the laps apart; the sequence word can.
__device__ inline bool warp_wait_full_at(const Ring& r, int slot, uint32_t par, uint32_t gs,
                                         bool need_seq, int* err, int* err_host,
                                         volatile int* s_abort) {
  uint64_t* bar = &r.full[slot];
  // usual case: the stage was queued long ago and has landed
  if (__all_sync(0xffffffffu, (!need_seq || r.seq[slot] == (int)(gs + 1u)) &&
                                  mbar_test_wait(bar, par)))
    return true;
  bool ok = true;
  if (need_seq && r.seq[slot] != (int)(gs + 1u)) {
    const bool leader = (threadIdx.x & 31) == 0;
    const uint64_t t0 = leader ? globaltimer_ns() : 0;
    for (uint32_t it = 1; r.seq[slot] != (int)(gs + 1u); ++it) {
      if (*s_abort) {
        ok = false;
        break;
      }
      if (leader && (it & 15u) == 0) {
        if ((err && ld_volatile_s32(err)) || globaltimer_ns() - t0 > kWaitLimitNs ||
            it > (1u << 26)) {
          if (!(err && ld_volatile_s32(err))) raise_error(err, err_host, kErrTimeout);
          *s_abort = 1;
          ok = false;
          break;
        }
      }
    }
  }
  __threadfence_block();
  if (!__any_sync(0xffffffffu, !ok)) ok = true;
  else return false;
  if (!mbar_try_wait(bar, par)) {
    const bool leader = (threadIdx.x & 31) == 0;
    const uint64_t t0 = leader ? globaltimer_ns() : 0;
    for (uint32_t it = 1;; ++it) {
      if (mbar_try_wait(bar, par)) break;
      if (*s_abort) {
        ok = false;
        break;
      }
      if (leader && (it & 15u) == 0) {
        if ((err && ld_volatile_s32(err)) || globaltimer_ns() - t0 > kWaitLimitNs ||
            it > (1u << 26)) {
          if (!(err && ld_volatile_s32(err))) raise_error(err, err_host, kErrTimeout);
          *s_abort = 1;
          ok = false;
          break;
        }
      }
    }
  }
  return !__any_sync(0xffffffffu, !ok);
}

// Consumer: one GEMV phase over the CTA's stage plan. The input vector xs is
// in shared memory; with S > 1 the matrix is viewed as [M*S x Kc] "virtual
// rows" (row r, K-chunk s) and virtual row v reads xs + (v % S) * Kc.
// epi.store(v, value) receives each finished (virtual) row, or
// epi.store_pair(v, value_v, value_v+1) two rows v (even with gran 2) and
// v + 1 computed together, from lane 0 of the warp that computed them, or
// (deferred rows) from the thread that adds the rows' partials at the end of
// the phase. seg is shared scratch for those partials. Ends with a barrier of the consumer
// warps; returns false on abort, identically in every consumer thread.
template <bool kXReg = true, bool kQ8 = false, bool kQ4 = false, class Epi>
__device__ inline bool consume_phase(const Ring& r, uint32_t& g, const StagePlan& p,
                                     const float* xs, int S, int Kc, float* seg, Epi& epi,
                                     int* err, int* err_host, volatile int* s_abort) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // Rows of at most 1024 floats (whole rows in a stage, one K-chunk): each lane
  // keeps its x slice in registers for the whole phase.
  const bool xreg = kXReg && !kQ8 && !kQ4 && (p.spr == 1) && (p.K <= 1024) && (S == 1);
  float4 xr[8];
  if (xreg) {
    const float4* x4 = reinterpret_cast<const float4*>(xs);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int e = lane + 32 * k;
      xr[k] = (e < (p.K >> 2)) ? x4[e] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  bool ok = true;
  // this warp's stages of the phase: global stage numbers g + j with (g + j) % 7 == warp
  int j = (int)((warp + kConsumerWarps - (int)(g % kConsumerWarps)) % kConsumerWarps);
  for (; j < p.nstages && ok; j += kConsumerWarps) {
    const uint32_t gs = g + (uint32_t)j;
    const int slot = (int)(gs % (uint32_t)r.nst);
    if (!warp_wait_full(r, slot, gs, err, err_host, s_abort)) {
      ok = false;
      break;
    }
    const StageDesc s = stage_desc(p, j);
    const int ncols = s.c1 - s.c0, n4 = ncols >> 2;
    const float* st = reinterpret_cast<const float*>(r.buf + (size_t)slot * kStageBytes);
    if (kQ8 || kQ4) {  // whole 8-bit or 4-bit rows (ncols = Kw words): y = scale * sum q x
      const float4* x4 = reinterpret_cast<const float4*>(xs);
      for (int ri = 0; ri < s.nrows; ri += 2) {
        const bool two = ri + 1 < s.nrows;
        const float* r0 = st + (size_t)ri * ncols;
        const float* r1 = r0 + ncols;
        const int* c0 = reinterpret_cast<const int*>(r0 + 4);
        const int* c1 = reinterpret_cast<const int*>(r1 + 4);
        float a0, a1 = 0.f;
        if (two) {
          const float2 t = kQ4 ? row2_partial_q4(c0, c1, x4, ncols - 4, lane)
                               : row2_partial_q8(c0, c1, x4, ncols - 4, lane);
          a0 = t.x;
          a1 = t.y;
        } else {
          a0 = kQ4 ? row_partial_q4(c0, x4, ncols - 4, lane) : row_partial_q8(c0, x4, ncols - 4, lane);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          a0 += __shfl_xor_sync(0xffffffffu, a0, o);
          a1 += __shfl_xor_sync(0xffffffffu, a1, o);
        }
        if (lane == 0) {
          if (p.defer) seg[s.row + ri - p.r0] = r0[0] * a0;
          else if (two) epi.store_pair(s.row + ri, r0[0] * a0, r1[0] * a1);
          else epi.store(s.row + ri, r0[0] * a0);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&r.empty[slot]);  // stage free for the producer
      continue;
    }
    for (int ri = 0; ri < s.nrows; ri += 2) {
      const bool two = ri + 1 < s.nrows;
      const int v0 = s.row + ri, v1 = v0 + 1;
      const float4* w0 = reinterpret_cast<const float4*>(st + (size_t)ri * ncols);
      const float4* w1 = w0 + n4;
      float a0, a1 = 0.f;
      if (xreg) {
        a0 = row_partial_xr(w0, xr, n4, lane);
        if (two) a1 = row_partial_xr(w1, xr, n4, lane);
      } else {
        const float* xb = xs + s.c0;
        const int o0 = S > 1 ? (v0 % S) * Kc : 0, o1 = S > 1 ? (v1 % S) * Kc : 0;
        if (two && o0 == o1) {  // same input columns: one pass for both rows
          const float2 r2 = row2_partial(w0, w1, reinterpret_cast<const float4*>(xb + o0), n4, lane);
          a0 = r2.x;
          a1 = r2.y;
        } else {
          a0 = row_partial(w0, reinterpret_cast<const float4*>(xb + o0), n4, lane);
          if (two) a1 = row_partial(w1, reinterpret_cast<const float4*>(xb + o1), n4, lane);
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        a0 += __shfl_xor_sync(0xffffffffu, a0, o);
        a1 += __shfl_xor_sync(0xffffffffu, a1, o);
      }
      if (lane == 0) {
        if (p.defer) {  // one row (or segment) per stage
          seg[(v0 - p.r0) * p.spr + j % p.spr] = a0;
        } else if (two) {
          epi.store_pair(v0, a0, a1);
        } else {
          epi.store(v0, a0);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&r.empty[slot]);  // stage free for the producer
  }
  g += (uint32_t)p.nstages;
  // every stage of the phase is consumed (or the CTA gives up together)
  if (named_bar_or(kBarConsumers, kConsumerThreads, !ok)) {
    if (tid == 0) *s_abort = 1;
    return false;
  }
  if (p.defer) {  // deferred rows: add each row's segments in order
    auto row_sum = [&](int ri) {
      float v = 0.f;
      for (int k = 0; k < p.spr; ++k) v += seg[ri * p.spr + k];
      return v;
    };
    const int nr = p.r1 - p.r0;
    for (int q = tid; q * p.gran < nr; q += kConsumerThreads) {
      if (p.gran == 2) epi.store_pair(p.r0 + 2 * q, row_sum(2 * q), row_sum(2 * q + 1));
      else epi.store(p.r0 + q, row_sum(q));
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
  }
  return true;
}

// ---- several input vectors (batched decode) ----------------------------------------

__host__ __device__ constexpr int pow2_at_least(int n) { return n <= 1 ? 1 : 2 * pow2_at_least((n + 1) / 2); }

// Sums N values (N a power of two, at most 32) over the warp at once: after
// the call lane l holds the warp's sum of v[l / (32 / N)]. Each halving step
// trades half of a lane's values with its partner, so the warp spends N - 1 +
// log2(32 / N) shuffles instead of 5 N.
template <int N>
__device__ __forceinline__ float warp_sum_transposed(float (&v)[N], int lane) {
#pragma unroll
  for (int t = 0; t < 5; ++t) {
    const int o = 16 >> t;
    const int cnt = (N >> t) > 1 ? (N >> t) : 1;
    if (cnt > 1) {
      const int half = cnt / 2;
      const bool up = (lane & o) != 0;
#pragma unroll
      for (int i = 0; i < half; ++i) {
        const float send = up ? v[i] : v[i + half];
        const float keep = up ? v[i + half] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
      }
    } else {
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
    }
  }
  return v[0];
}

// R rows of a stage (row r at w + r * ncols, ncols floats) times kB vectors
// (vector b at x + b * vs): every weight float4 read from shared memory meets
// all kB vectors, every x float4 all R rows. put(r, b, value, next) is called
// by the lane that holds the sum of row r with vector b; next is the sum of
// row r + 1 with vector b when r + 1 < R.
template <int R, int kB, class Put>
__device__ __forceinline__ void rows_times_vectors(const float* w, int ncols, const float* x,
                                                   int vs, int lane, bool pairs, Put put) {
  const int n4 = ncols >> 2, vs4 = vs >> 2;
  const float4* w4 = reinterpret_cast<const float4*>(w);
  const float4* x4 = reinterpret_cast<const float4*>(x);
  // Few products: a float4 of partial sums each (four independent chains);
  // many: one sum each (enough chains already, and fewer registers).
  constexpr bool kWide = R * kB < 8;
  constexpr int A = kWide ? 4 : 1;
  float acc[R * kB][A];
#pragma unroll
  for (int i = 0; i < R * kB; ++i)
#pragma unroll
    for (int k = 0; k < A; ++k) acc[i][k] = 0.f;
#pragma unroll 2
  for (int e = lane; e < n4; e += 32) {
    float4 wv[R];
#pragma unroll
    for (int r = 0; r < R; ++r) wv[r] = w4[r * n4 + e];
#pragma unroll
    for (int b = 0; b < kB; ++b) {
      const float4 xv = x4[b * vs4 + e];
#pragma unroll
      for (int r = 0; r < R; ++r) {
        float* a = acc[r * kB + b];
        if (kWide) {
          a[0] = fmaf(wv[r].x, xv.x, a[0]);
          a[A > 1 ? 1 : 0] = fmaf(wv[r].y, xv.y, a[A > 1 ? 1 : 0]);
          a[A > 2 ? 2 : 0] = fmaf(wv[r].z, xv.z, a[A > 2 ? 2 : 0]);
          a[A > 3 ? 3 : 0] = fmaf(wv[r].w, xv.w, a[A > 3 ? 3 : 0]);
        } else {
          a[0] = fmaf(wv[r].w, xv.w, fmaf(wv[r].z, xv.z, fmaf(wv[r].y, xv.y, fmaf(wv[r].x, xv.x, a[0]))));
        }
      }
    }
  }
  constexpr int N = pow2_at_least(R * kB);
  float v[N];
#pragma unroll
  for (int i = 0; i < N; ++i)
    v[i] = i >= R * kB ? 0.f : kWide ? (acc[i][0] + acc[i][A > 1 ? 1 : 0]) + (acc[i][A > 2 ? 2 : 0] + acc[i][A > 3 ? 3 : 0]) : acc[i][0];
  const float t = warp_sum_transposed<N>(v, lane);
  // the next row's sum for the same vector, for paired rows
  const float tn = pairs ? __shfl_down_sync(0xffffffffu, t, kB * (32 / N)) : 0.f;
  const int idx = lane / (32 / N);
  if (lane % (32 / N) == 0 && idx < R * kB) put(idx / kB, idx % kB, t, tn);
}

// The consumers' position in the stage stream, kept without divisions: g
// stages consumed so far, slot = g mod nst, lap = g / nst, w7 = g mod 7.
struct StageCursor {
  uint32_t g = 0, lap = 0;
  int slot = 0, w7 = 0;
  __device__ __forceinline__ void advance(int n, int nst) {
    g += (uint32_t)n;
    slot += n;
    while (slot >= nst) {
      slot -= nst;
      ++lap;
    }
    w7 = (w7 + n) % kConsumerWarps;
  }
};

// consume_phase for kB input vectors at once (vector b at xs + b * vs): the
// same stages, each weight read once from the ring for all kB products.
// epi.store_b(row, b, value) receives row `row` times vector b, or
// epi.store_pair_b(row, b, value, value of row + 1) paired rows. Deferred rows
// leave kB partials per segment in seg, added in segment order.
template <int kB, class Epi>
__device__ inline bool consume_phase_b(const Ring& r, StageCursor& cur, const StagePlan& p,
                                       const float* xs, int vs, float* seg, Epi& epi, int* err,
                                       int* err_host, volatile int* s_abort) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  bool ok = true;
  const bool pairs = p.gran == 2;
  int j = warp - cur.w7;
  if (j < 0) j += kConsumerWarps;
  int slot = cur.slot + j;
  uint32_t lap = cur.lap;
  while (slot >= r.nst) {
    slot -= r.nst;
    ++lap;
  }
  for (; j < p.nstages && ok; j += kConsumerWarps) {
    const uint32_t gs = cur.g + (uint32_t)j;
    if (!warp_wait_full_at(r, slot, lap & 1u, gs, j >= r.nst, err, err_host, s_abort)) {
      ok = false;
      break;
    }
    const StageDesc s = stage_desc(p, j);
    const int ncols = s.c1 - s.c0;
    const float* st = reinterpret_cast<const float*>(r.buf + (size_t)slot * kStageBytes);
    const float* xb = xs + s.c0;
    const int part = p.spr == 1 ? 0 : j % p.spr;
    int ri = 0;
    auto put_at = [&](int r0) {
      return [&, r0](int rr, int b, float v, float vn) {
        const int row = s.row + r0 + rr;
        if (p.defer) seg[((row - p.r0) * p.spr + part) * kB + b] = v;
        else if (p.gran == 2) {
          if ((rr & 1) == 0) epi.store_pair_b(row, b, v, vn);
        } else {
          epi.store_b(row, b, v);
        }
      };
    };
    for (; ri + 4 <= s.nrows; ri += 4)
      rows_times_vectors<4, kB>(st + (size_t)ri * ncols, ncols, xb, vs, lane, pairs, put_at(ri));
    if (s.nrows - ri == 3) {
      rows_times_vectors<3, kB>(st + (size_t)ri * ncols, ncols, xb, vs, lane, pairs, put_at(ri));
    } else if (s.nrows - ri == 2) {
      rows_times_vectors<2, kB>(st + (size_t)ri * ncols, ncols, xb, vs, lane, pairs, put_at(ri));
    } else if (s.nrows - ri == 1) {
      rows_times_vectors<1, kB>(st + (size_t)ri * ncols, ncols, xb, vs, lane, pairs, put_at(ri));
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&r.empty[slot]);  // stage free for the producer
    slot += kConsumerWarps;
    while (slot >= r.nst) {
      slot -= r.nst;
      ++lap;
    }
  }
  cur.advance(p.nstages, r.nst);
  if (named_bar_or(kBarConsumers, kConsumerThreads, !ok)) {
    if (tid == 0) *s_abort = 1;
    return false;
  }
  if (p.defer) {  // deferred rows: add each row's segments in order
    auto row_sum = [&](int ri, int b) {
      float v = 0.f;
      for (int k = 0; k < p.spr; ++k) v += seg[(ri * p.spr + k) * kB + b];
      return v;
    };
    const int nq = (p.r1 - p.r0) / p.gran;
    for (int q = tid; q < nq * kB; q += kConsumerThreads) {
      const int qi = q / kB, b = q - qi * kB;
      if (p.gran == 2)
        epi.store_pair_b(p.r0 + 2 * qi, b, row_sum(2 * qi, b), row_sum(2 * qi + 1, b));
      else
        epi.store_b(p.r0 + qi, b, row_sum(qi, b));
    }
    named_bar_sync(kBarConsumers, kConsumerThreads);
  }
  return true;
}

struct EpiStore {
  float* out;
  __device__ __forceinline__ void store(int row, float v) { out[row] = v; }
  __device__ __forceinline__ void store_pair(int row, float v0, float v1) {
    out[row] = v0;
    out[row + 1] = v1;
  }
};

}  // namespace tvl
