// stream_gemv.cuh — the weight-streaming GEMV engine shared by the decode
// kernel and the standalone GEMV (paper §3.1: y = W x reads every weight once,
// so the work is bound by memory; §6.1: one dot product per output row).
//
// Per CTA: a ring of shared-memory stages is filled with bulk asynchronous
// copies (the TMA engine) of a contiguous range of weight rows, each stage
// completing on an mbarrier; eight warps multiply each landed stage by the
// input vector held in shared memory. Thread 0 keeps the ring full: it issues
// the copy of stage g + nst as soon as stage g is consumed, walking a static
// schedule of phases that does not depend on activations, so the copies run
// ahead of whatever the warps are waiting for. This is the GPU form of the paper's two memory ideas: the
// weights flow as one aligned stream (§3.2, §4.1) and several independent
// loads are always in flight (§11.1's four accumulators become several
// 32 KB stages in flight per SM).
//
// Work split: CTA c owns rows [M*c/G, M*(c+1)/G) of an [M x K] matrix, which
// is one contiguous byte range. A stage holds whole rows (when a row fits in
// a stage) or one segment of a row. Inside a stage, each row is one unit of
// work for a warp, or 2/4/8 parts when the stage has fewer rows than warps;
// each unit sum is a fixed shuffle tree and each row sums its parts in order,
// so the result is bit-reproducible.
#pragma once
#include "ptx.cuh"

namespace tvl {

constexpr int kConsumerWarps = 8;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kThreads = kConsumerThreads;  // 2 warps per SM sub-partition: up to 255 registers
constexpr int kStageBytes = 32768;
constexpr int kStageFloats = kStageBytes / 4;
constexpr int kMaxRowsPerStage = 256;
constexpr int kMaxPieces = 256;       // per stage; see plan_stages
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
};

struct StageDesc {
  int row, nrows, c0, c1;  // rows [row, row+nrows), columns [c0, c1)
};

// Requires K % 4 == 0 (16-byte rows) and kStageFloats % 32 == 0. A stage has
// at most kMaxRowsPerStage rows; units per stage (rows x parts) stay below
// max(kMaxRowsPerStage, 2 * kConsumerWarps) <= kMaxPieces.
__host__ __device__ inline StagePlan plan_stages(long long M, int K, int G, int c) {
  StagePlan p;
  p.r0 = (int)(M * c / G);
  p.r1 = (int)(M * (c + 1) / G);
  p.K = K;
  const int nrows = p.r1 - p.r0;
  if (K <= kStageFloats) {
    p.rps = kStageFloats / K;
    if (p.rps > kMaxRowsPerStage) p.rps = kMaxRowsPerStage;
    p.spr = 1;
    p.seg = K;
    p.nstages = (nrows + p.rps - 1) / p.rps;
  } else {
    p.rps = 1;
    p.spr = (K + kStageFloats - 1) / kStageFloats;
    p.seg = ((K + p.spr - 1) / p.spr + 31) / 32 * 32;
    p.nstages = nrows * p.spr;
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
  uint64_t* full;  // [nst]
  int nst;
};

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

// Queues the stages of a static schedule of GEMV phases into the ring, in
// order. Sched::next(W, plan) yields the next phase's matrix and this CTA's
// stage plan, false at the end. Used by thread 0 only; the object lives in
// shared memory so that its state takes no registers in the stage loop.
template <class Sched>
struct Feeder {
  Sched sched;
  const float* W = nullptr;
  StagePlan p{};
  int j = 0;            // next stage of the current phase
  uint32_t issued = 0;  // stages queued so far
  bool done = false;
  uint64_t pol = 0;

  __device__ void start(const Ring& r) {
    pol = l2_evict_first();
    p.nstages = 0;
    for (int k = 0; k < r.nst; ++k) issue(r);
  }
  // Queue the next stage into slot issued % nst (its previous stage has been
  // consumed: the caller has passed the barrier that ends it).
  __device__ void issue(const Ring& r) {
    if (done) return;
    while (j >= p.nstages) {
      if (!sched.next(W, p)) {
        done = true;
        return;
      }
      j = 0;
    }
    const StageDesc s = stage_desc(p, j);
    const uint32_t bytes = (uint32_t)(s.nrows * (s.c1 - s.c0)) * 4u;
    const int slot = (int)(issued % (uint32_t)r.nst);
    mbar_arrive_expect_tx(&r.full[slot], bytes);
    bulk_g2s(r.buf + (size_t)slot * kStageBytes, W + (size_t)s.row * p.K + s.c0, bytes,
             &r.full[slot], pol);
    ++j;
    ++issued;
  }
  // Before the CTA leaves early: wait for the copies still in flight.
  __device__ void drain(const Ring& r, uint32_t consumed) {
    for (uint32_t k = consumed; k < issued; ++k)
      wait_bounded(&r.full[k % (uint32_t)r.nst], (k / (uint32_t)r.nst) & 1u, nullptr, nullptr,
                   false, nullptr);
  }
};

// All threads poll; thread 0 alone applies the limit and raises the abort
// flag, which the others observe. Returns true if the stage landed. The flag
// is only a hint to stop waiting: the decision to leave is taken by a vote at
// the next barrier.
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

// Lane part of one unit's dot product: n4 <= 256 float4 of weights and
// input; lane takes float4 lane + 32k (k < 8), in a fully unrolled loop whose
// loads the compiler hoists as far as registers allow.
__device__ __forceinline__ float unit_partial(const float4* w4, const float4* x4, int n4,
                                              int lane) {
  float4 c0 = make_float4(0.f, 0.f, 0.f, 0.f), c1 = c0;
#pragma unroll
  for (int k = 0; k < 8; k += 2) {
    const int e0 = lane + 32 * k, e1 = e0 + 32;
    if (e0 < n4) {
      const float4 w = w4[e0], x = x4[e0];
      c0.x = fmaf(w.x, x.x, c0.x);
      c0.y = fmaf(w.y, x.y, c0.y);
      c0.z = fmaf(w.z, x.z, c0.z);
      c0.w = fmaf(w.w, x.w, c0.w);
    }
    if (e1 < n4) {
      const float4 w = w4[e1], x = x4[e1];
      c1.x = fmaf(w.x, x.x, c1.x);
      c1.y = fmaf(w.y, x.y, c1.y);
      c1.z = fmaf(w.z, x.z, c1.z);
      c1.w = fmaf(w.w, x.w, c1.w);
    }
  }
  return ((c0.x + c0.y) + (c0.z + c0.w)) + ((c1.x + c1.y) + (c1.z + c1.w));
}

// Consumer: one GEMV phase over the CTA's stage plan. The input vector xs is
// in shared memory; with S > 1 the matrix is viewed as [M*S x Kc] "virtual
// rows" (row r, K-chunk s) and virtual row v reads xs + (v % S) * Kc.
// epi.store(v, value) receives each finished (virtual) row. Returns false on
// abort, identically in every consumer thread (a barrier vote).
//
// Work of one stage: its rows, each cut into P parts (P = 1, 2, 4 or 8, so
// that short stages still give every warp a part); a part ("unit") is at most
// 1024 floats: a row fits a stage (8192 floats), and P is chosen so that
// rows x P >= 8 whenever a row is longer than 1024 floats. Warp w takes units
// w, w+8, ...; each unit is one fully unrolled float4 stream and one shuffle
// tree; a row adds its parts in order.
template <class Epi, class Feed>
__device__ inline bool consume_phase(const Ring& r, uint32_t& g, Feed& feed, const StagePlan& p,
                                     const float* xs, int S, int Kc, float* pdot, Epi& epi,
                                     int* err, int* err_host, volatile int* s_abort) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float carry = 0.f;
  for (int j = 0; j < p.nstages; ++j, ++g) {
    const int slot = (int)(g % (uint32_t)r.nst);
    const uint32_t par = (g / (uint32_t)r.nst) & 1u;
    const bool ok = consumer_wait_full(&r.full[slot], par, err, err_host, s_abort);
    const StageDesc s = stage_desc(p, j);
    const int ncols = s.c1 - s.c0;
    int lp = 0;  // log2 of parts per row
    while (lp < 3 && (s.nrows << lp) < kConsumerWarps && (ncols >> (lp + 1)) >= 128) ++lp;
    const int units = s.nrows << lp;
    const int U = (((ncols + (1 << lp) - 1) >> lp) + 3) & ~3;  // floats per part
    float* pd = pdot + (g & 1u) * kMaxPieces;
    if (ok) {
      const float* st = reinterpret_cast<const float*>(r.buf + (size_t)slot * kStageBytes);
      auto unit = [&](int u) -> float {
        const int ri = u >> lp, pj = u & ((1 << lp) - 1);
        const int a = pj * U;
        const int b = (a + U < ncols) ? a + U : ncols;
        const int v = s.row + ri;
        const float* xr = xs + (S > 1 ? (v % S) * Kc : 0) + s.c0 + a;
        return unit_partial(reinterpret_cast<const float4*>(st + (size_t)ri * ncols + a),
                            reinterpret_cast<const float4*>(xr), (b - a) >> 2, lane);
      };
      // a warp takes units w and w+8 together: both loads in flight, both trees interleaved
      for (int u = warp; u < units; u += 2 * kConsumerWarps) {
        const bool two = u + kConsumerWarps < units;
        float s0 = unit(u);
        float s1 = two ? unit(u + kConsumerWarps) : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          s0 += __shfl_xor_sync(0xffffffffu, s0, o);
          s1 += __shfl_xor_sync(0xffffffffu, s1, o);
        }
        if (lane == 0) {
          pd[u] = s0;
          if (two) pd[u + kConsumerWarps] = s1;
        }
      }
    }
    // uniform decision: abort if any consumer thread gave up waiting
    if (named_bar_or(kBarConsumers, kConsumerThreads, !ok)) {
      if (tid == 0) {
        *s_abort = 1;
        feed.drain(r, g);
      }
      return false;
    }
    if (tid == 0) feed.issue(r);  // the slot is free: queue the stage nst ahead
    for (int ri = tid; ri < s.nrows; ri += kConsumerThreads) {
      float v = 0.f;
      for (int q = 0; q < (1 << lp); ++q) v += pd[(ri << lp) + q];
      if (p.spr > 1) {  // a segment of one row: thread 0 carries the row sum
        const int k = j % p.spr;
        carry = (k == 0) ? v : carry + v;
        if (k == p.spr - 1) epi.store(s.row, carry);
      } else {
        epi.store(s.row + ri, v);
      }
    }
  }
  return true;
}

struct EpiStore {
  float* out;
  __device__ __forceinline__ void store(int row, float v) { out[row] = v; }
};

}  // namespace tvl
