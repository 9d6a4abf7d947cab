// stream_gemv.cuh — the weight-streaming GEMV engine shared by the decode
// kernel and the standalone GEMV (paper §3.1: y = W x reads every weight once,
// so the work is bound by memory; §6.1: one dot product per output row).
//
// Per CTA: one producer warp streams a contiguous range of weight rows from
// global memory into a ring of shared-memory stages with bulk asynchronous
// copies (the TMA engine), each stage completing on an mbarrier; eight
// consumer warps multiply each landed stage by the input vector held in
// shared memory. This is the GPU form of the paper's two memory ideas: the
// weights flow as one aligned stream (§3.2, §4.1) and several independent
// loads are always in flight (§11.1's four accumulators become several
// 32 KB stages in flight per SM).
//
// Work split: CTA c owns rows [M*c/G, M*(c+1)/G) of an [M x K] matrix, which
// is one contiguous byte range. A stage holds whole rows (when a row fits in
// a stage) or one segment of a row. Inside a stage, rows are cut into pieces
// of at most kPiece floats; warps take pieces round-robin, each piece sum is
// a fixed shuffle tree, and each row sums its pieces in index order, so the
// result is bit-reproducible.
#pragma once
#include "ptx.cuh"

namespace tvl {

constexpr int kConsumerWarps = 8;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kThreads = kConsumerThreads + 32;  // + one producer warp
constexpr int kStageBytes = 32768;
constexpr int kStageFloats = kStageBytes / 4;
constexpr int kPiece = 256;           // floats one warp reduces at a time
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

// Requires K % 4 == 0 (16-byte rows) and kStageFloats % 32 == 0. Piece bound:
// K <= kPiece gives one piece per row and at most kMaxRowsPerStage rows;
// otherwise rows*ceil(K/kPiece) <= kStageFloats/kPiece + kStageFloats/K < 64.
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
  uint64_t* full;
  uint64_t* empty;
  int nst;
};

__device__ __forceinline__ void raise_error(int* err, int* err_host, int code) {
  if (err) atomicCAS(err, 0, code);
  if (err_host) *reinterpret_cast<volatile int*>(err_host) = code;
}

// Single-thread bounded wait (producer). Gives up on abort, on an error
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

// Producer: queue the stages of one phase. g counts stages over the launch.
__device__ inline bool produce_phase(const Ring& r, uint32_t& g, const float* W, const StagePlan& p,
                                     uint64_t pol, int* err, int* err_host,
                                     volatile int* s_abort) {
  for (int j = 0; j < p.nstages; ++j, ++g) {
    const int slot = (int)(g % (uint32_t)r.nst);
    if (g >= (uint32_t)r.nst) {
      bool to = false;
      const uint32_t par = ((g / (uint32_t)r.nst) - 1u) & 1u;
      if (!wait_bounded(&r.empty[slot], par, err, s_abort, true, &to)) {
        if (to) raise_error(err, err_host, kErrTimeout);
        *s_abort = 1;
        return false;
      }
    }
    const StageDesc s = stage_desc(p, j);
    const uint32_t bytes = (uint32_t)(s.nrows * (s.c1 - s.c0)) * 4u;
    mbar_arrive_expect_tx(&r.full[slot], bytes);
    bulk_g2s(r.buf + (size_t)slot * kStageBytes, W + (size_t)s.row * p.K + s.c0, bytes,
             &r.full[slot], pol);
  }
  return true;
}

// Producer epilogue: every copy it queued must land before the CTA may exit.
__device__ inline void drain_ring(const Ring& r, uint32_t g) {
  const uint32_t from = g > (uint32_t)r.nst ? g - (uint32_t)r.nst : 0u;
  for (uint32_t k = from; k < g; ++k)
    wait_bounded(&r.full[k % (uint32_t)r.nst], (k / (uint32_t)r.nst) & 1u, nullptr, nullptr,
                 false, nullptr);
}

// All consumer threads poll; thread 0 alone applies the limit and raises
// the abort flag, which the others observe (the producer may raise it too).
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

// Consumer: one GEMV phase over the CTA's stage plan. The input vector xs is
// in shared memory; with S > 1 the matrix is viewed as [M*S x Kc] "virtual
// rows" (row r, K-chunk s) and virtual row v reads xs + (v % S) * Kc.
// epi.store(v, value) receives each finished (virtual) row. Returns false on
// abort, identically in every consumer thread (a barrier vote).
template <class Epi>
__device__ inline bool consume_phase(const Ring& r, uint32_t& g, const StagePlan& p,
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
    const int npr = (ncols + kPiece - 1) / kPiece;
    const int npieces = s.nrows * npr;
    float* pd = pdot + (g & 1u) * kMaxPieces;
    if (ok) {
      const float* st = reinterpret_cast<const float*>(r.buf + (size_t)slot * kStageBytes);
      for (int q = warp; q < npieces; q += kConsumerWarps) {
        const int ri = q / npr, pj = q - ri * npr;
        const int a = pj * kPiece;
        const int b = (a + kPiece < ncols) ? a + kPiece : ncols;
        const int v = s.row + ri;
        const float* xr = xs + (S > 1 ? (v % S) * Kc : 0) + s.c0 + a;
        const float4* w4 = reinterpret_cast<const float4*>(st + (size_t)ri * ncols + a);
        const float4* x4 = reinterpret_cast<const float4*>(xr);
        const int n4 = (b - a) >> 2;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int e = lane; e < n4; e += 32) {
          const float4 w = w4[e], xv = x4[e];
          acc.x = fmaf(w.x, xv.x, acc.x);
          acc.y = fmaf(w.y, xv.y, acc.y);
          acc.z = fmaf(w.z, xv.z, acc.z);
          acc.w = fmaf(w.w, xv.w, acc.w);
        }
        const float sum = warp_sum((acc.x + acc.y) + (acc.z + acc.w));
        if (lane == 0) pd[q] = sum;
      }
    }
    // uniform decision: abort if any consumer thread gave up waiting
    if (named_bar_or(kBarConsumers, kConsumerThreads, !ok)) {
      if (tid == 0) *s_abort = 1;
      return false;
    }
    if (tid == 0) mbar_arrive(&r.empty[slot]);  // stage free for the producer
    for (int ri = tid; ri < s.nrows; ri += kConsumerThreads) {
      float v = 0.f;
      for (int q = 0; q < npr; ++q) v += pd[ri * npr + q];
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
