// gemv.cu — standalone y = W x (paper §6.1) on the weight-streaming engine.
//
// One CTA per SM streams its contiguous share of W through the shared-memory
// stage ring (a producer warp and seven consumer warps). Matrices with few
// rows are split along K into S chunks so that every SM gets work: virtual
// row v = (row v / S, chunk v % S); each virtual row's partial lands in a
// scratch buffer, and each row is summed over its S chunks in chunk order — by
// the CTA that owns the whole row, or for a row shared by two CTAs, by
// whichever of them finishes last (a per-row arrival counter tagged with the
// call's id, so that a call that gave up part-way leaves nothing the next
// call would count). The result does not depend on timing. Every wait in the
// kernel is bounded (one second); a CTA whose stage never lands raises
// TVL_E_TIMEOUT in the module's error word (tvl_gemv_status reports it) and
// leaves early, which only a broken device can cause.
#include <cstdio>
#include <map>
#include <mutex>
#include <string>
#include <utility>

#include "host_common.h"
#include "stream_gemv.cuh"

using namespace tvl;

namespace tvl {

// The standalone GEMV copies its stages without L2 prefetches ahead of them:
// measured over the sweep shapes, prefetching 4 or 12 stages ahead was slower
// on every shape (the copies already keep up to 12 stages in flight per SM).
constexpr int kGemvPrefetchAhead = 0;

struct GemvArgs {
  const float* W;
  const float* x;
  float* y;
  int M, K, S, Kc;
  long long nv;  // virtual rows = M * S
  float* part;   // [M * S] when S > 1
  unsigned* cnt; // [M]: (call id << 8) | chunks counted, for the call that last touched the row
  unsigned call_id;  // 1 .. 2^24 - 1, different for consecutive calls sharing cnt
  int* err;          // the module's error word (TVL_E_TIMEOUT after a wait ran out)
  int drop_last;     // self-test: CTA 0's producer never copies its last stage
  int nst;
  int sm_ring, sm_bars, sm_x, sm_seg, sm_misc;
};

struct EpiPart {
  float* part;
  __device__ __forceinline__ void store(int v, float val) { part[v] = val; }
  __device__ __forceinline__ void store_pair(int v, float v0, float v1) {
    part[v] = v0;
    part[v + 1] = v1;
  }
};

// The single phase of a standalone GEMV. Launched with a programmatic
// dependency on the stream's previous kernel: its first copies wait for that
// kernel (the L2 prefetches before them do not).
struct GemvSched {
  const float* W;
  uint32_t refill_delay_ns;
  StagePlan p;
  bool given;
  int prefetch_ahead;  // stages prefetched into L2 ahead of the copies
  // x [K] goes into shared memory by one bulk copy ahead of the weights
  float* xs;
  const float* x;
  uint32_t xbytes;
  uint64_t* xbar;
  __device__ void before_copies() {
    grid_wait_dependencies();
    mbar_arrive_expect_tx(xbar, xbytes);
    bulk_g2s(xs, x, xbytes, xbar, l2_evict_last());
  }
  __device__ bool next(const float*& w, StagePlan& plan) {
    if (given) return false;
    given = true;
    w = W;
    plan = p;
    return true;
  }
};

template <bool kQ8, bool kQ4 = false>
__global__ void __launch_bounds__(kThreads, 1) gemv_stream_kernel(const __grid_constant__ GemvArgs a) {
  extern __shared__ __align__(128) unsigned char smem[];
  Ring r;
  r.buf = smem + a.sm_ring;
  r.full = reinterpret_cast<uint64_t*>(smem + a.sm_bars);
  r.empty = r.full + a.nst;
  r.seq = reinterpret_cast<volatile int*>(r.empty + a.nst);
  r.nst = a.nst;
  volatile int* s_abort = reinterpret_cast<volatile int*>(smem + a.sm_misc);
  uint64_t* xbar = reinterpret_cast<uint64_t*>(smem + a.sm_misc + 64);
  float* xs = reinterpret_cast<float*>(smem + a.sm_x);
  const StagePlan p = plan_stages(a.nv, a.Kc, gridDim.x, blockIdx.x);
  if (threadIdx.x == 0) {
    for (int i = 0; i < a.nst; ++i) {
      mbar_init(&r.full[i], 1);
      mbar_init(&r.empty[i], 1);
      r.seq[i] = 0;
    }
    mbar_init(xbar, 1);
    *s_abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  // the stream's next kernel may launch now: with the ring sized to the work
  // its CTAs can start (and prefetch their rows) beside this one's
  grid_launch_dependents();
  uint32_t g = 0;
  if (threadIdx.x >= kConsumerThreads) {
    if (threadIdx.x == kConsumerThreads) {
      GemvSched sched{a.W, 0u, p, false, kGemvPrefetchAhead, xs, a.x, 4u * (uint32_t)a.K, xbar};
      if (a.drop_last && blockIdx.x == 0 && sched.p.nstages > 0) --sched.p.nstages;
      run_producer(r, sched, a.err, nullptr, s_abort);
      // the copy of x has landed before the CTA may exit
      wait_bounded(xbar, 0, nullptr, nullptr, false, nullptr);
    }
    return;
  }
  float* seg = reinterpret_cast<float*>(smem + a.sm_seg);
  grid_wait_dependencies();  // y and the scratch may still be in use by the previous kernel
  const bool xok = consumer_wait_full(xbar, 0, a.err, nullptr, s_abort);
  if (named_bar_or(kBarConsumers, kConsumerThreads, !xok)) return;
  if (a.S == 1) {
    EpiStore e{a.y};
    consume_phase<true, kQ8, kQ4>(r, g, p, xs, 1, a.Kc, seg, e, a.err, nullptr, s_abort);
    return;
  }
  EpiPart e{a.part};
  if (!consume_phase(r, g, p, xs, a.S, a.Kc, seg, e, a.err, nullptr, s_abort)) return;
  if (p.r1 <= p.r0) return;
  named_bar_sync(kBarConsumers, kConsumerThreads);
  const int S = a.S;
  const int ra = p.r0 / S, rb = (p.r1 - 1) / S;
  const unsigned id = a.call_id << 8;
  for (int row = ra + threadIdx.x; row <= rb; row += kConsumerThreads) {
    const int lo = max(p.r0, row * S), hi = min(p.r1, (row + 1) * S);
    const unsigned mine = (unsigned)(hi - lo);
    bool last = (mine == (unsigned)S);
    if (!last) {
      // add this CTA's chunks to the row's count for this call; a count left
      // by another call (one that gave up part-way) counts as zero
      __threadfence();
      unsigned* c = a.cnt + row;
      unsigned old = *reinterpret_cast<volatile unsigned*>(c), before = 0;
      bool added = false;
      for (int it = 0; it < (1 << 16) && !added; ++it) {
        before = (old & ~0xFFu) == id ? (old & 0xFFu) : 0u;
        const unsigned seen = atomicCAS(c, old, id | (before + mine));
        added = seen == old;
        old = seen;
      }
      if (!added) {  // cannot happen while calls sharing cnt are ordered
        raise_error(a.err, nullptr, kErrTimeout);
        continue;
      }
      last = (before + mine == (unsigned)S);
      if (last) __threadfence();
    }
    if (last) {
      float v = 0.f;
      for (int s = 0; s < S; ++s) v += __ldcg(a.part + (size_t)row * S + s);
      a.y[row] = v;
    }
  }
}

// Any shape or alignment: one warp per row, scalar loads.
__global__ void gemv_rowwise_kernel(const float* __restrict__ W, const float* __restrict__ x,
                                    float* __restrict__ y, int M, int K) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= M) return;
  const float* w = W + (size_t)warp * K;
  float acc = 0.f;
  for (int j = lane; j < K; j += 32) acc = fmaf(__ldg(w + j), __ldg(x + j), acc);
  acc = warp_sum(acc);
  if (lane == 0) y[warp] = acc;
}

// 8-bit codes of W [M x K] as packed rows (16 + K bytes: scale, 12 zero
// bytes, codes), one warp per row. Every decision is taken in float32 with
// IEEE division: s = max|w| / 127, code = nearest integer to w / s, ties to
// even (an all-zero row: s = 0, codes 0). Requires K % 16 == 0.
__global__ void quantize_q8_kernel(const float* __restrict__ W, unsigned char* __restrict__ Q,
                                   int M, int K) {
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (row >= M) return;
  const float4* w4 = reinterpret_cast<const float4*>(W + (size_t)row * K);
  const int n4 = K >> 2;
  float amax = 0.f;
  for (int e = lane; e < n4; e += 32) {
    const float4 v = w4[e];
    amax = fmaxf(amax, fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w))));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const float sc = __fdiv_rn(amax, 127.0f);
  unsigned char* out = Q + (size_t)row * (16 + K);
  if (lane < 4) reinterpret_cast<unsigned*>(out)[lane] = lane == 0 ? __float_as_uint(sc) : 0u;
  int* codes = reinterpret_cast<int*>(out + 16);
  auto code = [&](float v) -> int {
    if (sc == 0.f) return 0;
    int c = __float2int_rn(__fdiv_rn(v, sc));
    return c > 127 ? 127 : (c < -127 ? -127 : c);
  };
  for (int e = lane; e < n4; e += 32) {
    const float4 v = w4[e];
    codes[e] = (code(v.x) & 0xff) | ((code(v.y) & 0xff) << 8) | ((code(v.z) & 0xff) << 16) |
               (code(v.w) << 24);
  }
}

// 4-bit codes of W [M x K] as packed rows (16 + K/2 bytes: scale, 12 zero
// bytes, two codes per byte with the even column in the low nibble), one warp
// per row; lane takes code word e (columns 8e..8e+7). The same float32
// decisions as the 8-bit codes with 7 levels: s = max|w| / 7, code = nearest
// integer to w / s, ties to even, in [-7, 7]. Requires K % 32 == 0.
__global__ void quantize_q4_kernel(const float* __restrict__ W, unsigned char* __restrict__ Q,
                                   int M, int K) {
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (row >= M) return;
  const float4* w4 = reinterpret_cast<const float4*>(W + (size_t)row * K);
  const int n4 = K >> 2, nw = K >> 3;
  float amax = 0.f;
  for (int e = lane; e < n4; e += 32) {
    const float4 v = w4[e];
    amax = fmaxf(amax, fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w))));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const float sc = __fdiv_rn(amax, 7.0f);
  unsigned char* out = Q + (size_t)row * (16 + K / 2);
  if (lane < 4) reinterpret_cast<unsigned*>(out)[lane] = lane == 0 ? __float_as_uint(sc) : 0u;
  unsigned* words = reinterpret_cast<unsigned*>(out + 16);
  auto code = [&](float v) -> unsigned {
    if (sc == 0.f) return 0u;
    int c = __float2int_rn(__fdiv_rn(v, sc));
    c = c > 7 ? 7 : (c < -7 ? -7 : c);
    return (unsigned)c & 0xFu;
  };
  for (int e = lane; e < nw; e += 32) {
    const float4 a = w4[2 * e], b = w4[2 * e + 1];
    words[e] = code(a.x) | (code(a.y) << 4) | (code(a.z) << 8) | (code(a.w) << 12) |
               (code(b.x) << 16) | (code(b.y) << 20) | (code(b.z) << 24) | (code(b.w) << 28);
  }
}

}  // namespace tvl

namespace {

// The module's error word: every standalone GEMV kernel raises a timeout
// here; tvl_gemv_status reads and clears it. One per device.
static __device__ int g_gemv_err;

struct DevInfo {
  int sms = 0, max_optin = 0;
  int* err = nullptr;  // device address of g_gemv_err on this device
};
std::mutex g_dev_mu;
constexpr int kMaxDevices = 64;
DevInfo g_dev[kMaxDevices];  // fixed table: no heap use on any call

// Attributes of the current device and the address of its error word
// (looked up once per device).
tvl_status dev_info(const char* who, DevInfo* out) {
  int dev = 0;
  TVL_CK(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) {
    char msg[160];
    snprintf(msg, sizeof msg, "%s: device ordinal %d is beyond the %d-entry table", who, dev,
             kMaxDevices);
    set_error(msg);
    return TVL_E_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DevInfo& di = g_dev[dev];
  if (di.sms == 0) {
    void* e = nullptr;
    TVL_CK(cudaGetSymbolAddress(&e, g_gemv_err));
    TVL_CK(cudaDeviceGetAttribute(&di.max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev));
    int sms = 0;
    TVL_CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    di.err = reinterpret_cast<int*>(e);
    di.sms = sms;
  }
  *out = di;
  return TVL_OK;
}

// The next call id of a counter set (1 .. 2^24 - 1, never 0: zeroed counters
// belong to no call).
unsigned next_call_id(unsigned* next) {
  const unsigned id = *next;
  *next = id >= 0xFFFFFFu ? 1u : id + 1u;
  return id;
}

// Chunks along K: only when the matrix has fewer rows than there are SMs
// (each chunk at least 128 floats, the split a power of two dividing K / 4);
// otherwise every CTA owns whole rows and no partials cross CTAs.
int split_for(int M, int K, int G) {
  int S = 1;
  while ((long long)M * S < G && K % (8 * S) == 0 && K / (2 * S) >= 128) S *= 2;
  return S;
}

// Whether the streaming kernel takes W [M x K] (else the per-row kernel):
// 16-byte aligned W and x, K % 4 == 0, K <= 16384, and the segment partials
// of rows longer than a stage fit the shared scratch.
bool streams(const float* W, const float* x, int M, int K, int sms, int* S_out) {
  const bool aligned = ((uintptr_t)W % 16 == 0) && ((uintptr_t)x % 16 == 0) && K % 4 == 0;
  if (!aligned || K > 16384) return false;
  const int S = split_for(M, K, sms);
  const long long nv = (long long)M * S;
  const long long G = nv < sms ? nv : sms;
  const StagePlan pl = plan_stages(nv, K / S, (int)G, 0);
  *S_out = S;
  return pl.spr == 1 || ((nv + G - 1) / G) * pl.spr <= kMaxSegParts;
}

tvl_status launch_rowwise(const float* W, const float* x, float* y, int M, int K,
                          cudaStream_t s) {
  const int threads = 256, rows_per_block = threads / 32;
  gemv_rowwise_kernel<<<(M + rows_per_block - 1) / rows_per_block, threads, 0, s>>>(W, x, y, M,
                                                                                     K);
  TVL_CK(cudaGetLastError());
  return TVL_OK;
}

// Shared memory (ring | barriers | x | segment partials | misc, every region a
// 128-byte multiple) and launch of gemv_stream_kernel<kQ8, kQ4> for a.nv
// virtual rows of a.Kc words; a.K floats of x. The ring has as many stages as
// the busiest CTA copies (up to kMaxStages), the partial scratch only when rows
// are longer than a stage, so that small matrices leave room on each SM for
// the next kernel's CTAs. The launch carries a programmatic dependency on the
// stream's previous kernel (the kernel waits for it before its first copy).
template <bool kQ8, bool kQ4>
tvl_status launch_stream(GemvArgs& a, const DevInfo& di, cudaStream_t s, const char* who) {
  static std::mutex mu;
  static bool attr_set[kMaxDevices] = {};
  const int G = (int)(a.nv < di.sms ? a.nv : di.sms);
  int need = 1;
  bool defer = false;
  for (int c = 0; c < G; ++c) {
    const StagePlan pl = plan_stages(a.nv, a.Kc, G, c);
    need = pl.nstages > need ? pl.nstages : need;
    defer = defer || pl.defer;
  }
  const int xbytes = (int)a128(4LL * a.K), segb = defer ? (int)a128(kMaxSegParts * 4) : 128;
  const int bars = (int)a128(kRingBarBytes);
  const int misc = 128;
  int nst = (di.max_optin - xbytes - segb - bars - misc) / kStageBytes;
  if (nst > kMaxStages) nst = kMaxStages;
  if (nst > need) nst = need < 2 ? 2 : need;
  if (nst < 2) {
    set_error(std::string(who) + ": not enough shared memory");
    return TVL_E_UNSUPPORTED;
  }
  a.err = di.err;
  a.nst = nst;
  a.sm_ring = 0;
  a.sm_bars = nst * kStageBytes;
  a.sm_x = a.sm_bars + bars;
  a.sm_seg = a.sm_x + xbytes;
  a.sm_misc = a.sm_seg + segb;
  const int smem = a.sm_misc + misc;
  int dev = 0;
  TVL_CK(cudaGetDevice(&dev));
  {
    std::lock_guard<std::mutex> lk(mu);
    if (!attr_set[dev]) {
      TVL_CK(cudaFuncSetAttribute((const void*)gemv_stream_kernel<kQ8, kQ4>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, di.max_optin));
      attr_set[dev] = true;
    }
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = dim3(G);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = s;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  TVL_CK(cudaLaunchKernelEx(&cfg, gemv_stream_kernel<kQ8, kQ4>, (const GemvArgs)a));
  return TVL_OK;
}

// Per-stream split-K scratch of tvl_gemv, allocated on first use.
struct Workspace {
  float* part = nullptr;
  unsigned* cnt = nullptr;
  long long part_cap = 0;
  int cnt_cap = 0;
  unsigned next_id = 1;
};
std::mutex g_ws_mu;
std::map<std::pair<int, cudaStream_t>, Workspace> g_ws;

}  // namespace

extern "C" tvl_status tvl_gemv(const float* W, const float* x, float* y, int32_t d_out,
                               int32_t d_in, void* stream) {
  if (!W || !x || !y || d_out < 1 || d_in < 1) {
    set_error("tvl_gemv: null pointer or non-positive size");
    return TVL_E_INVAL;
  }
  cudaStream_t s = (cudaStream_t)stream;
  DevInfo di;
  tvl_status st = dev_info("tvl_gemv", &di);
  if (st != TVL_OK) return st;
  int S = 1;
  if (!streams(W, x, d_out, d_in, di.sms, &S)) return launch_rowwise(W, x, y, d_out, d_in, s);
  GemvArgs a{};
  a.W = W;
  a.x = x;
  a.y = y;
  a.M = d_out;
  a.K = d_in;
  a.S = S;
  a.Kc = d_in / S;
  a.nv = (long long)d_out * S;
  if (S > 1) {
    int dev = 0;
    TVL_CK(cudaGetDevice(&dev));
    std::lock_guard<std::mutex> lk(g_ws_mu);
    Workspace& ws = g_ws[{dev, s}];
    if (ws.part_cap < a.nv || ws.cnt_cap < d_out) {
      if (ws.part || ws.cnt) {  // earlier kernels on this stream may still use the old buffers
        TVL_CK(cudaStreamSynchronize(s));
        lib_free(ws.part);
        lib_free(ws.cnt);
        ws.part = nullptr;
        ws.cnt = nullptr;
        ws.part_cap = ws.cnt_cap = 0;
      }
      const long long pc = a.nv > 4096 ? a.nv : 4096;
      const int cc = d_out > 4096 ? d_out : 4096;
      cudaError_t e = lib_malloc((void**)&ws.part, 4 * pc + 256);
      if (e == cudaSuccess) e = lib_malloc((void**)&ws.cnt, 4LL * cc + 256);
      if (e == cudaSuccess) e = cudaMemsetAsync(ws.cnt, 0, 4LL * cc + 256, s);
      if (e != cudaSuccess) {
        lib_free(ws.part);
        lib_free(ws.cnt);
        ws.part = nullptr;
        ws.cnt = nullptr;
        return cuda_fail(e, "tvl_gemv: split-K scratch");
      }
      ws.part_cap = pc;
      ws.cnt_cap = cc;
    }
    a.part = ws.part;
    a.cnt = ws.cnt;
    a.call_id = next_call_id(&ws.next_id);
  }
  return launch_stream<false, false>(a, di, s, "tvl_gemv");
}

// ---- tvl_gemv_noalloc: the same GEMV with its split-K scratch in module memory ----

namespace {

// Split-K partials (floats) and per-row arrival counters of tvl_gemv_noalloc.
// split_for splits only matrices with fewer rows than SMs and keeps M * S
// below twice the SM count, so on a 152-SM part at most 302 partials and 151
// counters are live; the sizes below leave room for much larger parts.
constexpr int kNoAllocPart = 8192;
constexpr int kNoAllocRows = 4096;
constexpr size_t kNoAllocBytes = 4 * (size_t)kNoAllocPart + 4 * (size_t)kNoAllocRows;  // 48 KB
static __device__ __align__(256) unsigned char g_gemv_scratch[kNoAllocBytes];

struct NoAllocDev {
  bool ready;
  float* part;
  unsigned* cnt;
  unsigned next_id;
};
NoAllocDev g_noalloc[kMaxDevices];  // fixed table: no heap use on any call
std::mutex g_noalloc_mu;

// The static scratch of the current device (device addresses; the first call
// on a device looks them up and zeroes the counters on `s`, waiting for it),
// and the call's id. drop_last: see tvl_selftest_gemv_timeout.
tvl_status noalloc_gemv(const float* W, const float* x, float* y, int d_out, int d_in,
                        cudaStream_t s, int drop_last, const char* who) {
  DevInfo di;
  tvl_status st = dev_info(who, &di);
  if (st != TVL_OK) return st;
  int dev = 0;
  TVL_CK(cudaGetDevice(&dev));
  int S = 1;
  if (!streams(W, x, d_out, d_in, di.sms, &S)) {
    if (drop_last) {
      set_error(std::string(who) + ": the shape does not take the streaming kernel");
      return TVL_E_UNSUPPORTED;
    }
    return launch_rowwise(W, x, y, d_out, d_in, s);
  }
  const long long nv = (long long)d_out * S;
  if (S > 1 && (nv > kNoAllocPart || d_out > kNoAllocRows)) {
    char msg[192];
    snprintf(msg, sizeof msg,
             "%s: %d x %d splits into %lld partials over %d rows; the static scratch holds %d "
             "partials and %d rows (use tvl_gemv)",
             who, d_out, d_in, nv, d_out, kNoAllocPart, kNoAllocRows);
    set_error(msg);
    return TVL_E_UNSUPPORTED;
  }
  GemvArgs a{};
  {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    NoAllocDev& e = g_noalloc[dev];
    if (!e.ready) {  // once per device: address of the module array, counters to zero
      void* base = nullptr;
      TVL_CK(cudaGetSymbolAddress(&base, g_gemv_scratch));
      e.part = reinterpret_cast<float*>(base);
      e.cnt = reinterpret_cast<unsigned*>(reinterpret_cast<unsigned char*>(base) +
                                          4 * (size_t)kNoAllocPart);
      TVL_CK(cudaMemsetAsync(e.cnt, 0, 4 * (size_t)kNoAllocRows, s));
      TVL_CK(cudaStreamSynchronize(s));
      e.next_id = 1;
      e.ready = true;
    }
    a.part = e.part;
    a.cnt = e.cnt;
    a.call_id = next_call_id(&e.next_id);
  }
  a.W = W;
  a.x = x;
  a.y = y;
  a.M = d_out;
  a.K = d_in;
  a.S = S;
  a.Kc = d_in / S;
  a.nv = nv;
  a.drop_last = drop_last;
  return launch_stream<false, false>(a, di, s, who);
}

}  // namespace

extern "C" tvl_status tvl_gemv_noalloc(const float* W, const float* x, float* y, int32_t d_out,
                                       int32_t d_in, void* stream) {
  if (!W || !x || !y || d_out < 1 || d_in < 1) {
    set_error("tvl_gemv_noalloc: null pointer or non-positive size");
    return TVL_E_INVAL;
  }
  return noalloc_gemv(W, x, y, d_out, d_in, (cudaStream_t)stream, 0, "tvl_gemv_noalloc");
}

extern "C" tvl_status tvl_gemv_status(void* stream) {
  DevInfo di;
  tvl_status st = dev_info("tvl_gemv_status", &di);
  if (st != TVL_OK) return st;
  TVL_CK(cudaStreamSynchronize((cudaStream_t)stream));
  int code = 0;
  TVL_CK(cudaMemcpy(&code, di.err, sizeof(int), cudaMemcpyDeviceToHost));
  if (code == 0) return TVL_OK;
  TVL_CK(cudaMemset(di.err, 0, sizeof(int)));
  set_error("a bounded wait in a standalone GEMV kernel expired; the outputs of that call are "
            "incomplete");
  return (tvl_status)code;
}

extern "C" tvl_status tvl_selftest_gemv_timeout(const float* W, const float* x, float* y,
                                                int32_t d_out, int32_t d_in, void* stream) {
  if (!W || !x || !y || d_out < 1 || d_in < 1) {
    set_error("tvl_selftest_gemv_timeout: null pointer or non-positive size");
    return TVL_E_INVAL;
  }
  tvl_status st = noalloc_gemv(W, x, y, d_out, d_in, (cudaStream_t)stream, 1,
                               "tvl_selftest_gemv_timeout");
  if (st != TVL_OK) return st;
  st = tvl_gemv_status(stream);
  if (st == TVL_OK) {
    set_error("gemv self-test: the wait on the missing stage did not report a timeout");
    return TVL_E_CUDA;
  }
  return st;
}

// ---- weight-only 8-bit rows: quantization and GEMV --------------------------------

extern "C" size_t tvl_q8_bytes(int32_t rows, int32_t cols) {
  if (rows < 1 || cols < 16 || cols % 16 != 0) return 0;
  return (size_t)rows * (size_t)(16 + cols);
}

extern "C" tvl_status tvl_quantize_q8(const float* W, void* Wq8, int32_t rows, int32_t cols,
                                      void* stream) {
  if (!W || !Wq8 || tvl_q8_bytes(rows, cols) == 0) {
    set_error("tvl_quantize_q8: null pointer, or cols not a positive multiple of 16");
    return TVL_E_INVAL;
  }
  if ((uintptr_t)W % 16 || (uintptr_t)Wq8 % 16) {
    set_error("tvl_quantize_q8: W and Wq8 must be 16-byte aligned");
    return TVL_E_ALIGN;
  }
  const int threads = 256, rows_per_block = threads / 32;
  quantize_q8_kernel<<<(rows + rows_per_block - 1) / rows_per_block, threads, 0,
                       (cudaStream_t)stream>>>(W, (unsigned char*)Wq8, rows, cols);
  TVL_CK(cudaGetLastError());
  return TVL_OK;
}

extern "C" tvl_status tvl_gemv_q8(const void* Wq8, const float* x, float* y, int32_t d_out,
                                  int32_t d_in, void* stream) {
  if (!Wq8 || !x || !y || tvl_q8_bytes(d_out, d_in) == 0) {
    set_error("tvl_gemv_q8: null pointer, or d_in not a positive multiple of 16");
    return TVL_E_INVAL;
  }
  if ((uintptr_t)Wq8 % 16 || (uintptr_t)x % 16) {
    set_error("tvl_gemv_q8: Wq8 and x must be 16-byte aligned");
    return TVL_E_ALIGN;
  }
  const int Kw = 4 + d_in / 4;  // words per packed row
  if (Kw > kStageFloats) {
    set_error("tvl_gemv_q8: a packed row must fit one 16 KB stage (d_in <= 16368)");
    return TVL_E_UNSUPPORTED;
  }
  DevInfo di;
  tvl_status st = dev_info("tvl_gemv_q8", &di);
  if (st != TVL_OK) return st;
  GemvArgs a{};
  a.W = reinterpret_cast<const float*>(Wq8);
  a.x = x;
  a.y = y;
  a.M = d_out;
  a.K = d_in;
  a.S = 1;
  a.Kc = Kw;
  a.nv = d_out;
  return launch_stream<true, false>(a, di, (cudaStream_t)stream, "tvl_gemv_q8");
}

// ---- weight-only 4-bit rows: quantization and GEMV ---------------------------------

extern "C" size_t tvl_q4_bytes(int32_t rows, int32_t cols) {
  if (rows < 1 || cols < 32 || cols % 32 != 0) return 0;
  return (size_t)rows * (size_t)(16 + cols / 2);
}

extern "C" tvl_status tvl_quantize_q4(const float* W, void* Wq4, int32_t rows, int32_t cols,
                                      void* stream) {
  if (!W || !Wq4 || tvl_q4_bytes(rows, cols) == 0) {
    set_error("tvl_quantize_q4: null pointer, or cols not a positive multiple of 32");
    return TVL_E_INVAL;
  }
  if ((uintptr_t)W % 16 || (uintptr_t)Wq4 % 16) {
    set_error("tvl_quantize_q4: W and Wq4 must be 16-byte aligned");
    return TVL_E_ALIGN;
  }
  const int threads = 256, rows_per_block = threads / 32;
  quantize_q4_kernel<<<(rows + rows_per_block - 1) / rows_per_block, threads, 0,
                       (cudaStream_t)stream>>>(W, (unsigned char*)Wq4, rows, cols);
  TVL_CK(cudaGetLastError());
  return TVL_OK;
}

extern "C" tvl_status tvl_gemv_q4(const void* Wq4, const float* x, float* y, int32_t d_out,
                                  int32_t d_in, void* stream) {
  if (!Wq4 || !x || !y || tvl_q4_bytes(d_out, d_in) == 0) {
    set_error("tvl_gemv_q4: null pointer, or d_in not a positive multiple of 32");
    return TVL_E_INVAL;
  }
  if ((uintptr_t)Wq4 % 16 || (uintptr_t)x % 16) {
    set_error("tvl_gemv_q4: Wq4 and x must be 16-byte aligned");
    return TVL_E_ALIGN;
  }
  const int Kw = 4 + d_in / 8;  // words per packed row
  if (Kw > kStageFloats) {
    set_error("tvl_gemv_q4: a packed row must fit one 16 KB stage (d_in <= 32736)");
    return TVL_E_UNSUPPORTED;
  }
  DevInfo di;
  tvl_status st = dev_info("tvl_gemv_q4", &di);
  if (st != TVL_OK) return st;
  GemvArgs a{};
  a.W = reinterpret_cast<const float*>(Wq4);
  a.x = x;
  a.y = y;
  a.M = d_out;
  a.K = d_in;
  a.S = 1;
  a.Kc = Kw;
  a.nv = d_out;
  return launch_stream<false, true>(a, di, (cudaStream_t)stream, "tvl_gemv_q4");
}
