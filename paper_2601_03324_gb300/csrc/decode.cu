// decode.cu — model loading (one host-to-device copy into one arena) and the
// launches of the persistent decode kernel, behind the C ABI of include/tvl.h.
#include <fcntl.h>
#include <sys/mman.h>
#include <sys/stat.h>
#include <unistd.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>
#include <vector>

#include "decode_kernel.cuh"
#include "host_common.h"
#include "model.h"

using namespace tvl;


namespace tvl {

// Failure-detection self-test: one CTA polls a tagged word that nothing
// writes; the bounded wait must expire and report TVL_E_TIMEOUT.
__global__ void wait_selftest_kernel(unsigned long long* word, int* err,
                                     unsigned long long limit_ns) {
  __shared__ int s_abort;
  if (threadIdx.x == 0) s_abort = 0;
  __syncthreads();
  if (threadIdx.x >= kConsumerThreads) return;  // the consumer warps take part
  const Poll pc{err, nullptr, &s_abort, limit_ns};
  const bool ok = poll_pairs(word, 1, 1u, pc, [](int, float, float) {});
  vote_ok(ok, &s_abort);
}

// W[r][j] *= g[j] for rows [0, rows) of W [rows x cols] (cols % 4 == 0): an
// RMSNorm gain folded into the columns of a matrix that reads the normalised
// vector, W ((x * g) r) = r (W diag(g)) x.
__global__ void scale_columns_kernel(float* __restrict__ W, long long rows, int cols,
                                     const float* __restrict__ g) {
  const int c4 = cols >> 2;
  const long long n = rows * c4;
  float4* w4 = reinterpret_cast<float4*>(W);
  const float4* g4 = reinterpret_cast<const float4*>(g);
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x) {
    const float4 gv = g4[i % c4];
    float4 v = w4[i];
    v.x *= gv.x;
    v.y *= gv.y;
    v.z *= gv.z;
    v.w *= gv.w;
    w4[i] = v;
  }
}

}  // namespace tvl

namespace {

tvl_status scale_columns(unsigned char* W, long long rows, int cols, const unsigned char* g,
                         cudaStream_t st) {
  const long long n = rows * (cols / 4);
  const int blocks = (int)std::min<long long>((n + 255) / 256, 4096);
  scale_columns_kernel<<<blocks, 256, 0, st>>>(reinterpret_cast<float*>(W), rows, cols,
                                               reinterpret_cast<const float*>(g));
  TVL_CK(cudaGetLastError());
  return TVL_OK;
}

struct SmemPlan {
  int ring, bars, xs, vec, seg, att, misc, total, nst;
};

// Shared memory of one CTA for B sequences: the ring takes what the other
// regions leave, up to kMaxStages stages.
SmemPlan plan_smem(int d, int F, int hd, int nch_cap, int max_bytes, int B) {
  SmemPlan p{};
  const int att_floats = 3 * hd + kAttMaxChunk + 4 * kConsumerThreads + nch_cap * (hd + 2) + 16;
  // every region is a multiple of 128 bytes, so every region starts aligned
  const int xs = (int)a128(4LL * B * d), vec = (int)a128(4LL * B * std::max(d, F));
  const int seg = (int)a128(kMaxSegParts * 4), att = (int)a128(4LL * att_floats), misc = kMiscBytes;
  const int bars = (int)a128(kRingBarBytes);
  const int other = bars + xs + vec + seg + att + misc;
  int nst = (max_bytes - other) / kStageBytes;
  if (nst > kMaxStages) nst = kMaxStages;
  p.nst = nst;
  int off = 0;
  p.ring = off;
  off += nst * kStageBytes;
  p.bars = off;
  off += bars;
  p.xs = off;
  off += xs;
  p.vec = off;
  off += vec;
  p.seg = off;
  off += seg;
  p.att = off;
  off += att;
  p.misc = off;
  off += misc;
  p.total = off;
  return p;
}

int nch_cap_for(int S, int H, int G) {
  int cap = 1;
  for (int pos = 0; pos < S; ++pos) {
    int nch, clen;
    att_split(pos, H, G, &nch, &clen);
    cap = std::max(cap, nch);
  }
  return cap;
}

tvl_status check_device_error(tvl_model* m) {
  const int code = *reinterpret_cast<volatile int*>(m->err_host);
  if (code != 0) {
    m->sticky = (tvl_status)code;
    set_error("a bounded device-side wait expired (exchange poll or stage copy); "
              "the model's device state is no longer consistent");
    return m->sticky;
  }
  return TVL_OK;
}

void destroy(tvl_model* m) {
  if (!m) return;
  prefill_release(m);
  lib_free(m->arena);
  lib_free_host(m->err_host);
  if (m->own_stream && m->stream) cudaStreamDestroy(m->stream);
  delete m;
}

bool is_device_pointer(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

// The device address of pinned, mapped host memory (cudaHostAlloc, or
// registered with cudaHostRegister), else null: the kernel can store there
// directly, with no copy after it.
float* mapped_host_pointer(void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (at.type != cudaMemoryTypeHost || !at.devicePointer) return nullptr;
  return static_cast<float*>(at.devicePointer);
}

// Interleaves the rows of a [W1 | W3] block in place (F rows of row_bytes
// each, then F more): row 2i becomes W1's row i and row 2i + 1 W3's, so that
// one CTA computes both halves of each SwiGLU product. tmp holds the block.
tvl_status interleave_w13(unsigned char* block, size_t F, size_t row_bytes, unsigned char* tmp,
                          cudaStream_t st) {
  const size_t half = F * row_bytes;
  TVL_CK(cudaMemcpyAsync(tmp, block, 2 * half, cudaMemcpyDeviceToDevice, st));
  TVL_CK(cudaMemcpy2DAsync(block, 2 * row_bytes, tmp, row_bytes, row_bytes, F,
                           cudaMemcpyDeviceToDevice, st));
  TVL_CK(cudaMemcpy2DAsync(block + row_bytes, 2 * row_bytes, tmp + half, row_bytes, row_bytes, F,
                           cudaMemcpyDeviceToDevice, st));
  return TVL_OK;
}

tvl_status launch(tvl_model* m, int B, const int* tokens, int pos, int n_steps,
                  int final_token, float* logits_dst = nullptr) {
  DecodeArgs a = m->args;
  if (logits_dst) a.logits = logits_dst;  // the classifier writes there directly
  for (int b = 0; b < B; ++b) a.start_tokens[b] = tokens[b];
  a.start_pos = pos;
  a.n_steps = n_steps;
  a.final_token = final_token;
  // Every exchange of the launch has its own tag, above every tag a word may
  // still hold (words are published with an unsigned max, so a word's tag may
  // only grow); 0 marks a word never written.
  const uint64_t span = (uint64_t)n_steps * (uint64_t)(kPhasesPerLayer * m->cfg.n_layers + 1);
  if (span >= 0xFFFFFFFFull) {
    set_error("launch: too many exchanges in one launch for 32-bit tags");
    return TVL_E_RANGE;
  }
  if (m->next_tag + span > 0xFFFFFFFFull) {
    TVL_CK(cudaMemsetAsync(m->arena + m->xchg_off, 0, m->xchg_bytes, m->stream));
    m->next_tag = 1;
  }
  a.epoch0 = (unsigned)m->next_tag;
  const tvl_model::Plan& pl = m->plan[B];
  a.nst = pl.nst;
  a.sm_ring = pl.sm_ring; a.sm_bars = pl.sm_bars; a.sm_xs = pl.sm_xs; a.sm_vec = pl.sm_vec;
  a.sm_seg = pl.sm_seg; a.sm_att = pl.sm_att; a.sm_misc = pl.sm_misc;
  a.vs = m->vs;
  void* params[] = {&a};
  TVL_CK(cudaLaunchCooperativeKernel(m->kernel[B], dim3(a.G), dim3(kThreads), params,
                                     (size_t)pl.total, m->stream));
  m->next_tag += span;
  return TVL_OK;
}

}  // namespace

extern "C" {

tvl_status tvl_load(const tvl_config* cfg, const void* blob, size_t blob_bytes, void* stream,
                    tvl_model** out) {
  if (out) *out = nullptr;
  if (!out || !blob) {
    set_error("tvl_load: null argument");
    return TVL_E_INVAL;
  }
  if (!config_valid(cfg)) {
    set_error("tvl_load: invalid configuration");
    return TVL_E_INVAL;
  }
  const int d = cfg->dim, F = cfg->hidden_dim, H = cfg->n_heads, Hkv = cfg->n_kv_heads;
  const int hd = d / H, kvd = Hkv * hd, V = cfg->vocab_size, S = cfg->max_seq, L = cfg->n_layers;
  if (d % 32 != 0 || hd % 4 != 0 || hd > 128 || F % 4 != 0 || std::max(d, F) > 16384) {
    set_error("tvl_load: the GPU path needs dim % 32 == 0, head_dim % 4 == 0 and <= 128, "
              "hidden_dim % 4 == 0, max(dim, hidden_dim) <= 16384");
    return TVL_E_UNSUPPORTED;
  }
  const bool q4 = cfg->weight_bits == 4;
  const bool q8 = cfg->weight_bits == 8 || q4;  // quantized rows, 8-bit or 4-bit
  const int maxB = cfg->max_batch > 1 ? cfg->max_batch : 1;
  if (maxB > 1 && q8) {
    set_error("tvl_load: max_batch > 1 needs float32 weights (weight_bits 0)");
    return TVL_E_UNSUPPORTED;
  }
  if (q8 && (d % 16 != 0 || F % 16 != 0 || std::max(d, F) > 16368)) {
    set_error("tvl_load: 8-bit rows need dim and hidden_dim multiples of 16 and at most 16368");
    return TVL_E_UNSUPPORTED;
  }
  if (q4 && (d % 32 != 0 || F % 32 != 0)) {
    set_error("tvl_load: 4-bit rows need dim and hidden_dim multiples of 32");
    return TVL_E_UNSUPPORTED;
  }
  // §5.1 weight tying: explicit, or inferred from the blob size.
  const size_t tied_bytes = (size_t)blob_layout(cfg, true).total;
  const size_t untied_bytes = (size_t)blob_layout(cfg, false).total;
  bool tied;
  if (cfg->shared_classifier == 1) tied = true;
  else if (cfg->shared_classifier == 0) tied = false;
  else tied = blob_bytes < untied_bytes;
  if (blob_bytes != (tied ? tied_bytes : untied_bytes)) {
    set_error("tvl_load: blob_bytes " + std::to_string(blob_bytes) + " != expected " +
              std::to_string(tied ? tied_bytes : untied_bytes));
    return TVL_E_SIZE;
  }
  const BlobLayout bl = blob_layout(cfg, tied);
  // the kernel streams [Wq|Wk|Wv] and [W1|W3] as single matrices
  if (bl.wk != bl.wq + 4LL * d * d || bl.wv != bl.wk + 4LL * kvd * d ||
      bl.w3 != bl.w1 + 4LL * F * d) {
    set_error("tvl_load: layout has padding between fused matrices");
    return TVL_E_UNSUPPORTED;
  }

  tvl_model* m = new (std::nothrow) tvl_model();
  if (!m) return TVL_E_NOMEM;
  m->cfg = *cfg;
  m->tied = tied;
  m->max_batch = maxB;
  auto fail = [&](tvl_status s) {
    destroy(m);
    return s;
  };
  auto ck = [&](cudaError_t e, const char* what) -> tvl_status {
    return e == cudaSuccess ? TVL_OK : cuda_fail(e, what);
  };
  tvl_status st;
  m->kernel[1] = q4   ? (const void*)decode_kernel<true, 1, true>
                 : q8 ? (const void*)decode_kernel<true, 1>
                      : (const void*)decode_kernel<false, 1>;
  for (int B = 2; B <= maxB; ++B) m->kernel[B] = decode_kernel_for_batch(B);
  if ((st = ck(cudaGetDevice(&m->device), "cudaGetDevice")) != TVL_OK) return fail(st);
  int sms = 0, coop = 0, max_optin = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, m->device);
  cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, m->device);
  cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, m->device);
  if (!coop || sms <= 0) {
    set_error("tvl_load: device lacks cooperative launch");
    return fail(TVL_E_UNSUPPORTED);
  }
  const int G = sms;
  // a head gets the most attention chunks with one sequence: this bounds every B
  const int nch_cap = nch_cap_for(S, H, G);
  for (int B = 1; B <= maxB; ++B) {
    const SmemPlan sp = plan_smem(d, F, hd, nch_cap, max_optin, B);
    {  // segment partials of rows longer than a stage must fit the scratch
      const long long Ms[5] = {d + 2LL * kvd, d, 2LL * F, d, V};
      const int Ks[5] = {d, d, d, F, d};
      for (int i = 0; i < 5; ++i) {
        const StagePlan pl = plan_stages(Ms[i], Ks[i], G, 0, i == 2 ? 2 : 1);
        if (pl.defer && (long long)((Ms[i] + G - 1) / G + 1) * pl.spr * B > kMaxSegParts) {
          set_error("tvl_load: too many long rows per SM for the segment scratch");
          return fail(TVL_E_UNSUPPORTED);
        }
      }
    }
    // two stages at least; with several sequences four, or the stream stalls
    if (sp.nst < (B == 1 ? 2 : 4)) {
      set_error("tvl_load: not enough shared memory for the weight stages with " +
                std::to_string(B) + " sequence(s); lower max_batch");
      return fail(TVL_E_UNSUPPORTED);
    }
    if ((st = ck(cudaFuncSetAttribute(m->kernel[B],
                                      cudaFuncAttributeMaxDynamicSharedMemorySize, sp.total),
                 "cudaFuncSetAttribute")) != TVL_OK)
      return fail(st);
    int per_sm = 0;
    if ((st = ck(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, m->kernel[B],
                                                                kThreads, sp.total),
                 "cudaOccupancyMaxActiveBlocksPerMultiprocessor")) != TVL_OK)
      return fail(st);
    if (per_sm < 1) {
      set_error("tvl_load: decode kernel cannot be resident on an SM");
      return fail(TVL_E_UNSUPPORTED);
    }
    m->plan[B] = tvl_model::Plan{sp.ring, sp.bars, sp.xs, sp.vec, sp.seg, sp.att, sp.misc,
                                 sp.nst, sp.total};
  }
  m->smem_bytes = m->plan[1].total;
  m->vs = std::max(d, F);

  // ---- arena: weights | rope | K cache | V cache | scratch -------------------------
  const int att_stride = hd + 4;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = (size_t)a256((int64_t)(off + bytes));
    return at;
  };
  const size_t o_w = take(blob_bytes);
  // quantized rows: per layer [Wq|Wk|Wv], Wo, [W1|W3], W2; then E and the untied classifier
  const size_t rq = 16 + (size_t)(q4 ? d / 2 : d), rf = 16 + (size_t)(q4 ? F / 2 : F);
  size_t q_wqkv = 0, q_wo = 0, q_w13 = 0, q_w2 = 0, q_stride = 0, o_q = 0, o_qE = 0, o_qcls = 0;
  if (q8) {
    size_t lo = 0;
    auto ltake = [&](size_t bytes) {
      const size_t at = lo;
      lo = (size_t)a256((int64_t)(lo + bytes));
      return at;
    };
    q_wqkv = ltake((size_t)(d + 2 * kvd) * rq);
    q_wo = ltake((size_t)d * rq);
    q_w13 = ltake((size_t)2 * F * rq);
    q_w2 = ltake((size_t)d * rf);
    q_stride = lo;
    o_q = take(q_stride * (size_t)L);
    o_qE = take((size_t)V * rq);
    o_qcls = tied ? o_qE : take((size_t)V * rq);
  }
  const size_t o_rope = take((size_t)S * (hd / 2) * sizeof(float2));
  // K/V cache and exchange buffers: one of each per sequence slot
  const size_t kv_seq = (size_t)std::max(L, 1) * S * kvd;  // floats per sequence
  const size_t kv_bytes = kv_seq * 4 * maxB;
  const size_t o_kc = take(kv_bytes), o_vc = take(kv_bytes);
  const size_t o_scr = off;
  const size_t nB = (size_t)maxB;
  const size_t o_qkv = take(8ull * (d + 2 * kvd) * nB), o_o = take(8ull * d * nB);
  const size_t o_h13 = take(8ull * F * nB);
  const size_t o_f = take(8ull * d * nB), o_lg = take(4ull * V * nB);
  const size_t o_att = take(8ull * H * nch_cap * att_stride * nB);
  const size_t o_attn = take(8ull * d * nB);
  const size_t o_cand = take(8ull * 2 * G * 2 * nB), o_tok = take(4ull * S * nB);
  const size_t o_ts = take(8ull * S), o_err = take(4);
  m->arena_bytes = off;
  m->weight_bytes = blob_bytes;
  m->xchg_off = o_qkv;
  m->xchg_bytes = o_tok - o_qkv;
  if ((st = ck(lib_malloc((void**)&m->arena, m->arena_bytes), "cudaMalloc(arena)")) != TVL_OK)
    return fail(st);
  if (stream) {
    m->stream = (cudaStream_t)stream;
  } else {
    if ((st = ck(cudaStreamCreateWithFlags(&m->stream, cudaStreamNonBlocking),
                 "cudaStreamCreate")) != TVL_OK)
      return fail(st);
    m->own_stream = true;
  }
  if ((st = ck(lib_host_alloc((void**)&m->err_host, sizeof(int), cudaHostAllocMapped),
               "cudaHostAlloc(err)")) != TVL_OK)
    return fail(st);
  *m->err_host = 0;
  int* err_host_dev = nullptr;
  if ((st = ck(cudaHostGetDevicePointer((void**)&err_host_dev, m->err_host, 0),
               "cudaHostGetDevicePointer")) != TVL_OK)
    return fail(st);

  // ---- the single copy of the blob (pinned first, if it is not already) ------------
  const bool dev_blob = is_device_pointer(blob);
  bool registered = false;
  if (!dev_blob) {
    cudaPointerAttributes at{};
    const bool pinned = cudaPointerGetAttributes(&at, blob) == cudaSuccess &&
                        at.type == cudaMemoryTypeHost;
    cudaGetLastError();
    if (!pinned) {
      int ro = 0;
      cudaDeviceGetAttribute(&ro, cudaDevAttrHostRegisterReadOnlySupported, m->device);
      unsigned flags = ro ? cudaHostRegisterReadOnly : cudaHostRegisterDefault;
      registered = cudaHostRegister(const_cast<void*>(blob), blob_bytes, flags) == cudaSuccess;
      if (!registered && ro)
        registered =
            cudaHostRegister(const_cast<void*>(blob), blob_bytes, cudaHostRegisterDefault) ==
            cudaSuccess;
      cudaGetLastError();  // an unpinnable blob is still copied, from pageable memory
    }
  }
  st = ck(cudaMemcpyAsync(m->arena + o_w, blob, blob_bytes,
                          dev_blob ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, m->stream),
          "cudaMemcpyAsync(blob)");
  if (st == TVL_OK) st = ck(cudaStreamSynchronize(m->stream), "cudaStreamSynchronize(blob)");
  if (registered) cudaHostUnregister(const_cast<void*>(blob));
  if (st != TVL_OK) return fail(st);
  if (q8) {  // every weight matrix to 8-bit (or 4-bit) rows, on the device
    const unsigned char* Wf = m->arena + o_w;
    auto quant = [&](const unsigned char* src, size_t dst, int rows, int cols) {
      return q4 ? tvl_quantize_q4(reinterpret_cast<const float*>(src), m->arena + dst, rows, cols,
                                  m->stream)
                : tvl_quantize_q8(reinterpret_cast<const float*>(src), m->arena + dst, rows, cols,
                                  m->stream);
    };
    for (int l = 0; l < L && st == TVL_OK; ++l) {
      const unsigned char* lw = Wf + bl.l0 + (size_t)l * bl.stride;
      const size_t ql = o_q + (size_t)l * q_stride;
      st = quant(lw + bl.wq, ql + q_wqkv, d + 2 * kvd, d);
      if (st == TVL_OK) st = quant(lw + bl.wo, ql + q_wo, d, d);
      if (st == TVL_OK) st = quant(lw + bl.w1, ql + q_w13, 2 * F, d);
      if (st == TVL_OK) st = quant(lw + bl.w2, ql + q_w2, d, F);
    }
    if (st == TVL_OK) st = quant(Wf + bl.E, o_qE, V, d);
    if (st == TVL_OK && !tied) st = quant(Wf + bl.Wcls, o_qcls, V, d);
    if (st == TVL_OK) st = ck(cudaStreamSynchronize(m->stream), "cudaStreamSynchronize(q8)");
    if (st != TVL_OK) return fail(st);
  }
  {  // the streamed [W1 | W3] blocks get interleaved rows
    const size_t row_bytes = q8 ? rq : 4ull * d;
    unsigned char* tmp = nullptr;
    if (L > 0 && (st = ck(lib_malloc((void**)&tmp, 2 * (size_t)F * row_bytes),
                          "cudaMalloc(w13 scratch)")) != TVL_OK)
      return fail(st);
    for (int l = 0; l < L && st == TVL_OK; ++l) {
      unsigned char* blk = q8 ? m->arena + o_q + (size_t)l * q_stride + q_w13
                              : m->arena + o_w + bl.l0 + (size_t)l * bl.stride + bl.w1;
      st = interleave_w13(blk, (size_t)F, row_bytes, tmp, m->stream);
    }
    if (st == TVL_OK) st = ck(cudaStreamSynchronize(m->stream), "cudaStreamSynchronize(w13)");
    lib_free(tmp);
    if (st != TVL_OK) return fail(st);
  }
  if (!q8) {
    // float32 rows: the RMSNorm gains go into the columns of the matrices that
    // read the normalised vectors ([Wq|Wk|Wv] g_att, W1/W3 g_ffn, and the
    // classifier g_final unless it is the embedding table), so that the
    // kernel's phase input is x itself. (8-bit rows keep the gains apart: their
    // codes are those of the matrices as given.)
    for (int l = 0; l < L && st == TVL_OK; ++l) {
      unsigned char* lw = m->arena + o_w + bl.l0 + (size_t)l * bl.stride;
      st = scale_columns(lw + bl.wq, d + 2LL * kvd, d, lw + bl.g_att, m->stream);
      if (st == TVL_OK) st = scale_columns(lw + bl.w1, 2LL * F, d, lw + bl.g_ffn, m->stream);
    }
    if (st == TVL_OK && !tied)
      st = scale_columns(m->arena + o_w + bl.Wcls, V, d, m->arena + o_w + bl.g_final, m->stream);
    if (st == TVL_OK) st = ck(cudaStreamSynchronize(m->stream), "cudaStreamSynchronize(gains)");
    if (st != TVL_OK) return fail(st);
  }

  // ---- RoPE table: pair i at position p turns by p * theta^(-2i/hd) ------------------
  {
    std::vector<float2> rope((size_t)S * (hd / 2));
    for (int p = 0; p < S; ++p)
      for (int i = 0; i < hd / 2; ++i) {
        const double w = std::pow(cfg->rope_theta, -(2.0 * i) / (double)hd);
        const double ang = (double)p * w;
        rope[(size_t)p * (hd / 2) + i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
      }
    st = ck(cudaMemcpyAsync(m->arena + o_rope, rope.data(), rope.size() * sizeof(float2),
                            cudaMemcpyHostToDevice, m->stream),
            "cudaMemcpyAsync(rope)");
    if (st == TVL_OK)
      st = ck(cudaMemsetAsync(m->arena + o_kc, 0, m->arena_bytes - o_kc, m->stream),
              "cudaMemsetAsync(state)");
    if (st == TVL_OK) st = ck(cudaStreamSynchronize(m->stream), "cudaStreamSynchronize(rope)");
    if (st != TVL_OK) return fail(st);
  }
  (void)o_scr;

  // ---- kernel arguments that do not change between launches --------------------------
  DecodeArgs& a = m->args;
  unsigned char* W = m->arena + o_w;
  a.E = reinterpret_cast<const float*>(W + bl.E);
  a.g_final = reinterpret_cast<const float*>(W + bl.g_final);
  a.Wcls = reinterpret_cast<const float*>(W + (tied ? bl.E : bl.Wcls));
  a.layer0 = W + bl.l0;
  a.layer_stride = bl.stride;
  a.o_gatt = bl.g_att;
  a.o_wqkv = bl.wq;
  a.o_wo = bl.wo;
  a.o_gffn = bl.g_ffn;
  a.o_w13 = bl.w1;
  a.o_w2 = bl.w2;
  a.q_layer0 = q8 ? m->arena + o_q : nullptr;
  a.q_stride = (long long)q_stride;
  a.q_wqkv = (long long)q_wqkv;
  a.q_wo = (long long)q_wo;
  a.q_w13 = (long long)q_w13;
  a.q_w2 = (long long)q_w2;
  a.q_E = q8 ? m->arena + o_qE : nullptr;
  a.q_cls = q8 ? m->arena + o_qcls : nullptr;
  a.rope = reinterpret_cast<const float2*>(m->arena + o_rope);
  a.kc = reinterpret_cast<float*>(m->arena + o_kc);
  a.vc = reinterpret_cast<float*>(m->arena + o_vc);
  a.x_qkv = reinterpret_cast<unsigned long long*>(m->arena + o_qkv);
  a.x_o = reinterpret_cast<unsigned long long*>(m->arena + o_o);
  a.x_h13 = reinterpret_cast<unsigned long long*>(m->arena + o_h13);
  a.x_f = reinterpret_cast<unsigned long long*>(m->arena + o_f);
  a.logits = reinterpret_cast<float*>(m->arena + o_lg);
  a.x_att = reinterpret_cast<unsigned long long*>(m->arena + o_att);
  a.x_attn = reinterpret_cast<unsigned long long*>(m->arena + o_attn);
  a.x_cand = reinterpret_cast<unsigned long long*>(m->arena + o_cand);
  a.tokens = reinterpret_cast<int*>(m->arena + o_tok);
  a.ts = reinterpret_cast<unsigned long long*>(m->arena + o_ts);
  a.err = reinterpret_cast<int*>(m->arena + o_err);
  a.err_host = err_host_dev;
  a.d = d; a.F = F; a.V = V; a.L = L; a.H = H; a.Hkv = Hkv; a.hd = hd; a.kvd = kvd; a.S = S;
  a.G = G;
  a.att_stride = att_stride;
  a.nch_cap = nch_cap;
  a.eps = (float)cfg->norm_eps;
  a.gains_folded = !q8;
  a.final_gain_folded = !q8 && !tied;
  a.att_scale = (float)(1.0 / std::sqrt((double)hd));
  a.kv_seq = (long long)kv_seq;
  a.wait_limit_ns = kWaitLimitNs;
  m->streamed_bytes =
      q8 ? (int64_t)L * ((int64_t)(d + 2 * kvd) * (int64_t)rq + (int64_t)d * (int64_t)rq +
                         2LL * F * (int64_t)rq + (int64_t)d * (int64_t)rf + 8LL * d) +
               (int64_t)V * (int64_t)rq + (int64_t)rq + 4LL * d
         : 4LL * ((int64_t)L * ((int64_t)(d + 2 * kvd) * d + (int64_t)d * d + 3LL * F * d + 2LL * d) +
                  (int64_t)V * d + 2LL * d);
  *out = m;
  return TVL_OK;
}

tvl_status tvl_load_file(const tvl_config* cfg, const char* path, void* stream, tvl_model** out) {
  if (out) *out = nullptr;
  if (!path || !out) {
    set_error("tvl_load_file: null argument");
    return TVL_E_INVAL;
  }
  const int fd = open(path, O_RDONLY);
  if (fd < 0) {
    set_error(std::string("tvl_load_file: cannot open ") + path);
    return TVL_E_INVAL;
  }
  struct stat sb;
  if (fstat(fd, &sb) != 0 || sb.st_size <= 0) {
    close(fd);
    set_error("tvl_load_file: cannot stat file");
    return TVL_E_INVAL;
  }
  int flags = MAP_PRIVATE;
#ifdef MAP_POPULATE
  flags |= MAP_POPULATE;  // pre-fault the pages (the paper's Linux hint)
#endif
  void* p = mmap(nullptr, (size_t)sb.st_size, PROT_READ, flags, fd, 0);
  close(fd);
  if (p == MAP_FAILED) {
    set_error("tvl_load_file: mmap failed");
    return TVL_E_NOMEM;
  }
  const tvl_status st = tvl_load(cfg, p, (size_t)sb.st_size, stream, out);
  munmap(p, (size_t)sb.st_size);
  return st;
}

tvl_status tvl_forward_batch(tvl_model* m, int32_t batch, const int32_t* tokens, int32_t pos,
                             float* logits_out) {
  if (!m || !tokens) {
    set_error("tvl_forward_batch: null argument");
    return TVL_E_INVAL;
  }
  if (m->sticky != TVL_OK) return m->sticky;
  if (batch < 1 || batch > m->max_batch) {
    set_error("tvl_forward_batch: batch must be in [1, max_batch of the model]");
    return TVL_E_INVAL;
  }
  for (int b = 0; b < batch; ++b)
    if (tokens[b] < 0 || tokens[b] >= m->cfg.vocab_size) {
      set_error("tvl_forward_batch: token out of range");
      return TVL_E_RANGE;
    }
  if (pos < 0 || pos >= m->cfg.max_seq) {
    set_error("tvl_forward_batch: position out of range");
    return TVL_E_RANGE;
  }
  // pinned host logits: the classifier's epilogue writes them in place
  float* mapped = logits_out ? mapped_host_pointer(logits_out) : nullptr;
  tvl_status st = launch(m, batch, tokens, pos, 1, 0, mapped);
  if (st != TVL_OK) return st;
  if (!logits_out) return TVL_OK;
  if (mapped) {
    TVL_CK(cudaStreamSynchronize(m->stream));
    return check_device_error(m);
  }
  const size_t bytes = (size_t)m->cfg.vocab_size * 4 * batch;
  if (is_device_pointer(logits_out)) {
    TVL_CK(cudaMemcpyAsync(logits_out, m->args.logits, bytes, cudaMemcpyDeviceToDevice,
                           m->stream));
    return TVL_OK;
  }
  TVL_CK(cudaMemcpyAsync(logits_out, m->args.logits, bytes, cudaMemcpyDeviceToHost, m->stream));
  TVL_CK(cudaStreamSynchronize(m->stream));
  return check_device_error(m);
}

tvl_status tvl_forward(tvl_model* m, int32_t token, int32_t pos, float* logits_out) {
  if (!m) {
    set_error("tvl_forward: null model");
    return TVL_E_INVAL;
  }
  return tvl_forward_batch(m, 1, &token, pos, logits_out);
}

tvl_status tvl_decode_greedy_batch(tvl_model* m, int32_t batch, const int32_t* start_tokens,
                                   int32_t start_pos, int32_t n_steps, int32_t* tokens_out) {
  if (!m || !start_tokens) {
    set_error("tvl_decode_greedy_batch: null argument");
    return TVL_E_INVAL;
  }
  if (m->sticky != TVL_OK) return m->sticky;
  if (batch < 1 || batch > m->max_batch) {
    set_error("tvl_decode_greedy_batch: batch must be in [1, max_batch of the model]");
    return TVL_E_INVAL;
  }
  for (int b = 0; b < batch; ++b)
    if (start_tokens[b] < 0 || start_tokens[b] >= m->cfg.vocab_size) {
      set_error("tvl_decode_greedy_batch: token out of range");
      return TVL_E_RANGE;
    }
  if (start_pos < 0 || n_steps < 1 || (int64_t)start_pos + n_steps > m->cfg.max_seq) {
    set_error("tvl_decode_greedy_batch: position or step count out of range");
    return TVL_E_RANGE;
  }
  tvl_status st = launch(m, batch, start_tokens, start_pos, n_steps, 1);
  if (st != TVL_OK) return st;
  if (!tokens_out) return TVL_OK;
  TVL_CK(cudaMemcpyAsync(tokens_out, m->args.tokens, 4ull * n_steps * batch,
                         cudaMemcpyDeviceToHost, m->stream));
  TVL_CK(cudaStreamSynchronize(m->stream));
  return check_device_error(m);
}

tvl_status tvl_decode_greedy(tvl_model* m, int32_t start_token, int32_t start_pos,
                             int32_t n_steps, int32_t* tokens_out) {
  if (!m) {
    set_error("tvl_decode_greedy: null model");
    return TVL_E_INVAL;
  }
  return tvl_decode_greedy_batch(m, 1, &start_token, start_pos, n_steps, tokens_out);
}

tvl_status tvl_sync(tvl_model* m) {
  if (!m) {
    set_error("tvl_sync: null model");
    return TVL_E_INVAL;
  }
  TVL_CK(cudaStreamSynchronize(m->stream));
  if (m->sticky != TVL_OK) return m->sticky;
  return check_device_error(m);
}

void tvl_free(tvl_model* m) {
  if (!m) return;
  if (m->stream) cudaStreamSynchronize(m->stream);
  destroy(m);
}

tvl_status tvl_get_info(const tvl_model* m, tvl_model_info* out) {
  if (!m || !out) {
    set_error("tvl_get_info: null argument");
    return TVL_E_INVAL;
  }
  out->arena_bytes = (int64_t)m->arena_bytes;
  out->weight_bytes = (int64_t)m->weight_bytes;
  out->streamed_bytes = m->streamed_bytes;
  out->grid = m->args.G;
  out->threads = kThreads;
  out->smem_bytes = m->smem_bytes;
  out->ring_stages = m->plan[1].nst;
  out->stage_bytes = kStageBytes;
  out->tied = m->tied ? 1 : 0;
  out->exchanges_per_step = kPhasesPerLayer * m->cfg.n_layers + 1;
  out->next_tag = (int64_t)m->next_tag;
  out->max_batch = m->max_batch;
  return TVL_OK;
}

tvl_status tvl_step_times(tvl_model* m, uint64_t* ns_out, int32_t n) {
  if (!m || !ns_out || n < 1 || n > m->cfg.max_seq) {
    set_error("tvl_step_times: bad argument");
    return TVL_E_INVAL;
  }
  TVL_CK(cudaMemcpyAsync(ns_out, m->args.ts, 8ull * n, cudaMemcpyDeviceToHost, m->stream));
  TVL_CK(cudaStreamSynchronize(m->stream));
  return TVL_OK;
}

tvl_status tvl_debug_set_next_tag(tvl_model* m, uint64_t tag) {
  if (!m || tag < 1 || tag > 0xFFFFFFFFull) {
    set_error("tvl_debug_set_next_tag: null model or tag outside [1, 2^32 - 1]");
    return TVL_E_INVAL;
  }
  if (tag < m->next_tag)  // the words may hold larger tags: clear them
    TVL_CK(cudaMemsetAsync(m->arena + m->xchg_off, 0, m->xchg_bytes, m->stream));
  m->next_tag = tag;
  return TVL_OK;
}

tvl_status tvl_selftest_barrier_timeout(int32_t limit_ms) {
  if (limit_ms < 1 || limit_ms > 10000) {
    set_error("tvl_selftest_barrier_timeout: limit_ms out of [1, 10000]");
    return TVL_E_INVAL;
  }
  unsigned char* buf = nullptr;
  TVL_CK(lib_malloc((void**)&buf, 256));
  tvl_status st = TVL_OK;
  cudaError_t e = cudaMemset(buf, 0, 256);  // tag 0: never the awaited tag 1
  if (e == cudaSuccess) {
    wait_selftest_kernel<<<1, kThreads>>>(reinterpret_cast<unsigned long long*>(buf),
                                          reinterpret_cast<int*>(buf + 64),
                                          (unsigned long long)limit_ms * 1000000ull);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  int code = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&code, buf + 64, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) st = cuda_fail(e, "wait self-test");
  lib_free(buf);
  if (st != TVL_OK) return st;
  if (code == 0) {
    set_error("wait self-test: the wait did not report a timeout");
    return TVL_E_CUDA;
  }
  set_error("wait self-test: the bounded wait expired as intended");
  return (tvl_status)code;
}

}  // extern "C"
