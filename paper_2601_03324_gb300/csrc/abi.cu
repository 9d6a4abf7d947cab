// abi.cu — status strings, per-thread error messages, blob layout and size.
#include <atomic>
#include <cstdio>
#include <string>

#include "host_common.h"

namespace tvl {

static thread_local std::string g_last_error;

// Allocation accounting and the failure injector (test hooks of include/tvl.h).
static std::atomic<long long> g_live_allocs{0};
static std::atomic<int> g_fail_countdown{-1};  // < 0: off; k: fail the k-th attempt from now

static bool injected_failure() {
  int k = g_fail_countdown.load();
  while (k >= 0) {
    if (g_fail_countdown.compare_exchange_weak(k, k - 1)) return k == 0;
  }
  return false;
}

cudaError_t lib_malloc(void** p, size_t bytes) {
  *p = nullptr;
  if (injected_failure()) return cudaErrorMemoryAllocation;
  const cudaError_t e = cudaMalloc(p, bytes);
  if (e == cudaSuccess) ++g_live_allocs;
  return e;
}

void lib_free(void* p) {
  if (!p) return;
  cudaFree(p);
  --g_live_allocs;
}

cudaError_t lib_host_alloc(void** p, size_t bytes, unsigned flags) {
  *p = nullptr;
  if (injected_failure()) return cudaErrorMemoryAllocation;
  const cudaError_t e = cudaHostAlloc(p, bytes, flags);
  if (e == cudaSuccess) ++g_live_allocs;
  return e;
}

void lib_free_host(void* p) {
  if (!p) return;
  cudaFreeHost(p);
  --g_live_allocs;
}

void set_error(const std::string& msg) { g_last_error = msg; }

tvl_status cuda_fail(cudaError_t e, const char* what) {
  char buf[512];
  std::snprintf(buf, sizeof buf, "%s failed: %s (%s)", what, cudaGetErrorName(e),
                cudaGetErrorString(e));
  set_error(buf);
  if (e == cudaErrorMemoryAllocation) return TVL_E_NOMEM;
  return TVL_E_CUDA;
}

bool config_valid(const tvl_config* c) {
  if (!c) return false;
  if (c->dim <= 0 || c->hidden_dim <= 0 || c->n_layers < 0 || c->n_heads <= 0 ||
      c->n_kv_heads <= 0 || c->vocab_size <= 0 || c->max_seq <= 0)
    return false;
  if (c->dim % c->n_heads != 0 || c->n_heads % c->n_kv_heads != 0) return false;
  if ((c->dim / c->n_heads) % 2 != 0) return false;  // RoPE turns pairs
  if (!(c->rope_theta > 0.0) || !(c->norm_eps >= 0.0)) return false;
  if (c->shared_classifier < -1 || c->shared_classifier > 1) return false;
  if (c->weight_bits != 0 && c->weight_bits != 8 && c->weight_bits != 4) return false;
  if (c->max_batch < 0 || c->max_batch > 4) return false;
  return true;
}

BlobLayout blob_layout(const tvl_config* c, bool tied) {
  BlobLayout b;
  const int64_t d = c->dim, F = c->hidden_dim, V = c->vocab_size;
  const int64_t kvd = (int64_t)c->n_kv_heads * (d / c->n_heads);
  int64_t off = 0;
  auto take = [&](int64_t nfloats) {
    const int64_t at = off;
    off = a128(off + 4 * nfloats);
    return at;
  };
  b.E = take(V * d);
  b.l0 = off;
  // one layer, placed at offset 0 of its own block (every layer is alike)
  int64_t lo = 0;
  auto ltake = [&](int64_t nfloats) {
    const int64_t at = lo;
    lo = a128(lo + 4 * nfloats);
    return at;
  };
  b.g_att = ltake(d);
  b.wq = ltake(d * d);
  b.wk = ltake(kvd * d);
  b.wv = ltake(kvd * d);
  b.wo = ltake(d * d);
  b.g_ffn = ltake(d);
  b.w1 = ltake(F * d);
  b.w3 = ltake(F * d);
  b.w2 = ltake(d * F);
  b.stride = lo;
  off += (int64_t)c->n_layers * b.stride;
  b.g_final = take(d);
  if (!tied) b.Wcls = take(V * d);
  b.total = off;
  return b;
}

}  // namespace tvl

extern "C" {

size_t tvl_blob_bytes(const tvl_config* cfg, int32_t tied) {
  if (!tvl::config_valid(cfg)) return 0;
  return (size_t)tvl::blob_layout(cfg, tied != 0).total;
}

const char* tvl_status_string(tvl_status s) {
  switch (s) {
    case TVL_OK: return "ok";
    case TVL_E_INVAL: return "invalid argument";
    case TVL_E_SIZE: return "blob size does not match the configuration";
    case TVL_E_ALIGN: return "pointer not aligned as required";
    case TVL_E_NOMEM: return "out of memory";
    case TVL_E_CUDA: return "CUDA runtime error";
    case TVL_E_RANGE: return "token, position or step count out of range";
    case TVL_E_TIMEOUT: return "device-side wait timed out";
    case TVL_E_UNSUPPORTED: return "shape not supported by the GPU path";
  }
  return "unknown status";
}

const char* tvl_last_error(void) { return tvl::g_last_error.c_str(); }

void tvl_debug_fail_allocation(int32_t k) { tvl::g_fail_countdown.store(k < 0 ? -1 : k); }

int64_t tvl_debug_live_allocations(void) { return (int64_t)tvl::g_live_allocs.load(); }

}  // extern "C"
