// host_common.h — host-side helpers shared by the library's .cu files:
// the per-thread error message and the blob layout as the library reads it.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>
#include <string>

#include "../../include/tvl.h"

namespace tvl {

void set_error(const std::string& msg);
tvl_status cuda_fail(cudaError_t e, const char* what);

#define TVL_CK(call)                                             \
  do {                                                           \
    cudaError_t e_ = (call);                                     \
    if (e_ != cudaSuccess) return ::tvl::cuda_fail(e_, #call);   \
  } while (0)

inline int64_t a128(int64_t b) { return (b + 127) / 128 * 128; }
inline int64_t a256(int64_t b) { return (b + 255) / 256 * 256; }

// Byte offsets of the packed blob (definition in include/tvl.h).
struct BlobLayout {
  int64_t E = 0, g_final = 0, Wcls = -1, total = 0;
  int64_t l0 = 0, stride = 0;  // first layer's start, bytes per layer
  int64_t g_att = 0, wq = 0, wk = 0, wv = 0, wo = 0, g_ffn = 0, w1 = 0, w3 = 0, w2 = 0;  // in a layer
};

// Every device and pinned-host allocation of the library goes through these:
// they count the allocations held (tvl_debug_live_allocations) and can be told
// to fail one attempt (tvl_debug_fail_allocation), so that tests can reach
// every failure point of the allocating calls and check their clean-up.
cudaError_t lib_malloc(void** p, size_t bytes);
void lib_free(void* p);
cudaError_t lib_host_alloc(void** p, size_t bytes, unsigned flags);
void lib_free_host(void* p);

bool config_valid(const tvl_config* c);
BlobLayout blob_layout(const tvl_config* c, bool tied);

}  // namespace tvl
