// model.h — the loaded-model state shared by the library's host files
// (decode.cu: loading and decode launches; prefill.cu: multi-token prefill).
#pragma once
#include "decode_kernel.cuh"
#include "host_common.h"

using tvl::DecodeArgs;
using tvl::kMaxBatch;

struct tvl_model {
  tvl_config cfg{};
  bool tied = false;
  int device = 0;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  unsigned char* arena = nullptr;
  size_t arena_bytes = 0;
  size_t weight_bytes = 0;
  int64_t streamed_bytes = 0;
  DecodeArgs args{};
  int max_batch = 1;
  // per batch size B = 1..max_batch: the kernel (decode_kernel<q8, B>), its
  // shared-memory plan and the words between two sequences' phase inputs
  const void* kernel[kMaxBatch + 1] = {};
  struct Plan {
    int sm_ring, sm_bars, sm_xs, sm_vec, sm_seg, sm_att, sm_misc, nst, total;
  } plan[kMaxBatch + 1] = {};
  int vs = 0;
  int smem_bytes = 0;
  int* err_host = nullptr;  // pinned, mapped: the kernel writes its error code here too
  // Tag of the next launch's first exchange. Tags are 32-bit and 0 means never
  // written; before a launch whose tags would pass 2^32 - 1 the exchange words
  // [xchg_off, xchg_off + xchg_bytes) of the arena are zeroed and tags start at 1
  // again, so a tag is never reused while a word may still hold it.
  uint64_t next_tag = 1;
  size_t xchg_off = 0, xchg_bytes = 0;
  tvl_status sticky = TVL_OK;
  // multi-token prefill (prefill.cu): created on first use
  float* pf = nullptr;          // activations of up to max_seq positions
  size_t pf_bytes = 0;
  unsigned char* pf_w = nullptr;  // bf16 parts of every layer's weight matrices
};

// Releases what prefill created (prefill.cu).
void prefill_release(tvl_model* m);
