// tc.cuh — inline-PTX building blocks of the fifth-generation tensor cores on
// sm_103a: tensor-memory (TMEM) allocation, tcgen05.mma issued by one thread
// with shared-memory matrix descriptors, completion through tcgen05.commit on
// an mbarrier, tcgen05.ld of the accumulator, and 2-D TMA tensor loads.
#pragma once
#include <cuda.h>

#include "ptx.cuh"

namespace tvl {

// ---- tensor memory --------------------------------------------------------------

// Allocates ncols columns (a power of two, at least 32) of this SM's tensor
// memory for the CTA; the TMEM address lands in *slot (shared memory). Warp-wide.
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_addr(slot)),
               "r"(ncols)
               : "memory");
}

// Lets other CTAs on the SM allocate (this CTA allocates only once). Warp-wide.
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// Ordering of tcgen05 operations across a thread synchronisation.
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// ---- matrix descriptors and the MMA ------------------------------------------------

// Shared-memory descriptor of a K-major operand tile stored with the 128-byte
// swizzle (rows of 128 bytes, groups of 8 rows 1024 bytes apart, the tile
// 1024-byte aligned; what a TMA load with CU_TENSOR_MAP_SWIZZLE_128B writes).
// Fields: start address >> 4 (bits 0-13), leading-dimension byte offset >> 4
// (bits 16-29; unused for this layout), stride-dimension byte offset >> 4
// (bits 32-45: 1024 bytes between 8-row groups), descriptor version 1 (bits
// 46-47), layout 2 = 128-byte swizzle (bits 61-63). p may point 32, 64 or 96
// bytes into a row to select the K step inside the swizzle span.
__device__ __forceinline__ uint64_t umma_desc_sw128(const void* p) {
  const uint32_t a = smem_addr(p);
  uint64_t d = (uint64_t)((a >> 4) & 0x3FFFu);
  d |= (uint64_t)1u << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}

// Instruction descriptor of tcgen05.mma kind::f16 with bf16 A and B, an fp32
// accumulator, both operands K-major: D format f32 (bits 4-5 = 1), A format
// bf16 (bits 7-9 = 1), B format bf16 (bits 10-12 = 1), no negation, K-major
// A and B (bits 15, 16 = 0), N >> 3 (bits 17-22), M >> 4 (bits 24-28).
__host__ __device__ constexpr uint32_t umma_idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

// D[tmem] (+)= A * B^T over one K step (16 bf16): A [M x 16] and B [N x 16]
// from their descriptors. accumulate 0 overwrites D. One thread issues it.
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives once on bar when every tcgen05.mma this thread issued before has
// completed (their shared-memory operands may then be overwritten).
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_addr(bar))
      : "memory");
}

// Sixteen consecutive 32-bit columns of TMEM lane (lane_base + laneid) into v,
// waiting for the load inside the same statement so that no use of v can be
// scheduled before the data is there. Warp-wide; the warp may only address
// the 32 lanes of its quarter of the SM (warp w % 4).
__device__ __forceinline__ void tc_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15}, [%16];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// ---- TMA tensor loads -----------------------------------------------------------

// Box at coordinates (x, y) of a 2-D tensor map (x: inner dimension, in
// elements; x * element size must be a multiple of 16 bytes) into dst, which
// must be aligned as the map's swizzle needs; completion on bar (the full box
// size counts, zeros included for coordinates outside the tensor).
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, "
      "{%2, %3}], [%4];" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

}  // namespace tvl
