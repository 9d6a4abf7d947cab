// decode_batch.cu — the persistent decode kernel for two to four sequences at
// once (float32 weights), in a translation unit of its own so that it
// compiles in parallel with the single-sequence kernels of decode.cu.
#include "decode_kernel.cuh"

namespace tvl {

const void* decode_kernel_for_batch(int B) {
  switch (B) {
    case 2: return (const void*)decode_kernel<false, 2>;
    case 3: return (const void*)decode_kernel<false, 3>;
    case 4: return (const void*)decode_kernel<false, 4>;
    default: return nullptr;
  }
}

}  // namespace tvl
