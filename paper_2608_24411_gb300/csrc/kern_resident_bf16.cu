// Instantiations of the resident verification kernel for bf16 logits.
#include "kernels.h"
#include "verify_kernel.cuh"

namespace rs {
const void* resident_entry_bf16(int threads) {
  return threads == 512 ? (const void*)verify_kernel<512, true> : (const void*)verify_kernel<256, true>;
}
}  // namespace rs
