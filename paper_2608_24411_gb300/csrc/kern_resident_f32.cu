// Instantiations of the resident verification kernel for f32 logits.
#include "kernels.h"
#include "verify_kernel.cuh"

namespace rs {
const void* resident_entry_f32(int threads) {
  return threads == 512 ? (const void*)verify_kernel<512, false> : (const void*)verify_kernel<256, false>;
}
}  // namespace rs
