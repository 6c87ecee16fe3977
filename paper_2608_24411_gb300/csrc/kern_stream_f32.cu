// Instantiations of the stream verification kernel for f32 logits.
#include "kernels.h"
#include "verify_stream.cuh"

namespace rs {
const void* stream_entry_f32(int threads) {
  return threads == 512 ? (const void*)stream_kernel<512, false, false>
                       : (const void*)stream_kernel<256, false, false>;
}
}  // namespace rs
