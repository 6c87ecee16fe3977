// Instantiations of the stream verification kernel for bf16 logits.
#include "kernels.h"
#include "verify_stream.cuh"

namespace rs {
const void* stream_entry_bf16(int threads) {
  return threads == 512 ? (const void*)stream_kernel<512, true, false>
                       : (const void*)stream_kernel<256, true, false>;
}
}  // namespace rs
