// Instantiations of the stream verification kernel for bf16 logits: the
// ResiSpec instance and the SpecInfer instance (specinfer.cuh).
#include "kernels.h"
#include "verify_stream.cuh"

namespace rs {
const void* stream_entry_bf16(int threads, bool spec) {
  if (spec)
    return threads == 512 ? (const void*)stream_kernel<512, true, false, true>
                          : (const void*)stream_kernel<256, true, false, true>;
  return threads == 512 ? (const void*)stream_kernel<512, true, false, false>
                        : (const void*)stream_kernel<256, true, false, false>;
}
}  // namespace rs
