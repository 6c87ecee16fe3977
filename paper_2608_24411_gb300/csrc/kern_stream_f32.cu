// Instantiations of the stream verification kernel for f32 logits: the
// ResiSpec instance and the SpecInfer instance (specinfer.cuh).
#include "kernels.h"
#include "verify_stream.cuh"

namespace rs {
const void* stream_entry_f32(int threads, bool spec) {
  if (spec)
    return threads == 512 ? (const void*)stream_kernel<512, false, false, true>
                          : (const void*)stream_kernel<256, false, false, true>;
  return threads == 512 ? (const void*)stream_kernel<512, false, false, false>
                        : (const void*)stream_kernel<256, false, false, false>;
}
}  // namespace rs
