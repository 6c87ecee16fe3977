// Instantiations of the stream verification kernel for bf16 logits with the
// optional paths compiled in (Z_applied, proxy denominator, level fill,
// drafting, phase counters), for ResiSpec and for SpecInfer.
#include "kernels.h"
#include "verify_stream.cuh"

namespace rs {
const void* stream_var_entry_bf16(int threads, bool spec) {
  if (spec)
    return threads == 512 ? (const void*)stream_kernel<512, true, true, true>
                          : (const void*)stream_kernel<256, true, true, true>;
  return threads == 512 ? (const void*)stream_kernel<512, true, true, false>
                        : (const void*)stream_kernel<256, true, true, false>;
}
}  // namespace rs
