// Instantiations of the stream verification kernel for f32 logits with the
// optional paths compiled in (Z_applied, proxy denominator, level fill,
// drafting, phase counters).
#include "kernels.h"
#include "verify_stream.cuh"

namespace rs {
const void* stream_var_entry_f32(int threads) {
  return threads == 512 ? (const void*)stream_kernel<512, false, true>
                        : (const void*)stream_kernel<256, false, true>;
}
}  // namespace rs
