// Instantiations of the stream verification kernel for bf16 logits with the
// optional paths compiled in (Z_applied, proxy denominator, level fill,
// drafting, phase counters).
#include "kernels.h"
#include "verify_stream.cuh"

namespace rs {
const void* stream_var_entry_bf16(int threads) {
  return threads == 512 ? (const void*)stream_kernel<512, true, true>
                        : (const void*)stream_kernel<256, true, true>;
}
}  // namespace rs
