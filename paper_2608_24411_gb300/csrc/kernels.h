// Entry points of the kernel translation units (one per kernel and dtype,
// compiled in parallel).  Each returns the __global__ function for a block
// size of 256 or 512 threads; the streaming kernel's for ResiSpec or, with
// spec, for SpecInfer.
#pragma once

namespace rs {
const void* resident_entry_f32(int threads);
const void* resident_entry_bf16(int threads);
const void* stream_entry_f32(int threads, bool spec);
const void* stream_entry_bf16(int threads, bool spec);
const void* stream_var_entry_f32(int threads, bool spec);   // with the optional paths
const void* stream_var_entry_bf16(int threads, bool spec);
}  // namespace rs
