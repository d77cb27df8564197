// Instantiations of the production row kernel (kernel_row.cuh) for fp32
// logits: 256-thread CTAs two to an SM (fp32 slices of Qwen3-sized rows
// take 114 KB of shared memory even in clusters of 16).
#include "kernel_row.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* row_kernel_f32(int nt, int minb) {
  if (nt == 256 && minb == 2) return reinterpret_cast<const void*>(&fuse_verify_row<float, 256, 2>);
  return nullptr;
}

}  // namespace asymspec_impl
