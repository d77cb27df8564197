// Instantiations of the production row kernel (kernel_row.cuh) for
// __nv_bfloat16 logits: 224-thread CTAs three to an SM, 192-thread CTAs
// four to an SM, 256-thread CTAs three or two to an SM.
#include "kernel_row.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* row_kernel_bf16(int nt, int minb) {
  if (nt == 224 && minb == 3) return reinterpret_cast<const void*>(&fuse_verify_row<__nv_bfloat16, 224, 3>);
  if (nt == 256 && minb == 3) return reinterpret_cast<const void*>(&fuse_verify_row<__nv_bfloat16, 256, 3>);
  if (nt == 256 && minb == 2) return reinterpret_cast<const void*>(&fuse_verify_row<__nv_bfloat16, 256, 2>);
  if (nt == 192 && minb == 4) return reinterpret_cast<const void*>(&fuse_verify_row<__nv_bfloat16, 192, 4>);
  return nullptr;
}

}  // namespace asymspec_impl
