// Instantiation of the production row kernel (kernel_row.cuh) for
// __nv_bfloat16 logits.
#include "kernel_row.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* row_kernel_bf16() { return reinterpret_cast<const void*>(&fuse_verify_row<__nv_bfloat16>); }


}  // namespace asymspec_impl
