// Instantiation of the production row kernel (kernel_row.cuh) for fp32
// logits.
#include "kernel_row.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* row_kernel_f32() { return reinterpret_cast<const void*>(&fuse_verify_row<float>); }


}  // namespace asymspec_impl
