// Instantiation of the streaming kernel for __nv_bfloat16 logits, stoch mode (see kernel_stream.cuh).
#include "kernel_stream.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* stream_kernel_bf16_stoch() {
  return reinterpret_cast<const void*>(&fuse_verify_stream<__nv_bfloat16, true>);
}

}  // namespace asymspec_impl
