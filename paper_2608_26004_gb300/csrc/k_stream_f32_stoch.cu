// Instantiation of the streaming kernel for float logits, stoch mode (see kernel_stream.cuh).
#include "kernel_stream.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* stream_kernel_f32_stoch() {
  return reinterpret_cast<const void*>(&fuse_verify_stream<float, true>);
}

}  // namespace asymspec_impl
