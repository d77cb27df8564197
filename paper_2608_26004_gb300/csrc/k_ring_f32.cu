// Instantiations of the persistent cluster kernel for float logits (see kernel_ring.cuh).
#include "kernel_ring.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* ring_kernel_f32(bool stoch) {
  return stoch ? reinterpret_cast<const void*>(&fuse_verify_ring<float, true>)
               : reinterpret_cast<const void*>(&fuse_verify_ring<float, false>);
}

}  // namespace asymspec_impl
