// Instantiations of the persistent cluster kernel for __nv_bfloat16 logits (see kernel_ring.cuh).
#include "kernel_ring.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* ring_kernel_bf16(bool stoch) {
  return stoch ? reinterpret_cast<const void*>(&fuse_verify_ring<__nv_bfloat16, true>)
               : reinterpret_cast<const void*>(&fuse_verify_ring<__nv_bfloat16, false>);
}

}  // namespace asymspec_impl
