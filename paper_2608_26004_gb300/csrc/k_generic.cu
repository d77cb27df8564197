// Instantiations of the generic cluster kernel (see kernel_generic.cuh).
#include "kernel_generic.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* generic_kernel(int dtype, bool vector_path, bool stoch) {
  if (dtype == ASYMSPEC_FP32) {
    if (vector_path)
      return stoch ? reinterpret_cast<const void*>(&fuse_verify_generic<float, 4, true>)
                   : reinterpret_cast<const void*>(&fuse_verify_generic<float, 4, false>);
    return stoch ? reinterpret_cast<const void*>(&fuse_verify_generic<float, 1, true>)
                 : reinterpret_cast<const void*>(&fuse_verify_generic<float, 1, false>);
  }
  if (vector_path)
    return stoch ? reinterpret_cast<const void*>(&fuse_verify_generic<__nv_bfloat16, 8, true>)
                 : reinterpret_cast<const void*>(&fuse_verify_generic<__nv_bfloat16, 8, false>);
  return stoch ? reinterpret_cast<const void*>(&fuse_verify_generic<__nv_bfloat16, 1, true>)
               : reinterpret_cast<const void*>(&fuse_verify_generic<__nv_bfloat16, 1, false>);
}

}  // namespace asymspec_impl
