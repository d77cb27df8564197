// Instantiations of the drafter's draw (see kernel_draft.cuh).
#include "kernel_draft.cuh"
#include "kernels.h"

namespace asymspec_impl {

template <typename T, int VE>
const void* draft_pick(bool stoch) {
  return stoch ? reinterpret_cast<const void*>(&draft_kernel<T, VE, true>)
               : reinterpret_cast<const void*>(&draft_kernel<T, VE, false>);
}

const void* draft_kernel_ptr(int dtype, bool vector_path, bool stoch) {
  if (dtype == ASYMSPEC_FP32)
    return vector_path ? draft_pick<float, 4>(stoch) : draft_pick<float, 1>(stoch);
  return vector_path ? draft_pick<__nv_bfloat16, 8>(stoch) : draft_pick<__nv_bfloat16, 1>(stoch);
}

}  // namespace asymspec_impl
