// Instantiations of the cluster TMA kernel and its decision kernel for float logits (see kernel_tma.cuh).
#include "kernel_tma.cuh"
#include "kernels.h"

namespace asymspec_impl {

// Program set 0 (run-time dispatch); the production sets are in k_tma_f32_prod.cu.
// (the stochastic one in k_tma_f32_any_s.cu, built in parallel)
const void* tma_kernel_f32_any(bool stoch) {
  return stoch ? tma_kernel_f32_any_stoch()
               : reinterpret_cast<const void*>(&fuse_verify_tma<float, false, 0>);
}

const void* decide_kernel_f32(bool stoch) {
  return stoch ? reinterpret_cast<const void*>(&decide_rows<float, true>)
               : reinterpret_cast<const void*>(&decide_rows<float, false>);
}

}  // namespace asymspec_impl
