// Instantiations of the cluster TMA kernel and its decision kernel for __nv_bfloat16 logits (see kernel_tma.cuh).
#include "kernel_tma.cuh"
#include "kernels.h"

namespace asymspec_impl {

// Program set 0 (run-time dispatch); the production sets are in k_tma_bf16_prod.cu.
// (the stochastic one in k_tma_bf16_any_s.cu, built in parallel)
const void* tma_kernel_bf16_any(bool stoch) {
  return stoch ? tma_kernel_bf16_any_stoch()
               : reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 0>);
}

const void* decide_kernel_bf16(bool stoch) {
  return stoch ? reinterpret_cast<const void*>(&decide_rows<__nv_bfloat16, true>)
               : reinterpret_cast<const void*>(&decide_rows<__nv_bfloat16, false>);
}

}  // namespace asymspec_impl
