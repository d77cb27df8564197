// Program set 0 (run-time dispatch) of the cluster TMA kernel for float logits,
// stochastic mode (see kernel_tma.cuh); in its own translation unit so that
// the build compiles it in parallel with the greedy one.
#include "kernel_tma.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* tma_kernel_f32_any_stoch() {
  return reinterpret_cast<const void*>(&fuse_verify_tma<float, true, 0>);
}

}  // namespace asymspec_impl
