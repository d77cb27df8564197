// The production program sets of the cluster TMA kernel for float logits
// (see tma_program_set in kernel_tma.cuh).
#include "kernel_tma.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* tma_kernel_f32(bool stoch, int sel) {
  if (sel <= 0 || sel >= kTmaProgramSets || (stoch && sel > 3)) return tma_kernel_f32_any(stoch);
  if (stoch) {
    switch (sel) {
      case 1: return reinterpret_cast<const void*>(&fuse_verify_tma<float, true, 1>);
      case 2: return reinterpret_cast<const void*>(&fuse_verify_tma<float, true, 2>);
      case 3: return reinterpret_cast<const void*>(&fuse_verify_tma<float, true, 3>);
    }
  }
  switch (sel) {
    case 1: return reinterpret_cast<const void*>(&fuse_verify_tma<float, false, 1>);
    case 2: return reinterpret_cast<const void*>(&fuse_verify_tma<float, false, 2>);
    case 3: return reinterpret_cast<const void*>(&fuse_verify_tma<float, false, 3>);
    case 4: return reinterpret_cast<const void*>(&fuse_verify_tma<float, false, 4>);
    case 5: return reinterpret_cast<const void*>(&fuse_verify_tma<float, false, 5>);
    case 6: return reinterpret_cast<const void*>(&fuse_verify_tma<float, false, 6>);
  }
  return tma_kernel_f32_any(stoch);
}

}  // namespace asymspec_impl
