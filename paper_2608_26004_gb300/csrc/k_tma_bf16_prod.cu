// The production program sets of the cluster TMA kernel for __nv_bfloat16 logits
// (see tma_program_set in kernel_tma.cuh).
#include "kernel_tma.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* tma_kernel_bf16(bool stoch, int sel) {
  if (sel <= 0 || sel >= kTmaProgramSets || (stoch && sel > 3)) return tma_kernel_bf16_any(stoch);
  if (stoch) {
    switch (sel) {
      case 1: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, true, 1>);
      case 2: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, true, 2>);
      case 3: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, true, 3>);
    }
  }
  switch (sel) {
    case 1: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 1>);
    case 2: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 2>);
    case 3: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 3>);
    case 4: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 4>);
    case 5: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 5>);
    case 6: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 6>);
  }
  return tma_kernel_bf16_any(stoch);
}

}  // namespace asymspec_impl
