// The production program sets 1..6 of the persistent cluster kernel,
// fuse_verify_tma<T, STOCH, SEL, true>, for __nv_bfloat16 logits (see kernel_tma.cuh).
// There is no persistent form of program set 0 (run-time dispatch).
#include "kernel_tma.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* tmap_kernel_bf16(bool stoch, int sel) {
  if (sel <= 0 || sel >= kTmaProgramSets || (stoch && sel > 3)) return nullptr;
  if (stoch) {
    switch (sel) {
      case 1: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, true, 1, true>);
      case 2: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, true, 2, true>);
      case 3: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, true, 3, true>);
    }
  }
  switch (sel) {
    case 1: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 1, true>);
    case 2: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 2, true>);
    case 3: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 3, true>);
    case 4: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 4, true>);
    case 5: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 5, true>);
    case 6: return reinterpret_cast<const void*>(&fuse_verify_tma<__nv_bfloat16, false, 6, true>);
  }
  return nullptr;
}

}  // namespace asymspec_impl
