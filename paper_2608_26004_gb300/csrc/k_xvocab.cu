// Instantiations of the cross-family gather and emission (see kernel_xvocab.cuh).
#include "kernel_xvocab.cuh"
#include "kernels.h"

namespace asymspec_impl {

const void* xvocab_gather_ptr(int dtype, bool with_t) {
  if (dtype == ASYMSPEC_FP32)
    return with_t ? reinterpret_cast<const void*>(&xvocab_gather<float, true>)
                  : reinterpret_cast<const void*>(&xvocab_gather<float, false>);
  return with_t ? reinterpret_cast<const void*>(&xvocab_gather<__nv_bfloat16, true>)
                : reinterpret_cast<const void*>(&xvocab_gather<__nv_bfloat16, false>);
}

const void* xvocab_gather_inv_ptr(int dtype) {
  return dtype == ASYMSPEC_FP32 ? reinterpret_cast<const void*>(&xvocab_gather_inv<float>)
                                : reinterpret_cast<const void*>(&xvocab_gather_inv<__nv_bfloat16>);
}

const void* xvocab_emit_ptr() { return reinterpret_cast<const void*>(&xvocab_emit<int32_t>); }

const void* xvocab_inv_fill_ptr() { return reinterpret_cast<const void*>(&xvocab_inv_fill<int>); }

const void* xvocab_inv_build_ptr() { return reinterpret_cast<const void*>(&xvocab_inv_build<int>); }

}  // namespace asymspec_impl
