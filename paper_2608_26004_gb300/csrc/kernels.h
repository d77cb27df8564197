// Host accessors of the kernels, each compiled in its own translation unit
// (k_*.cu) so that the build compiles them in parallel.  The pointers are
// passed to cudaLaunchKernelExC and the occupancy queries.
#pragma once

namespace asymspec_impl {

// fuse_verify_generic<T, VE, STOCH> (k_generic.cu)
const void* generic_kernel(int dtype, bool vector_path, bool stoch);
// fuse_verify_tma<T, STOCH, SEL>: program set 0 (k_tma_bf16.cu, k_tma_f32.cu) and the
// production sets 1..6 (k_tma_bf16_prod.cu, k_tma_f32_prod.cu); tma_kernel_* falls
// back to set 0 for any other sel
const void* tma_kernel_bf16_any(bool stoch);
const void* tma_kernel_f32_any(bool stoch);
const void* tma_kernel_bf16_any_stoch();  // k_tma_bf16_any_s.cu
const void* tma_kernel_f32_any_stoch();   // k_tma_f32_any_s.cu
const void* tma_kernel_bf16(bool stoch, int sel);
const void* tma_kernel_f32(bool stoch, int sel);
// fuse_verify_row<T>, the production kernel of the stochastic JSD step
// (k_row_bf16.cu, k_row_f32.cu)
const void* row_kernel_bf16();
const void* row_kernel_f32();
// decide_rows<T, STOCH>, launched after fuse_verify_tma or fuse_verify_row (k_tma_*.cu)
const void* decide_kernel_bf16(bool stoch);
const void* decide_kernel_f32(bool stoch);
// draft_kernel<T, VE, STOCH>, the drafter's draw (k_draft.cu)
const void* draft_kernel_ptr(int dtype, bool vector_path, bool stoch);
// the cross-family vocabulary map (k_xvocab.cu): xvocab_gather<T, WITH_T>,
// xvocab_gather_inv<T>, xvocab_inv_fill, xvocab_inv_build, xvocab_emit
const void* xvocab_gather_ptr(int dtype, bool with_t);
const void* xvocab_gather_inv_ptr(int dtype);
const void* xvocab_inv_fill_ptr();
const void* xvocab_inv_build_ptr();
const void* xvocab_emit_ptr();

}  // namespace asymspec_impl
