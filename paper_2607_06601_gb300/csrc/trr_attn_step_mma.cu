// trr_attn_step_mma.cu - the tensor-core kernels of trr_decode_step (query groups as
// for trr_decode_attn's tensor-core path), one instance per head size and groups per
// head; their split partials are merged by the same combine kernel.
#include "trr_attn.cuh"

namespace trr {

cudaError_t launch_attn_step_mma(const Layout& l, dim3 grid, dim3 block, size_t smem, cudaStream_t s, const AttnKernelArgs& k) {
  const int ng = l.d / l.G;
  if (l.d == 64) {
    if (ng == 1) return launch_pdl(attn_mma_kernel<64, 1, true>, grid, block, smem, s, k);
    return launch_pdl(attn_mma_kernel<64, 2, true>, grid, block, smem, s, k);
  }
  if (ng == 1) return launch_pdl(attn_mma_kernel<128, 1, true>, grid, block, smem, s, k);
  if (ng == 2) return launch_pdl(attn_mma_kernel<128, 2, true>, grid, block, smem, s, k);
  return launch_pdl(attn_mma_kernel<128, 4, true>, grid, block, smem, s, k);
}

cudaError_t configure_attn_step_mma() {
  const void* ks[] = {reinterpret_cast<const void*>(attn_mma_kernel<64, 1, true>),
                      reinterpret_cast<const void*>(attn_mma_kernel<64, 2, true>),
                      reinterpret_cast<const void*>(attn_mma_kernel<128, 1, true>),
                      reinterpret_cast<const void*>(attn_mma_kernel<128, 2, true>),
                      reinterpret_cast<const void*>(attn_mma_kernel<128, 4, true>)};
  for (const void* f : ks) {
    const cudaError_t e =
        cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, attn_smem_limit(kMmaCtasPerSm));
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace trr
