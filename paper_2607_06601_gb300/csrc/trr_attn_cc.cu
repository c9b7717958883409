// trr_attn_cc.cu - the CUDA-core attention kernels of trr_decode_attn (one mode per
// query): one instance per head size and page size, so that the page loop unrolls and
// a kernel's code holds only the four width classes it can meet.
#include "trr_attn.cuh"

namespace trr {

cudaError_t launch_attn_cc(const Layout& l, dim3 grid, dim3 block, size_t smem, cudaStream_t s, const AttnKernelArgs& k) {
  if (l.d == 64) {
    if (l.P == 16) return launch_pdl(attn_kernel<64, 16, false, false>, grid, block, smem, s, k);
    if (l.P == 32) return launch_pdl(attn_kernel<64, 32, false, false>, grid, block, smem, s, k);
    return launch_pdl(attn_kernel<64, 64, false, false>, grid, block, smem, s, k);
  }
  if (l.P == 16) return launch_pdl(attn_kernel<128, 16, false, false>, grid, block, smem, s, k);
  if (l.P == 32) return launch_pdl(attn_kernel<128, 32, false, false>, grid, block, smem, s, k);
  return launch_pdl(attn_kernel<128, 64, false, false>, grid, block, smem, s, k);
}

cudaError_t configure_attn_cc() {
  const void* k64[] = {reinterpret_cast<const void*>(attn_kernel<64, 16, false, false>),
                       reinterpret_cast<const void*>(attn_kernel<64, 32, false, false>),
                       reinterpret_cast<const void*>(attn_kernel<64, 64, false, false>)};
  const void* k128[] = {reinterpret_cast<const void*>(attn_kernel<128, 16, false, false>),
                        reinterpret_cast<const void*>(attn_kernel<128, 32, false, false>),
                        reinterpret_cast<const void*>(attn_kernel<128, 64, false, false>)};
  for (const void* f : k64) {
    const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               attn_smem_limit(cc_ctas_per_sm(64)));
    if (e != cudaSuccess) return e;
  }
  for (const void* f : k128) {
    const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               attn_smem_limit(cc_ctas_per_sm(128)));
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace trr
