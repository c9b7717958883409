// trr_attn_mma.cu - the tensor-core attention kernels of trr_decode_attn (query groups
// g >= 2 whose (head, group) columns fit one 8-wide mma tile), one instance per head
// size and groups per head, and the kernel that merges their split partials.
#include "trr_attn.cuh"

namespace trr {

cudaError_t launch_attn_mma(const Layout& l, dim3 grid, dim3 block, size_t smem, cudaStream_t s, const AttnKernelArgs& k) {
  const int ng = l.d / l.G;
  if (l.d == 64) {
    if (ng == 1) return launch_pdl(attn_mma_kernel<64, 1, false>, grid, block, smem, s, k);
    return launch_pdl(attn_mma_kernel<64, 2, false>, grid, block, smem, s, k);
  }
  if (ng == 1) return launch_pdl(attn_mma_kernel<128, 1, false>, grid, block, smem, s, k);
  if (ng == 2) return launch_pdl(attn_mma_kernel<128, 2, false>, grid, block, smem, s, k);
  return launch_pdl(attn_mma_kernel<128, 4, false>, grid, block, smem, s, k);
}

cudaError_t launch_attn_combine(int d, dim3 grid, dim3 block, cudaStream_t s, const CombineArgs& ca) {
  return d == 64 ? launch_pdl(attn_combine_kernel<64>, grid, block, 0, s, ca)
                 : launch_pdl(attn_combine_kernel<128>, grid, block, 0, s, ca);
}

cudaError_t configure_attn_mma() {
  const void* ks[] = {reinterpret_cast<const void*>(attn_mma_kernel<64, 1, false>),
                      reinterpret_cast<const void*>(attn_mma_kernel<64, 2, false>),
                      reinterpret_cast<const void*>(attn_mma_kernel<128, 1, false>),
                      reinterpret_cast<const void*>(attn_mma_kernel<128, 2, false>),
                      reinterpret_cast<const void*>(attn_mma_kernel<128, 4, false>)};
  for (const void* f : ks) {
    const cudaError_t e =
        cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, attn_smem_limit(kMmaCtasPerSm));
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace trr
