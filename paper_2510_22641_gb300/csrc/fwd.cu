// Instantiations and launcher of the persistent forward kernel (head_dim 64 and 128).
#include "fwd.cuh"

namespace ssd {

cudaError_t fwd_attrs() {
  cudaError_t e = cudaFuncSetAttribute(fwd_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       FwdSmem<64>::kTotal);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(fwd_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, FwdSmem<128>::kTotal);
}

// CTAs of the kernel that fit on one SM (the grid must be fully resident).
cudaError_t fwd_ctas_per_sm(int head_dim, int* n) {
  return head_dim == 64
             ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, fwd_kernel<64>, kFwdThreads, FwdSmem<64>::kTotal)
             : cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, fwd_kernel<128>, kFwdThreads, FwdSmem<128>::kTotal);
}

cudaError_t fwd_launch(int head_dim, const FwdParams& p, int grid, cudaStream_t stream, bool cooperative) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kFwdThreads);
  cfg.dynamicSmemBytes = head_dim == 64 ? FwdSmem<64>::kTotal : FwdSmem<128>::kTotal;
  cfg.stream = stream;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;
  at[0].val.cooperative = cooperative ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return head_dim == 64 ? cudaLaunchKernelEx(&cfg, fwd_kernel<64>, p) : cudaLaunchKernelEx(&cfg, fwd_kernel<128>, p);
}

}  // namespace ssd
