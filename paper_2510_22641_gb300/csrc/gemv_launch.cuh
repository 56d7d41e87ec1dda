// Host-side launch helpers for ssd_wstream_kernel instantiations (one translation
// unit per epilogue kind keeps compile times parallel).
#pragma once

#include "gemv.cuh"

namespace ssd {

template <int M, Epi EPI>
cudaError_t gemv_launch_m(const CUtensorMap* maps, const GemvParams& p, int grid, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kGemvThreads);
  cfg.dynamicSmemBytes = GemvSmem<M>::kTotal;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, ssd_wstream_kernel<M, EPI>, maps[0], maps[1], maps[2], p);
}

template <int M, Epi EPI>
cudaError_t gemv_attr_m() {
  return cudaFuncSetAttribute(ssd_wstream_kernel<M, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              GemvSmem<M>::kTotal);
}

}  // namespace ssd

// Defines gemv_launch_<name>(M, ...) and gemv_attrs_<name>() for M = 1..16.
#define SSD_GEMV_CASE(M_, EPI_) \
  case M_:                      \
    return gemv_launch_m<M_, EPI_>(maps, p, grid, s, pdl);
#define SSD_GEMV_ATTR(M_, EPI_)               \
  if ((e = gemv_attr_m<M_, EPI_>()) != cudaSuccess) return e;

#define SSD_DEFINE_GEMV_16(NAME, EPI_)                                                                        \
  namespace ssd {                                                                                           \
  cudaError_t gemv_launch_##NAME(int M, const CUtensorMap* maps, const GemvParams& p, int grid, cudaStream_t s, \
                                 bool pdl) {                                                                \
    switch (M) {                                                                                            \
      SSD_GEMV_CASE(1, EPI_) SSD_GEMV_CASE(2, EPI_) SSD_GEMV_CASE(3, EPI_) SSD_GEMV_CASE(4, EPI_)            \
      SSD_GEMV_CASE(5, EPI_) SSD_GEMV_CASE(6, EPI_) SSD_GEMV_CASE(7, EPI_) SSD_GEMV_CASE(8, EPI_)            \
      SSD_GEMV_CASE(9, EPI_) SSD_GEMV_CASE(10, EPI_) SSD_GEMV_CASE(11, EPI_) SSD_GEMV_CASE(12, EPI_)         \
      SSD_GEMV_CASE(13, EPI_) SSD_GEMV_CASE(14, EPI_) SSD_GEMV_CASE(15, EPI_) SSD_GEMV_CASE(16, EPI_)        \
      default:                                                                                              \
        return cudaErrorInvalidValue;                                                                       \
    }                                                                                                       \
  }                                                                                                         \
  cudaError_t gemv_attrs_##NAME() {                                                                         \
    cudaError_t e;                                                                                          \
    SSD_GEMV_ATTR(1, EPI_) SSD_GEMV_ATTR(2, EPI_) SSD_GEMV_ATTR(3, EPI_) SSD_GEMV_ATTR(4, EPI_)              \
    SSD_GEMV_ATTR(5, EPI_) SSD_GEMV_ATTR(6, EPI_) SSD_GEMV_ATTR(7, EPI_) SSD_GEMV_ATTR(8, EPI_)              \
    SSD_GEMV_ATTR(9, EPI_) SSD_GEMV_ATTR(10, EPI_) SSD_GEMV_ATTR(11, EPI_) SSD_GEMV_ATTR(12, EPI_)           \
    SSD_GEMV_ATTR(13, EPI_) SSD_GEMV_ATTR(14, EPI_) SSD_GEMV_ATTR(15, EPI_) SSD_GEMV_ATTR(16, EPI_)          \
    return cudaSuccess;                                                                                     \
  }                                                                                                         \
  }
