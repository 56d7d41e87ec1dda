// ssd_splitkv_attn_kernel instantiations (M = 1..kAttnMaxRows query rows per request, head_dim
// 64 / 128, causal or EXT) and their host-side launchers.
#include "attention.cuh"

namespace ssd {

namespace {

template <int M, int DH>
cudaError_t launch_md(bool ext, const AttnParams& a, dim3 grid, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kAttnThreads);
  cfg.dynamicSmemBytes = AttnSmem<M, DH>::kTotal;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return ext ? cudaLaunchKernelEx(&cfg, ssd_splitkv_attn_kernel<M, DH, true>, a)
             : cudaLaunchKernelEx(&cfg, ssd_splitkv_attn_kernel<M, DH, false>, a);
}

template <int M>
cudaError_t launch_m(int head_dim, bool ext, const AttnParams& a, dim3 grid, cudaStream_t s, bool pdl) {
  return head_dim == 128 ? launch_md<M, 128>(ext, a, grid, s, pdl) : launch_md<M, 64>(ext, a, grid, s, pdl);
}

template <int M, int DH>
cudaError_t attr_md() {
  cudaError_t e = cudaFuncSetAttribute(ssd_splitkv_attn_kernel<M, DH, false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, AttnSmem<M, DH>::kTotal);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(ssd_splitkv_attn_kernel<M, DH, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              AttnSmem<M, DH>::kTotal);
}

template <int M>
cudaError_t attrs_upto() {
  if constexpr (M > 1) {
    cudaError_t e = attrs_upto<M - 1>();
    if (e != cudaSuccess) return e;
  }
  cudaError_t e = attr_md<M, 128>();
  return e != cudaSuccess ? e : attr_md<M, 64>();
}

}  // namespace

// One launch over M rows per request of nreq requests: grid (kAttnSplit, n_heads, nreq).  EXT: fixed
// key sets / absolute positions / relative-position bias (the encoder-decoder model).
cudaError_t attn_launch(int M, int head_dim, const AttnParams& a, int nreq, cudaStream_t s, bool pdl) {
  const dim3 grid(kAttnSplit, a.n_heads, nreq);
  const bool ext = a.fixed_keys || a.abs_pos || a.bias;
  switch (M) {
    case 1: return launch_m<1>(head_dim, ext, a, grid, s, pdl);
    case 2: return launch_m<2>(head_dim, ext, a, grid, s, pdl);
    case 3: return launch_m<3>(head_dim, ext, a, grid, s, pdl);
    case 4: return launch_m<4>(head_dim, ext, a, grid, s, pdl);
    case 5: return launch_m<5>(head_dim, ext, a, grid, s, pdl);
    case 6: return launch_m<6>(head_dim, ext, a, grid, s, pdl);
    case 7: return launch_m<7>(head_dim, ext, a, grid, s, pdl);
    case 8: return launch_m<8>(head_dim, ext, a, grid, s, pdl);
    case 9: return launch_m<9>(head_dim, ext, a, grid, s, pdl);
    case 10: return launch_m<10>(head_dim, ext, a, grid, s, pdl);
    case 11: return launch_m<11>(head_dim, ext, a, grid, s, pdl);
    case 12: return launch_m<12>(head_dim, ext, a, grid, s, pdl);
    case 13: return launch_m<13>(head_dim, ext, a, grid, s, pdl);
    case 14: return launch_m<14>(head_dim, ext, a, grid, s, pdl);
    case 15: return launch_m<15>(head_dim, ext, a, grid, s, pdl);
    case 16: return launch_m<16>(head_dim, ext, a, grid, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t attn_attrs() { return attrs_upto<kAttnMaxRows>(); }

}  // namespace ssd
