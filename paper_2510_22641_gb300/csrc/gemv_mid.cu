// ssd_wstream_mid_kernel instantiations (one per epilogue kind) and the activation split, with
// their host-side launchers.
#include "gemv_mid.cuh"

namespace ssd {

namespace {
template <Epi EPI>
cudaError_t mid_launch_e(const CUtensorMap* wmaps, const CUtensorMap* amaps, const GemvParams& p, int M, int grid,
                         cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);  // persistent: min(units, kMidCtasPerSm x #SMs)
  cfg.blockDim = dim3(kMidThreads);
  cfg.dynamicSmemBytes = MidSmem::kTotal;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, ssd_wstream_mid_kernel<EPI>, wmaps[0], wmaps[1], wmaps[2], amaps[0], amaps[1], p, M);
}

template <Epi EPI>
cudaError_t mid_reduce_launch_e(const GemvParams& p, int M, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((M + kNPad - 1) / kNPad, p.n_rt);
  cfg.blockDim = dim3(kDrainThreads);
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, ssd_mid_reduce_kernel<EPI>, p, M);
}

template <Epi EPI>
cudaError_t mid_attr_e() {
  return cudaFuncSetAttribute(ssd_wstream_mid_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              MidSmem::kTotal);
}
}  // namespace

// CTAs of one streaming launch (at most): the partial buffer needs that many + the site's row
// tiles slots of kMaxMidRows x kTileN floats.
int mid_max_ctas(int num_sms) { return kMidCtasPerSm * num_sms; }

// M in 1..kMaxMidRows; amaps: the split activations' hi and lo tensor maps ([NP][64] boxes).  Two
// launches: the stream (grid min(units, kMidCtasPerSm x num_sms)) writing partials, then the
// reduction + epilogue (grid chunks x row tiles).
cudaError_t mid_launch(Epi e, const CUtensorMap* wmaps, const CUtensorMap* amaps, const GemvParams& p0, int M,
                       int num_sms, cudaStream_t s, bool pdl) {
  if (M < 1 || M > kMaxMidRows) return cudaErrorInvalidValue;
  GemvParams p = p0;
  p.grid_ctas = p.units < kMidCtasPerSm * num_sms ? p.units : kMidCtasPerSm * num_sms;
  const int grid = p.grid_ctas;
  cudaError_t r;
  switch (e) {
    case Epi::QKV: r = mid_launch_e<Epi::QKV>(wmaps, amaps, p, M, grid, s, pdl); break;
    case Epi::GATE_SILU: r = mid_launch_e<Epi::GATE_SILU>(wmaps, amaps, p, M, grid, s, pdl); break;
    case Epi::SILU: r = mid_launch_e<Epi::SILU>(wmaps, amaps, p, M, grid, s, pdl); break;
    case Epi::RESID: r = mid_launch_e<Epi::RESID>(wmaps, amaps, p, M, grid, s, pdl); break;
    default: r = mid_launch_e<Epi::ARGMAX>(wmaps, amaps, p, M, grid, s, pdl); break;
  }
  if (r != cudaSuccess) return r;
  switch (e) {
    case Epi::QKV: return mid_reduce_launch_e<Epi::QKV>(p, M, s, pdl);
    case Epi::GATE_SILU: return mid_reduce_launch_e<Epi::GATE_SILU>(p, M, s, pdl);
    case Epi::SILU: return mid_reduce_launch_e<Epi::SILU>(p, M, s, pdl);
    case Epi::RESID: return mid_reduce_launch_e<Epi::RESID>(p, M, s, pdl);
    default: return mid_reduce_launch_e<Epi::ARGMAX>(p, M, s, pdl);
  }
}

cudaError_t mid_attrs() {
  cudaError_t e;
  if ((e = mid_attr_e<Epi::QKV>()) != cudaSuccess) return e;
  if ((e = mid_attr_e<Epi::GATE_SILU>()) != cudaSuccess) return e;
  if ((e = mid_attr_e<Epi::SILU>()) != cudaSuccess) return e;
  if ((e = mid_attr_e<Epi::RESID>()) != cudaSuccess) return e;
  return mid_attr_e<Epi::ARGMAX>();
}

cudaError_t split_act_launch(const float* x, int x_stride, int K, const __nv_bfloat16* gain, float eps,
                             __nv_bfloat16* hi, __nv_bfloat16* lo, int ld, float* rs, int rows, cudaStream_t s,
                             bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(rows);
  cfg.blockDim = dim3(kDrainThreads);
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, ssd_split_act_kernel, x, x_stride, K, gain, eps, hi, lo, ld, rs);
}

}  // namespace ssd
