// Launchers of the prefill kernels (tcgen05 GEMM, activation split, causal attention).
#include "prefill.cuh"

namespace ssd {

template <typename Kern, typename... Args>
static cudaError_t launch_pdl(Kern kern, dim3 grid, dim3 block, size_t smem, cudaStream_t s, bool pdl,
                              Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

template <Epi EPI, int NT>
static cudaError_t tc_attr() {
  return cudaFuncSetAttribute(ssd_prefill_tc_kernel<EPI, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              TcShape<NT>::kSmem);
}

cudaError_t prefill_attrs() {
  cudaError_t e;
  if ((e = tc_attr<Epi::QKV, 128>()) || (e = tc_attr<Epi::QKV, 256>()) || (e = tc_attr<Epi::GATE_SILU, 128>()) ||
      (e = tc_attr<Epi::GATE_SILU, 256>()) || (e = tc_attr<Epi::RESID, 128>()))
    return e;
  if ((e = cudaFuncSetAttribute(ssd_prefill_attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                FaSmem<128>::kTotal)))
    return e;
  return cudaFuncSetAttribute(ssd_prefill_attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              FaSmem<64>::kTotal);
}

// nt: output tile width, 128 or 256 (QKV and gate/up only).
cudaError_t tc_gemm_launch(Epi e, int nt, const CUtensorMap* a, const CUtensorMap* b, const TcParams& p, int grid,
                           cudaStream_t s, bool pdl) {
  const dim3 g(grid), blk(kTcThreads);
  switch (e) {
    case Epi::QKV:
      return nt == 256 ? launch_pdl(ssd_prefill_tc_kernel<Epi::QKV, 256>, g, blk, TcShape<256>::kSmem, s, pdl, a[0],
                                    a[1], b[0], b[1], b[2], p)
                       : launch_pdl(ssd_prefill_tc_kernel<Epi::QKV, 128>, g, blk, TcShape<128>::kSmem, s, pdl, a[0],
                                    a[1], b[0], b[1], b[2], p);
    case Epi::GATE_SILU:
      return nt == 256 ? launch_pdl(ssd_prefill_tc_kernel<Epi::GATE_SILU, 256>, g, blk, TcShape<256>::kSmem, s, pdl,
                                    a[0], a[1], b[0], b[1], b[2], p)
                       : launch_pdl(ssd_prefill_tc_kernel<Epi::GATE_SILU, 128>, g, blk, TcShape<128>::kSmem, s, pdl,
                                    a[0], a[1], b[0], b[1], b[2], p);
    case Epi::RESID:
      return launch_pdl(ssd_prefill_tc_kernel<Epi::RESID, 128>, g, blk, TcShape<128>::kSmem, s, pdl, a[0], a[1], b[0],
                        b[1], b[2], p);
    default:
      return cudaErrorInvalidValue;
  }
}

cudaError_t split_rows_launch(const float* x, int x_stride, int K, const __nv_bfloat16* gain, float eps,
                              __nv_bfloat16* hi, __nv_bfloat16* lo, int rows, cudaStream_t s, bool pdl) {
  return launch_pdl(ssd_split_rows_kernel, dim3(rows), dim3(256), 0, s, pdl, x, x_stride, K, gain, eps, hi, lo);
}

cudaError_t attn_parts_launch(int head_dim, const float* q, int q_stride, const float* kc, const float* vc, int max_seq,
                              int P, int n_heads, __nv_bfloat16* parts, size_t q_elems, size_t kv_elems, int qs_stride,
                              int s_pad, cudaStream_t s, bool pdl) {
  const dim3 grid((P + 63) / 64, n_heads);
  __nv_bfloat16 *qh = parts, *ql = parts + q_elems, *kh = parts + 2 * q_elems, *kl = kh + kv_elems,
                *vh = kh + 2 * kv_elems, *vl = kh + 3 * kv_elems;
  if (head_dim == 128)
    return launch_pdl(ssd_attn_parts_kernel<128>, grid, dim3(256), 0, s, pdl, q, q_stride, kc, vc, max_seq, P, qh, ql,
                      qs_stride, kh, kl, vh, vl, s_pad);
  return launch_pdl(ssd_attn_parts_kernel<64>, grid, dim3(256), 0, s, pdl, q, q_stride, kc, vc, max_seq, P, qh, ql,
                    qs_stride, kh, kl, vh, vl, s_pad);
}

cudaError_t prefill_attn_launch(int head_dim, const CUtensorMap* maps, float* o, int o_stride, int P, int n_heads,
                                int s_pad, float scale, DevState* st, cudaStream_t s, bool pdl) {
  const dim3 grid((P + kFaQ - 1) / kFaQ, n_heads);
  if (head_dim == 128)
    return launch_pdl(ssd_prefill_attn_kernel<128>, grid, dim3(kFaThreads), FaSmem<128>::kTotal, s, pdl, maps[0],
                      maps[1], maps[2], maps[3], maps[4], maps[5], o, o_stride, P, s_pad, scale, st);
  return launch_pdl(ssd_prefill_attn_kernel<64>, grid, dim3(kFaThreads), FaSmem<64>::kTotal, s, pdl, maps[0], maps[1],
                    maps[2], maps[3], maps[4], maps[5], o, o_stride, P, s_pad, scale, st);
}

}  // namespace ssd
