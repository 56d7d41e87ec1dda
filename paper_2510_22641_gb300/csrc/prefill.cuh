// Prefill kernels: the decoder's projections over all P prompt rows as a dense
// tensor-core contraction (tcgen05 / TMEM), and causal attention over the rows.
//
// Prefill (Sec. "SSD Setup for VLMs": z and the prompt enter the decoder) runs
// every layer at M = P rows (P = 640 for the LLaVA-1.5 shape), which makes the
// projections real dense GEMMs.  They run on the 5th-generation tensor cores:
//   * activations a (fp32) are split into bf16 hi + lo parts (a = hi + lo up to
//     2^-17 relative), weights are bf16, and each K step issues two
//     kind::f16 MMAs (hi x W, lo x W) accumulating in fp32 in TMEM -- fp32-class
//     accuracy at bf16 tensor-core rate;
//   * 128 x 128 output tiles, K steps of 64 (one 128-byte swizzled row), a
//     4-stage TMA ring (A hi, A lo, W: 48 KB per stage), a double-buffered TMEM
//     accumulator (2 x 128 columns);
//   * warp 0 issues TMA, warp 1 owns TMEM and one thread of it issues the MMAs,
//     warps 2-5 drain TMEM with tcgen05.ld and apply the same fused epilogues as
//     the decode path (RoPE + KV write, SiLU(gate)*up, scaled residual).
#pragma once

#include "common.cuh"
#include "gemv.cuh"

#include "prefill_params.cuh"

namespace ssd {


// ------------------------------------------------------------------ activation split

// Row r of `out_hi` / `out_lo` (bf16 [rows][K]) = split of x[r] (fp32), optionally
// RMSNorm-scaled: v = x * rs * gain with rs = 1/sqrt(mean(x^2) + eps).
// hi = bf16(v), lo = bf16(v - hi).
__global__ void __launch_bounds__(256) ssd_split_rows_kernel(const float* __restrict__ x, int x_stride, int K,
                                                         const __nv_bfloat16* __restrict__ gain, float eps,
                                                         __nv_bfloat16* __restrict__ out_hi,
                                                         __nv_bfloat16* __restrict__ out_lo) {
  __shared__ float red[8];
  __shared__ float rs_s;
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x, tid = threadIdx.x;
  const float* xr = x + static_cast<size_t>(r) * x_stride;
  float rs = 1.f;
  if (gain) {
    float ss = 0.f;
    for (int i = tid; i < (K >> 2); i += 256) {
      const float4 v = __ldcg(reinterpret_cast<const float4*>(xr) + i);
      ss = fmaf(v.x, v.x, ss);
      ss = fmaf(v.y, v.y, ss);
      ss = fmaf(v.z, v.z, ss);
      ss = fmaf(v.w, v.w, ss);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    if ((tid & 31) == 0) red[tid >> 5] = ss;
    __syncthreads();
    if (tid == 0) {
      float t = 0.f;
      for (int w = 0; w < 8; ++w) t += red[w];
      rs_s = rsqrtf(t / static_cast<float>(K) + eps);
    }
    __syncthreads();
    rs = rs_s;
  }
  __nv_bfloat16* hr = out_hi + static_cast<size_t>(r) * K;
  __nv_bfloat16* lr = out_lo + static_cast<size_t>(r) * K;
  for (int i = tid; i < K; i += 256) {
    float v = __ldcg(xr + i);
    if (gain) v = v * rs * __bfloat162float(gain[i]);
    const __nv_bfloat16 h = __float2bfloat16_rn(v);
    hr[i] = h;
    lr[i] = __float2bfloat16_rn(v - __bfloat162float(h));
  }
}

// ------------------------------------------------------------------ tcgen05 GEMM

template <Epi EPI>
__device__ __forceinline__ void tc_epilogue_row(const TcParams& p, int n_t, int r, const float* acc) {
  // acc: the 128 fp32 outputs of token row r in output tile n_t (columns of the tile)
  const int pos = p.pos0 + r;
  if constexpr (EPI == Epi::QKV) {
    const int c0 = n_t * kTcN, seg = c0 / p.seg_rows, mat = seg + p.seg_base, local0 = c0 - seg * p.seg_rows;
    const int Dh = p.head_dim, half = Dh >> 1;
    if (pos < 0 || pos >= p.max_seq) {
      set_error(p.st, DERR_POS);
      return;
    }
    if (mat < 2) {
      for (int hh = 0; hh < kTcN / Dh; ++hh) {
        const int h = local0 / Dh + hh;
        float* kr = mat == 1 ? p.k_cache + (static_cast<size_t>(h) * p.max_seq + pos) * Dh : nullptr;
        float* qr = mat == 0 ? p.q_out + static_cast<size_t>(r) * p.q_stride + h * Dh : nullptr;
        for (int j = 0; j < half; ++j) {
          const float a = acc[hh * Dh + j], b = acc[hh * Dh + j + half];
          float va = a, vb = b;
          if (p.rope_cs) {
            const float2 cs = p.rope_cs[static_cast<size_t>(pos) * half + j];
            va = a * cs.x - b * cs.y;
            vb = a * cs.y + b * cs.x;
          }
          if (mat == 0) {
            qr[j] = va;
            qr[j + half] = vb;
          } else {
            kr[j] = va;
            kr[j + half] = vb;
          }
        }
      }
    } else {
      for (int c = 0; c < kTcN; ++c) {
        const int row = local0 + c, h = row / Dh, d = row - h * Dh;
        p.v_cache[(static_cast<size_t>(h) * p.max_seq + pos) * Dh + d] = acc[c];
      }
    }
  } else if constexpr (EPI == Epi::GATE_SILU) {
    float* hr = p.h_out + static_cast<size_t>(r) * p.h_stride + n_t * (kTcN / 2);
    for (int j = 0; j < kTcN / 2; ++j) {
      if (n_t * (kTcN / 2) + j >= p.N) break;
      hr[j] = (p.act ? gelu_tanh_f(acc[j]) : silu_f(acc[j])) * acc[kTcN / 2 + j];
    }
  } else {  // RESID
    const float s = __ldg(p.scale);
    const float* br = p.base + static_cast<size_t>(r) * p.base_stride + n_t * kTcN;
    float* dr = p.dst + static_cast<size_t>(r) * p.dst_stride + n_t * kTcN;
    for (int c = 0; c < kTcN; ++c) {
      if (n_t * kTcN + c >= p.N) break;
      dr[c] = br[c] + s * acc[c];
    }
  }
}

template <Epi EPI>
__global__ void __launch_bounds__(kTcThreads, 1)
    ssd_prefill_tc_kernel(const __grid_constant__ CUtensorMap map_ahi, const __grid_constant__ CUtensorMap map_alo,
                   const __grid_constant__ CUtensorMap map_b0, const __grid_constant__ CUtensorMap map_b1,
                   const __grid_constant__ CUtensorMap map_b2, const TcParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte aligned base for the swizzled tiles
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kTcStages * kTcStage);
  uint64_t* empty = full + kTcStages;
  uint64_t* tfull = empty + kTcStages;   // [2]
  uint64_t* tempty = tfull + 2;          // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_tiles = p.tiles_m * p.tiles_n;

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < kTcStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {  // TMEM: 2 x 128 fp32 columns
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kTcTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int g = 0;
      for (int t = blockIdx.x; t < n_tiles && !*reinterpret_cast<volatile int*>(abort_flag); t += gridDim.x) {
        const int m_t = t % p.tiles_m, n_t = t / p.tiles_m;
        for (int ks = 0; ks < p.k_steps; ++ks, ++g) {
          const int s = g % kTcStages;
          if (!mbar_wait(&empty[s], ((g / kTcStages) & 1) ^ 1)) {
            set_error(p.st, DERR_TIMEOUT);
            *reinterpret_cast<volatile int*>(abort_flag) = 1;
            break;
          }
          uint8_t* st = smem + s * kTcStage;
          mbar_arrive_expect_tx(&full[s], kTcStage);
          const int kx = ks * kTcK;
          tma_load_2d(st, &map_ahi, &full[s], kx, m_t * kTcM);
          tma_load_2d(st + kTcATile, &map_alo, &full[s], kx, m_t * kTcM);
          uint8_t* bs = st + 2 * kTcATile;
          if constexpr (EPI == Epi::GATE_SILU) {
            tma_load_2d(bs, &map_b0, &full[s], kx, n_t * (kTcN / 2));
            tma_load_2d(bs + kTcBTile / 2, &map_b1, &full[s], kx, n_t * (kTcN / 2));
          } else if constexpr (EPI == Epi::QKV) {
            const int r0 = n_t * kTcN, mat = r0 / p.seg_rows;
            tma_load_2d(bs, mat == 0 ? &map_b0 : (mat == 1 ? &map_b1 : &map_b2), &full[s], kx, r0 - mat * p.seg_rows);
          } else {
            tma_load_2d(bs, &map_b0, &full[s], kx, n_t * kTcN);
          }
        }
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_bf16(kTcM, kTcN);
      int g = 0, it = 0;
      for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++it) {
        const int b = it & 1;
        if (!mbar_wait(&tempty[b], ((it >> 1) & 1) ^ 1)) {
          set_error(p.st, DERR_TIMEOUT);
          *reinterpret_cast<volatile int*>(abort_flag) = 1;
          break;
        }
        tmem_fence_after();
        const uint32_t d = tmem + b * kTcN;
        bool ok = true;
        for (int ks = 0; ks < p.k_steps; ++ks, ++g) {
          const int s = g % kTcStages;
          if (!mbar_wait(&full[s], (g / kTcStages) & 1)) {
            set_error(p.st, DERR_TIMEOUT);
            *reinterpret_cast<volatile int*>(abort_flag) = 1;
            ok = false;
            break;
          }
          tmem_fence_after();
          const uint32_t sa = smem_u32(smem + s * kTcStage);
          const uint64_t ahi = umma_desc_sw128(sa), alo = umma_desc_sw128(sa + kTcATile),
                         bw = umma_desc_sw128(sa + 2 * kTcATile);
#pragma unroll
          for (int kk = 0; kk < kTcK / 16; ++kk) {
            // +32 bytes per 16-element K slice inside the 128-byte swizzled row
            umma_f16(d, ahi + 2 * kk, bw + 2 * kk, idesc, (ks > 0 || kk > 0) ? 1u : 0u);
            umma_f16(d, alo + 2 * kk, bw + 2 * kk, idesc, 1u);
          }
          umma_commit(&empty[s]);  // stage s is free once these MMAs have read it
        }
        if (!ok) break;
        umma_commit(&tfull[b]);    // accumulator b is complete
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue (warps 2..5)
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    int it = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++it) {
      const int b = it & 1;
      const int m_t = t % p.tiles_m, n_t = t / p.tiles_m;
      if (!mbar_wait(&tfull[b], (it >> 1) & 1)) {
        set_error(p.st, DERR_TIMEOUT);
        break;
      }
      tmem_fence_after();
      float acc[kTcN];
      const uint32_t base = tmem + (static_cast<uint32_t>(q * 32) << 16) + b * kTcN;
#pragma unroll
      for (int c = 0; c < kTcN / 32; ++c) tmem_ld32(base + c * 32, acc + c * 32);
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[b]);  // accumulator b may be overwritten
      const int r = m_t * kTcM + q * 32 + lane;
      if (r < p.M) tc_epilogue_row<EPI>(p, n_t, r, acc);
    }
  }
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcTmemCols) : "memory");
  }
}

}  // namespace ssd

namespace ssd {

// ------------------------------------------------------------------ causal prefill attention
// One CTA per (64-query block, head), the blocks with the most key blocks launched
// first: keys in blocks of 64 up to the query block (causal), brought into shared
// memory with 16-byte asynchronous copies, double-buffered (block kb + 1 loads while
// block kb is computed).  Scores 4 rows x 4 keys per thread in fp32 (keys tc, tc + 16,
// tc + 32, tc + 48: with K rows padded to Dh + 4 floats, the 16-byte K reads of a
// quarter warp hit 8 different bank groups), online softmax per row (a row's 64
// scores live on 16 consecutive lanes), O += P V with 4 rows x Dh/16 dims per thread.
// q: [P][q_stride] rotated queries; K, V: the fp32 cache.
constexpr int kPaQ = 64;
constexpr int kPaK = 64;
constexpr int kPaPad = 68;  // Q^T and P rows: 64 + 4 floats

template <int DH>
struct PaSmem {
  static constexpr int kKs = DH + 4;                            // padded K row
  static constexpr int kQt = 0;                                 // [DH][kPaPad]
  static constexpr int kK = kQt + DH * kPaPad * 4;              // [2][64][DH + 4]
  static constexpr int kV = kK + 2 * kPaK * kKs * 4;            // [2][64][DH]
  static constexpr int kP = kV + 2 * kPaK * DH * 4;             // [64][kPaPad]
  static constexpr int kTotal = kP + kPaQ * kPaPad * 4;
};

template <int DH>
__global__ void __launch_bounds__(256) ssd_prefill_attn_kernel(const float* __restrict__ q, int q_stride,
                                                           const float* __restrict__ k_cache,
                                                           const float* __restrict__ v_cache, float* __restrict__ o,
                                                           int o_stride, int P, int max_seq, float scale) {
  using S = PaSmem<DH>;
  constexpr int DPT = DH / 16;  // output dims per thread
  constexpr int KS = S::kKs;
  extern __shared__ __align__(128) uint8_t pa_smem[];
  float* Qt = reinterpret_cast<float*>(pa_smem + S::kQt);
  float* Kb = reinterpret_cast<float*>(pa_smem + S::kK);
  float* Vb = reinterpret_cast<float*>(pa_smem + S::kV);
  float* Ps = reinterpret_cast<float*>(pa_smem + S::kP);
  const int nqb = gridDim.x, qb = nqb - 1 - static_cast<int>(blockIdx.x), h = blockIdx.y, tid = threadIdx.x;
  const int q0 = qb * kPaQ;
  const int tr = tid >> 4, tc = tid & 15;  // rows 4tr..4tr+3; score keys tc + 16b; output dims tc*DPT..
  const float* kh = k_cache + static_cast<size_t>(h) * max_seq * DH;
  const float* vh = v_cache + static_cast<size_t>(h) * max_seq * DH;
  const int n_kb = min(qb + 1, (P + kPaK - 1) / kPaK);
  // key block kb -> buffer kb & 1; rows at or past P are zero-filled (nothing read)
  auto issue = [&](int kb) {
    const int j0 = kb * kPaK;
    float* kd = Kb + (kb & 1) * kPaK * KS;
    float* vd = Vb + (kb & 1) * kPaK * DH;
    for (int c = tid; c < kPaK * (DH / 4); c += 256) {
      const int j = c / (DH / 4), d4 = (c - j * (DH / 4)) * 4;
      const bool in = j0 + j < P;
      const size_t off = in ? static_cast<size_t>(j0 + j) * DH + d4 : 0;
      cp_async16_fill(kd + j * KS + d4, kh + off, in ? 16u : 0u);
      cp_async16_fill(vd + j * DH + d4, vh + off, in ? 16u : 0u);
    }
    cp_async_commit();
  };
  pdl_trigger();
  pdl_wait();
  issue(0);
  if (n_kb > 1) issue(1);
  else cp_async_commit();  // keep one group per block for the waits below

  // Q block, transposed: Qt[d][i] = q[q0 + i][h*DH + d] (rows past P read as 0)
  for (int idx = tid; idx < kPaQ * DH; idx += 256) {
    const int i = idx / DH, d = idx - i * DH;
    Qt[d * kPaPad + i] = (q0 + i < P) ? __ldcg(q + static_cast<size_t>(q0 + i) * q_stride + h * DH + d) : 0.f;
  }
  float m_run[4], l_run[4], acc[4][DPT];
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    m_run[a] = -INFINITY;
    l_run[a] = 0.f;
#pragma unroll
    for (int e = 0; e < DPT; ++e) acc[a][e] = 0.f;
  }
  for (int kb = 0; kb < n_kb; ++kb) {
    const int j0 = kb * kPaK;
    const float* Ks = Kb + (kb & 1) * kPaK * KS;
    const float* Vs = Vb + (kb & 1) * kPaK * DH;
    cp_async_wait_group<1>();  // block kb has landed (block kb + 1 may still be in flight)
    __syncthreads();
    // scores s[a][b] = q_{4tr+a} . k_{tc+16b}
    float s[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) s[a][b] = 0.f;
#pragma unroll 2
    for (int d = 0; d < DH; d += 4) {
      float4 qv[4], kv[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) qv[e] = *reinterpret_cast<const float4*>(Qt + (d + e) * kPaPad + 4 * tr);
#pragma unroll
      for (int b = 0; b < 4; ++b) kv[b] = *reinterpret_cast<const float4*>(Ks + (tc + 16 * b) * KS + d);
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        s[0][b] = fmaf(qv[0].x, kv[b].x, s[0][b]);
        s[1][b] = fmaf(qv[0].y, kv[b].x, s[1][b]);
        s[2][b] = fmaf(qv[0].z, kv[b].x, s[2][b]);
        s[3][b] = fmaf(qv[0].w, kv[b].x, s[3][b]);
        s[0][b] = fmaf(qv[1].x, kv[b].y, s[0][b]);
        s[1][b] = fmaf(qv[1].y, kv[b].y, s[1][b]);
        s[2][b] = fmaf(qv[1].z, kv[b].y, s[2][b]);
        s[3][b] = fmaf(qv[1].w, kv[b].y, s[3][b]);
        s[0][b] = fmaf(qv[2].x, kv[b].z, s[0][b]);
        s[1][b] = fmaf(qv[2].y, kv[b].z, s[1][b]);
        s[2][b] = fmaf(qv[2].z, kv[b].z, s[2][b]);
        s[3][b] = fmaf(qv[2].w, kv[b].z, s[3][b]);
        s[0][b] = fmaf(qv[3].x, kv[b].w, s[0][b]);
        s[1][b] = fmaf(qv[3].y, kv[b].w, s[1][b]);
        s[2][b] = fmaf(qv[3].z, kv[b].w, s[2][b]);
        s[3][b] = fmaf(qv[3].w, kv[b].w, s[3][b]);
      }
    }
    // online softmax per row over this key block (16 lanes share a row)
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int qi = q0 + 4 * tr + a;
      float mx = -INFINITY;
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int kj = j0 + tc + 16 * b;
        s[a][b] = (kj <= qi && kj < P) ? s[a][b] * scale : -INFINITY;
        mx = fmaxf(mx, s[a][b]);
      }
#pragma unroll
      for (int off = 8; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      const float m_new = fmaxf(m_run[a], mx);
      float rsum = 0.f;
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const float e = (m_new == -INFINITY || s[a][b] == -INFINITY) ? 0.f : expf(s[a][b] - m_new);
        Ps[(4 * tr + a) * kPaPad + tc + 16 * b] = e;
        rsum += e;
      }
#pragma unroll
      for (int off = 8; off > 0; off >>= 1) rsum += __shfl_xor_sync(0xffffffffu, rsum, off);
      const float corr = (m_run[a] == -INFINITY) ? 0.f : expf(m_run[a] - m_new);
      l_run[a] = l_run[a] * corr + rsum;
#pragma unroll
      for (int e = 0; e < DPT; ++e) acc[a][e] *= corr;
      m_run[a] = m_new;
    }
    __syncthreads();
    // O += P V
    const int kn = min(kPaK, P - j0);
    for (int j = 0; j < kn; ++j) {
      float vv[DPT];
#pragma unroll
      for (int e = 0; e < DPT; e += 4) {
        const float4 t = *reinterpret_cast<const float4*>(Vs + j * DH + tc * DPT + e);
        vv[e] = t.x;
        vv[e + 1] = t.y;
        vv[e + 2] = t.z;
        vv[e + 3] = t.w;
      }
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const float pj = Ps[(4 * tr + a) * kPaPad + j];
#pragma unroll
        for (int e = 0; e < DPT; ++e) acc[a][e] = fmaf(pj, vv[e], acc[a][e]);
      }
    }
    __syncthreads();  // buffer kb & 1 and Ps are free again
    if (kb + 2 < n_kb) issue(kb + 2);
    else cp_async_commit();
  }
  cp_async_wait_all();
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    const int qi = q0 + 4 * tr + a;
    if (qi >= P) continue;
    const float inv = 1.0f / l_run[a];
    float* orow = o + static_cast<size_t>(qi) * o_stride + h * DH + tc * DPT;
#pragma unroll
    for (int e = 0; e < DPT; ++e) orow[e] = acc[a][e] * inv;
  }
}

}  // namespace ssd
