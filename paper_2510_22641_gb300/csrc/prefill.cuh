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

// p.tiles_n counts 128-column sub-tiles; a CTA tile is NT columns (kSub sub-tiles, the last one of a
// row of tiles possibly past the end, then neither loaded nor stored).
template <Epi EPI, int NT>
__global__ void __launch_bounds__(kTcThreads, 1)
    ssd_prefill_tc_kernel(const __grid_constant__ CUtensorMap map_ahi, const __grid_constant__ CUtensorMap map_alo,
                   const __grid_constant__ CUtensorMap map_b0, const __grid_constant__ CUtensorMap map_b1,
                   const __grid_constant__ CUtensorMap map_b2, const TcParams p) {
  using TS = TcShape<NT>;
  constexpr int kStagesT = TS::kStages;
  constexpr uint32_t kStageT = TS::kStage;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte aligned base for the swizzled tiles
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStagesT * kStageT);
  uint64_t* empty = full + kStagesT;
  uint64_t* tfull = empty + kStagesT;     // [2]
  uint64_t* tempty = tfull + 2;          // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  int* abort_flag = reinterpret_cast<int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tiles_nt = (p.tiles_n + TS::kSub - 1) / TS::kSub;  // NT-column tiles
  const int n_tiles = p.tiles_m * tiles_nt;

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesT; ++s) {
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
  if (warp == 1) {  // TMEM: 2 x NT fp32 columns
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(TS::kTmemCols)
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
        const int m_t = t % p.tiles_m, n_t0 = (t / p.tiles_m) * TS::kSub;
        const int n_sub = min(TS::kSub, p.tiles_n - n_t0);  // sub-tiles inside the matrix
        for (int ks = 0; ks < p.k_steps; ++ks, ++g) {
          const int s = g % kStagesT;
          if (!mbar_wait(&empty[s], ((g / kStagesT) & 1) ^ 1)) {
            set_error(p.st, DERR_TIMEOUT);
            *reinterpret_cast<volatile int*>(abort_flag) = 1;
            break;
          }
          uint8_t* st = smem + s * kStageT;
          mbar_arrive_expect_tx(&full[s], 2 * kTcATile + n_sub * kTcBTile);
          const int kx = ks * kTcK;
          tma_load_2d(st, &map_ahi, &full[s], kx, m_t * kTcM);
          tma_load_2d(st + kTcATile, &map_alo, &full[s], kx, m_t * kTcM);
          for (int sub = 0; sub < n_sub; ++sub) {
            const int n_t = n_t0 + sub;
            uint8_t* bs = st + 2 * kTcATile + sub * kTcBTile;
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
      if (*reinterpret_cast<volatile int*>(abort_flag)) drain_ring(full, kStagesT, g);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_bf16(kTcM, NT);
      int g = 0, it = 0;
      for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++it) {
        const int b = it & 1;
        if (!mbar_wait(&tempty[b], ((it >> 1) & 1) ^ 1)) {
          set_error(p.st, DERR_TIMEOUT);
          *reinterpret_cast<volatile int*>(abort_flag) = 1;
          break;
        }
        tmem_fence_after();
        const uint32_t d = tmem + b * NT;
        bool ok = true;
        for (int ks = 0; ks < p.k_steps; ++ks, ++g) {
          const int s = g % kStagesT;
          if (!mbar_wait(&full[s], (g / kStagesT) & 1)) {
            set_error(p.st, DERR_TIMEOUT);
            *reinterpret_cast<volatile int*>(abort_flag) = 1;
            ok = false;
            break;
          }
          tmem_fence_after();
          const uint32_t sa = smem_u32(smem + s * kStageT);
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
      const int m_t = t % p.tiles_m, n_t0 = (t / p.tiles_m) * TS::kSub;
      if (!mbar_wait(&tfull[b], (it >> 1) & 1)) {
        set_error(p.st, DERR_TIMEOUT);
        break;
      }
      tmem_fence_after();
      const int r = m_t * kTcM + q * 32 + lane;
#pragma unroll 1
      for (int sub = 0; sub < TS::kSub; ++sub) {
        if (n_t0 + sub >= p.tiles_n) break;
        float acc[kTcN];
        const uint32_t base = tmem + (static_cast<uint32_t>(q * 32) << 16) + b * NT + sub * kTcN;
#pragma unroll
        for (int c = 0; c < kTcN / 32; ++c) tmem_ld32(base + c * 32, acc + c * 32);
        if (r < p.M) tc_epilogue_row<EPI>(p, n_t0 + sub, r, acc);
      }
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[b]);  // accumulator b may be overwritten
    }
  }
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TS::kTmemCols) : "memory");
  }
}

}  // namespace ssd

namespace ssd {

// ------------------------------------------------------------------ causal prefill attention
// One CTA per (128-query block, head), the blocks with the most key blocks launched first.
// Both products run on the 5th-generation tensor cores with fp32-class accuracy: every fp32
// operand x is split into bf16 parts x = hi + lo and a product a.b is taken as
// hi(a) hi(b) + hi(a) lo(b) + lo(a) hi(b) in fp32 (the lo lo term is below fp32 rounding).
// ssd_attn_parts_kernel writes the parts once per layer (q rows, K rows, V transposed), so here
// every operand arrives by TMA in the 128-byte swizzled layout the MMA reads:
//   * warp 0 (one thread): the Q block, then each 64-key block's K and V^T parts into a 2-stage ring;
//   * warp 1 (one thread): S_j = Q K_j^T, 3 x Dh/16 MMAs (M = 128 queries, N = 64 keys) into one of
//     two TMEM score buffers, issued while the softmax works on the previous block; then
//     O_j = P_j V_j, 3 x 4 MMAs (N = Dh) into the TMEM output block;
//   * warps 2..5, one thread per query row (its TMEM lane): causal mask, online softmax in
//     registers (exp2 of the scores times scale * log2 e), P_j as bf16 parts into shared memory,
//     and O = O * alpha + O_j folded into the row's fp32 registers.
// Every step of a row depends on the keys' positions only; rows are independent.
constexpr int kFaThreads = 192;
constexpr int kFaTmemCols = 256;  // S: 2 x 64 columns, O block: Dh columns

template <int DH>
struct FaSmem {
  static constexpr int kNA = DH / 64;                    // 64-column atoms along the head dimension
  static constexpr int kQAtom = kFaQ * 128;              // one atom of the Q block (hi or lo)
  static constexpr int kKAtom = kFaK * 128;              // one atom of a K block
  static constexpr int kQh = 0;                          // [kNA][128 rows][128 B]
  static constexpr int kQl = kQh + kNA * kQAtom;
  static constexpr int kStage = 2 * kNA * kKAtom + 2 * DH * 128;  // K hi, K lo, V^T hi, V^T lo
  static constexpr int kKV = kQl + kNA * kQAtom;         // [2 stages]
  static constexpr int kPh = kKV + 2 * kStage;           // P: [128 rows][64 keys x 2 B]
  static constexpr int kPl = kPh + kFaQ * 128;
  static constexpr int kBar = kPl + kFaQ * 128;          // q_full, kv_full[2], kv_empty[2], s_full[2], p_full, o_full, o_empty
  static constexpr int kTmemSlot = kBar + 10 * 8;
  static constexpr int kTotal = kTmemSlot + 16 + 1024;   // + slack for the 1024-byte alignment
  // within a stage
  static constexpr int kKh = 0, kKl = kNA * kKAtom, kVh = 2 * kNA * kKAtom, kVl = kVh + DH * 128;
};

// 8 fp32 values -> bf16 hi and lo parts, packed two per word.
__device__ __forceinline__ void split8_bf16(const float* v, uint4& hi, uint4& lo) {
  uint32_t hw[4], lw[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const __nv_bfloat16 h0 = __float2bfloat16_rn(v[2 * e]), h1 = __float2bfloat16_rn(v[2 * e + 1]);
    hw[e] = pack_bf16x2(h0, h1);
    lw[e] = pack_bf16x2(__float2bfloat16_rn(v[2 * e] - __bfloat162float(h0)),
                        __float2bfloat16_rn(v[2 * e + 1] - __bfloat162float(h1)));
  }
  hi = make_uint4(hw[0], hw[1], hw[2], hw[3]);
  lo = make_uint4(lw[0], lw[1], lw[2], lw[3]);
}

// Byte offset of 16-byte chunk ch of row r in a 128-byte swizzled tile.
__device__ __forceinline__ int sw128_off(int r, int ch) { return r * 128 + ((ch ^ (r & 7)) << 4); }

// The attention's operand parts of one layer, once per prefill: for the 64 positions
// r0 .. r0 + 63 of head h, the q rows and the cache's K rows as bf16 hi / lo rows
// (qs [rows][qs_stride], ks [H][s_pad][Dh]) and the V rows transposed through shared memory
// (vt [H][Dh][s_pad], positions at or past P written as zeros), all with 16-byte stores.
template <int DH>
__global__ void __launch_bounds__(256) ssd_attn_parts_kernel(const float* __restrict__ q, int q_stride,
                                                            const float* __restrict__ k_cache,
                                                            const float* __restrict__ v_cache, int max_seq, int P,
                                                            __nv_bfloat16* qs_hi, __nv_bfloat16* qs_lo, int qs_stride,
                                                            __nv_bfloat16* ks_hi, __nv_bfloat16* ks_lo,
                                                            __nv_bfloat16* vt_hi, __nv_bfloat16* vt_lo, int s_pad) {
  __shared__ float vt[DH][65];
  const int r0 = blockIdx.x * 64, h = blockIdx.y, tid = threadIdx.x;
  pdl_trigger();
  pdl_wait();
  for (int t = tid; t < 64 * (DH / 8); t += 256) {
    const int r = t / (DH / 8), c8 = t - r * (DH / 8), pos = r0 + r;
    if (pos >= P) {
#pragma unroll
      for (int e = 0; e < 8; ++e) vt[c8 * 8 + e][r] = 0.f;
      continue;
    }
    uint4 hi, lo;
    float v[8];
    const float4* qr = reinterpret_cast<const float4*>(q + static_cast<size_t>(pos) * q_stride + h * DH + c8 * 8);
    float4 a = __ldcg(qr), b = __ldcg(qr + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    split8_bf16(v, hi, lo);
    const size_t qo = static_cast<size_t>(pos) * qs_stride + h * DH + c8 * 8;
    *reinterpret_cast<uint4*>(qs_hi + qo) = hi;
    *reinterpret_cast<uint4*>(qs_lo + qo) = lo;
    const size_t ko = (static_cast<size_t>(h) * max_seq + pos) * DH + c8 * 8;
    a = __ldcg(reinterpret_cast<const float4*>(k_cache + ko));
    b = __ldcg(reinterpret_cast<const float4*>(k_cache + ko) + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    split8_bf16(v, hi, lo);
    const size_t kso = (static_cast<size_t>(h) * s_pad + pos) * DH + c8 * 8;
    *reinterpret_cast<uint4*>(ks_hi + kso) = hi;
    *reinterpret_cast<uint4*>(ks_lo + kso) = lo;
    a = __ldcg(reinterpret_cast<const float4*>(v_cache + ko));
    b = __ldcg(reinterpret_cast<const float4*>(v_cache + ko) + 1);
    vt[c8 * 8 + 0][r] = a.x; vt[c8 * 8 + 1][r] = a.y; vt[c8 * 8 + 2][r] = a.z; vt[c8 * 8 + 3][r] = a.w;
    vt[c8 * 8 + 4][r] = b.x; vt[c8 * 8 + 5][r] = b.y; vt[c8 * 8 + 6][r] = b.z; vt[c8 * 8 + 7][r] = b.w;
  }
  __syncthreads();
  for (int t = tid; t < DH * 8; t += 256) {
    const int d = t >> 3, p8 = t & 7;
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = vt[d][p8 * 8 + e];
    uint4 hi, lo;
    split8_bf16(v, hi, lo);
    const size_t o = (static_cast<size_t>(h) * DH + d) * s_pad + r0 + p8 * 8;
    *reinterpret_cast<uint4*>(vt_hi + o) = hi;
    *reinterpret_cast<uint4*>(vt_lo + o) = lo;
  }
}

// maps: q hi, q lo ([rows][H*Dh], 128-row boxes), k hi, k lo ([H*s_pad][Dh], 64-row boxes),
// v^T hi, v^T lo ([H*Dh][s_pad], Dh-row boxes), all with 64-column boxes.
template <int DH>
__global__ void __launch_bounds__(kFaThreads, 1)
    ssd_prefill_attn_kernel(const __grid_constant__ CUtensorMap mqh, const __grid_constant__ CUtensorMap mql,
                            const __grid_constant__ CUtensorMap mkh, const __grid_constant__ CUtensorMap mkl,
                            const __grid_constant__ CUtensorMap mvh, const __grid_constant__ CUtensorMap mvl,
                            float* __restrict__ o, int o_stride, int P, int s_pad, float scale, DevState* st) {
  using S = FaSmem<DH>;
  extern __shared__ __align__(1024) uint8_t fa_raw[];
  const uint32_t raw = smem_u32(fa_raw);
  uint8_t* smem = fa_raw + (((raw + 1023u) & ~1023u) - raw);
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + S::kBar);
  uint64_t* kv_full = q_full + 1;
  uint64_t* kv_empty = kv_full + 2;
  uint64_t* s_full = kv_empty + 2;
  uint64_t* p_full = s_full + 2;
  uint64_t* o_full = p_full + 1;
  uint64_t* o_empty = o_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + S::kTmemSlot);
  const int nqb = gridDim.x, qb = nqb - 1 - static_cast<int>(blockIdx.x), h = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q0 = qb * kFaQ;
  const int n_keys = min(q0 + kFaQ, P);  // keys 0 .. n_keys - 1 reach some row of the block
  const int n_kb = (n_keys + kFaK - 1) / kFaK;

  pdl_trigger();
  if (tid == 0) {
    mbar_init(q_full, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&kv_full[b], 1);
      mbar_init(&kv_empty[b], 1);
      mbar_init(&s_full[b], 1);
    }
    mbar_init(p_full, 4);
    mbar_init(o_full, 1);
    mbar_init(o_empty, 4);
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kFaTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      prefetch_tensormap(&mkh);
      pdl_wait();  // the parts come from the upstream QKV projection
      mbar_arrive_expect_tx(q_full, 2 * S::kNA * S::kQAtom);
#pragma unroll
      for (int a = 0; a < S::kNA; ++a) {
        tma_load_2d(smem + S::kQh + a * S::kQAtom, &mqh, q_full, h * DH + a * 64, q0);
        tma_load_2d(smem + S::kQl + a * S::kQAtom, &mql, q_full, h * DH + a * 64, q0);
      }
      int issued = 0;
      for (int j = 0; j < n_kb; ++j) {
        const int b = j & 1;
        if (j >= 2 && !mbar_wait(&kv_empty[b], static_cast<uint32_t>((j - 2) >> 1) & 1u)) {
          set_error(st, DERR_TIMEOUT);
          break;
        }
        uint8_t* sb = smem + S::kKV + b * S::kStage;
        mbar_arrive_expect_tx(&kv_full[b], S::kStage);
#pragma unroll
        for (int a = 0; a < S::kNA; ++a) {
          tma_load_2d(sb + S::kKh + a * S::kKAtom, &mkh, &kv_full[b], a * 64, h * s_pad + j * kFaK);
          tma_load_2d(sb + S::kKl + a * S::kKAtom, &mkl, &kv_full[b], a * 64, h * s_pad + j * kFaK);
        }
        tma_load_2d(sb + S::kVh, &mvh, &kv_full[b], j * kFaK, h * DH);
        tma_load_2d(sb + S::kVl, &mvl, &kv_full[b], j * kFaK, h * DH);
        issued = j + 1;
      }
      if (__ldcg(&st->error) & DERR_TIMEOUT) {  // a wait gave up somewhere: bounded waits for the copies
        mbar_wait_for(q_full, 0u, 100000000ull);
        drain_ring(kv_full, 2, issued);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_s = umma_idesc_bf16(kFaQ, kFaK);
      constexpr uint32_t idesc_o = umma_idesc_bf16(kFaQ, DH);
      auto issue_s = [&](int j) {  // S_j into score buffer j & 1
        const int b = j & 1;
        const uint8_t* sb = smem + S::kKV + b * S::kStage;
        const uint32_t d = tmem + static_cast<uint32_t>(b * kFaK);
        tmem_fence_after();
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const int at = kk >> 2, sub = 2 * (kk & 3);
          const uint64_t qh = umma_desc_sw128(smem_u32(smem + S::kQh + at * S::kQAtom)) + sub;
          const uint64_t ql = umma_desc_sw128(smem_u32(smem + S::kQl + at * S::kQAtom)) + sub;
          const uint64_t kh = umma_desc_sw128(smem_u32(sb + S::kKh + at * S::kKAtom)) + sub;
          const uint64_t kl = umma_desc_sw128(smem_u32(sb + S::kKl + at * S::kKAtom)) + sub;
          umma_f16(d, qh, kh, idesc_s, kk > 0 ? 1u : 0u);
          umma_f16(d, qh, kl, idesc_s, 1u);
          umma_f16(d, ql, kh, idesc_s, 1u);
        }
        umma_commit(&s_full[b]);
      };
      auto issue_o = [&](int j) {  // O_j = P_j V_j; frees stage j & 1
        const uint8_t* sb = smem + S::kKV + (j & 1) * S::kStage;
        const uint32_t d = tmem + static_cast<uint32_t>(2 * kFaK);
        tmem_fence_after();
#pragma unroll
        for (int kk = 0; kk < kFaK / 16; ++kk) {
          const uint64_t ph = umma_desc_sw128(smem_u32(smem + S::kPh)) + 2 * kk;
          const uint64_t pl = umma_desc_sw128(smem_u32(smem + S::kPl)) + 2 * kk;
          const uint64_t vh = umma_desc_sw128(smem_u32(sb + S::kVh)) + 2 * kk;
          const uint64_t vl = umma_desc_sw128(smem_u32(sb + S::kVl)) + 2 * kk;
          umma_f16(d, ph, vh, idesc_o, kk > 0 ? 1u : 0u);
          umma_f16(d, ph, vl, idesc_o, 1u);
          umma_f16(d, pl, vh, idesc_o, 1u);
        }
        umma_commit(o_full);
        umma_commit(&kv_empty[j & 1]);
      };
      bool ok = n_kb > 0 && mbar_wait(q_full, 0) && mbar_wait(&kv_full[0], 0);
      if (ok) issue_s(0);
      for (int j = 0; ok && j < n_kb; ++j) {
        if (j + 1 < n_kb) {  // S_{j+1} runs while the softmax works on S_j: its score buffer held S_{j-1},
                             // which the softmax read before it released P_{j-1} (waited for below, last round)
          if (!mbar_wait(&kv_full[(j + 1) & 1], static_cast<uint32_t>((j + 1) >> 1) & 1u)) {
            ok = false;
            break;
          }
          issue_s(j + 1);
        }
        // O_j once P_j is written and O_{j-1} has been folded
        if (!mbar_wait(p_full, static_cast<uint32_t>(j) & 1u) ||
            (j >= 1 && !mbar_wait(o_empty, static_cast<uint32_t>(j - 1) & 1u))) {
          ok = false;
          break;
        }
        issue_o(j);
      }
      if (!ok && n_kb > 0) set_error(st, DERR_TIMEOUT);
    }
  } else {
    // ---------------------------------------------------------------- softmax (warps 2..5)
    const int quad = warp & 3;
    const int row = quad * 32 + lane, qi = q0 + row;
    const float sl2 = scale * 1.4426950408889634f;  // scores in log2 units: exp(x) = exp2(x log2 e)
    const uint32_t tl = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    float m_run = -INFINITY, l_run = 0.f, alpha_prev = 0.f;
    float acc[DH];
#pragma unroll
    for (int d = 0; d < DH; ++d) acc[d] = 0.f;
    bool ok = true;
    auto fold = [&](int j) {  // acc = acc * alpha_j + O_j
      if (ok && !mbar_wait(o_full, static_cast<uint32_t>(j) & 1u)) ok = false;
      tmem_fence_after();
#pragma unroll
      for (int c = 0; c < DH / 32; ++c) {
        float ov[32];
        tmem_ld32(tl + static_cast<uint32_t>(2 * kFaK + c * 32), ov);
#pragma unroll
        for (int e = 0; e < 32; ++e) acc[c * 32 + e] = fmaf(acc[c * 32 + e], alpha_prev, ov[e]);
      }
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(o_empty);
    };
    for (int j = 0; j < n_kb; ++j) {
      const int j0 = j * kFaK;
      const bool full = j0 + kFaK - 1 <= q0 && j0 + kFaK <= P;  // every key visible to every row
      if (ok && !mbar_wait(&s_full[j & 1], static_cast<uint32_t>(j >> 1) & 1u)) ok = false;
      tmem_fence_after();
      const uint32_t ts = tl + static_cast<uint32_t>((j & 1) * kFaK);
      float sv[2][32];
      tmem_ld32(ts, sv[0]);
      tmem_ld32(ts + 32, sv[1]);
      float bm = -INFINITY;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf)
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const int kj = j0 + hf * 32 + c;
          if (!full && (kj > qi || kj >= P)) sv[hf][c] = -INFINITY;
          bm = fmaxf(bm, sv[hf][c]);
        }
      const float m_new = fmaxf(m_run, bm * sl2);  // scale > 0: the max commutes with it
      const float alpha = m_run == -INFINITY ? 0.f : exp2f(m_run - m_new);
      float ls = 0.f;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf)
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const float e = sv[hf][c] == -INFINITY ? 0.f : exp2f(fmaf(sv[hf][c], sl2, -m_new));
          sv[hf][c] = e;
          ls += e;
        }
      tmem_fence_before();
      if (j >= 1) fold(j - 1);  // O_{j-1} is done, so P_{j-1} has been read: P_j may be written
#pragma unroll
      for (int hf = 0; hf < 2; ++hf)
#pragma unroll
        for (int c8 = 0; c8 < 4; ++c8) {
          uint4 hi, lo;
          split8_bf16(sv[hf] + 8 * c8, hi, lo);
          const int off = sw128_off(row, hf * 4 + c8);
          *reinterpret_cast<uint4*>(smem + S::kPh + off) = hi;
          *reinterpret_cast<uint4*>(smem + S::kPl + off) = lo;
        }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
      l_run = l_run * alpha + ls;
      m_run = m_new;
      alpha_prev = alpha;
    }
    if (n_kb > 0) fold(n_kb - 1);
    if (!ok) set_error(st, DERR_TIMEOUT);
    if (qi < P && ok) {
      const float inv = 1.0f / l_run;
      float4* orow = reinterpret_cast<float4*>(o + static_cast<size_t>(qi) * o_stride + h * DH);
#pragma unroll
      for (int d4 = 0; d4 < DH / 4; ++d4)
        orow[d4] = make_float4(acc[4 * d4] * inv, acc[4 * d4 + 1] * inv, acc[4 * d4 + 2] * inv, acc[4 * d4 + 3] * inv);
    }
  }
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kFaTmemCols) : "memory");
  }
}

}  // namespace ssd
