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
// One CTA per (128-query block, head), the blocks with the most key blocks launched first.
// Both products run on the 5th-generation tensor cores with fp32-class accuracy: every fp32
// operand x is split into bf16 parts x = hi + lo, and a product a.b is taken as
// hi(a) hi(b) + hi(a) lo(b) + lo(a) hi(b) in fp32 (the lo lo term is below fp32 rounding).
//   * Q block (128 rows x Dh) -> bf16 hi / lo, 128-byte swizzled K-major (rows = queries), once;
//   * per 64-key block (causal: up to the query block): thread 0 bulk-copies the block's fp32 K and
//     V rows into a staging buffer one block ahead; all threads turn them into bf16 hi / lo K
//     (rows = keys) and V^T (rows = head dimensions, keys along K);
//   * S = Q K^T: 3 x Dh/16 tcgen05.mma (M = 128 queries, N = 64 keys) into TMEM columns 0..63;
//   * warps 0..3, one thread per query row (its TMEM lane): scale, causal mask, online softmax
//     (running max and sum in registers), P = exp(S - max) -> bf16 hi / lo, 128-byte swizzled
//     (rows = queries, keys along K);
//   * O_blk = P V: 3 x 4 tcgen05.mma (M = 128, N = Dh, K = 64 keys) into TMEM columns 64..64+Dh;
//     the same threads fold it into their row's fp32 output registers, O = O * alpha + O_blk.
// Every step of a row depends on the keys' positions only; rows are independent.
// q: [P][q_stride] rotated queries; K, V: the fp32 cache [H][max_seq][Dh]; o: [P][o_stride].
constexpr int kFaQ = 128;       // query rows per CTA (the MMA's M)
constexpr int kFaK = 64;        // keys per block (the S MMA's N, the P.V MMA's K)
constexpr int kFaThreads = 256;
constexpr int kFaTmemCols = 256;  // S: 64 columns, O block: Dh columns

template <int DH>
struct FaSmem {
  static constexpr int kNA = DH / 64;                    // 64-column atoms along the head dimension
  static constexpr int kQAtom = kFaQ * 128;              // one atom of the Q block (hi or lo)
  static constexpr int kKAtom = kFaK * 128;              // one atom of the K block
  static constexpr int kQh = 0;                          // [kNA][128 rows][128 B]
  static constexpr int kQl = kQh + kNA * kQAtom;
  static constexpr int kKh = kQl + kNA * kQAtom;         // [kNA][64 keys][128 B]
  static constexpr int kKl = kKh + kNA * kKAtom;
  static constexpr int kVh = kKl + kNA * kKAtom;         // V^T: [Dh rows][64 keys x 2 B]
  static constexpr int kVl = kVh + DH * 128;
  static constexpr int kPh = kVl + DH * 128;             // P: [128 rows][64 keys x 2 B]
  static constexpr int kPl = kPh + kFaQ * 128;
  static constexpr int kStK = kPl + kFaQ * 128;          // fp32 staging of one block: K [64][Dh]
  static constexpr int kStV = kStK + kFaK * DH * 4;      //                            V [64][Dh]
  static constexpr int kBar = kStV + kFaK * DH * 4;      // staging full, MMA done
  static constexpr int kTmemSlot = kBar + 16;
  static constexpr int kTotal = kTmemSlot + 16 + 1024;   // + slack for the 1024-byte alignment
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

// Byte offset of 16-byte chunk ch of row r in a 128-byte swizzled atom.
__device__ __forceinline__ int sw128_off(int r, int ch) { return r * 128 + ((ch ^ (r & 7)) << 4); }

template <int DH>
__global__ void __launch_bounds__(kFaThreads, 1)
    ssd_prefill_attn_kernel(const float* __restrict__ q, int q_stride, const float* __restrict__ k_cache,
                            const float* __restrict__ v_cache, float* __restrict__ o, int o_stride, int P,
                            int max_seq, float scale, DevState* st) {
  using S = FaSmem<DH>;
  extern __shared__ __align__(1024) uint8_t fa_raw[];
  const uint32_t raw = smem_u32(fa_raw);
  uint8_t* smem = fa_raw + (((raw + 1023u) & ~1023u) - raw);
  uint64_t* bar_ld = reinterpret_cast<uint64_t*>(smem + S::kBar);
  uint64_t* bar_mma = bar_ld + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + S::kTmemSlot);
  const float* stk = reinterpret_cast<const float*>(smem + S::kStK);
  const float* stv = reinterpret_cast<const float*>(smem + S::kStV);
  const int nqb = gridDim.x, qb = nqb - 1 - static_cast<int>(blockIdx.x), h = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q0 = qb * kFaQ;
  const int n_keys = min(q0 + kFaQ, P);  // keys 0 .. n_keys - 1 reach some row of the block
  const int n_kb = (n_keys + kFaK - 1) / kFaK;
  const float* kh = k_cache + static_cast<size_t>(h) * max_seq * DH;
  const float* vh = v_cache + static_cast<size_t>(h) * max_seq * DH;

  pdl_trigger();
  if (tid == 0) {
    mbar_init(bar_ld, 1);
    mbar_init(bar_mma, 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kFaTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();  // q, K and V come from the upstream projection

  // block kb's K and V rows (the keys below P) into the staging buffer
  auto issue = [&](int kb) {
    const int j0 = kb * kFaK, nk = min(kFaK, n_keys - j0);
    const uint32_t bytes = static_cast<uint32_t>(nk * DH * 4);
    mbar_arrive_expect_tx(bar_ld, 2 * bytes);
    bulk_load(smem + S::kStK, kh + static_cast<size_t>(j0) * DH, bytes, bar_ld);
    bulk_load(smem + S::kStV, vh + static_cast<size_t>(j0) * DH, bytes, bar_ld);
  };
  int pending = -1;  // thread 0: the block whose staging copy has not been waited for
  if (tid == 0) {
    issue(0);
    pending = 0;
  }

  // Q block -> hi / lo (rows past P are zero)
  for (int t = tid; t < kFaQ * (DH / 8); t += kFaThreads) {
    const int r = t / (DH / 8), c8 = t - r * (DH / 8);
    float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (q0 + r < P) {
      const float4* src = reinterpret_cast<const float4*>(q + static_cast<size_t>(q0 + r) * q_stride + h * DH + c8 * 8);
      const float4 a = __ldcg(src), b = __ldcg(src + 1);
      v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
    uint4 hi, lo;
    split8_bf16(v, hi, lo);
    const int off = (c8 >> 3) * S::kQAtom + sw128_off(r, c8 & 7);
    *reinterpret_cast<uint4*>(smem + S::kQh + off) = hi;
    *reinterpret_cast<uint4*>(smem + S::kQl + off) = lo;
  }

  const int row = (warp & 3) * 32 + lane;  // softmax threads (warps 0..3): query row = TMEM lane
  const int qi = q0 + row;
  float m_run = -INFINITY, l_run = 0.f;
  float acc[DH];
#pragma unroll
  for (int d = 0; d < DH; ++d) acc[d] = 0.f;
  bool ok = true;
  uint32_t mma_phase = 0;
  constexpr uint32_t idesc_s = umma_idesc_bf16(kFaQ, kFaK);
  constexpr uint32_t idesc_o = umma_idesc_bf16(kFaQ, DH);

  for (int kb = 0; kb < n_kb; ++kb) {
    const int j0 = kb * kFaK, nk = min(kFaK, n_keys - j0);
    // ---- the block's K and V: staging -> bf16 hi / lo operands (keys past nk are zero)
    if (ok && !mbar_wait(bar_ld, static_cast<uint32_t>(kb) & 1u)) ok = false;
    if (ok && tid == 0) pending = -1;
    for (int t = tid; t < kFaK * (DH / 8); t += kFaThreads) {  // K: rows = keys
      const int j = t / (DH / 8), c8 = t - j * (DH / 8);
      float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      if (j < nk) {
        const float4 a = *reinterpret_cast<const float4*>(stk + j * DH + c8 * 8);
        const float4 b = *reinterpret_cast<const float4*>(stk + j * DH + c8 * 8 + 4);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
      }
      uint4 hi, lo;
      split8_bf16(v, hi, lo);
      const int off = (c8 >> 3) * S::kKAtom + sw128_off(j, c8 & 7);
      *reinterpret_cast<uint4*>(smem + S::kKh + off) = hi;
      *reinterpret_cast<uint4*>(smem + S::kKl + off) = lo;
    }
    for (int t = tid; t < DH * (kFaK / 8); t += kFaThreads) {  // V^T: rows = dimensions, keys along K
      const int c8 = t / DH, d = t - c8 * DH;
      float v[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = (c8 * 8 + e < nk) ? stv[(c8 * 8 + e) * DH + d] : 0.f;
      uint4 hi, lo;
      split8_bf16(v, hi, lo);
      const int off = sw128_off(d, c8);
      *reinterpret_cast<uint4*>(smem + S::kVh + off) = hi;
      *reinterpret_cast<uint4*>(smem + S::kVl + off) = lo;
    }
    fence_proxy_async_smem();
    if (!__syncthreads_and(ok)) {
      ok = false;
      break;
    }
    if (tid == 0) {
      if (kb + 1 < n_kb) {  // the staging buffer is free: the next block's rows go out now
        issue(kb + 1);
        pending = kb + 1;
      }
      // ---- S = Q K^T
      tmem_fence_after();
#pragma unroll
      for (int kk = 0; kk < DH / 16; ++kk) {
        const int at = kk >> 2, sub = 2 * (kk & 3);
        const uint64_t qh = umma_desc_sw128(smem_u32(smem + S::kQh + at * S::kQAtom)) + sub;
        const uint64_t ql = umma_desc_sw128(smem_u32(smem + S::kQl + at * S::kQAtom)) + sub;
        const uint64_t kh_ = umma_desc_sw128(smem_u32(smem + S::kKh + at * S::kKAtom)) + sub;
        const uint64_t kl_ = umma_desc_sw128(smem_u32(smem + S::kKl + at * S::kKAtom)) + sub;
        umma_f16(tmem, qh, kh_, idesc_s, kk > 0 ? 1u : 0u);
        umma_f16(tmem, qh, kl_, idesc_s, 1u);
        umma_f16(tmem, ql, kh_, idesc_s, 1u);
      }
      umma_commit(bar_mma);
    }
    // ---- softmax of the block's scores, one row per thread of warps 0..3
    if (ok && !mbar_wait(bar_mma, mma_phase)) ok = false;
    mma_phase ^= 1u;
    tmem_fence_after();
    float alpha = 1.f;
    if (warp < 4) {
      const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
      float sv[32];
      float bm = -INFINITY;
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        tmem_ld32(trow + half * 32, sv);
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const int kj = j0 + half * 32 + c;
          if (kj <= qi && kj < P) bm = fmaxf(bm, sv[c] * scale);
        }
      }
      const float m_new = fmaxf(m_run, bm);
      alpha = m_run == -INFINITY ? 0.f : expf(m_run - m_new);
      float ls = 0.f;
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        tmem_ld32(trow + half * 32, sv);
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const int kj = j0 + half * 32 + c;
          sv[c] = (kj <= qi && kj < P) ? expf(sv[c] * scale - m_new) : 0.f;
          ls += sv[c];
        }
#pragma unroll
        for (int c8 = 0; c8 < 4; ++c8) {
          uint4 hi, lo;
          split8_bf16(sv + 8 * c8, hi, lo);
          const int off = sw128_off(row, half * 4 + c8);
          *reinterpret_cast<uint4*>(smem + S::kPh + off) = hi;
          *reinterpret_cast<uint4*>(smem + S::kPl + off) = lo;
        }
      }
      l_run = l_run * alpha + ls;
      m_run = m_new;
    }
    tmem_fence_before();
    fence_proxy_async_smem();
    if (!__syncthreads_and(ok)) {
      ok = false;
      break;
    }
    if (tid == 0) {
      // ---- O_blk = P V
      tmem_fence_after();
#pragma unroll
      for (int kk = 0; kk < kFaK / 16; ++kk) {
        const uint64_t ph = umma_desc_sw128(smem_u32(smem + S::kPh)) + 2 * kk;
        const uint64_t pl = umma_desc_sw128(smem_u32(smem + S::kPl)) + 2 * kk;
        const uint64_t vh_ = umma_desc_sw128(smem_u32(smem + S::kVh)) + 2 * kk;
        const uint64_t vl_ = umma_desc_sw128(smem_u32(smem + S::kVl)) + 2 * kk;
        umma_f16(tmem + kFaK, ph, vh_, idesc_o, kk > 0 ? 1u : 0u);
        umma_f16(tmem + kFaK, ph, vl_, idesc_o, 1u);
        umma_f16(tmem + kFaK, pl, vh_, idesc_o, 1u);
      }
      umma_commit(bar_mma);
    }
    if (ok && !mbar_wait(bar_mma, mma_phase)) ok = false;
    mma_phase ^= 1u;
    tmem_fence_after();
    if (warp < 4) {
      const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16) + kFaK;
#pragma unroll
      for (int c = 0; c < DH / 32; ++c) {
        float ov[32];
        tmem_ld32(trow + c * 32, ov);
#pragma unroll
        for (int e = 0; e < 32; ++e) acc[c * 32 + e] = fmaf(acc[c * 32 + e], alpha, ov[e]);
      }
    }
    tmem_fence_before();
    if (!__syncthreads_and(ok)) {  // the operands and the accumulators are free for the next block
      ok = false;
      break;
    }
  }
  if (!ok && tid == 0) {
    set_error(st, DERR_TIMEOUT);
    if (pending >= 0)  // a staging copy may still be landing: a bounded wait before the CTA leaves
      mbar_wait_for(bar_ld, static_cast<uint32_t>(pending) & 1u, 100000000ull);
  }
  if (warp < 4 && qi < P && ok) {
    const float inv = 1.0f / l_run;
    float4* orow = reinterpret_cast<float4*>(o + static_cast<size_t>(qi) * o_stride + h * DH);
#pragma unroll
    for (int d4 = 0; d4 < DH / 4; ++d4)
      orow[d4] = make_float4(acc[4 * d4] * inv, acc[4 * d4 + 1] * inv, acc[4 * d4 + 2] * inv, acc[4 * d4 + 3] * inv);
  }
  tmem_fence_before();
  __syncthreads();
  if (warp == 0) {
    tmem_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kFaTmemCols) : "memory");
  }
}

}  // namespace ssd
