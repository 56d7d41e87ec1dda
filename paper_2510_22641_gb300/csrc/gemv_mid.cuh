// Medium-M weight-streaming GEMM on the 5th-generation tensor cores: the
// verification pass of batched requests, M = 17..128 activation rows.
//
//   out[m][n] = sum_k W[n][k] * a[m][k],   W bf16 [N][K] (nn.Linear layout), a fp32
//
// In the serving form of Algorithm 1 every request of a batch verifies its
// gamma + 1 rows in the same full-depth pass, so one projection carries
// B * (gamma + 1) rows (112 for 16 requests at gamma = 6).  Each weight byte now
// meets up to 128 rows: a real dense contraction, still bound by the weight
// stream.  The kernel keeps ssd_wstream_kernel's stream-K unit partition (units of
// 128 weight rows x 64 columns, contiguous CTA ranges, split row tiles summed in
// CTA order by the CTA that takes the tile's last ticket), its MMA orientation
// (the weight unit is A, M = 128; the activations are B) and its fused epilogues,
// and changes what the row count makes expensive:
//  * the B operand is no longer converted inside every CTA: ssd_split_act_kernel
//    turns the M rows into bf16 hi + lo parts once per projection (RMSNorm gain
//    folded in, exactly as the GEMV's converter warps do) and computes the rows'
//    RMSNorm scales; warp 0 TMA-loads the parts as 128-byte swizzled [NP][64]
//    tiles beside each weight unit (NP = M rounded up to 16 is the MMA's N);
//  * one CTA per SM; the weight units stream through an 8-stage ring of 16 KB fed by warp 0
//    (issued ahead of the upstream wait), the B tiles through a 3-stage ring of
//    2 x NP x 128 B fed by warp 6, so the weight stream keeps 8 units in flight
//    whatever the B ring holds;
//  * one MMA of N = 2 NP per 16-column K slice takes a stage's hi rows and the
//    lo rows stored right after them, so a row tile's accumulator is 2 NP TMEM
//    columns (two buffers of up to 256), the hi products in the first NP and the
//    lo products in the last NP; warps 2..5 read back 16 columns -- 16
//    activation rows -- of each half at a time and store their sum as the CTA's
//    partial of that tile;
//  * the reduction and the fused epilogue run in a second kernel,
//    ssd_mid_reduce_kernel, one CTA per (row tile, 16-row chunk): a tile's 112
//    rows are finished by 7 CTAs at once instead of one CTA's 128 threads after
//    the stream (measured: about 3 us per 16-row chunk, which made the serial
//    tail as long as the stream itself).
// The per-element arithmetic is the GEMV's up to rounding order: a = hi + lo,
// fp32 accumulation, the RMSNorm scale applied after the products, and the
// split-tile sums in CTA order; the hi and lo products accumulate separately
// over a CTA's K range and are added at the drain.  The grid is its own (one CTA
// per SM), so the split points differ from the GEMV's too: a row through this
// kernel equals the same row through the GEMV up to rounding, and every row is
// still independent of the launch's other rows.
#pragma once

#include "gemv.cuh"

namespace ssd {

constexpr int kMidWStages = 8;      // weight ring
constexpr int kMidBStages = 3;      // activation (B) ring
constexpr int kMidCtasPerSm = 1;
constexpr int kMidThreads = 224;    // warp 0 weight TMA, warp 1 MMA + TMEM, warps 2..5 drain, warp 6 B TMA
constexpr int kMidTmemCols = 512;   // two accumulators of up to 256 columns (hi rows, then lo rows)
constexpr uint32_t kMidBBytes = kMaxMidRows * kTileK * 2;  // one B part (hi or lo) of up to 128 rows: 16 KB
constexpr int kMidSlot = kMaxMidRows * kTileN;             // floats of one partial row tile, [m][128]

struct MidSmem {
  static constexpr int kW = 0;                                  // [wstages][16 KB] weight units
  // [bstages][2 NP][64] bf16: a stage holds the NP hi rows, then the NP lo rows right after them,
  // so one MMA of N = 2 NP takes both parts
  static constexpr int kB = kW + kMidWStages * kWTileBytes;
  static constexpr int kBar = kB + kMidBStages * 2 * kMidBBytes;  // wfull, wempty [wstages]; bfull, bempty [bstages]; afull, aempty [2]
  static constexpr int kTmemSlot = kBar + (2 * kMidWStages + 2 * kMidBStages + 4) * 8;
  static constexpr int kTotal = kTmemSlot + 16 + 1024;          // + slack for the 1024-byte alignment
};

// ------------------------------------------------------------------ activation split
// Row r of hi / lo (bf16 [rows][ld]) = the split of x[r] * gain (gain null: x[r]): v = x * g,
// hi = bf16(v), lo = bf16(v - hi); rs[r] = 1/sqrt(mean(x[r]^2) + eps) with gain, 1 without.
// 128 threads per row and the same summation order as the GEMV's drain warps, so the scale is
// bitwise the one the GEMV computes for the row.
__global__ void __launch_bounds__(kDrainThreads) ssd_split_act_kernel(const float* __restrict__ x, int x_stride,
                                                                      int K, const __nv_bfloat16* __restrict__ gain,
                                                                      float eps, __nv_bfloat16* __restrict__ hi,
                                                                      __nv_bfloat16* __restrict__ lo, int ld,
                                                                      float* __restrict__ rs) {
  __shared__ float red[4];
  pdl_trigger();
  pdl_wait();
  const int r = blockIdx.x, t = threadIdx.x, lane = t & 31;
  const float* xr = x + static_cast<size_t>(r) * x_stride;
  if (gain) {
    float ss = 0.f;
    for (int i = t; i < (K >> 2); i += kDrainThreads) {
      const float4 v = __ldcg(reinterpret_cast<const float4*>(xr) + i);
      ss = fmaf(v.x, v.x, ss);
      ss = fmaf(v.y, v.y, ss);
      ss = fmaf(v.z, v.z, ss);
      ss = fmaf(v.w, v.w, ss);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    if (lane == 0) red[t >> 5] = ss;
    __syncthreads();
    if (t == 0) {
      float s = 0.f;
      for (int w = 0; w < 4; ++w) s += red[w];
      rs[r] = rsqrtf(s / static_cast<float>(K) + eps);
    }
  } else if (t == 0) {
    rs[r] = 1.0f;
  }
  __nv_bfloat16* hr = hi + static_cast<size_t>(r) * ld;
  __nv_bfloat16* lr = lo + static_cast<size_t>(r) * ld;
  for (int i = t; i < (K >> 3); i += kDrainThreads) {
    const float4 a0 = __ldcg(reinterpret_cast<const float4*>(xr) + 2 * i);
    const float4 a1 = __ldcg(reinterpret_cast<const float4*>(xr) + 2 * i + 1);
    float v[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
    if (gain) {
      const uint4 gv = __ldg(reinterpret_cast<const uint4*>(gain) + i);
      const float2 g0 = bf16x2_to_float2(gv.x), g1 = bf16x2_to_float2(gv.y), g2 = bf16x2_to_float2(gv.z),
                   g3 = bf16x2_to_float2(gv.w);
      v[0] *= g0.x; v[1] *= g0.y; v[2] *= g1.x; v[3] *= g1.y;
      v[4] *= g2.x; v[5] *= g2.y; v[6] *= g3.x; v[7] *= g3.y;
    }
    uint32_t hw[4], lw[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const __nv_bfloat16 h0 = __float2bfloat16_rn(v[2 * e]), h1 = __float2bfloat16_rn(v[2 * e + 1]);
      const __nv_bfloat16 l0 = __float2bfloat16_rn(v[2 * e] - __bfloat162float(h0));
      const __nv_bfloat16 l1 = __float2bfloat16_rn(v[2 * e + 1] - __bfloat162float(h1));
      hw[e] = pack_bf16x2(h0, h1);
      lw[e] = pack_bf16x2(l0, l1);
    }
    reinterpret_cast<uint4*>(hr)[i] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    reinterpret_cast<uint4*>(lr)[i] = make_uint4(lw[0], lw[1], lw[2], lw[3]);
  }
}

// ------------------------------------------------------------------ kernel
// map0..2: the site's weight matrices (as for ssd_wstream_kernel); map_hi / map_lo: the split
// activations [128][K] with [NP][64] boxes.  M rows, NP = M rounded up to 16.
template <Epi EPI>
__global__ void __launch_bounds__(kMidThreads, kMidCtasPerSm)
    ssd_wstream_mid_kernel(const __grid_constant__ CUtensorMap map0, const __grid_constant__ CUtensorMap map1,
                           const __grid_constant__ CUtensorMap map2, const __grid_constant__ CUtensorMap map_hi,
                           const __grid_constant__ CUtensorMap map_lo, const GemvParams p, int M) {
  using S = MidSmem;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  uint64_t* wfull = reinterpret_cast<uint64_t*>(smem + S::kBar);
  uint64_t* wempty = wfull + kMidWStages;
  uint64_t* bfull = wempty + kMidWStages;
  uint64_t* bempty = bfull + kMidBStages;
  uint64_t* afull = bempty + kMidBStages;
  uint64_t* aempty = afull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + S::kTmemSlot);

  const int G = gridDim.x, c = blockIdx.x;
  const int u0 = unit_begin(c, p.units, G), u1 = unit_begin(c + 1, p.units, G);
  const int n_units = u1 - u0;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int NP = (M + 15) & ~15;

  if (!p.late_trigger) pdl_trigger();
  if (*reinterpret_cast<volatile int*>(&p.st->error) & DERR_TIMEOUT) return;

  if (tid == 0) {
    for (int s = 0; s < kMidWStages; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], 1);
    }
    for (int s = 0; s < kMidBStages; ++s) {
      mbar_init(&bfull[s], 1);
      mbar_init(&bempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&afull[b], 1);
      mbar_init(&aempty[b], 4);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kMidTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- weight TMA producer
    if (lane == 0) {
      auto issue_weights = [&](int s, int u) {
        const int rt = u / p.n_kt, kt = u - rt * p.n_kt;
        uint8_t* wdst = smem + S::kW + s * kWTileBytes;
        const int x = kt * kTileK;
        mbar_arrive_expect_tx(&wfull[s], kWTileBytes);
        if constexpr (EPI == Epi::GATE_SILU) {
          tma_load_2d(wdst, &map0, &wfull[s], x, rt * kHalfN);
          tma_load_2d(wdst + kWTileBytes / 2, &map1, &wfull[s], x, rt * kHalfN);
        } else if constexpr (EPI == Epi::QKV) {
          const int r0 = rt * kTileN, mat = r0 / p.seg_rows;
          tma_load_2d(wdst, mat == 0 ? &map0 : (mat == 1 ? &map1 : &map2), &wfull[s], x, r0 - mat * p.seg_rows);
        } else {
          tma_load_2d(wdst, &map0, &wfull[s], x, rt * kTileN);
        }
      };
      prefetch_tensormap(&map0);
      // weights do not depend on the previous kernel: the first stages go out before its end
      int issued = 0;
      for (int i = 0; i < n_units; ++i, ++issued) {
        const int s = i % kMidWStages;
        if (i >= kMidWStages && !mbar_wait(&wempty[s], static_cast<uint32_t>((i / kMidWStages) - 1) & 1u)) {
          set_error(p.st, DERR_TIMEOUT);
          break;
        }
        issue_weights(s, u0 + i);
      }
      if (__ldcg(&p.st->error) & DERR_TIMEOUT) drain_ring(wfull, kMidWStages, issued);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(kTileN, 2 * NP);
      int sg = 0;
      bool seg_open = false;
      uint32_t d = tmem;
      for (int i = 0; i < n_units; ++i) {
        const int u = u0 + i, kt = u % p.n_kt, s = i % kMidWStages, sb = i % kMidBStages;
        if (!seg_open) {  // a new row-tile segment: take a free accumulator
          const int b = sg & 1;
          if (!mbar_wait(&aempty[b], static_cast<uint32_t>(((sg >> 1) & 1) ^ 1))) {
            set_error(p.st, DERR_TIMEOUT);
            break;
          }
          tmem_fence_after();
          d = tmem + static_cast<uint32_t>(b * 2 * kMaxMidRows);
        }
        if (!mbar_wait(&wfull[s], static_cast<uint32_t>(i / kMidWStages) & 1u) ||
            !mbar_wait(&bfull[sb], static_cast<uint32_t>(i / kMidBStages) & 1u)) {
          set_error(p.st, DERR_TIMEOUT);
          break;
        }
        tmem_fence_after();
        const uint64_t adesc = umma_desc_sw128(smem_u32(smem + S::kW + s * kWTileBytes));
        const uint64_t bdesc = umma_desc_sw128(smem_u32(smem + S::kB + sb * 2 * kMidBBytes));
#pragma unroll
        for (int kk = 0; kk < kTileK / 16; ++kk) {
          // +32 bytes (2 descriptor units) per 16-element K slice inside the swizzled row; columns
          // 0..NP-1 of the accumulator take the hi products, NP..2NP-1 the lo products
          umma_f16(d, adesc + 2 * kk, bdesc + 2 * kk, idesc, (seg_open || kk > 0) ? 1u : 0u);
          seg_open = true;
        }
        umma_commit(&wempty[s]);  // the stages may be refilled once these MMAs have read them
        umma_commit(&bempty[sb]);
        if (kt == p.n_kt - 1 || i == n_units - 1) {
          umma_commit(&afull[sg & 1]);  // the row tile's accumulator is complete
          ++sg;
          seg_open = false;
        }
      }
    }
  } else if (warp == 6) {
    // ---------------------------------------------------------------- B TMA producer (split activations)
    if (lane == 0) {
      const uint32_t bbytes = static_cast<uint32_t>(NP) * kTileK * 2;
      pdl_wait();  // the split kernel's rows
      if (p.late_trigger) pdl_trigger();
      int issued = 0;
      for (int i = 0; i < n_units; ++i, ++issued) {
        const int sb = i % kMidBStages;
        if (i >= kMidBStages && !mbar_wait(&bempty[sb], static_cast<uint32_t>((i / kMidBStages) - 1) & 1u)) {
          set_error(p.st, DERR_TIMEOUT);
          break;
        }
        const int x = ((u0 + i) % p.n_kt) * kTileK;
        mbar_arrive_expect_tx(&bfull[sb], 2 * bbytes);
        uint8_t* bdst = smem + S::kB + sb * 2 * kMidBBytes;
        tma_load_2d(bdst, &map_hi, &bfull[sb], x, 0);
        tma_load_2d(bdst + bbytes, &map_lo, &bfull[sb], x, 0);
      }
      if (__ldcg(&p.st->error) & DERR_TIMEOUT) drain_ring(bfull, kMidBStages, issued);
    }
  } else {
    // ---------------------------------------------------------------- drain (warps 2..5)
    // Every finished accumulator -- row tile rt's share of this CTA's unit range -- goes to
    // partial slot c + rt, 16 columns (activation rows) at a time, [m][128] fp32.  Along the
    // partition the pairs (CTA, tile) never decrease in either index, so c + rt is unique;
    // ssd_mid_reduce_kernel sums each tile's slots in CTA order and runs the epilogue.
    const int q = warp & 3;  // TMEM lane quadrant: tile rows 32q .. 32q+31
    const int n_ch = (M + kNPad - 1) / kNPad;
    int sg = 0;
    for (int i = 0; i < n_units; ++i) {
      const int u = u0 + i, rt = u / p.n_kt, kt = u - rt * p.n_kt;
      if (!(kt == p.n_kt - 1 || i == n_units - 1)) continue;
      const int b = sg & 1;
      if (!mbar_wait(&afull[b], static_cast<uint32_t>((sg >> 1) & 1))) {
        set_error(p.st, DERR_TIMEOUT);
        break;
      }
      tmem_fence_after();
      const uint32_t tbase =
          tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(b * 2 * kMaxMidRows);
      float* dstp = p.partials + static_cast<size_t>(c + rt) * kMidSlot;
      for (int ch = 0; ch < n_ch; ++ch) {
        float v[kNPad], vl[kNPad];
        tmem_ld16(tbase + ch * kNPad, v);
        tmem_ld16(tbase + NP + ch * kNPad, vl);
#pragma unroll
        for (int m = 0; m < kNPad; ++m)
          if (ch * kNPad + m < M) __stcg(dstp + (ch * kNPad + m) * kTileN + q * 32 + lane, v[m] + vl[m]);
      }
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&aempty[b]);  // the MMA warp may reuse accumulator b
      ++sg;
    }
  }
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kMidTmemCols) : "memory");
  }
}

// ------------------------------------------------------------------ reduction + epilogue
// One CTA per (16-row chunk ch = blockIdx.x, row tile rt = blockIdx.y) of a medium-M projection
// streamed by `G = p.grid_ctas` CTAs: sums the tile's partials (slots c + rt for the CTAs c that
// held its units) in CTA order, then applies the RMSNorm scale and the fused epilogue to rows
// 16 ch .. 16 ch + 15 -- the GEMV's epilogue code, with its inputs (rotation table rows, residual
// base rows) loaded up front.  The LM head's argmax keys of a chunk are finished by the last of
// the chunk's n_rt CTAs.
template <Epi EPI>
__global__ void __launch_bounds__(kDrainThreads) ssd_mid_reduce_kernel(const GemvParams p, int M) {
  __shared__ __align__(16) float outb[kNPad * kTileN];
  __shared__ __align__(16) float pre[kNPad * kTileN];  // QKV: [16][head_dim / 2] float2; RESID: [16][128]
  __shared__ float rs[kNPad];
  __shared__ int rmap[2 * kMaxMidRows];                // positions, requests of all M rows
  const int ch = blockIdx.x, rt = blockIdx.y, tid = threadIdx.x;
  const int m0 = ch * kNPad, mc = min(kNPad, M - m0);
  const int G = p.grid_ctas;
  pdl_trigger();
  pdl_wait();
  if (__ldcg(&p.st->error) & DERR_TIMEOUT) return;  // the stream gave up: partials are incomplete
  const int base_pos = (p.abs_pos || p.batch_rows ? 0 : __ldcg(&p.st->kv_len)) + p.pos_off;
  int* rpos = p.batch_rows ? rmap : nullptr;
  int* rreq = p.batch_rows ? rmap + kMaxMidRows : nullptr;
  if (rpos)
    for (int m = tid; m < M; m += kDrainThreads) {
      const int b = m / p.batch_rows;
      rreq[m] = b;
      rpos[m] = __ldcg(&p.req_st[b].kv_len) + batch_offset(p, m, b);
    }
  if (p.rs_parts) {
    // 1/rms from the producer's per-tile sums of squares: 8 lanes per row, lane l summing tiles
    // l, l + 8, ... (loads issued together), then a fixed xor tree over the 8 lanes
    static_assert(kDrainThreads == 8 * kNPad, "8 lanes per row");
    const int r = tid >> 3, l = tid & 7;
    const float* src = p.rs_parts + (m0 + r) * p.rs_nparts;
    float t = 0.f;
    if (r < mc)
      for (int i0 = l; i0 < p.rs_nparts; i0 += 64) {
        float v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) v[k] = i0 + 8 * k < p.rs_nparts ? __ldcg(src + i0 + 8 * k) : 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) t += v[k];
      }
#pragma unroll
    for (int off = 4; off > 0; off >>= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
    if (r < mc && l == 0) rs[r] = rsqrtf(t / static_cast<float>(p.K) + p.eps);
  } else if (tid < mc) {
    rs[tid] = p.rs_in ? __ldcg(p.rs_in + m0 + tid) : 1.0f;
  }
  __syncthreads();
  // epilogue inputs, all loads independent
  bool use_pre = false;
  if constexpr (EPI == Epi::QKV) {
    const int half = p.head_dim >> 1;
    use_pre = p.rope_cs != nullptr && (rt * kTileN) / p.seg_rows + p.seg_base < 2;
    if (use_pre)
      for (int t = tid; t < mc * half; t += kDrainThreads) {
        const int m = t / half, j = t - m * half;
        const int pos = rpos ? rpos[m0 + m] : base_pos + m0 + m;
        reinterpret_cast<float2*>(pre)[t] =
            (pos >= 0 && pos < p.max_seq) ? __ldg(p.rope_cs + static_cast<size_t>(pos) * half + j) : make_float2(1.f, 0.f);
      }
  } else if constexpr (EPI == Epi::RESID) {
    use_pre = true;
    for (int t = tid; t < mc * kTileN; t += kDrainThreads) {
      const int m = t / kTileN, n = rt * kTileN + (t - m * kTileN);
      pre[t] = n < p.N ? __ldcg(p.base + static_cast<size_t>(m0 + m) * p.base_stride + n) : 0.f;
    }
  }
  // the tile's partials in CTA order, four contributors' loads in flight per row slice
  const int c_first = unit_owner(rt * p.n_kt, p.units, G);
  const int c_last = unit_owner(rt * p.n_kt + p.n_kt - 1, p.units, G);
  const int nsp = c_last - c_first + 1;
  const float4* part = reinterpret_cast<const float4*>(p.partials);
  constexpr int kSlotF4 = kMidSlot / 4;
  const int nf = mc * (kTileN / 4), f0 = m0 * (kTileN / 4);
  for (int f = tid; f < nf; f += kDrainThreads) {
    float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k0 = 0; k0 < nsp; k0 += 4) {
      float4 pv[4];
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        pv[kk] = k0 + kk < nsp ? __ldcg(part + static_cast<size_t>(c_first + k0 + kk + rt) * kSlotF4 + f0 + f)
                               : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        if (k0 + kk >= nsp) break;
        if (k0 + kk == 0) {
          sum = pv[kk];
        } else {
          sum.x += pv[kk].x;
          sum.y += pv[kk].y;
          sum.z += pv[kk].z;
          sum.w += pv[kk].w;
        }
      }
    }
    reinterpret_cast<float4*>(outb)[f] = sum;
  }
  __syncthreads();
  gemv_epilogue<kNPad, EPI, true>(p, rt, outb, rs, use_pre ? pre : nullptr, base_pos, rpos, rreq, tid, m0, mc);
  if constexpr (EPI == Epi::ARGMAX) gemv_argmax_finish(p, rreq, tid, p.n_rt, m0, mc);
}

}  // namespace ssd
