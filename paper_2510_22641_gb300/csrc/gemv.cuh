// Weight-streaming skinny GEMM ("GEMV" for M = 1..kMaxRows activation rows).
//
//   out[m][n] = sum_k W[n][k] * a[m][k],   W bf16 [N][K] (nn.Linear layout), a fp32
//
// Every decode-time projection of the decoder (Sec. "SSD Setup for VLMs",
// x_{l+1} = x_l + f_l(x_l)), of the imitation network and of the LM head g
// runs through this kernel; at batch 1 it is bound by HBM bandwidth, since each
// weight byte is used for M <= 9 rows only.
//
// Design (sm_103a):
//  * persistent grid of min(#SMs, units) CTAs; the weight matrix is cut into
//    units of 128 rows x 64 columns (16 KB of bf16) and CTA c streams the
//    contiguous unit range [c*U/G, (c+1)*U/G) -- stream-K, so every SM moves
//    the same number of bytes whatever N and K are;
//  * thread 0 issues 2D TMA loads of the weight units (and 1D bulk copies of
//    the matching 64-column slice of each activation row and of the RMSNorm
//    gain) into a 5-stage shared-memory ring guarded by mbarriers; weight
//    loads for the first stages are issued before griddepcontrol.wait, so they
//    overlap the tail of the previous kernel (programmatic dependent launch);
//    a stage is refilled as soon as all eight warps have released it;
//  * eight warps read the tile with 128-bit shared loads and accumulate in
//    fp32 with packed FFMA2 (__ffma2_rn); activations stay fp32; with 256
//    threads and two CTAs per SM every thread may hold 128 registers;
//  * a row tile split across CTAs is reduced from a workspace in fixed CTA
//    order by the CTA that finishes it last (atomic ticket, no spinning);
//  * the fused epilogue applies the RMSNorm scale and then RoPE + KV-cache
//    write (QKV), SiLU(gate)*up, SiLU, a scaled residual add, or the LM-head
//    argmax.
//
// Batch invariance: the unit partition, the order of FMAs feeding each output
// and the reduction trees do not depend on M, so row m of an M-row launch is
// bitwise equal to the same row computed alone.  This makes the verify pass
// (M = gamma+1) reproduce greedy decoding (M = 1) exactly.
#pragma once

#include "common.cuh"

namespace ssd {

constexpr int kTileN = 128;          // weight rows per unit
constexpr int kTileK = 64;           // weight columns per unit (128 bytes of bf16)
constexpr int kConsumerWarps = 8;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kGemvThreads = kConsumerThreads;
constexpr int kStages = 5;
constexpr uint32_t kWTileBytes = kTileN * kTileK * 2;

enum class Epi : int { QKV = 0, GATE_SILU = 1, SILU = 2, RESID = 3, ARGMAX = 4 };

struct GemvParams {
  int K, n_kt, n_rt, units;
  int N;           // valid output rows (GATE_SILU: d_ff; tiles hold 64 gate + 64 up rows)
  int seg_rows;    // QKV: rows per source matrix (q, k, v)
  const float* x;  // activations [M][x_stride] (fp32)
  int x_stride;
  const __nv_bfloat16* gain;  // RMSNorm gain [K], or null (no norm)
  float eps;
  float* partials;      // [2 * grid][kMaxRows][kTileN]
  unsigned* counters;   // [n_rt]
  DevState* st;
  int pos_off;          // row m sits at position st->kv_len + pos_off + m
  // QKV
  float* q_out;
  int q_stride;
  __nv_bfloat16* k_cache;  // this layer's [H][max_seq][head_dim]
  __nv_bfloat16* v_cache;
  int head_dim, max_seq;
  const float2* rope_cs;   // [max_seq][head_dim/2] (cos, sin)
  // GATE_SILU / SILU
  float* h_out;
  int h_stride;
  // RESID: dst[m][n] = base[m][n] + (*scale) * out[m][n]
  const float* base;
  int base_stride;
  float* dst;
  int dst_stride;
  const float* scale;
  // ARGMAX
  int* tok_dst;        // tok_dst[m] = argmax of row m
  float* logits;       // optional [logits_rows][N] capture
  int logits_rows;
};

template <int M>
struct GemvSmem {
  static constexpr int kActBytes = M * kTileK * 4;
  static constexpr int kW = 0;
  static constexpr int kA = kW + kStages * kWTileBytes;
  static constexpr int kG = kA + kStages * kActBytes;
  static constexpr int kOut = kG + kStages * kTileK * 2;
  static constexpr int kRs = kOut + M * kTileN * 4;
  static constexpr int kRed = kRs + kMaxRows * 4;
  static constexpr int kFlag = kRed + kConsumerWarps * kMaxRows * 4;
  static constexpr int kBar = (kFlag + 16 + 7) & ~7;
  static constexpr int kTotal = kBar + 2 * kStages * 8;
};

// Which CTA of a G-CTA grid owns unit u (ranges [floor(cU/G), floor((c+1)U/G))).
__device__ __forceinline__ int unit_owner(int u, int units, int G) {
  return static_cast<int>((static_cast<long long>(u + 1) * G - 1) / units);
}
__device__ __forceinline__ int unit_begin(int c, int units, int G) {
  return static_cast<int>((static_cast<long long>(c) * units) / G);
}

// ------------------------------------------------------------------ epilogues
// All run on the 256 consumer threads with the finished row tile in out_s
// ([M][kTileN], fp32, before the RMSNorm scale) and rs[m] (1 if no norm).

template <int M, Epi EPI>
__device__ __forceinline__ void gemv_epilogue(const GemvParams& p, int rt, const float* out_s, const float* rs,
                                              int tid) {
  if constexpr (EPI == Epi::QKV) {
    const int r0 = rt * kTileN;
    const int mat = r0 / p.seg_rows;  // 0 = q, 1 = k, 2 = v
    const int local0 = r0 - mat * p.seg_rows;
    const int Dh = p.head_dim, half = Dh >> 1;
    const int base_pos = __ldcg(&p.st->kv_len) + p.pos_off;
    if (mat < 2) {
      for (int idx = tid; idx < M * (kTileN / 2); idx += kConsumerThreads) {
        const int m = idx / (kTileN / 2), pr = idx - m * (kTileN / 2);
        const int hh = pr / half, j = pr - hh * half;
        const int ra = hh * Dh + j, rb = ra + half;
        const int pos = base_pos + m;
        if (pos < 0 || pos >= p.max_seq) {
          set_error(p.st, DERR_POS);
          continue;
        }
        const float a = out_s[m * kTileN + ra] * rs[m];
        const float b = out_s[m * kTileN + rb] * rs[m];
        const float2 cs = p.rope_cs[static_cast<size_t>(pos) * half + j];
        const float va = a * cs.x - b * cs.y;
        const float vb = a * cs.y + b * cs.x;
        if (mat == 0) {
          p.q_out[m * p.q_stride + local0 + ra] = va;
          p.q_out[m * p.q_stride + local0 + rb] = vb;
        } else {
          const int h = local0 / Dh + hh;
          __nv_bfloat16* kr = p.k_cache + (static_cast<size_t>(h) * p.max_seq + pos) * Dh;
          kr[j] = __float2bfloat16_rn(va);
          kr[j + half] = __float2bfloat16_rn(vb);
        }
      }
    } else {
      for (int idx = tid; idx < M * kTileN; idx += kConsumerThreads) {
        const int m = idx / kTileN, i = idx - m * kTileN;
        const int pos = base_pos + m;
        if (pos < 0 || pos >= p.max_seq) {
          set_error(p.st, DERR_POS);
          continue;
        }
        const int row = local0 + i, h = row / Dh, d = row - h * Dh;
        p.v_cache[(static_cast<size_t>(h) * p.max_seq + pos) * Dh + d] =
            __float2bfloat16_rn(out_s[idx] * rs[m]);
      }
    }
  } else if constexpr (EPI == Epi::GATE_SILU) {
    for (int idx = tid; idx < M * (kTileN / 2); idx += kConsumerThreads) {
      const int m = idx / (kTileN / 2), j = idx - m * (kTileN / 2);
      const int n = rt * (kTileN / 2) + j;
      if (n >= p.N) continue;
      const float g = out_s[m * kTileN + j] * rs[m];
      const float u = out_s[m * kTileN + (kTileN / 2) + j] * rs[m];
      p.h_out[m * p.h_stride + n] = silu_f(g) * u;
    }
  } else if constexpr (EPI == Epi::SILU) {
    for (int idx = tid; idx < M * kTileN; idx += kConsumerThreads) {
      const int m = idx / kTileN, i = idx - m * kTileN;
      const int n = rt * kTileN + i;
      if (n >= p.N) continue;
      p.h_out[m * p.h_stride + n] = silu_f(out_s[idx] * rs[m]);
    }
  } else if constexpr (EPI == Epi::RESID) {
    const float s = __ldg(p.scale);
    for (int idx = tid; idx < M * kTileN; idx += kConsumerThreads) {
      const int m = idx / kTileN, i = idx - m * kTileN;
      const int n = rt * kTileN + i;
      if (n >= p.N) continue;
      const float b = __ldcg(p.base + m * p.base_stride + n);
      p.dst[m * p.dst_stride + n] = b + s * (out_s[idx] * rs[m]);
    }
  } else {  // ARGMAX (LM head): argmax over the vocabulary, lowest index on ties
    const int lane = tid & 31;
    const int base_pos = __ldcg(&p.st->kv_len) + p.pos_off;
    const int P = __ldcg(&p.st->prompt_len);
    if (tid < kTileN) {
      const int n = rt * kTileN + tid;
      const bool valid = n < p.N;
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const float logit = out_s[m * kTileN + tid] * rs[m];
        if (p.logits != nullptr && valid) {
          const int row = base_pos + m + 1 - P;
          if (row >= 0 && row < p.logits_rows) p.logits[static_cast<size_t>(row) * p.N + n] = logit;
        }
        unsigned long long key = valid ? argmax_key(logit, static_cast<uint32_t>(n)) : 0ull;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const unsigned long long o = __shfl_xor_sync(0xffffffffu, key, off);
          key = o > key ? o : key;
        }
        if (lane == 0) atomicMax(&p.st->am_key[m], key);
      }
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) {
      const unsigned prev = atomicAdd(&p.st->am_count, 1u);
      if (prev == static_cast<unsigned>(p.n_rt - 1)) {
        __threadfence();
        for (int m = 0; m < M; ++m) {
          const unsigned long long key = atomicExch(&p.st->am_key[m], 0ull);
          p.tok_dst[m] = static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull));
        }
        atomicExch(&p.st->am_count, 0u);
      }
    }
  }
}

// ------------------------------------------------------------------ kernel

template <int M, Epi EPI>
__global__ void __launch_bounds__(kGemvThreads, (M <= 6 ? 2 : 1))
    gemv_kernel(const __grid_constant__ CUtensorMap map0, const __grid_constant__ CUtensorMap map1,
                const __grid_constant__ CUtensorMap map2, const GemvParams p) {
  using S = GemvSmem<M>;
  extern __shared__ __align__(128) uint8_t smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBar);
  uint64_t* empty = full + kStages;
  float* out_s = reinterpret_cast<float*>(smem + S::kOut);
  float* rs = reinterpret_cast<float*>(smem + S::kRs);
  float* red = reinterpret_cast<float*>(smem + S::kRed);
  int* flag = reinterpret_cast<int*>(smem + S::kFlag);

  const int G = gridDim.x, c = blockIdx.x;
  const int u0 = unit_begin(c, p.units, G), u1 = unit_begin(c + 1, p.units, G);
  const int n_units = u1 - u0;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rsub = lane >> 3, ch = lane & 7;
  const uint32_t tx = kWTileBytes + S::kActBytes + (p.gain ? kTileK * 2 : 0);

  // ---- producer helpers (thread 0 only)
  auto issue_weights = [&](int s, int u) {
    const int rt = u / p.n_kt, kt = u - rt * p.n_kt;
    uint8_t* wdst = smem + S::kW + s * kWTileBytes;
    if constexpr (EPI == Epi::GATE_SILU) {
      tma_load_2d(wdst, &map0, &full[s], kt * kTileK, rt * (kTileN / 2));
      tma_load_2d(wdst + kWTileBytes / 2, &map1, &full[s], kt * kTileK, rt * (kTileN / 2));
    } else if constexpr (EPI == Epi::QKV) {
      const int r0 = rt * kTileN, mat = r0 / p.seg_rows;
      const CUtensorMap* mp = mat == 0 ? &map0 : (mat == 1 ? &map1 : &map2);
      tma_load_2d(wdst, mp, &full[s], kt * kTileK, r0 - mat * p.seg_rows);
    } else {
      tma_load_2d(wdst, &map0, &full[s], kt * kTileK, rt * kTileN);
    }
    if (p.gain) bulk_load(smem + S::kG + s * kTileK * 2, p.gain + kt * kTileK, kTileK * 2, &full[s]);
  };
  auto issue_acts = [&](int s, int u) {
    const int kt = u % p.n_kt;
    uint8_t* adst = smem + S::kA + s * S::kActBytes;
#pragma unroll
    for (int m = 0; m < M; ++m)
      bulk_load(adst + m * kTileK * 4, p.x + static_cast<size_t>(m) * p.x_stride + kt * kTileK, kTileK * 4,
                &full[s]);
  };

  pdl_trigger();
  // After a timed-out wait anywhere in the decode, later kernels do nothing
  // (best-effort read before any copy is issued).
  if (*reinterpret_cast<volatile int*>(&p.st->error) & DERR_TIMEOUT) return;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kConsumerWarps);
    }
    flag[0] = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const int npre = n_units < kStages ? n_units : kStages;
  if (tid == 0) {
    prefetch_tensormap(&map0);
    // weights do not depend on the previous kernel: start streaming before the wait
    for (int i = 0; i < npre; ++i) {
      mbar_arrive_expect_tx(&full[i], tx);
      issue_weights(i, u0 + i);
    }
  }
  pdl_wait();  // activations, residuals and state are written by the previous kernel
  if (tid == 0)
    for (int i = 0; i < npre; ++i) issue_acts(i, u0 + i);

  // RMSNorm scale per row: rs[m] = 1/sqrt(mean(x^2) + eps), fixed reduction order.
  if (p.gain) {
#pragma unroll 1
    for (int m = 0; m < M; ++m) {
      const float4* xr = reinterpret_cast<const float4*>(p.x + static_cast<size_t>(m) * p.x_stride);
      float ss = 0.f;
      for (int i = tid; i < (p.K >> 2); i += kConsumerThreads) {
        const float4 v = __ldcg(xr + i);
        ss = fmaf(v.x, v.x, ss);
        ss = fmaf(v.y, v.y, ss);
        ss = fmaf(v.z, v.z, ss);
        ss = fmaf(v.w, v.w, ss);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
      if (lane == 0) red[warp * kMaxRows + m] = ss;
    }
    __syncthreads();
    if (tid < M) {
      float t = 0.f;
      for (int w = 0; w < kConsumerWarps; ++w) t += red[w * kMaxRows + tid];
      rs[tid] = rsqrtf(t / static_cast<float>(p.K) + p.eps);
    }
  } else if (tid < M) {
    rs[tid] = 1.0f;
  }
  __syncthreads();

  float2 acc[4][M];
#pragma unroll
  for (int j = 0; j < 4; ++j)
#pragma unroll
    for (int m = 0; m < M; ++m) acc[j][m] = make_float2(0.f, 0.f);

  const int rt_first = u0 / p.n_kt;
  int seg_kt0 = u0 - rt_first * p.n_kt;
  const uint8_t* wbase = smem + S::kW + (warp * 16 + rsub) * (kTileK * 2) + ch * 16;

  for (int i = 0; i < n_units; ++i) {
    const int u = u0 + i;
    const int rt = u / p.n_kt, kt = u - rt * p.n_kt;
    const int s = i % kStages;
    const uint32_t par = static_cast<uint32_t>(i / kStages) & 1u;
    if (!mbar_wait(&full[s], par)) {
      set_error(p.st, DERR_TIMEOUT);
      return;  // every warp times out on the same stage
    }
    // weights: rows 16w + rsub + 4j (j < 4), columns ch*8 .. ch*8+7 of the 128 x 64 unit
    uint4 wv[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      wv[j] = *reinterpret_cast<const uint4*>(wbase + s * kWTileBytes + j * 4 * (kTileK * 2));
    float2 gs[4];
    if (p.gain) {
      const uint4 gv = *reinterpret_cast<const uint4*>(smem + S::kG + s * kTileK * 2 + ch * 16);
      gs[0] = bf16x2_to_float2(gv.x);
      gs[1] = bf16x2_to_float2(gv.y);
      gs[2] = bf16x2_to_float2(gv.z);
      gs[3] = bf16x2_to_float2(gv.w);
    }
    float2 w2[4][4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      w2[j][0] = bf16x2_to_float2(wv[j].x);
      w2[j][1] = bf16x2_to_float2(wv[j].y);
      w2[j][2] = bf16x2_to_float2(wv[j].z);
      w2[j][3] = bf16x2_to_float2(wv[j].w);
    }
    const float* abase = reinterpret_cast<const float*>(smem + S::kA + s * S::kActBytes) + ch * 8;
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const float4 a0 = *reinterpret_cast<const float4*>(abase + m * kTileK);
      const float4 a1 = *reinterpret_cast<const float4*>(abase + m * kTileK + 4);
      float2 x2[4] = {make_float2(a0.x, a0.y), make_float2(a0.z, a0.w), make_float2(a1.x, a1.y),
                      make_float2(a1.z, a1.w)};
      if (p.gain) {
#pragma unroll
        for (int q = 0; q < 4; ++q) x2[q] = make_float2(x2[q].x * gs[q].x, x2[q].y * gs[q].y);
      }
#pragma unroll
      for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[j][m] = __ffma2_rn(w2[j][q], x2[q], acc[j][m]);
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);
    if (tid == 0 && i + kStages < n_units) {
      // refill this stage once every warp has released it
      if (!mbar_wait(&empty[s], par)) {
        set_error(p.st, DERR_TIMEOUT);
      } else {
        mbar_arrive_expect_tx(&full[s], tx);
        issue_weights(s, u + kStages);
        issue_acts(s, u + kStages);
      }
    }

    const bool seg_end = (kt == p.n_kt - 1) || (i == n_units - 1);
    if (!seg_end) continue;

    // ---- finish this row-tile segment: reduce over the 8 column lanes
#pragma unroll
    for (int j = 0; j < 4; ++j) {
#pragma unroll
      for (int m = 0; m < M; ++m) {
        float v = acc[j][m].x + acc[j][m].y;
        v += __shfl_xor_sync(0xffffffffu, v, 1);
        v += __shfl_xor_sync(0xffffffffu, v, 2);
        v += __shfl_xor_sync(0xffffffffu, v, 4);
        if (ch == 0) out_s[m * kTileN + warp * 16 + rsub + 4 * j] = v;
        acc[j][m] = make_float2(0.f, 0.f);
      }
    }
    __syncthreads();
    const bool whole = (seg_kt0 == 0) && (kt == p.n_kt - 1);
    if (whole) {
      gemv_epilogue<M, EPI>(p, rt, out_s, rs, tid);
    } else {
      const int slot = 2 * c + (rt == rt_first ? 0 : 1);
      float* dstp = p.partials + static_cast<size_t>(slot) * (kMaxRows * kTileN);
      for (int idx = tid; idx < M * kTileN; idx += kConsumerThreads) __stcg(dstp + idx, out_s[idx]);
      __threadfence();
      __syncthreads();
      const int c_first = unit_owner(rt * p.n_kt, p.units, G);
      const int c_last = unit_owner(rt * p.n_kt + p.n_kt - 1, p.units, G);
      if (tid == 0) {
        const unsigned prev = atomicAdd(&p.counters[rt], 1u);
        flag[0] = (prev == static_cast<unsigned>(c_last - c_first)) ? 1 : 0;
      }
      __syncthreads();
      if (flag[0]) {
        __threadfence();
        for (int idx = tid; idx < M * kTileN; idx += kConsumerThreads) {
          float sum = 0.f;
          for (int cc = c_first; cc <= c_last; ++cc) {
            const int rt_cc = unit_begin(cc, p.units, G) / p.n_kt;
            const int sl = 2 * cc + (rt == rt_cc ? 0 : 1);
            const float v = __ldcg(p.partials + static_cast<size_t>(sl) * (kMaxRows * kTileN) + idx);
            sum = (cc == c_first) ? v : sum + v;
          }
          out_s[idx] = sum;
        }
        __syncthreads();
        gemv_epilogue<M, EPI>(p, rt, out_s, rs, tid);
        if (tid == 0) p.counters[rt] = 0u;
      }
    }
    __syncthreads();
    seg_kt0 = 0;  // the next segment starts at a row-tile boundary
  }
}

}  // namespace ssd
