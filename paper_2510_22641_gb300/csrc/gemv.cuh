// Weight-streaming skinny GEMM ("GEMV" for M = 1..9 activation rows).
//
//   out[m][n] = sum_k W[n][k] * a[m][k],   W bf16 [N][K] (nn.Linear layout), a fp32
//
// Every decode-time projection of the decoder (Sec. "SSD Setup for VLMs",
// x_{l+1} = x_l + f_l(x_l)), of the imitation network and of the LM head g
// runs through this kernel; at batch 1 it is bound by HBM bandwidth, since each
// weight byte is used for M <= 9 rows only.
//
// Design (sm_103a):
//  * persistent grid of min(2 x #SMs, units) CTAs; the weight matrix is cut
//    into units of 32 rows x 256 columns (16 KB of bf16, 512-byte runs per row)
//    and CTA c streams the contiguous unit range [c*U/G, (c+1)*U/G) -- stream-K,
//    so every SM moves the same number of bytes whatever N and K are;
//  * thread 0 issues 2D TMA loads of the weight units (plus 1D bulk copies of
//    the matching 256-column slice of each activation row and of the RMSNorm
//    gain) into a 4-stage shared-memory ring guarded by mbarriers; the first
//    stages' weights are requested before griddepcontrol.wait, so they overlap
//    the previous kernel (programmatic dependent launch); a stage is refilled
//    as soon as its eight warps have released it;
//  * warp w owns rows 4w..4w+3 of the unit, lane l columns 8l..8l+7; weights
//    are read with 128-bit shared loads and accumulated in fp32 with packed
//    FFMA2 (__ffma2_rn); activations stay fp32;
//  * finished row tiles are parked in shared memory and their epilogues (and
//    the cross-CTA reduction of row tiles split between CTAs, in fixed CTA
//    order by the CTA that finishes last -- an atomic ticket, no spinning) run
//    after the stream, so the weight stream never pauses mid-kernel;
//  * the fused epilogue applies the RMSNorm scale 1/rms(x) (the gain is folded
//    into the activations) and then RoPE + KV-cache write (QKV; the cache holds
//    fp32), SiLU(gate)*up, SiLU, a scaled residual add, or the LM-head argmax.
//    For QKV and gate/up a unit holds two 16-row halves: rows i and i+Dh/2 of
//    a head (a RoPE pair), or gate row i and up row i.
//
// Batch invariance: the unit partition, the order of FMAs feeding each output
// and the reduction trees do not depend on M, so row m of an M-row launch is
// bitwise equal to the same row computed alone.  This makes the verify pass
// (M = gamma+1) reproduce greedy decoding (M = 1) exactly.
#pragma once

#include "common.cuh"

namespace ssd {

constexpr int kTileN = 32;           // weight rows per unit
constexpr int kHalfN = kTileN / 2;   // rows per half box (paired units)
constexpr int kTileK = 256;          // weight columns per unit (512 bytes of bf16)
constexpr int kConsumerWarps = 8;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kGemvThreads = kConsumerThreads;
constexpr int kStages = 4;
constexpr int kMaxSeg = 8;           // parked row-tile results before a flush
constexpr uint32_t kWTileBytes = kTileN * kTileK * 2;

enum class Epi : int { QKV = 0, GATE_SILU = 1, SILU = 2, RESID = 3, ARGMAX = 4 };

struct GemvParams {
  int K, n_kt, n_rt, units;
  int N;           // valid output rows (GATE_SILU: d_ff; a unit holds 16 gate + 16 up rows)
  int seg_rows;    // QKV: rows per source matrix (q, k, v)
  const float* x;  // activations [M][x_stride] (fp32, columns K..x_stride-1 zero)
  int x_stride;
  const __nv_bfloat16* gain;  // RMSNorm gain, zero-padded to a multiple of kTileK, or null (no norm)
  float eps;
  float* partials;      // [2 * grid][kMaxRows][kTileN]
  unsigned* counters;   // [n_rt]
  DevState* st;
  int pos_off;          // row m sits at position st->kv_len + pos_off + m
  int pf_dist;          // units prefetched into L2 ahead of the shared-memory ring
  // QKV
  float* q_out;
  int q_stride;
  float* k_cache;  // this layer's [H][max_seq][head_dim], fp32
  float* v_cache;
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
  static constexpr int kSeg = kG + kStages * kTileK * 2;          // parked tiles [kMaxSeg][M][kTileN]
  static constexpr int kSegRt = kSeg + kMaxSeg * M * kTileN * 4;  // [kMaxSeg] row tile, [kMaxSeg] whole flag
  static constexpr int kOut = kSegRt + 2 * kMaxSeg * 4;          // reduction buffer [M][kTileN]
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
// All run on the 256 threads with the finished row tile in out ([M][kTileN],
// fp32, before the RMSNorm scale) and rs[m] (1 if no norm).

template <int M, Epi EPI>
__device__ __forceinline__ void gemv_epilogue(const GemvParams& p, int rt, const float* out, const float* rs,
                                              int tid) {
  if constexpr (EPI == Epi::QKV) {
    const int tiles_per_mat = p.seg_rows / kTileN;
    const int mat = rt / tiles_per_mat;  // 0 = q, 1 = k, 2 = v
    const int rtm = rt - mat * tiles_per_mat;
    const int Dh = p.head_dim, half = Dh >> 1, tph = half / kHalfN;  // paired tiles per head
    const int base_pos = __ldcg(&p.st->kv_len) + p.pos_off;
    if (mat < 2) {
      const int h = rtm / tph, j0 = (rtm - h * tph) * kHalfN;
      for (int idx = tid; idx < M * kHalfN; idx += kConsumerThreads) {
        const int m = idx / kHalfN, i = idx - m * kHalfN;
        const int pos = base_pos + m;
        if (pos < 0 || pos >= p.max_seq) {
          set_error(p.st, DERR_POS);
          continue;
        }
        const int j = j0 + i;  // rotation pair (j, j + half) of head h
        const float a = out[m * kTileN + i] * rs[m];
        const float b = out[m * kTileN + kHalfN + i] * rs[m];
        const float2 cs = p.rope_cs[static_cast<size_t>(pos) * half + j];
        const float va = a * cs.x - b * cs.y;
        const float vb = a * cs.y + b * cs.x;
        if (mat == 0) {
          p.q_out[m * p.q_stride + h * Dh + j] = va;
          p.q_out[m * p.q_stride + h * Dh + j + half] = vb;
        } else {
          float* kr = p.k_cache + (static_cast<size_t>(h) * p.max_seq + pos) * Dh;
          kr[j] = va;
          kr[j + half] = vb;
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
        const int row = rtm * kTileN + i, h = row / Dh, d = row - h * Dh;
        p.v_cache[(static_cast<size_t>(h) * p.max_seq + pos) * Dh + d] = out[idx] * rs[m];
      }
    }
  } else if constexpr (EPI == Epi::GATE_SILU) {
    for (int idx = tid; idx < M * kHalfN; idx += kConsumerThreads) {
      const int m = idx / kHalfN, j = idx - m * kHalfN;
      const int n = rt * kHalfN + j;
      if (n >= p.N) continue;
      const float g = out[m * kTileN + j] * rs[m];
      const float u = out[m * kTileN + kHalfN + j] * rs[m];
      p.h_out[m * p.h_stride + n] = silu_f(g) * u;
    }
  } else if constexpr (EPI == Epi::SILU) {
    for (int idx = tid; idx < M * kTileN; idx += kConsumerThreads) {
      const int m = idx / kTileN, i = idx - m * kTileN;
      const int n = rt * kTileN + i;
      if (n >= p.N) continue;
      p.h_out[m * p.h_stride + n] = silu_f(out[idx] * rs[m]);
    }
  } else if constexpr (EPI == Epi::RESID) {
    const float s = __ldg(p.scale);
    for (int idx = tid; idx < M * kTileN; idx += kConsumerThreads) {
      const int m = idx / kTileN, i = idx - m * kTileN;
      const int n = rt * kTileN + i;
      if (n >= p.N) continue;
      const float b = __ldcg(p.base + m * p.base_stride + n);
      p.dst[m * p.dst_stride + n] = b + s * (out[idx] * rs[m]);
    }
  } else {  // ARGMAX (LM head): argmax over the vocabulary, lowest index on ties
    const int warp = tid >> 5, lane = tid & 31;
    const int base_pos = __ldcg(&p.st->kv_len) + p.pos_off;
    const int P = __ldcg(&p.st->prompt_len);
    for (int m = warp; m < M; m += kConsumerWarps) {  // warp per row, lane per tile row
      const int n = rt * kTileN + lane;
      const bool valid = n < p.N;
      const float logit = out[m * kTileN + lane] * rs[m];
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
  float* seg = reinterpret_cast<float*>(smem + S::kSeg);
  int* seg_rt = reinterpret_cast<int*>(smem + S::kSegRt);
  int* seg_whole = seg_rt + kMaxSeg;
  float* outb = reinterpret_cast<float*>(smem + S::kOut);
  float* rs = reinterpret_cast<float*>(smem + S::kRs);
  float* red = reinterpret_cast<float*>(smem + S::kRed);
  int* flag = reinterpret_cast<int*>(smem + S::kFlag);

  const int G = gridDim.x, c = blockIdx.x;
  const int u0 = unit_begin(c, p.units, G), u1 = unit_begin(c + 1, p.units, G);
  const int n_units = u1 - u0;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t tx = kWTileBytes + S::kActBytes + (p.gain ? kTileK * 2 : 0);

  // ---- producer helpers (thread 0 only)
  auto weight_box = [&](int u, auto&& op) {
    const int rt = u / p.n_kt, kt = u - rt * p.n_kt;
    const int x = kt * kTileK;
    if constexpr (EPI == Epi::GATE_SILU) {
      op(&map0, x, rt * kHalfN, 0);
      op(&map1, x, rt * kHalfN, static_cast<int>(kWTileBytes / 2));
    } else if constexpr (EPI == Epi::QKV) {
      const int tiles_per_mat = p.seg_rows / kTileN;
      const int mat = rt / tiles_per_mat, rtm = rt - mat * tiles_per_mat;
      if (mat < 2) {
        const int half = p.head_dim >> 1, tph = half / kHalfN;
        const int h = rtm / tph, r1 = h * p.head_dim + (rtm - h * tph) * kHalfN;
        const CUtensorMap* mp = mat == 0 ? &map0 : &map1;
        op(mp, x, r1, 0);
        op(mp, x, r1 + half, static_cast<int>(kWTileBytes / 2));
      } else {
        op(&map2, x, rtm * kTileN, 0);
      }
    } else {
      op(&map0, x, rt * kTileN, 0);
    }
  };
  auto issue_weights = [&](int s, int u) {
    uint8_t* wdst = smem + S::kW + s * kWTileBytes;
    weight_box(u, [&](const CUtensorMap* mp, int x, int y, int off) { tma_load_2d(wdst + off, mp, &full[s], x, y); });
    if (p.gain) {
      const int kt = u % p.n_kt;
      bulk_load(smem + S::kG + s * kTileK * 2, p.gain + kt * kTileK, kTileK * 2, &full[s]);
    }
  };
  auto prefetch_unit = [&](int u) {
    weight_box(u, [&](const CUtensorMap* mp, int x, int y, int) { tma_prefetch_2d(mp, x, y); });
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
    const int pf_end = min(n_units, npre + p.pf_dist);
    for (int i = npre; i < pf_end; ++i) prefetch_unit(u0 + i);
  }
  pdl_wait();  // activations, residuals and state are written by the previous kernel
  if (tid == 0)
    for (int i = 0; i < npre; ++i) issue_acts(i, u0 + i);

  float2 acc[4][M];
#pragma unroll
  for (int j = 0; j < 4; ++j)
#pragma unroll
    for (int m = 0; m < M; ++m) acc[j][m] = make_float2(0.f, 0.f);

  const int rt_first = u0 / p.n_kt;
  int seg_kt0 = u0 - rt_first * p.n_kt;
  int nseg = 0;
  bool rs_done = false;
  const uint8_t* wbase = smem + S::kW + (warp * 4) * (kTileK * 2) + lane * 16;

  // Runs the epilogues / cross-CTA reductions of the parked row tiles (all threads).
  auto flush = [&]() {
    __syncthreads();
    if (!rs_done) {
      // RMSNorm scale per row: rs[m] = 1/sqrt(mean(x^2) + eps), fixed reduction order
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
      rs_done = true;
    }
    for (int k = 0; k < nseg; ++k) {
      const int rt = seg_rt[k];
      const float* so = seg + k * (M * kTileN);
      if (seg_whole[k]) {
        gemv_epilogue<M, EPI>(p, rt, so, rs, tid);
      } else {
        const int slot = 2 * c + (rt == rt_first ? 0 : 1);
        float* dstp = p.partials + static_cast<size_t>(slot) * (kMaxRows * kTileN);
        for (int idx = tid; idx < M * kTileN; idx += kConsumerThreads) __stcg(dstp + idx, so[idx]);
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
            outb[idx] = sum;
          }
          __syncthreads();
          gemv_epilogue<M, EPI>(p, rt, outb, rs, tid);
          if (tid == 0) p.counters[rt] = 0u;
        }
      }
      __syncthreads();
    }
    nseg = 0;
  };

  for (int i = 0; i < n_units; ++i) {
    const int u = u0 + i;
    const int rt = u / p.n_kt, kt = u - rt * p.n_kt;
    const int s = i % kStages;
    const uint32_t par = static_cast<uint32_t>(i / kStages) & 1u;
    if (!mbar_wait(&full[s], par)) {
      set_error(p.st, DERR_TIMEOUT);
      return;  // every warp times out on the same stage
    }
    // weights: rows 4w + j (j < 4), columns 8*lane .. 8*lane+7 of the 32 x 256 unit
    uint4 wv[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) wv[j] = *reinterpret_cast<const uint4*>(wbase + s * kWTileBytes + j * (kTileK * 2));
    float2 gs[4];
    if (p.gain) {
      const uint4 gv = *reinterpret_cast<const uint4*>(smem + S::kG + s * kTileK * 2 + lane * 16);
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
    const float* abase = reinterpret_cast<const float*>(smem + S::kA + s * S::kActBytes) + lane * 8;
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
        if (p.pf_dist > 0 && i + kStages + p.pf_dist < n_units) prefetch_unit(u + kStages + p.pf_dist);
      }
    }

    const bool seg_end = (kt == p.n_kt - 1) || (i == n_units - 1);
    if (!seg_end) continue;

    // ---- park this row-tile segment: reduce over the 32 column lanes (warp-local)
    float* so = seg + nseg * (M * kTileN);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
#pragma unroll
      for (int m = 0; m < M; ++m) {
        float v = acc[j][m].x + acc[j][m].y;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if (lane == 0) so[m * kTileN + warp * 4 + j] = v;
        acc[j][m] = make_float2(0.f, 0.f);
      }
    }
    if (tid == 0) {
      seg_rt[nseg] = rt;
      seg_whole[nseg] = (seg_kt0 == 0) && (kt == p.n_kt - 1);
    }
    ++nseg;
    seg_kt0 = 0;  // the next segment starts at a row-tile boundary
    if (nseg == kMaxSeg && i + 1 < n_units) flush();
  }
  flush();
}

}  // namespace ssd
