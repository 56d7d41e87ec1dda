// Weight-streaming skinny GEMM ("GEMV" for M = 1..16 activation rows) on the
// 5th-generation tensor cores.
//
//   out[m][n] = sum_k W[n][k] * a[m][k],   W bf16 [N][K] (nn.Linear layout), a fp32
//
// Every decode-time projection of the decoder (Sec. "SSD Setup for VLMs",
// x_{l+1} = x_l + f_l(x_l)), of the imitation network and of the LM head g
// runs through this kernel; at batch 1 it is bound by HBM bandwidth, since each
// weight byte is used for M <= 9 rows only.  The arithmetic runs on tcgen05 so
// that issue slots never limit the weight stream:
//  * persistent grid of min(2 x #SMs, units) CTAs; the weight matrix is cut
//    into units of 128 rows x 64 columns (16 KB, one 128-byte swizzled row per
//    weight row) and CTA c streams the contiguous unit range [c*U/G, (c+1)*U/G)
//    -- stream-K, so every SM moves the same number of bytes;
//  * warp 0 issues TMA: the weight unit (SWIZZLE_128B), the fp32 slice of each
//    activation row and of the RMSNorm gain, into a 4-stage mbarrier ring; the
//    first stages' weights are requested before griddepcontrol.wait, so they
//    overlap the previous kernel (programmatic dependent launch);
//  * warps 2-3 turn each activation slice into the MMA's B operand: a = hi + lo
//    in bf16 (a to 2^-17 relative), rows padded to N = 16 with zeros, written in
//    the swizzled K-major layout;
//  * one thread of warp 1 issues tcgen05.mma.kind::f16 with the weight unit as
//    A (M = 128 weight rows) and the activations as B (N = 16): per unit 4 K
//    slices x (hi, lo) = 8 MMAs accumulating in fp32 in TMEM; a row tile's
//    accumulator (128 lanes x 16 columns) is double-buffered;
//  * warps 4-7 drain finished accumulators with tcgen05.ld while the stream
//    goes on, reduce row tiles split between CTAs in fixed CTA order (the CTA
//    that finishes a tile last does it -- an atomic ticket, no spinning), and
//    apply the fused epilogue: the RMSNorm scale 1/rms(x) (the gain is folded
//    into the activations), then RoPE + KV-cache write (QKV), SiLU(gate)*up
//    (a unit holds 64 gate + the same 64 up rows), SiLU, a scaled residual
//    add, or the LM-head argmax.
//
// Batch invariance: the unit partition, the MMA shape (always N = 16), the K
// order and the reduction order do not depend on M, and each output element
// is an independent dot product, so row m of an M-row launch is bitwise equal
// to the same row computed alone.  This makes the verify pass (M = gamma+1)
// reproduce greedy decoding (M = 1) exactly.
#pragma once

#include "common.cuh"
#include "tcgen05.cuh"

namespace ssd {

constexpr int kTileN = 128;          // weight rows per unit (the MMA's M)
constexpr int kHalfN = kTileN / 2;   // gate or up rows of a paired unit
constexpr int kTileK = 64;           // weight columns per unit (one 128-byte swizzled row)
constexpr int kNPad = 16;            // activation rows padded to the MMA's N
constexpr int kStages = 4;
constexpr int kGemvThreads = 256;
constexpr int kGemvCtasPerSm = 2;   // persistent grid: min(units, 2 x #SMs) CTAs
constexpr int kDrainThreads = 128;   // warps 4..7
constexpr int kTmemCols = 32;        // two 16-column accumulators
constexpr uint32_t kWTileBytes = kTileN * kTileK * 2;   // 16 KB
constexpr uint32_t kBOpBytes = kNPad * kTileK * 2;      // 2 KB (hi or lo)

enum class Epi : int { QKV = 0, GATE_SILU = 1, SILU = 2, RESID = 3, ARGMAX = 4, XATTN = 5 };

struct GemvParams {
  int K, n_kt, n_rt, units;
  int N;           // valid output rows (GATE_SILU: d_ff; a unit holds 64 gate + 64 up rows)
  int seg_rows;    // QKV: rows per source matrix (q, k, v)
  const float* x;  // activations [M][x_stride] (fp32)
  int x_stride;
  const __nv_bfloat16* gain;  // RMSNorm gain (zero-padded), or null (no norm)
  float eps;
  float* partials;      // [2 * grid][kMaxRows][kTileN]
  unsigned* counters;   // [n_rt]
  DevState* st;
  int pos_off;          // row m sits at position st->kv_len + pos_off + m
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
  float* logits;       // optional [logits_rows][N] capture: row m's logits go to row position + 1 - P
                       // (the index of the token it predicts), or with logits_step_rows > 0 to row
                       // st->steps * logits_step_rows + pos_off + m (draft rows by step)
  int logits_rows;
  int logits_step_rows;
  // Trigger the dependent launch only once the upstream grid has completed (from the weight
  // producer, after its wait), so that everything older than this launch is complete when the
  // dependent grid starts: the split-KV attention after the QKV projection reads older cache rows
  // before its own wait.
  int late_trigger;
  int seg_base;  // QKV: segment of the site's first matrix (0 = q; 1 = k, for a [k; v] site)
  // Batched requests (batch_rows = 0: one request, whose state is st).  With batch_rows = R > 0,
  // row m belongs to request b = m / R at offset i = pos_off + m % R within the request's rows:
  // it sits at position req_st[b].kv_len + i, its K/V rows are at k_cache / v_cache + b * req_kv,
  // its argmax goes to tok_dst[b * tok_stride + m % R], and a logits capture writes
  // logits[b][row][N] (full-model rows by the index of the predicted token within the request,
  // draft rows by req_st[b].steps * logits_step_rows + i).  st still holds the error word and the
  // argmax keys of the launch.
  int batch_rows;
  DevState* req_st;
  long long req_kv;
  int tok_stride;
  // Medium-M kernel only: the rows' RMSNorm scales 1/rms(x_m), computed by the split kernel
  // (the gain is folded into its bf16 hi/lo parts).
  const float* rs_in;
  // Medium-M, when the producing kernel has already split this launch's rows: their sums of squares
  // per 128-column tile of the producer, [row][rs_nparts], summed here in tile order for 1/rms.
  const float* rs_parts;
  int rs_nparts;
  // Medium-M reduction as the producer of the next medium-M projection's input (nx_hi null: none):
  // the RESID / GATE_SILU outputs also go out as bf16 parts of value * nx_gain[n] (no gain: value),
  // [row][nx_ld], and RESID rows' sums of squares per tile to nx_ssq[row][n_rt].
  __nv_bfloat16* nx_hi;
  __nv_bfloat16* nx_lo;
  int nx_ld;
  const __nv_bfloat16* nx_gain;
  float* nx_ssq;
  int grid_ctas;  // medium-M reduction: the CTAs of the streaming launch
  int abs_pos;   // row m sits at position pos_off + m, st->kv_len ignored (the encoder's rows)
  int act;       // GATE_SILU: 0 = SiLU(gate) * up, 1 = GELU_tanh(gate) * up (gated GELU)
  // XATTN (a q-only site: the encoder-decoder model's cross-attention query): instead of writing
  // q, the tile's owner attends with it over the st->enc_len <= kXattnKeys cross keys xk / xv
  // ([H][x_max][head_dim] fp32, every key visible, scores times x_scale) and writes the attention
  // output rows to xo (row stride xo_stride).
  const float* xk;
  const float* xv;
  int x_max;
  float x_scale;
  float* xo;
  int xo_stride;
};

constexpr int kXattnKeys = 128;  // cross keys the folded cross-attention takes

template <int M>
struct GemvSmem {
  static constexpr int kPreRows = M <= 9 ? M : 0;  // epilogue inputs fetched early (rows up to 9)
  static constexpr int kActBytes = M * kTileK * 4;
  static constexpr int kW = 0;                                  // [stages][16 KB] weight units (1024-aligned)
  static constexpr int kB = kW + kStages * kWTileBytes;         // [stages][hi | lo] B operands (1024-aligned)
  static constexpr int kA = kB + kStages * 2 * kBOpBytes;       // [stages][M][64] fp32 activation slices
  static constexpr int kG = kA + kStages * kActBytes;           // [stages][64] bf16 gain slices
  static constexpr int kOut = kG + kStages * kTileK * 2;        // drained row tile [M][128]
  static constexpr int kPre = kOut + M * kTileN * 4;             // epilogue inputs fetched early: [2][M][128] fp32
  static constexpr int kRowPos = kPre + 2 * kPreRows * kTileN * 4;  // batched rows: position, request [2][kMaxRows]
  static constexpr int kRs = kRowPos + 2 * kMaxRows * 4;
  static constexpr int kRed = kRs + kMaxRows * 4;               // [4][kMaxRows]
  static constexpr int kFlag = kRed + 4 * kMaxRows * 4;
  static constexpr int kBar = (kFlag + 16 + 7) & ~7;            // full, empty, bready [stages]; afull, aempty [2]
  static constexpr int kTmemSlot = kBar + (3 * kStages + 4) * 8;
  static constexpr int kTotal = kTmemSlot + 16 + 1024;          // + slack for the 1024-byte alignment
};

// Which CTA of a G-CTA grid owns unit u (ranges [floor(cU/G), floor((c+1)U/G))).
__device__ __forceinline__ int unit_owner(int u, int units, int G) {
  return static_cast<int>((static_cast<long long>(u + 1) * G - 1) / units);
}
__device__ __forceinline__ int unit_begin(int c, int units, int G) {
  return static_cast<int>((static_cast<long long>(c) * units) / G);
}

// ------------------------------------------------------------------ epilogues
// Run on the 128 drain threads with a finished row tile in out ([MT][kTileN],
// fp32, before the RMSNorm scale) and rs[m] (1 if no norm) for the mc <= MT
// rows m0 .. m0 + mc - 1 of the launch (local row m is launch row m0 + m).
// pre: inputs fetched into shared memory after the upstream wait, or null --
// QKV: the rotation table rows of the rows' positions ([mc][head_dim / 2]
// float2); RESID: the tile's base rows ([mc][kTileN]).  base_pos: position of
// launch row 0 (st->kv_len + pos_off, or pos_off with abs_pos; read once per
// CTA) for one request; with batch_rows, rpos[m] / rreq[m] hold the position
// and the request of launch row m instead (rpos is null for one request).

__device__ __forceinline__ void drain_sync() { named_bar_sync(1, kDrainThreads); }

// The medium-M RESID epilogue's per-warp sums of squares of a tile's rows, [drain warp][row].
__device__ __forceinline__ float* argmax_warp_ssq() {
  __shared__ float sq[(kDrainThreads / 32) * kNPad];
  return sq;
}

// The LM head epilogue's per-warp argmax keys of a tile's rows, [drain warp][row] (16 rows).
__device__ __forceinline__ unsigned long long* argmax_warp_keys() {
  __shared__ unsigned long long keys[(kDrainThreads / 32) * kNPad];
  return keys;
}

// Launch row mg's request and offset within the request's rows (batch_rows > 0).
__device__ __forceinline__ int batch_offset(const GemvParams& p, int mg, int b) {
  return p.pos_off + mg - b * p.batch_rows;
}

// Cross-attention folded into the cross-q projection's epilogue (see GemvParams::xk): for the
// tile's heads (128 / head_dim of them) and rows m0 .. m0 + mc - 1, with q = out * rs,
//   s_j = x_scale * q . K_j,  p_j = exp(s_j - max_j s),  o = (sum_j p_j V_j) / (sum_j p_j),
// keys in order, each row on its own (the result does not depend on the launch's other rows).
template <int MT>
__device__ __forceinline__ void gemv_cross_attention(const GemvParams& p, int rt, const float* out, const float* rs,
                                                     int tid, int m0, int mc) {
  __shared__ float xs[kNPad * 2 * kXattnKeys];  // [row][head of the tile][key] scores, then exponentials
  __shared__ float xl[kNPad * 2];               // [row][head] sums
  const int Dh = p.head_dim, hpt = kTileN / Dh, h0 = (rt * kTileN) / Dh;
  const int nk = min(__ldcg(&p.st->enc_len), kXattnKeys);
  // 1. scores: one (head, key) item per thread, its key row read once for all rows
  for (int it = tid; it < hpt * nk; it += kDrainThreads) {
    const int hh = it / nk, j = it - hh * nk;
    const float4* kr = reinterpret_cast<const float4*>(p.xk + (static_cast<size_t>(h0 + hh) * p.x_max + j) * Dh);
    float a[MT];
#pragma unroll
    for (int m = 0; m < MT; ++m) a[m] = 0.f;
    for (int d4 = 0; d4 < (Dh >> 2); ++d4) {
      const float4 k4 = __ldg(kr + d4);
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        if (m >= mc) break;
        const float* q = out + m * kTileN + hh * Dh + 4 * d4;
        a[m] = fmaf(q[0], k4.x, a[m]);
        a[m] = fmaf(q[1], k4.y, a[m]);
        a[m] = fmaf(q[2], k4.z, a[m]);
        a[m] = fmaf(q[3], k4.w, a[m]);
      }
    }
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      if (m >= mc) break;
      xs[(m * 2 + hh) * kXattnKeys + j] = (a[m] * rs[m]) * p.x_scale;
    }
  }
  drain_sync();
  // 2. per (row, head), one warp: max, exponentials in place, their sum
  const int lane = tid & 31, w = tid >> 5;
  for (int r = w; r < mc * hpt; r += kDrainThreads / 32) {
    const int m = r / hpt, hh = r - m * hpt;
    float* sr = xs + (m * 2 + hh) * kXattnKeys;
    float mx = -INFINITY;
    for (int j = lane; j < nk; j += 32) mx = fmaxf(mx, sr[j]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    float sum = 0.f;
    for (int j = lane; j < nk; j += 32) {
      const float e = expf(sr[j] - mx);
      sr[j] = e;
      sum += e;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
    if (lane == 0) xl[m * 2 + hh] = sum;
  }
  drain_sync();
  // 3. P.V: one (head, dimension) item per thread, the keys in order
  for (int it = tid; it < hpt * Dh; it += kDrainThreads) {
    const int hh = it / Dh, d = it - hh * Dh;
    const float* vc = p.xv + static_cast<size_t>(h0 + hh) * p.x_max * Dh + d;
    float o[MT];
#pragma unroll
    for (int m = 0; m < MT; ++m) o[m] = 0.f;
    for (int j = 0; j < nk; ++j) {
      const float v = __ldg(vc + static_cast<size_t>(j) * Dh);
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        if (m >= mc) break;
        o[m] = fmaf(xs[(m * 2 + hh) * kXattnKeys + j], v, o[m]);
      }
    }
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      if (m >= mc) break;
      const float L = xl[m * 2 + hh];
      p.xo[(m0 + m) * p.xo_stride + (h0 + hh) * Dh + d] = L > 0.f ? o[m] / L : 0.f;
    }
  }
}

// NX: the medium-M reduction's instance, which may also write the next projection's operand parts
// (GemvParams nx_*); the GEMV's instances compile without that code.
template <int MT, Epi EPI, bool NX = false>
__device__ __forceinline__ void gemv_epilogue(const GemvParams& p, int rt, const float* out, const float* rs,
                                              const float* pre, int base_pos, const int* rpos, const int* rreq,
                                              int tid, int m0, int mc) {
  if constexpr (EPI == Epi::XATTN) {
    gemv_cross_attention<MT>(p, rt, out, rs, tid, m0, mc);
  } else if constexpr (EPI == Epi::QKV) {
    const int r0 = rt * kTileN;
    const int seg = r0 / p.seg_rows;       // source matrix of this row tile within the site
    const int mat = seg + p.seg_base;      // 0 = q, 1 = k, 2 = v
    const int local0 = r0 - seg * p.seg_rows;
    const int Dh = p.head_dim, half = Dh >> 1;
    if (mat < 2) {
      // four (row, pair) items per thread at a time: their rotation coefficients are fetched
      // first (from shared memory, or from the table in global memory), then rotated and stored
      constexpr int kPairs = kTileN / 2;
      const int n_items = mc * kPairs;
      for (int i0 = tid; i0 < n_items; i0 += 4 * kDrainThreads) {
        float2 cs[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int idx = i0 + u * kDrainThreads;
          cs[u] = make_float2(1.f, 0.f);
          if (idx < n_items && p.rope_cs) {
            const int m = idx / kPairs, pr = idx - m * kPairs, mg = m0 + m;
            const int j = pr - (pr / half) * half;
            const int pos = rpos ? rpos[mg] : base_pos + mg;
            if (pre) cs[u] = reinterpret_cast<const float2*>(pre)[m * half + j];
            else if (pos >= 0 && pos < p.max_seq) cs[u] = __ldg(p.rope_cs + static_cast<size_t>(pos) * half + j);
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int idx = i0 + u * kDrainThreads;
          if (idx >= n_items) break;
          const int m = idx / kPairs, pr = idx - m * kPairs, mg = m0 + m;
          const int hh = pr / half, j = pr - hh * half;
          const int ra = hh * Dh + j, rb = ra + half;
          const int pos = rpos ? rpos[mg] : base_pos + mg;
          if (pos < 0 || pos >= p.max_seq) {
            set_error(p.st, DERR_POS);
            continue;
          }
          const float a = out[m * kTileN + ra] * rs[m];
          const float b = out[m * kTileN + rb] * rs[m];
          float va = a, vb = b;  // no rotation without a table (relative-position-bias models)
          if (p.rope_cs) {
            va = a * cs[u].x - b * cs[u].y;
            vb = a * cs[u].y + b * cs[u].x;
          }
          if (mat == 0) {
            p.q_out[mg * p.q_stride + local0 + ra] = va;
            p.q_out[mg * p.q_stride + local0 + rb] = vb;
          } else {
            const int h = local0 / Dh + hh;
            float* kr = p.k_cache + (rreq ? rreq[mg] * p.req_kv : 0ll) + (static_cast<size_t>(h) * p.max_seq + pos) * Dh;
            kr[j] = va;
            kr[j + half] = vb;
          }
        }
      }
    } else {
      for (int idx = tid; idx < mc * kTileN; idx += kDrainThreads) {
        const int m = idx / kTileN, i = idx - m * kTileN, mg = m0 + m;
        const int pos = rpos ? rpos[mg] : base_pos + mg;
        if (pos < 0 || pos >= p.max_seq) {
          set_error(p.st, DERR_POS);
          continue;
        }
        const int row = local0 + i, h = row / Dh, d = row - h * Dh;
        p.v_cache[(rreq ? rreq[mg] * p.req_kv : 0ll) + (static_cast<size_t>(h) * p.max_seq + pos) * Dh + d] =
            out[idx] * rs[m];
      }
    }
  } else if constexpr (EPI == Epi::GATE_SILU) {
    for (int idx = tid; idx < mc * kHalfN; idx += kDrainThreads) {
      const int m = idx / kHalfN, j = idx - m * kHalfN;
      const int n = rt * kHalfN + j;
      if (n >= p.N) continue;
      const float g = out[m * kTileN + j] * rs[m];
      const float u = out[m * kTileN + kHalfN + j] * rs[m];
      const float hv = (p.act ? gelu_tanh_f(g) : silu_f(g)) * u;
      p.h_out[(m0 + m) * p.h_stride + n] = hv;
      if (NX && p.nx_hi) {
        const __nv_bfloat16 hh = __float2bfloat16_rn(hv);
        p.nx_hi[(m0 + m) * p.nx_ld + n] = hh;
        p.nx_lo[(m0 + m) * p.nx_ld + n] = __float2bfloat16_rn(hv - __bfloat162float(hh));
      }
    }
  } else if constexpr (EPI == Epi::SILU) {
    for (int idx = tid; idx < mc * kTileN; idx += kDrainThreads) {
      const int m = idx / kTileN, i = idx - m * kTileN;
      const int n = rt * kTileN + i;
      if (n >= p.N) continue;
      p.h_out[(m0 + m) * p.h_stride + n] = silu_f(out[idx] * rs[m]);
    }
  } else if constexpr (EPI == Epi::RESID) {
    // thread tid owns column tid of every row; the base rows are loaded before any store
    // (dst may alias base, so the stores would otherwise serialize the loads)
    static_assert(kDrainThreads == kTileN, "one thread per tile column");
    const float s = __ldg(p.scale);
    const int n = rt * kTileN + tid;
    float xv[MT];
#pragma unroll
    for (int m = 0; m < MT; ++m) xv[m] = 0.f;
    if (n < p.N) {
      float bv[MT];
#pragma unroll
      for (int m = 0; m < MT; ++m)
        if (m < mc) bv[m] = pre ? pre[m * kTileN + tid] : __ldcg(p.base + (m0 + m) * p.base_stride + n);
#pragma unroll
      for (int m = 0; m < MT; ++m)
        if (m < mc) {
          xv[m] = bv[m] + s * (out[m * kTileN + tid] * rs[m]);
          p.dst[(m0 + m) * p.dst_stride + n] = xv[m];
        }
      if (NX && p.nx_hi) {  // the next projection's input parts: x * gain
        const float gn = p.nx_gain ? __bfloat162float(p.nx_gain[n]) : 1.0f;
#pragma unroll
        for (int m = 0; m < MT; ++m)
          if (m < mc) {
            const float v = xv[m] * gn;
            const __nv_bfloat16 hh = __float2bfloat16_rn(v);
            p.nx_hi[(m0 + m) * p.nx_ld + n] = hh;
            p.nx_lo[(m0 + m) * p.nx_ld + n] = __float2bfloat16_rn(v - __bfloat162float(hh));
          }
      }
    }
    if (NX && p.nx_ssq) {  // the rows' sums of squares over this tile: warps, then the 4 warps in order
      float* red = argmax_warp_ssq();
      const int lane = tid & 31, w = tid >> 5;
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        float q = xv[m] * xv[m];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) q += __shfl_xor_sync(0xffffffffu, q, off);
        if (lane == 0) red[w * kNPad + m] = q;
      }
      drain_sync();
      if (tid < mc)
        p.nx_ssq[(m0 + tid) * p.n_rt + rt] = ((red[tid] + red[kNPad + tid]) + red[2 * kNPad + tid]) + red[3 * kNPad + tid];
      drain_sync();
    }
  } else {  // ARGMAX (LM head): this tile's keys of the rows; gemv_argmax_finish turns them into tokens
    const int lane = tid & 31;
    const int row0 = (p.logits == nullptr || rpos) ? 0
                     : p.logits_step_rows > 0 ? __ldcg(&p.st->steps) * p.logits_step_rows + p.pos_off
                                              : base_pos + 1 - __ldcg(&p.st->prompt_len);
    const int n = rt * kTileN + tid;  // thread per tile row
    const bool valid = n < p.N;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      if (m >= mc) break;
      const int mg = m0 + m;
      const float logit = out[m * kTileN + tid] * rs[m];
      if (p.logits != nullptr && valid) {
        if (rpos) {  // batched: rows [request][logits_rows]
          const int b = rreq[mg];
          const int row = p.logits_step_rows > 0
                              ? __ldcg(&p.req_st[b].steps) * p.logits_step_rows + batch_offset(p, mg, b)
                              : rpos[mg] + 1 - __ldcg(&p.req_st[b].prompt_len);
          if (row >= 0 && row < p.logits_rows)
            p.logits[(static_cast<size_t>(b) * p.logits_rows + row) * p.N + n] = logit;
        } else {
          const int row = row0 + mg;
          if (row >= 0 && row < p.logits_rows) p.logits[static_cast<size_t>(row) * p.N + n] = logit;
        }
      }
      unsigned long long key = valid ? argmax_key(logit, static_cast<uint32_t>(n)) : 0ull;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const unsigned long long o = __shfl_xor_sync(0xffffffffu, key, off);
        key = o > key ? o : key;
      }
      if (lane == 0) argmax_warp_keys()[(tid >> 5) * kNPad + m] = key;
    }
  }
}

// LM head, after the epilogue of a row tile: each drain warp left its maxima of the tile's rows
// m0 .. m0 + mc - 1 in shared memory; thread r folds the four warps' keys of row m0 + r into the
// row's global key with one atomic (rows on separate 128-byte lines).  The maxima are released
// by one acq_rel ticket of the rows' 16-row chunk after the CTA barrier; the tile that completes
// the chunk's count of `tiles` reads and resets the chunk's keys, one thread per row, and writes
// the tokens (-1 once a bounded wait anywhere has given up: the keys may miss tiles).
__device__ __forceinline__ void gemv_argmax_finish(const GemvParams& p, const int* rreq, int tid, int tiles,
                                                   int m0, int mc) {
  __shared__ int am_last;
  const unsigned long long* wk = argmax_warp_keys();
  unsigned int* count = &p.st->am_count[(m0 / kNPad) * kAmCountStride];
  drain_sync();
  if (tid < mc) {
    unsigned long long key = wk[tid];
#pragma unroll
    for (int w = 1; w < kDrainThreads / 32; ++w) key = max(key, wk[w * kNPad + tid]);
    atomicMax(&p.st->am_key[(m0 + tid) * kAmKeyStride], key);
  }
  drain_sync();
  if (tid == 0) am_last = atom_add_acq_rel_gpu(count, 1u) == static_cast<unsigned>(tiles - 1);
  drain_sync();
  if (am_last) {
    const bool stopped = (__ldcg(&p.st->error) & DERR_TIMEOUT) != 0;
    for (int r = m0 + tid; r < m0 + mc; r += kDrainThreads) {
      const unsigned long long key = atomicExch(&p.st->am_key[r * kAmKeyStride], 0ull);
      const int tok = stopped ? -1 : static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull));
      if (rreq) {
        const int b = rreq[r];
        p.tok_dst[b * p.tok_stride + (r - b * p.batch_rows)] = tok;
      } else {
        p.tok_dst[r * (p.tok_stride ? p.tok_stride : 1)] = tok;
      }
    }
    if (tid == 0) atomicExch(count, 0u);
  }
}

// ------------------------------------------------------------------ kernel

template <int M, Epi EPI>
__global__ void __launch_bounds__(kGemvThreads, 2)
    ssd_wstream_kernel(const __grid_constant__ CUtensorMap map0, const __grid_constant__ CUtensorMap map1,
                const __grid_constant__ CUtensorMap map2, const GemvParams p) {
  static_assert(M >= 1 && M <= kNPad, "activation rows");
  using S = GemvSmem<M>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBar);
  uint64_t* empty = full + kStages;
  uint64_t* bready = empty + kStages;
  uint64_t* afull = bready + kStages;
  uint64_t* aempty = afull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + S::kTmemSlot);
  float* outb = reinterpret_cast<float*>(smem + S::kOut);
  float* rs = reinterpret_cast<float*>(smem + S::kRs);
  float* red = reinterpret_cast<float*>(smem + S::kRed);
  int* flag = reinterpret_cast<int*>(smem + S::kFlag);

  const int G = gridDim.x, c = blockIdx.x;
  const int u0 = unit_begin(c, p.units, G), u1 = unit_begin(c + 1, p.units, G);
  const int n_units = u1 - u0;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t tx = kWTileBytes + S::kActBytes + (p.gain ? kTileK * 2 : 0);

  if (!p.late_trigger) pdl_trigger();
  // After a timed-out wait anywhere in the decode, later kernels do nothing
  // (best-effort read before any copy is issued or TMEM is taken).
  if (*reinterpret_cast<volatile int*>(&p.st->error) & DERR_TIMEOUT) return;

  // zero the B operands once: rows M..15 stay zero for the whole kernel
  for (int i = tid; i < kStages * 2 * static_cast<int>(kBOpBytes) / 16; i += kGemvThreads)
    reinterpret_cast<uint4*>(smem + S::kB)[i] = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&bready[s], 2);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&afull[b], 1);
      mbar_init(&aempty[b], 4);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kTmemCols)
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
      auto issue_weights = [&](int s, int u) {
        const int rt = u / p.n_kt, kt = u - rt * p.n_kt;
        uint8_t* wdst = smem + S::kW + s * kWTileBytes;
        const int x = kt * kTileK;
        if constexpr (EPI == Epi::GATE_SILU) {
          tma_load_2d(wdst, &map0, &full[s], x, rt * kHalfN);
          tma_load_2d(wdst + kWTileBytes / 2, &map1, &full[s], x, rt * kHalfN);
        } else if constexpr (EPI == Epi::QKV) {
          const int r0 = rt * kTileN, mat = r0 / p.seg_rows;
          tma_load_2d(wdst, mat == 0 ? &map0 : (mat == 1 ? &map1 : &map2), &full[s], x, r0 - mat * p.seg_rows);
        } else {
          tma_load_2d(wdst, &map0, &full[s], x, rt * kTileN);
        }
        if (p.gain) bulk_load(smem + S::kG + s * kTileK * 2, p.gain + x, kTileK * 2, &full[s]);
      };
      auto issue_acts = [&](int s, int u) {
        const int kt = u % p.n_kt;
        uint8_t* adst = smem + S::kA + s * S::kActBytes;
#pragma unroll
        for (int m = 0; m < M; ++m)
          bulk_load(adst + m * kTileK * 4, p.x + static_cast<size_t>(m) * p.x_stride + kt * kTileK, kTileK * 4,
                    &full[s]);
      };
      prefetch_tensormap(&map0);
      const int npre = n_units < kStages ? n_units : kStages;
      for (int i = 0; i < npre; ++i) {
        mbar_arrive_expect_tx(&full[i], tx);
        issue_weights(i, u0 + i);  // weights do not depend on the previous kernel
      }
      pdl_wait();
      if (p.late_trigger) pdl_trigger();
      for (int i = 0; i < npre; ++i) issue_acts(i, u0 + i);
      int issued = npre;
      for (int i = npre; i < n_units; ++i, ++issued) {
        const int s = i % kStages;
        if (!mbar_wait(&empty[s], static_cast<uint32_t>((i / kStages) - 1) & 1u)) {
          set_error(p.st, DERR_TIMEOUT);
          break;
        }
        mbar_arrive_expect_tx(&full[s], tx);
        issue_weights(s, u0 + i);
        issue_acts(s, u0 + i);
      }
      if (__ldcg(&p.st->error) & DERR_TIMEOUT) drain_ring(full, kStages, issued);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_bf16(kTileN, kNPad);
      int sg = 0;
      bool seg_open = false;
      uint32_t d = tmem;
      for (int i = 0; i < n_units; ++i) {
        const int u = u0 + i, kt = u % p.n_kt, s = i % kStages;
        if (!seg_open) {  // a new row-tile segment: take a free accumulator
          const int b = sg & 1;
          if (!mbar_wait(&aempty[b], static_cast<uint32_t>(((sg >> 1) & 1) ^ 1))) {
            set_error(p.st, DERR_TIMEOUT);
            break;
          }
          tmem_fence_after();
          d = tmem + static_cast<uint32_t>(b * kNPad);
        }
        if (!mbar_wait(&bready[s], static_cast<uint32_t>(i / kStages) & 1u)) {
          set_error(p.st, DERR_TIMEOUT);
          break;
        }
        tmem_fence_after();
        const uint32_t wa = smem_u32(smem + S::kW + s * kWTileBytes);
        const uint32_t ba = smem_u32(smem + S::kB + s * 2 * kBOpBytes);
        const uint64_t adesc = umma_desc_sw128(wa), hdesc = umma_desc_sw128(ba), ldesc = umma_desc_sw128(ba + kBOpBytes);
#pragma unroll
        for (int kk = 0; kk < kTileK / 16; ++kk) {
          // +32 bytes (2 descriptor units) per 16-element K slice inside the swizzled row
          umma_f16(d, adesc + 2 * kk, hdesc + 2 * kk, idesc, (seg_open || kk > 0) ? 1u : 0u);
          umma_f16(d, adesc + 2 * kk, ldesc + 2 * kk, idesc, 1u);
          seg_open = true;
        }
        umma_commit(&empty[s]);  // stage s may be refilled once these MMAs have read it
        if (kt == p.n_kt - 1 || i == n_units - 1) {
          umma_commit(&afull[sg & 1]);  // the row tile's accumulator is complete
          ++sg;
          seg_open = false;
        }
      }
    }
  } else if (warp < 4) {
    // ---------------------------------------------------------------- B operand: fp32 -> bf16 hi + lo, swizzled
    const int ct = tid - 64;  // 0..63
    for (int i = 0; i < n_units; ++i) {
      const int s = i % kStages;
      if (!mbar_wait(&full[s], static_cast<uint32_t>(i / kStages) & 1u)) {
        set_error(p.st, DERR_TIMEOUT);
        break;
      }
      const float* a = reinterpret_cast<const float*>(smem + S::kA + s * S::kActBytes);
      const __nv_bfloat16* g = reinterpret_cast<const __nv_bfloat16*>(smem + S::kG + s * kTileK * 2);
      uint8_t* bh = smem + S::kB + s * 2 * kBOpBytes;
      for (int task = ct; task < M * 8; task += 64) {
        const int m = task >> 3, ch = task & 7;
        const float4 a0 = *reinterpret_cast<const float4*>(a + m * kTileK + ch * 8);
        const float4 a1 = *reinterpret_cast<const float4*>(a + m * kTileK + ch * 8 + 4);
        float v[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
        if (p.gain) {
          const uint4 gv = *reinterpret_cast<const uint4*>(g + ch * 8);
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
        const int off = m * 128 + ((ch ^ (m & 7)) << 4);  // 128-byte swizzle of row m
        *reinterpret_cast<uint4*>(bh + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        *reinterpret_cast<uint4*>(bh + kBOpBytes + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
      }
      fence_proxy_async_smem();  // make the generic-proxy writes visible to the tensor core
      __syncwarp();
      if (lane == 0) mbar_arrive(&bready[s]);
    }
  } else {
    // ---------------------------------------------------------------- drain + epilogues (warps 4..7)
    const int dt = tid - 128;  // 0..127
    const int q = warp & 3;    // TMEM lane quadrant: tile rows 32q .. 32q+31
    pdl_wait();
    // RMSNorm scale per row: rs[m] = 1/sqrt(mean(x^2) + eps), fixed reduction order
    if (p.gain) {
#pragma unroll 1
      for (int m = 0; m < M; ++m) {
        const float4* xr = reinterpret_cast<const float4*>(p.x + static_cast<size_t>(m) * p.x_stride);
        float ss = 0.f;
        for (int i = dt; i < (p.K >> 2); i += kDrainThreads) {
          const float4 v = __ldcg(xr + i);
          ss = fmaf(v.x, v.x, ss);
          ss = fmaf(v.y, v.y, ss);
          ss = fmaf(v.z, v.z, ss);
          ss = fmaf(v.w, v.w, ss);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
        if (lane == 0) red[(warp - 4) * kMaxRows + m] = ss;
      }
      drain_sync();
      if (dt < M) {
        float t = 0.f;
        for (int w = 0; w < 4; ++w) t += red[w * kMaxRows + dt];
        rs[dt] = rsqrtf(t / static_cast<float>(p.K) + p.eps);
      }
    } else if (dt < M) {
      rs[dt] = 1.0f;
    }
    // epilogue inputs fetched now, off the tail: the rotation rows of the M positions (QKV),
    // the base rows of this CTA's first and last row tiles (RESID; every contributor of a split
    // tile fetches them, whichever ends up owning it, before its ticket)
    const int rt_first = u0 / p.n_kt, rt_last = (u1 - 1) / p.n_kt;
    const int base_pos = (p.abs_pos || p.batch_rows ? 0 : __ldcg(&p.st->kv_len)) + p.pos_off;
    float* pre = reinterpret_cast<float*>(smem + S::kPre);
    // batched rows: each row's position and request, once per CTA
    int* rpos = p.batch_rows ? reinterpret_cast<int*>(smem + S::kRowPos) : nullptr;
    int* rreq = p.batch_rows ? rpos + kMaxRows : nullptr;
    if (rpos && dt < M) {
      const int b = dt / p.batch_rows;
      rreq[dt] = b;
      rpos[dt] = __ldcg(&p.req_st[b].kv_len) + batch_offset(p, dt, b);
    }
    bool pre_rope = false;
    if constexpr (EPI == Epi::QKV && S::kPreRows > 0) {
      const int half = p.head_dim >> 1;
      pre_rope = p.rope_cs != nullptr && !p.batch_rows && base_pos >= 0 && base_pos + M <= p.max_seq &&
                 half <= kTileN;
      if (pre_rope)
        for (int idx = dt; idx < M * half; idx += kDrainThreads) {
          const int m = idx / half, j = idx - m * half;
          reinterpret_cast<float2*>(pre)[idx] = p.rope_cs[static_cast<size_t>(base_pos + m) * half + j];
        }
    } else if constexpr (EPI == Epi::RESID && S::kPreRows > 0) {
      const int nb = rt_last == rt_first ? 1 : 2;
      for (int idx = dt; idx < nb * M * kTileN; idx += kDrainThreads) {
        const int b = idx / (M * kTileN), r = idx - b * (M * kTileN), m = r / kTileN, i = r - m * kTileN;
        const int n = (b == 0 ? rt_first : rt_last) * kTileN + i;
        pre[idx] = n < p.N ? __ldcg(p.base + m * p.base_stride + n) : 0.f;
      }
    }
    drain_sync();
    auto pre_of = [&](int rt) -> const float* {
      if constexpr (EPI == Epi::QKV) return pre_rope ? pre : nullptr;
      if constexpr (EPI == Epi::RESID && S::kPreRows > 0) {
        if (rt == rt_first) return pre;
        if (rt == rt_last) return pre + M * kTileN;
      }
      return nullptr;
    };

    int seg_kt0 = u0 - rt_first * p.n_kt;
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
      float v[kNPad];
      tmem_ld16(tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(b * kNPad), v);
      tmem_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&aempty[b]);  // the MMA warp may reuse accumulator b
#pragma unroll
      for (int m = 0; m < M; ++m) outb[m * kTileN + q * 32 + lane] = v[m];
      drain_sync();
      const bool whole = (seg_kt0 == 0) && (kt == p.n_kt - 1);
      if (whole) {
        gemv_epilogue<M, EPI>(p, rt, outb, rs, pre_of(rt), base_pos, rpos, rreq, dt, 0, M);
        if constexpr (EPI == Epi::ARGMAX) gemv_argmax_finish(p, rreq, dt, p.n_rt, 0, M);
      } else {
        const int slot = 2 * c + (rt == rt_first ? 0 : 1);
        float* dstp = p.partials + static_cast<size_t>(slot) * (kMaxRows * kTileN);
        for (int idx = dt; idx < M * kTileN; idx += kDrainThreads) __stcg(dstp + idx, outb[idx]);
        // Release / acquire through the tile's ticket: the CTA barrier orders every drain thread's
        // partial stores before thread 0's acq_rel atomic, and the barrier after it orders the
        // owner's loads after its acquire (no per-thread fences).
        drain_sync();
        const int c_first = unit_owner(rt * p.n_kt, p.units, G);
        const int c_last = unit_owner(rt * p.n_kt + p.n_kt - 1, p.units, G);
        if (dt == 0) {
          const unsigned prev = atom_add_acq_rel_gpu(&p.counters[rt], 1u);
          flag[0] = (prev == static_cast<unsigned>(c_last - c_first)) ? 1 : 0;
        }
        drain_sync();
        if (flag[0]) {
          // Sum the partials in CTA order, all rows at once.  Every CTA after c_first starts its
          // range inside this tile (slot 2 cc); c_first's slot depends on whether the tile is its
          // first one.  When this is the CTA's last segment its weight ring is idle (every MMA
          // has completed), so all partials land there with one round of 16-byte asynchronous
          // copies; otherwise 16 CTAs' 16-byte loads are kept in flight per round.
          const int nsp = c_last - c_first + 1;
          const int slot0 = 2 * c_first + (unit_begin(c_first, p.units, G) / p.n_kt == rt ? 0 : 1);
          const float4* part = reinterpret_cast<const float4*>(p.partials);
          constexpr int kSlotF4 = kMaxRows * kTileN / 4;
          constexpr int kF4 = M * (kTileN / 4);  // float4s of one partial
          if (i == n_units - 1 && nsp * kF4 * 16 <= kStages * static_cast<int>(kWTileBytes)) {
            float4* land = reinterpret_cast<float4*>(smem + S::kW);  // [nsp][kF4]
            for (int t = dt; t < nsp * kF4; t += kDrainThreads) {
              const int k = t / kF4, f = t - k * kF4;
              const int sl = k == 0 ? slot0 : 2 * (c_first + k);
              cp_async16(land + t, part + static_cast<size_t>(sl) * kSlotF4 + f);
            }
            cp_async_commit();
            cp_async_wait_all();
            drain_sync();
            for (int f = dt; f < kF4; f += kDrainThreads) {
              float4 sum = land[f];
              for (int k = 1; k < nsp; ++k) {
                const float4 v = land[k * kF4 + f];
                sum.x += v.x;
                sum.y += v.y;
                sum.z += v.z;
                sum.w += v.w;
              }
              reinterpret_cast<float4*>(outb)[f] = sum;
            }
          } else {
            for (int f = dt; f < kF4; f += kDrainThreads) {
              float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
              for (int b0 = 0; b0 < nsp; b0 += 16) {
                float4 pv[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                  const int k = b0 + j;
                  const int sl = k == 0 ? slot0 : 2 * (c_first + k);
                  pv[j] = k < nsp ? __ldcg(part + static_cast<size_t>(sl) * kSlotF4 + f) : make_float4(0.f, 0.f, 0.f, 0.f);
                }
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                  if (b0 + j >= nsp) continue;
                  if (b0 + j == 0) {
                    sum = pv[j];
                  } else {
                    sum.x += pv[j].x;
                    sum.y += pv[j].y;
                    sum.z += pv[j].z;
                    sum.w += pv[j].w;
                  }
                }
              }
              reinterpret_cast<float4*>(outb)[f] = sum;
            }
          }
          drain_sync();
          gemv_epilogue<M, EPI>(p, rt, outb, rs, pre_of(rt), base_pos, rpos, rreq, dt, 0, M);
          if constexpr (EPI == Epi::ARGMAX) gemv_argmax_finish(p, rreq, dt, p.n_rt, 0, M);
          if (dt == 0) p.counters[rt] = 0u;
        }
      }
      drain_sync();
      seg_kt0 = 0;
      ++sg;
    }
  }
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

}  // namespace ssd
