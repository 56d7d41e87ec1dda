// Per-warp attention state over fixed 16 KB key chunks (Sec. "Methodology": the
// draft and verification passes attend over one shared KV cache).  Used by the
// split-KV decode attention kernel and by the persistent forward kernel.
#pragma once

#include "common.cuh"

namespace ssd {

constexpr int kAttnMaxRows = 9;           // query rows of one call (gamma_max + 1)
constexpr int kAttnChunkBytes = 16384;    // one K (or V) chunk: 32 keys of head_dim 128, 64 of 64

// Attention state of one warp for the query rows of one work item.  Within every
// chunk the warp owns a fixed quarter of the keys (8 of 32 for head_dim 128, 16 of
// 64 for 64): scores with TPK lanes per key (32 dimensions each, summed with a
// fixed xor tree), an online softmax over the warp's keys, and P.V with each lane
// holding DH/32 output dimensions.  The key -> (split, warp) assignment depends on
// key positions only, so every row's result is independent of the number of rows.
template <int DH>
struct AttnWarp {
  static constexpr int KPC = kAttnChunkBytes / (DH * 4);  // keys per chunk
  static constexpr int KPW = KPC / 4;            // keys per warp
  static constexpr int TPK = 32 / KPW;           // lanes per key (4 or 2)
  static constexpr int DPL = DH / 32;            // output dimensions per lane (4 or 2)
  float mx[kAttnMaxRows], l[kAttnMaxRows], o[kAttnMaxRows][DPL];

  __device__ __forceinline__ void init() {
#pragma unroll
    for (int m = 0; m < kAttnMaxRows; ++m) {
      mx[m] = -INFINITY;
      l[m] = 0.f;
#pragma unroll
      for (int e = 0; e < DPL; ++e) o[m][e] = 0.f;
    }
  }

  // Fold the warp's keys of one chunk (K rows Ks, V rows Vs, keys j0 .. j0+nk-1 valid) into the state,
  // for a row count M known at compile time.  The steps run across all rows at once (scores, maxima, exponentials, sums, then P.V), so the
  // shuffle trees of different rows overlap; the probabilities go through pw ([kAttnMaxRows][KPW],
  // this warp's shared scratch) and are read back as broadcasts.
  __device__ __forceinline__ void chunk(const float* Ks, const float* Vs, const float* Qs, int M, int j0, int nk,
                                        int base, float scale, int w, int lane, float* pw) {
    const int kk = lane / TPK, part = lane - kk * TPK, rot = lane & 7;
    const int j = w * KPW + kk;  // this lane's key within the chunk
    const float* kr = Ks + j * DH + part * 32;
    float kv[32];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float4 t = *reinterpret_cast<const float4*>(kr + ((e + rot) & 7) * 4);
      kv[4 * e] = t.x;
      kv[4 * e + 1] = t.y;
      kv[4 * e + 2] = t.z;
      kv[4 * e + 3] = t.w;
    }
    float sc[kAttnMaxRows];
#pragma unroll
    for (int m = 0; m < kAttnMaxRows; ++m) {
      sc[m] = 0.f;
      if (m >= M) continue;
      const float* qr = Qs + m * DH + part * 32;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float4 q = *reinterpret_cast<const float4*>(qr + ((e + rot) & 7) * 4);
        sc[m] = fmaf(kv[4 * e], q.x, sc[m]);
        sc[m] = fmaf(kv[4 * e + 1], q.y, sc[m]);
        sc[m] = fmaf(kv[4 * e + 2], q.z, sc[m]);
        sc[m] = fmaf(kv[4 * e + 3], q.w, sc[m]);
      }
    }
#pragma unroll
    for (int off = 1; off < TPK; off <<= 1)
#pragma unroll
      for (int m = 0; m < kAttnMaxRows; ++m)
        if (m < M) sc[m] += __shfl_xor_sync(0xffffffffu, sc[m], off);
    float cmx[kAttnMaxRows];
#pragma unroll
    for (int m = 0; m < kAttnMaxRows; ++m) {
      const bool vis = j < nk && j0 + j <= base + m;
      sc[m] = vis ? sc[m] * scale : -INFINITY;
      cmx[m] = sc[m];
    }
#pragma unroll
    for (int off = TPK; off < 32; off <<= 1)
#pragma unroll
      for (int m = 0; m < kAttnMaxRows; ++m)
        if (m < M) cmx[m] = fmaxf(cmx[m], __shfl_xor_sync(0xffffffffu, cmx[m], off));
    float cs[kAttnMaxRows];
#pragma unroll
    for (int m = 0; m < kAttnMaxRows; ++m) {
      const float pj = (m < M && sc[m] != -INFINITY) ? expf(sc[m] - cmx[m]) : 0.f;
      if (part == 0 && m < M) pw[m * KPW + kk] = pj;
      cs[m] = part == 0 ? pj : 0.f;
    }
#pragma unroll
    for (int off = 1; off < 32; off <<= 1)
#pragma unroll
      for (int m = 0; m < kAttnMaxRows; ++m)
        if (m < M) cs[m] += __shfl_xor_sync(0xffffffffu, cs[m], off);
    __syncwarp();
    const int d0 = lane * DPL;
    float acc[kAttnMaxRows][DPL];
#pragma unroll
    for (int m = 0; m < kAttnMaxRows; ++m)
#pragma unroll
      for (int e = 0; e < DPL; ++e) acc[m][e] = 0.f;
#pragma unroll
    for (int t = 0; t < KPW; ++t) {
      if (w * KPW + t >= nk) break;  // rows past the chunk's keys hold stale shared memory
      const float* vr = Vs + (w * KPW + t) * DH + d0;
      float vv[DPL];
      if constexpr (DPL == 4) {
        const float4 v4 = *reinterpret_cast<const float4*>(vr);
        vv[0] = v4.x;
        vv[1] = v4.y;
        vv[2] = v4.z;
        vv[3] = v4.w;
      } else {
        const float2 v2 = *reinterpret_cast<const float2*>(vr);
        vv[0] = v2.x;
        vv[1] = v2.y;
      }
#pragma unroll
      for (int m = 0; m < kAttnMaxRows; ++m) {
        if (m >= M) break;
        const float pt = pw[m * KPW + t];
#pragma unroll
        for (int e = 0; e < DPL; ++e) acc[m][e] = fmaf(pt, vv[e], acc[m][e]);
      }
    }
    __syncwarp();  // pw is rewritten by the next chunk
#pragma unroll
    for (int m = 0; m < kAttnMaxRows; ++m) {
      if (m >= M || cmx[m] == -INFINITY) continue;  // no visible key of row m among this warp's keys
      const float nmx = fmaxf(mx[m], cmx[m]);
      const float so = expf(mx[m] - nmx), sn = expf(cmx[m] - nmx);
      l[m] = l[m] * so + cs[m] * sn;
#pragma unroll
      for (int e = 0; e < DPL; ++e) o[m][e] = o[m][e] * so + acc[m][e] * sn;
      mx[m] = nmx;
    }
  }

  // Same fold, one row after another: for a row count known only at run time (the batched
  // form would run every step for all kAttnMaxRows rows).
  __device__ __forceinline__ void chunk_rows(const float* Ks, const float* Vs, const float* Qs, int M, int j0, int nk,
                                        int base, float scale, int w, int lane) {
    const int kk = lane / TPK, part = lane - kk * TPK, rot = lane & 7;
    const int j = w * KPW + kk;  // this lane's key within the chunk
    const float* kr = Ks + j * DH + part * 32;
    float kv[32];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float4 t = *reinterpret_cast<const float4*>(kr + ((e + rot) & 7) * 4);
      kv[4 * e] = t.x;
      kv[4 * e + 1] = t.y;
      kv[4 * e + 2] = t.z;
      kv[4 * e + 3] = t.w;
    }
    const int d0 = lane * DPL;
#pragma unroll
    for (int m = 0; m < kAttnMaxRows; ++m) {
      if (m >= M) break;
      const float* qr = Qs + m * DH + part * 32;
      float sc = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float4 q = *reinterpret_cast<const float4*>(qr + ((e + rot) & 7) * 4);
        sc = fmaf(kv[4 * e], q.x, sc);
        sc = fmaf(kv[4 * e + 1], q.y, sc);
        sc = fmaf(kv[4 * e + 2], q.z, sc);
        sc = fmaf(kv[4 * e + 3], q.w, sc);
      }
#pragma unroll
      for (int off = 1; off < TPK; off <<= 1) sc += __shfl_xor_sync(0xffffffffu, sc, off);
      const bool vis = j < nk && j0 + j <= base + m;
      const float v = vis ? sc * scale : -INFINITY;
      float cmx = v;
#pragma unroll
      for (int off = TPK; off < 32; off <<= 1) cmx = fmaxf(cmx, __shfl_xor_sync(0xffffffffu, cmx, off));
      if (cmx == -INFINITY) continue;  // no visible key of row m among this warp's keys
      const float pj = vis ? expf(v - cmx) : 0.f;
      float csum = part == 0 ? pj : 0.f;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) csum += __shfl_xor_sync(0xffffffffu, csum, off);
      float acc[DPL];
#pragma unroll
      for (int e = 0; e < DPL; ++e) acc[e] = 0.f;
#pragma unroll
      for (int t = 0; t < KPW; ++t) {
        const float pt = __shfl_sync(0xffffffffu, pj, t * TPK);
        if (w * KPW + t >= nk) break;  // rows past the chunk's keys hold stale shared memory
        const float* vr = Vs + (w * KPW + t) * DH + d0;
        if constexpr (DPL == 4) {
          const float4 vv = *reinterpret_cast<const float4*>(vr);
          acc[0] = fmaf(pt, vv.x, acc[0]);
          acc[1] = fmaf(pt, vv.y, acc[1]);
          acc[2] = fmaf(pt, vv.z, acc[2]);
          acc[3] = fmaf(pt, vv.w, acc[3]);
        } else {
          const float2 vv = *reinterpret_cast<const float2*>(vr);
          acc[0] = fmaf(pt, vv.x, acc[0]);
          acc[1] = fmaf(pt, vv.y, acc[1]);
        }
      }
      const float nmx = fmaxf(mx[m], cmx);
      const float so = expf(mx[m] - nmx), sn = expf(cmx - nmx);
      l[m] = l[m] * so + csum * sn;
#pragma unroll
      for (int e = 0; e < DPL; ++e) o[m][e] = o[m][e] * so + acc[e] * sn;
      mx[m] = nmx;
    }
  }
};

}  // namespace ssd
