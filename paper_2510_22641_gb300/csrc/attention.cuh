// Split-KV decode attention over the shared KV cache, causal over a block of
// M query rows (Sec. "Methodology", KV cache: draft and verify read one cache).
//
// Row m sits at position base + m (base = st->kv_len + pos_off) and attends
// to keys 0 .. base + m.  Keys are cut into fixed 64-key chunks at absolute
// positions; one warp handles one (head, chunk) item for all M rows, writes a
// partial (running max, sum of exp, unnormalised output), and the warp that
// finishes the head's last item combines the partials in chunk order.
// Chunk boundaries and the combine order do not depend on M, so each row's
// output equals the single-row (M = 1) result bitwise.
#pragma once

#include "common.cuh"

namespace ssd {

constexpr int kAttnChunk = 64;
constexpr int kAttnWarps = 4;

struct AttnParams {
  const float* q;  // [M][q_stride], rotated queries
  int q_stride;
  const __nv_bfloat16* k_cache;  // this layer's [H][max_seq][Dh]
  const __nv_bfloat16* v_cache;
  float* o;  // [M][o_stride]
  int o_stride;
  float* part;          // [H][max_chunks][kMaxRows][Dh + 4]
  unsigned* counters;   // [H]
  DevState* st;
  int pos_off;
  int n_heads, max_seq, max_chunks;
  float scale;  // 1/sqrt(Dh)
};

template <int M, int DH>
__global__ void __launch_bounds__(kAttnWarps * 32) attn_kernel(const AttnParams p) {
  constexpr int PER = DH / 32;       // output dims per lane
  constexpr int PS = DH + 4;         // partial record stride (floats)
  __shared__ __align__(16) float q_s[kAttnWarps][M][DH];
  pdl_trigger();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (__ldcg(&p.st->error) & DERR_TIMEOUT) return;
  const int base = __ldcg(&p.st->kv_len) + p.pos_off;
  const int n_keys = base + M;  // keys 0 .. base+M-1 exist for the last row
  if (base < 0 || n_keys > p.max_seq) {
    if (threadIdx.x == 0 && blockIdx.x == 0) set_error(p.st, DERR_POS);
    return;
  }
  const int n_chunks = (n_keys + kAttnChunk - 1) / kAttnChunk;
  const int items = p.n_heads * n_chunks;
  const int gw = blockIdx.x * kAttnWarps + warp, nw = gridDim.x * kAttnWarps;

  for (int item = gw; item < items; item += nw) {
    const int h = item / n_chunks, c = item - h * n_chunks;
#pragma unroll
    for (int m = 0; m < M; ++m)
      for (int d = lane; d < DH; d += 32) q_s[warp][m][d] = __ldcg(p.q + m * p.q_stride + h * DH + d);
    __syncwarp();

    const int j0 = c * kAttnChunk;
    const int jA = j0 + lane, jB = j0 + 32 + lane;
    const bool inA = jA < n_keys, inB = jB < n_keys;
    const __nv_bfloat16* kbase = p.k_cache + static_cast<size_t>(h) * p.max_seq * DH;
    const uint4* kA = reinterpret_cast<const uint4*>(kbase + static_cast<size_t>(inA ? jA : 0) * DH);
    const uint4* kB = reinterpret_cast<const uint4*>(kbase + static_cast<size_t>(inB ? jB : 0) * DH);

    float sA[M], sB[M];
#pragma unroll
    for (int m = 0; m < M; ++m) sA[m] = sB[m] = 0.f;
#pragma unroll 4
    for (int d8 = 0; d8 < DH / 8; ++d8) {
      const uint4 ka = inA ? __ldcg(kA + d8) : make_uint4(0, 0, 0, 0);
      const uint4 kb = inB ? __ldcg(kB + d8) : make_uint4(0, 0, 0, 0);
      const float2 a0 = bf16x2_to_float2(ka.x), a1 = bf16x2_to_float2(ka.y), a2 = bf16x2_to_float2(ka.z),
                   a3 = bf16x2_to_float2(ka.w);
      const float2 b0 = bf16x2_to_float2(kb.x), b1 = bf16x2_to_float2(kb.y), b2 = bf16x2_to_float2(kb.z),
                   b3 = bf16x2_to_float2(kb.w);
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const float4 q0 = *reinterpret_cast<const float4*>(&q_s[warp][m][d8 * 8]);
        const float4 q1 = *reinterpret_cast<const float4*>(&q_s[warp][m][d8 * 8 + 4]);
        float s = sA[m];
        s = fmaf(a0.x, q0.x, s); s = fmaf(a0.y, q0.y, s); s = fmaf(a1.x, q0.z, s); s = fmaf(a1.y, q0.w, s);
        s = fmaf(a2.x, q1.x, s); s = fmaf(a2.y, q1.y, s); s = fmaf(a3.x, q1.z, s); s = fmaf(a3.y, q1.w, s);
        sA[m] = s;
        float t = sB[m];
        t = fmaf(b0.x, q0.x, t); t = fmaf(b0.y, q0.y, t); t = fmaf(b1.x, q0.z, t); t = fmaf(b1.y, q0.w, t);
        t = fmaf(b2.x, q1.x, t); t = fmaf(b2.y, q1.y, t); t = fmaf(b3.x, q1.z, t); t = fmaf(b3.y, q1.w, t);
        sB[m] = t;
      }
    }

    // softmax statistics of this chunk, per row (keys beyond the row's position masked)
    float pA[M], pB[M], mxv[M], lv[M];
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const bool vA = jA <= base + m, vB = jB <= base + m;
      const float a = vA ? sA[m] * p.scale : -INFINITY;
      const float b = vB ? sB[m] * p.scale : -INFINITY;
      float mx = fmaxf(a, b);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      float ea = 0.f, eb = 0.f;
      if (mx != -INFINITY) {
        ea = vA ? expf(a - mx) : 0.f;
        eb = vB ? expf(b - mx) : 0.f;
      }
      float l = ea + eb;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
      pA[m] = ea;
      pB[m] = eb;
      mxv[m] = mx;
      lv[m] = l;
    }

    // unnormalised P.V over the chunk's keys, lane owns dims lane*PER ..
    float oacc[M][PER];
#pragma unroll
    for (int m = 0; m < M; ++m)
#pragma unroll
      for (int e = 0; e < PER; ++e) oacc[m][e] = 0.f;
    const int nk = min(kAttnChunk, n_keys - j0);
    const __nv_bfloat16* vbase = p.v_cache + (static_cast<size_t>(h) * p.max_seq + j0) * DH + lane * PER;
#pragma unroll 4
    for (int t = 0; t < nk; ++t) {
      float v[PER];
      if constexpr (PER == 4) {
        const uint2 raw = __ldcg(reinterpret_cast<const uint2*>(vbase + static_cast<size_t>(t) * DH));
        const float2 v0 = bf16x2_to_float2(raw.x), v1 = bf16x2_to_float2(raw.y);
        v[0] = v0.x; v[1] = v0.y; v[2] = v1.x; v[3] = v1.y;
      } else {
        const uint32_t raw = __ldcg(reinterpret_cast<const unsigned int*>(vbase + static_cast<size_t>(t) * DH));
        const float2 v0 = bf16x2_to_float2(raw);
        v[0] = v0.x; v[1] = v0.y;
      }
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const float pm = __shfl_sync(0xffffffffu, t < 32 ? pA[m] : pB[m], t & 31);
#pragma unroll
        for (int e = 0; e < PER; ++e) oacc[m][e] = fmaf(pm, v[e], oacc[m][e]);
      }
    }

    float* rec = p.part + (static_cast<size_t>(h) * p.max_chunks + c) * kMaxRows * PS;
#pragma unroll
    for (int m = 0; m < M; ++m) {
#pragma unroll
      for (int e = 0; e < PER; ++e) __stcg(rec + m * PS + 4 + lane * PER + e, oacc[m][e]);
      if (lane == 0) {
        __stcg(rec + m * PS, mxv[m]);
        __stcg(rec + m * PS + 1, lv[m]);
      }
    }
    __threadfence();
    __syncwarp();
    unsigned prev = 0;
    if (lane == 0) prev = atomicAdd(&p.counters[h], 1u);
    prev = __shfl_sync(0xffffffffu, prev, 0);
    if (prev == static_cast<unsigned>(n_chunks - 1)) {
      // last item of head h: combine the chunks in order
      __threadfence();
      const float* hrec = p.part + static_cast<size_t>(h) * p.max_chunks * kMaxRows * PS;
#pragma unroll 1
      for (int m = 0; m < M; ++m) {
        float mt = -INFINITY;
        for (int cc = 0; cc < n_chunks; ++cc) mt = fmaxf(mt, __ldcg(hrec + (cc * kMaxRows + m) * PS));
        float L = 0.f, O[PER];
#pragma unroll
        for (int e = 0; e < PER; ++e) O[e] = 0.f;
        for (int cc = 0; cc < n_chunks; ++cc) {
          const float* r = hrec + (cc * kMaxRows + m) * PS;
          const float mc = __ldcg(r);
          if (mc == -INFINITY) continue;
          const float w = expf(mc - mt);
          L = fmaf(w, __ldcg(r + 1), L);
#pragma unroll
          for (int e = 0; e < PER; ++e) O[e] = fmaf(w, __ldcg(r + 4 + lane * PER + e), O[e]);
        }
        const float inv = 1.0f / L;
#pragma unroll
        for (int e = 0; e < PER; ++e) p.o[m * p.o_stride + h * DH + lane * PER + e] = O[e] * inv;
      }
      if (lane == 0) p.counters[h] = 0u;
    }
    __syncwarp();
  }
}

}  // namespace ssd
