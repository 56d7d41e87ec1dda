// Split-KV decode attention over the shared KV cache, causal over a block of
// M query rows (Sec. "Methodology", KV cache: draft and verify read one cache).
//
// Row m sits at position base + m (base = st->kv_len + pos_off) and attends
// to keys 0 .. base + m.  Keys are cut into fixed 32-key chunks at absolute
// positions.  Each head is served by one thread-block cluster of kAttnSplit
// CTAs; CTA r of the cluster takes chunks r, r + kAttnSplit, ... in order:
// thread 0 brings each chunk's K and V rows (contiguous in the [H][max_seq][Dh]
// fp32 cache) into shared memory with bulk copies, double-buffered, and the
// CTA folds the chunk into a running softmax state per row (max, sum of exp,
// unnormalised output).  The cluster then merges its kAttnSplit states through
// distributed shared memory in rank order.  The chunk grid, the per-CTA chunk
// order and the merge order depend only on key positions, never on M, so each
// row's output equals the single-row (M = 1) result bitwise.
#pragma once

#include <cooperative_groups.h>

#include "common.cuh"

namespace ssd {

constexpr int kAttnChunk = 32;
constexpr int kAttnThreads = 128;
constexpr int kAttnSplit = 8;  // CTAs per head (cluster size)

struct AttnParams {
  const float* q;  // [M][q_stride], rotated queries
  int q_stride;
  const float* k_cache;  // this layer's [H][max_seq][Dh], fp32
  const float* v_cache;
  float* o;  // [M][o_stride]
  int o_stride;
  DevState* st;
  int pos_off;
  int n_heads, max_seq;
  float scale;  // 1/sqrt(Dh)
};

template <int M, int DH>
struct AttnSmem {
  static constexpr int kKV = kAttnChunk * DH * 4;         // one K (or V) chunk
  static constexpr int kQ = 0;                            // q rows [M][DH]
  static constexpr int kBuf0 = kQ + M * DH * 4;           // two {K, V} buffers
  static constexpr int kP = kBuf0 + 4 * kKV;              // probabilities [M][32]
  static constexpr int kCs = kP + M * kAttnChunk * 4;     // chunk max / sum [2][M]
  static constexpr int kFin = kCs + 2 * kMaxRows * 4;     // final state: mx[M], l[M], o[M][DH]
  static constexpr int kBar = (kFin + (2 * M + M * DH) * 4 + 7) & ~7;
  static constexpr int kTotal = kBar + 3 * 8;
};

template <int M, int DH>
__global__ void __cluster_dims__(kAttnSplit, 1, 1) __launch_bounds__(kAttnThreads)
    attn_kernel(const AttnParams p) {
  namespace cg = cooperative_groups;
  using S = AttnSmem<M, DH>;
  constexpr int GROUPS = kAttnThreads / DH;  // row groups in P.V: 1 (Dh 128) or 2 (Dh 64)
  constexpr int RPG = (M + GROUPS - 1) / GROUPS;
  extern __shared__ __align__(128) uint8_t smem[];
  float* Qs = reinterpret_cast<float*>(smem + S::kQ);
  float* Ps = reinterpret_cast<float*>(smem + S::kP);
  float* cs = reinterpret_cast<float*>(smem + S::kCs);
  float* fin = reinterpret_cast<float*>(smem + S::kFin);
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + S::kBar);
  cg::cluster_group cluster = cg::this_cluster();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rank = static_cast<int>(cluster.block_rank());
  const int h = blockIdx.y;

  pdl_trigger();
  if (tid == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    mbar_init(&bar[2], 1);
    fence_mbar_init();
  }
  __syncthreads();
  pdl_wait();
  int base = __ldcg(&p.st->kv_len) + p.pos_off;
  bool bad = (__ldcg(&p.st->error) & DERR_TIMEOUT) != 0;
  if (base < 0 || base + M > p.max_seq) {
    if (tid == 0 && rank == 0 && h == 0) set_error(p.st, DERR_POS);
    bad = true;
  }
  const int n_keys = bad ? 0 : base + M;  // keys 0 .. base+M-1 exist for the last row
  const int n_chunks = (n_keys + kAttnChunk - 1) / kAttnChunk;
  const int my_chunks = n_chunks > rank ? (n_chunks - rank + kAttnSplit - 1) / kAttnSplit : 0;

  auto issue = [&](int buf, int c) {
    const int j0 = c * kAttnChunk, nk = min(kAttnChunk, n_keys - j0);
    uint8_t* b = smem + S::kBuf0 + buf * 2 * S::kKV;
    const uint32_t kv_bytes = static_cast<uint32_t>(nk * DH * 4);
    mbar_arrive_expect_tx(&bar[buf], 2 * kv_bytes);
    const size_t off = (static_cast<size_t>(h) * p.max_seq + j0) * DH;
    bulk_load(b, p.k_cache + off, kv_bytes, &bar[buf]);
    bulk_load(b + S::kKV, p.v_cache + off, kv_bytes, &bar[buf]);
  };
  if (tid == 0 && my_chunks > 0) {
    mbar_arrive_expect_tx(&bar[2], M * DH * 4);
#pragma unroll
    for (int m = 0; m < M; ++m)
      bulk_load(Qs + m * DH, p.q + static_cast<size_t>(m) * p.q_stride + h * DH, DH * 4, &bar[2]);
    issue(0, rank);
  }

  // running state: thread (d, g) owns o[m][d] for m = g, g + GROUPS, ...; row stats kept per thread
  const int d = tid % DH, g = tid / DH;
  float o_run[RPG], mx_run[RPG], l_run[RPG];
#pragma unroll
  for (int r = 0; r < RPG; ++r) {
    o_run[r] = 0.f;
    mx_run[r] = -INFINITY;
    l_run[r] = 0.f;
  }
  bool ok = true;
  if (my_chunks > 0 && !mbar_wait(&bar[2], 0)) ok = false;

  for (int i = 0; ok && i < my_chunks; ++i) {
    const int c = rank + i * kAttnSplit, buf = i & 1;
    const int j0 = c * kAttnChunk, nk = min(kAttnChunk, n_keys - j0);
    if (tid == 0 && i + 1 < my_chunks) issue(buf ^ 1, c + kAttnSplit);
    if (!mbar_wait(&bar[buf], static_cast<uint32_t>(i >> 1) & 1u)) {
      ok = false;
      break;
    }
    const float* Ks = reinterpret_cast<const float*>(smem + S::kBuf0 + buf * 2 * S::kKV);
    const float* Vs = Ks + kAttnChunk * DH;

    // scores of the chunk: warp w, lane j -> key j, rows m = w, w+4, w+8 (columns read in a rotated order)
    {
      const int j = lane;
      const bool have = j < nk;
      for (int m = warp; m < M; m += 4) {
        float s = 0.f;
        if (have) {
          const float* kr = Ks + j * DH;
          const float* qr = Qs + m * DH;
#pragma unroll 8
          for (int t = 0; t < DH / 4; ++t) {
            const int c4 = ((t + j) & (DH / 4 - 1)) * 4;
            const float4 kv = *reinterpret_cast<const float4*>(kr + c4);
            const float4 qv = *reinterpret_cast<const float4*>(qr + c4);
            s = fmaf(kv.x, qv.x, s);
            s = fmaf(kv.y, qv.y, s);
            s = fmaf(kv.z, qv.z, s);
            s = fmaf(kv.w, qv.w, s);
          }
        }
        const bool vis = have && (j0 + j <= base + m);
        const float v = vis ? s * p.scale : -INFINITY;
        float mx = v;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        const float e = (vis && mx != -INFINITY) ? expf(v - mx) : 0.f;
        float l = e;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
        Ps[m * kAttnChunk + j] = e;
        if (lane == 0) {
          cs[m] = mx;
          cs[kMaxRows + m] = l;
        }
      }
    }
    __syncthreads();
    // chunk P.V and merge into the running state (chunks in increasing position)
#pragma unroll
    for (int r = 0; r < RPG; ++r) {
      const int m = g + r * GROUPS;
      if (m >= M) continue;
      float acc = 0.f;
      for (int j = 0; j < nk; ++j) acc = fmaf(Ps[m * kAttnChunk + j], Vs[j * DH + d], acc);
      const float cmx = cs[m];
      if (cmx == -INFINITY) continue;  // no visible key of row m in this chunk
      const float nmx = fmaxf(mx_run[r], cmx);
      const float so = expf(mx_run[r] - nmx), sc = expf(cmx - nmx);
      l_run[r] = l_run[r] * so + cs[kMaxRows + m] * sc;
      o_run[r] = o_run[r] * so + acc * sc;
      mx_run[r] = nmx;
    }
    __syncthreads();  // buffers and Ps/cs are rewritten by the next chunk
  }
  if (!ok) set_error(p.st, DERR_TIMEOUT);

  // publish this CTA's state, then rank 0 merges the cluster's states in rank order
#pragma unroll
  for (int r = 0; r < RPG; ++r) {
    const int m = g + r * GROUPS;
    if (m >= M) continue;
    fin[2 * M + m * DH + d] = o_run[r];
    if (d == 0) {
      fin[m] = mx_run[r];
      fin[M + m] = l_run[r];
    }
  }
  cluster.sync();
  if (rank == 0 && !bad) {
#pragma unroll
    for (int r = 0; r < RPG; ++r) {
      const int m = g + r * GROUPS;
      if (m >= M) continue;
      float mt = -INFINITY;
      for (int q = 0; q < kAttnSplit; ++q) mt = fmaxf(mt, cluster.map_shared_rank(fin, q)[m]);
      float L = 0.f, O = 0.f;
      for (int q = 0; q < kAttnSplit; ++q) {
        const float* f = cluster.map_shared_rank(fin, q);
        const float mq = f[m];
        if (mq == -INFINITY) continue;
        const float w = expf(mq - mt);
        L = fmaf(w, f[M + m], L);
        O = fmaf(w, f[2 * M + m * DH + d], O);
      }
      p.o[m * p.o_stride + h * DH + d] = O / L;
    }
  }
  cluster.sync();  // keep every CTA's shared memory alive until rank 0 has read it
}

}  // namespace ssd
