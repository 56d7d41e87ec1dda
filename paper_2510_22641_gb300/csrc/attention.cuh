// Split-KV decode attention over the shared KV cache, causal over a block of
// M query rows (Sec. "Methodology", KV cache: draft and verify read one cache).
//
// Row m sits at position base + m (base = st->kv_len + pos_off) and attends
// to keys 0 .. base + m.  Keys are cut into fixed 16 KB chunks at absolute
// positions (32 keys for head_dim 128, 64 for 64).  Each head is served by one
// thread-block cluster of kAttnSplit CTAs; CTA r of the cluster takes chunks r,
// r + kAttnSplit, ... in order: thread 0 brings each chunk's K and V rows
// (contiguous in the [H][max_seq][Dh] fp32 cache) into shared memory with bulk
// copies, double-buffered.  Within a chunk, each of the 4 warps owns a fixed
// quarter of the keys and folds them into its own running softmax state per row
// (max, sum of exp, unnormalised output), so a chunk costs one CTA barrier.  The
// cluster then merges the 4 x kAttnSplit states through distributed shared
// memory, each CTA a slice of the output columns, in (CTA, warp) order.  The chunk grid, the key -> (CTA, warp)
// assignment and the merge order depend only on key positions, never on M, so
// each row's output equals the single-row (M = 1) result bitwise.
#pragma once

#include <cooperative_groups.h>

#include "attn_warp.cuh"

namespace ssd {

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
  static constexpr int kKV = kAttnChunkBytes;                       // one K (or V) chunk
  static constexpr int kQ = 0;                                      // q rows [M][DH]
  static constexpr int kBuf0 = (kQ + M * DH * 4 + 15) & ~15;        // two {K, V} buffers
  static constexpr int kFin = kBuf0 + 4 * kKV;                      // warp states [4][M][DH + 2]
  static constexpr int kPw = kFin + 4 * M * (DH + 2) * 4;           // per-warp probabilities [4][rows][KPW]
  static constexpr int kWq = kPw + 4 * kAttnMaxRows * (AttnWarp<DH>::KPW) * 4;  // merge weights [M][32], sums [M]
  static constexpr int kBar = (kWq + M * 33 * 4 + 7) & ~7;
  static constexpr int kTotal = kBar + 3 * 8;
};

template <int M, int DH>
__global__ void __cluster_dims__(kAttnSplit, 1, 1) __launch_bounds__(kAttnThreads)
    attn_kernel(const AttnParams p) {
  namespace cg = cooperative_groups;
  using S = AttnSmem<M, DH>;
  using AW = AttnWarp<DH>;
  constexpr int KPC = AW::KPC, DPL = AW::DPL;
  static_assert(M <= kAttnMaxRows, "query rows");
  extern __shared__ __align__(128) uint8_t smem[];
  float* Qs = reinterpret_cast<float*>(smem + S::kQ);
  float* fin = reinterpret_cast<float*>(smem + S::kFin);
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + S::kBar);
  cg::cluster_group cluster = cg::this_cluster();
  const int tid = threadIdx.x, w = tid >> 5, lane = tid & 31;
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
  const int n_chunks = (n_keys + KPC - 1) / KPC;
  const int my_chunks = n_chunks > rank ? (n_chunks - rank + kAttnSplit - 1) / kAttnSplit : 0;

  auto issue = [&](int buf, int c) {
    const int j0 = c * KPC, nk = min(KPC, n_keys - j0);
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

  AW st;
  st.init();
  bool ok = true;
  if (my_chunks > 0 && !mbar_wait(&bar[2], 0)) ok = false;
  for (int i = 0; ok && i < my_chunks; ++i) {
    const int c = rank + i * kAttnSplit, buf = i & 1;
    const int j0 = c * KPC, nk = min(KPC, n_keys - j0);
    if (tid == 0 && i + 1 < my_chunks) issue(buf ^ 1, c + kAttnSplit);
    if (!mbar_wait(&bar[buf], static_cast<uint32_t>(i >> 1) & 1u)) {
      ok = false;
      break;
    }
    const float* Ks = reinterpret_cast<const float*>(smem + S::kBuf0 + buf * 2 * S::kKV);
    st.chunk(Ks, Ks + KPC * DH, Qs, M, j0, nk, base, p.scale, w, lane,
             reinterpret_cast<float*>(smem + S::kPw) + w * kAttnMaxRows * AW::KPW);
    __syncthreads();  // buffer buf is refilled by the next iteration's copy
  }
  if (!ok) set_error(p.st, DERR_TIMEOUT);

  // publish the warps' states; the cluster then merges the 4 x kAttnSplit states of each row.
  // State s = 4 * CTA + warp.  Per row, one warp forms the weights exp(mx_s - max) and their sum
  // with fixed shuffle trees; then CTA r combines columns [r * DH / kAttnSplit, (r + 1) * DH /
  // kAttnSplit) of all rows, summing the states in s order.  None of it depends on M.
#pragma unroll
  for (int m = 0; m < M; ++m) {
    float* e = fin + (w * M + m) * (DH + 2);
#pragma unroll
    for (int d = 0; d < DPL; ++d) e[lane * DPL + d] = st.o[m][d];
    if (lane == 0) {
      e[DH] = st.mx[m];
      e[DH + 1] = st.l[m];
    }
  }
  cluster.sync();
  static_assert(4 * kAttnSplit == 32, "one merge lane per state");
  if (!bad) {
    float* wq = reinterpret_cast<float*>(smem + S::kWq);  // [M][32]
    float* ls = wq + M * 32;                              // [M]
    const float* fs = cluster.map_shared_rank(fin, lane >> 2);
    for (int m = w; m < M; m += 4) {
      const float* e = fs + ((lane & 3) * M + m) * (DH + 2);
      const float mq = e[DH], lq = e[DH + 1];
      float mt = mq;
#pragma unroll
      for (int o = 16; o; o >>= 1) mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, o));
      const float g = mq == -INFINITY ? 0.f : expf(mq - mt);
      float L = g * lq;
#pragma unroll
      for (int o = 16; o; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
      wq[m * 32 + lane] = g;
      if (lane == 0) ls[m] = L;
    }
    __syncthreads();
    constexpr int DS = DH / kAttnSplit;
    for (int idx = tid; idx < M * DS; idx += kAttnThreads) {
      const int m = idx / DS, d = rank * DS + (idx - m * DS);
      float v[32];
#pragma unroll
      for (int s = 0; s < 32; ++s)
        v[s] = cluster.map_shared_rank(fin, s >> 2)[((s & 3) * M + m) * (DH + 2) + d];
      float O = 0.f;
#pragma unroll
      for (int s = 0; s < 32; ++s) O = fmaf(wq[m * 32 + s], v[s], O);
      const float L = ls[m];
      p.o[m * p.o_stride + h * DH + d] = L > 0.f ? O / L : 0.f;
    }
  }
  cluster.sync();  // keep every CTA's shared memory alive until rank 0 has read it
}

}  // namespace ssd
