// Split-KV decode attention over the shared KV cache, causal over a block of
// M query rows (Sec. "Methodology", KV cache: draft and verify read one cache).
//
// Row m sits at position base + m (base = st->kv_len + pos_off) and attends
// to keys 0 .. base + m.  Keys are cut into fixed 16 KB chunks at absolute
// positions (32 keys for head_dim 128, 64 for 64).  Each head is served by
// kAttnSplit CTAs; CTA r of the head takes chunks r, r + kAttnSplit, ... in
// order, in groups of kAttnBufs chunks: thread 0 brings a
// group's K and V rows (contiguous in the [H][max_seq][Dh] fp32 cache) into
// shared memory with bulk copies.  Per group the CTA
//   1. scores every key of the group for every row (warp w owns a fixed 1/8 of
//      each chunk's keys, TPK lanes per key with a fixed xor tree),
//   2. updates each row's running max and sum once for the whole group (one warp
//      per row; exponentials written back in place of the scores),
//   3. folds P.V into the warps' output accumulators, rescaled by the row's
//      running-max change.
// All warps share one running max per row, so the CTA's state is the warps'
// accumulators summed in warp order.  Each CTA stores its state and takes the
// head's ticket (one acq_rel atomic after a CTA barrier); the CTA that completes
// the count merges the kAttnSplit states in CTA order and writes the head's
// output, so the other CTAs leave without waiting for each other.  When all of
// a head's keys fit one chunk (short caches: the encoder-decoder's decoder,
// early positions) CTA 0 holds the whole state and writes the output itself,
// with no state store, ticket or merge: the merge would return that state's
// O / L unchanged, so the result is the same bits.  The chunk
// grid, the grouping, the key -> (CTA, warp)
// assignment and every summation order depend only on key positions, never on
// M, so each row's output equals the single-row (M = 1) result bitwise.
//
// Batched requests (batch_rows > 0) add a grid dimension: blockIdx.z is the
// request z, whose M rows are rows z*M .. z*M+M-1 of q and o, whose keys are
// its own cache rows (k_cache / v_cache + z * req_kv) and whose base is
// req_st[z].kv_len + pos_off; requests never share a CTA, a state or a ticket.
// A request that is done reads no keys (its output rows are zero and unused).
//
// With prefetch_old set, the launch before this one triggered its dependents
// only after its own upstream grid had completed, so everything older than that
// launch is complete here: the chunks holding only keys below base (written by
// earlier launches) are fetched before the wait on the upstream grid, and only
// q and the chunk with this step's keys after it.
#pragma once

#include "common.cuh"

namespace ssd {

constexpr int kAttnMaxRows = SSD_MAX_GAMMA + 1;  // query rows per request of one call (gamma_max + 1)
constexpr int kAttnChunkBytes = 16384;    // one K (or V) chunk: 32 keys of head_dim 128, 64 of 64
constexpr int kAttnWarps = 8;
constexpr int kAttnThreads = 32 * kAttnWarps;
constexpr int kAttnSplit = 8;  // CTAs per head
constexpr int kAttnBufs = 3;   // chunks per group = {K, V} buffers per CTA

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
  float scale;       // 1/sqrt(Dh)
  int prefetch_old;  // the previous launch triggered after its own upstream completed (see above)
  float* part;        // [requests][n_heads][kAttnSplit][kAttnMaxRows][Dh + 2] CTA states (output, max, sum)
  unsigned* tickets;  // [requests][n_heads], zero between launches
  // Non-causal key sets and relative-position bias (encoder-decoder models; read only by the EXT
  // instantiations, so the causal kernels compile without them):
  int fixed_keys;     // 1: keys 0 .. st->enc_len - 1, every one visible to every row (cross-attention,
                      // bidirectional encoder self-attention); 0: causal over the cache (above)
  int abs_pos;        // row m sits at position pos_off + m (st->kv_len ignored): the encoder's rows
  const float* bias;  // null, or [n_heads][bias_stride]: score(row at i, key j) += bias[h][j - i + bias_zero]
  int bias_stride, bias_zero;
  // Batched requests (0: one request; else the rows per request, = M): see the header.
  int batch_rows;
  const DevState* req_st;
  long long req_kv;
  // Null, or the merged output rows also go out as bf16 hi / lo parts, [request * M + row][xo_ld]
  // (the medium-M o projection's operand, so it needs no split launch of its own).
  __nv_bfloat16* xo_hi;
  __nv_bfloat16* xo_lo;
  int xo_ld;
};

template <int DH>
struct AttnGeo {
  static constexpr int KPC = kAttnChunkBytes / (DH * 4);  // keys per chunk (32 or 64)
  static constexpr int KPW = KPC / kAttnWarps;            // keys per warp and chunk (4 or 8)
  static constexpr int TPK = 32 / KPW;                    // lanes per key (8 or 4)
  static constexpr int DPP = DH / TPK;                    // key dimensions per lane in the scores
  static constexpr int NF = DPP / 4;                      // 16-byte loads per lane and row
  static constexpr int DPL = DH / 32;                     // output dimensions per lane (4 or 2)
  static constexpr int GK = kAttnBufs * KPC;              // keys per group
  static constexpr int KPL = GK / 32;                     // keys per lane in the row statistics
  static_assert(NF == 4 && KPW % 4 == 0 && KPW * kAttnWarps == KPC && GK % 32 == 0, "chunk split");
};

template <int M, int DH>
struct AttnSmem {
  using G = AttnGeo<DH>;
  static constexpr int kKV = kAttnChunkBytes;                    // one K (or V) chunk
  static constexpr int kQ = 0;                                   // q rows [M][DH]
  static constexpr int kBuf0 = (kQ + M * DH * 4 + 127) & ~127;   // kAttnBufs {K, V} buffers
  static constexpr int kWs = kBuf0;  // warp accumulators [kAttnWarps][M][DH], over the buffers after the last group
  static_assert(kAttnWarps * M * DH * 4 <= kAttnBufs * 2 * kKV, "warp accumulators fit the chunk buffers");
  static constexpr int kS = kBuf0 + kAttnBufs * 2 * kKV;         // scores, then probabilities [M][GK]
  static constexpr int kRow = kS + M * G::GK * 4;                // per row: running max, sum, rescale, - [M][4]
  static constexpr int kWq = kRow + M * 4 * 4;                   // merge weights [M][kAttnSplit], totals [M]
  static constexpr int kFlag = kWq + M * (kAttnSplit + 1) * 4;   // last-CTA flag
  static constexpr int kBar = (kFlag + 4 + 7) & ~7;
  static constexpr int kTotal = kBar + (kAttnBufs + 1) * 8;
};

// Up to 9 rows two CTAs share an SM; beyond that one CTA holds the larger q rows and accumulators.
template <int M, int DH, bool EXT>
__global__ void __launch_bounds__(kAttnThreads, M <= 9 ? 2 : 1) ssd_splitkv_attn_kernel(const AttnParams p) {
  using S = AttnSmem<M, DH>;
  using G = AttnGeo<DH>;
  constexpr int KPC = G::KPC, KPW = G::KPW, TPK = G::TPK, DPP = G::DPP, NF = G::NF, DPL = G::DPL;
  constexpr int GK = G::GK, E = DH + 2;
  static_assert(M <= kAttnMaxRows, "query rows");
  extern __shared__ __align__(128) uint8_t smem[];
  float* Qs = reinterpret_cast<float*>(smem + S::kQ);
  float* ss = reinterpret_cast<float*>(smem + S::kS);
  float* rowst = reinterpret_cast<float*>(smem + S::kRow);
  float* ws = reinterpret_cast<float*>(smem + S::kWs);
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + S::kBar);  // [kAttnBufs] chunks, then q
  const int tid = threadIdx.x, w = tid >> 5, lane = tid & 31;
  const int rank = blockIdx.x;
  const int h = blockIdx.y;
  const int z = blockIdx.z;  // request (0 for one request)
  const float* k_cache = p.k_cache + z * p.req_kv;
  const float* v_cache = p.v_cache + z * p.req_kv;
  const float* q_rows = p.q + static_cast<size_t>(z) * M * p.q_stride;
  float* o_rows = p.o + static_cast<size_t>(z) * M * p.o_stride;

  pdl_trigger();
  if (tid == 0) {
    for (int b = 0; b <= kAttnBufs; ++b) mbar_init(&bar[b], 1);
    fence_mbar_init();
  }
  if (tid < M) {
    rowst[4 * tid] = -INFINITY;
    rowst[4 * tid + 1] = 0.f;
  }
  __syncthreads();

  int base = 0, n_keys = 0, my_chunks = 0;
  bool bad = false;
  auto geometry = [&]() {
    base = ((EXT && p.abs_pos) ? 0 : __ldcg(p.batch_rows ? &p.req_st[z].kv_len : &p.st->kv_len)) + p.pos_off;
    if (p.batch_rows && __ldcg(&p.req_st[z].done)) {  // a finished request's rows are never used
      n_keys = my_chunks = 0;
      return;
    }
    if (EXT && p.fixed_keys) {
      const int ne = __ldcg(&p.st->enc_len);
      bad = base < 0 || ne < 1 || ne > p.max_seq;
      n_keys = bad ? 0 : ne;
    } else {
      bad = base < 0 || base + M > p.max_seq;
      n_keys = bad ? 0 : base + M;  // keys 0 .. base+M-1 exist for the last row
    }
    const int n_chunks = (n_keys + KPC - 1) / KPC;
    my_chunks = n_chunks > rank ? (n_chunks - rank + kAttnSplit - 1) / kAttnSplit : 0;
  };
  auto issue = [&](int buf, int c) {
    const int j0 = c * KPC, nk = min(KPC, n_keys - j0);
    uint8_t* b = smem + S::kBuf0 + buf * 2 * S::kKV;
    const uint32_t kv_bytes = static_cast<uint32_t>(nk * DH * 4);
    mbar_arrive_expect_tx(&bar[buf], 2 * kv_bytes);
    const size_t off = (static_cast<size_t>(h) * p.max_seq + j0) * DH;
    bulk_load(b, k_cache + off, kv_bytes, &bar[buf]);
    bulk_load(b + S::kKV, v_cache + off, kv_bytes, &bar[buf]);
  };
  int issued = 0;  // thread 0: chunks of the first group already requested
  if (p.prefetch_old) {
    geometry();
    if (tid == 0)
      for (; issued < kAttnBufs && issued < my_chunks; ++issued) {
        const int c = rank + issued * kAttnSplit;
        if ((EXT && p.fixed_keys) || (c + 1) * KPC > base) break;  // holds keys the upstream grid writes
        issue(issued, c);
      }
  }
  pdl_wait();
  if (!p.prefetch_old) geometry();
  if (bad && tid == 0 && rank == 0 && h == 0) set_error(p.st, DERR_POS);
  const bool timed_out = (__ldcg(&p.st->error) & DERR_TIMEOUT) != 0;
  if (tid == 0 && my_chunks > 0) {
    mbar_arrive_expect_tx(&bar[kAttnBufs], M * DH * 4);
#pragma unroll
    for (int m = 0; m < M; ++m)
      bulk_load(Qs + m * DH, q_rows + static_cast<size_t>(m) * p.q_stride + h * DH, DH * 4, &bar[kAttnBufs]);
    for (; issued < kAttnBufs && issued < my_chunks; ++issued) issue(issued, rank + issued * kAttnSplit);
  }

  const int kk = lane / TPK, part = lane - kk * TPK, rot = ((lane & 7) >> 1) & 3;
  const int jw = w * KPW + kk;  // this lane's key within a chunk (scores)
  float acc[M][DPL];
#pragma unroll
  for (int m = 0; m < M; ++m)
#pragma unroll
    for (int e = 0; e < DPL; ++e) acc[m][e] = 0.f;
  bool ok = true;
  if (my_chunks > 0 && !mbar_wait(&bar[kAttnBufs], 0)) ok = false;
  for (int g0 = 0; ok && g0 < my_chunks; g0 += kAttnBufs) {
    const int gn = min(kAttnBufs, my_chunks - g0);
    const uint32_t parity = static_cast<uint32_t>(g0 / kAttnBufs) & 1u;
    // 1. scores of the group's keys for every row (-inf where masked): the lane's key slices of
    // all the group's chunks are held in registers, so each q row is read once per group
    float kv[kAttnBufs][DPP];
    int nkc[kAttnBufs], j0c[kAttnBufs];
#pragma unroll
    for (int i = 0; i < kAttnBufs; ++i) {
      j0c[i] = (rank + (g0 + i) * kAttnSplit) * KPC;
      nkc[i] = i < gn ? min(KPC, n_keys - j0c[i]) : 0;
      if (i >= gn) continue;
      if (!mbar_wait(&bar[i], parity)) {
        ok = false;
        continue;
      }
      const float* kr = reinterpret_cast<const float*>(smem + S::kBuf0 + i * 2 * S::kKV) + jw * DH + part * DPP;
#pragma unroll
      for (int e = 0; e < NF; ++e) {
        const float4 t = *reinterpret_cast<const float4*>(kr + ((e + rot) & (NF - 1)) * 4);
        kv[i][4 * e] = t.x;
        kv[i][4 * e + 1] = t.y;
        kv[i][4 * e + 2] = t.z;
        kv[i][4 * e + 3] = t.w;
      }
    }
    // all (row, chunk) partial dots first, then the xor trees level by level, then the stores:
    // no shared-memory store sits between one row's q loads and the next's
    float a[M][kAttnBufs];
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const float* qr = Qs + m * DH + part * DPP;
      float4 q4[NF];
#pragma unroll
      for (int e = 0; e < NF; ++e) q4[e] = *reinterpret_cast<const float4*>(qr + ((e + rot) & (NF - 1)) * 4);
#pragma unroll
      for (int i = 0; i < kAttnBufs; ++i) {
        float t = 0.f;
#pragma unroll
        for (int e = 0; e < NF; ++e) {
          t = fmaf(kv[i][4 * e], q4[e].x, t);
          t = fmaf(kv[i][4 * e + 1], q4[e].y, t);
          t = fmaf(kv[i][4 * e + 2], q4[e].z, t);
          t = fmaf(kv[i][4 * e + 3], q4[e].w, t);
        }
        a[m][i] = t;
      }
    }
#pragma unroll
    for (int off = 1; off < TPK; off <<= 1)
#pragma unroll
      for (int m = 0; m < M; ++m)
#pragma unroll
        for (int i = 0; i < kAttnBufs; ++i) a[m][i] += __shfl_xor_sync(0xffffffffu, a[m][i], off);
    if (part == 0) {
#pragma unroll
      for (int m = 0; m < M; ++m)
#pragma unroll
        for (int i = 0; i < kAttnBufs; ++i) {
          if (i >= gn) break;
          const int j = j0c[i] + jw;
          const bool vis = jw < nkc[i] && ((EXT && p.fixed_keys) || j <= base + m);
          float sv = a[m][i] * p.scale;
          if constexpr (EXT) {
            if (vis && p.bias) {
              const int bi = min(max(j - (base + m) + p.bias_zero, 0), p.bias_stride - 1);
              sv += __ldg(p.bias + static_cast<size_t>(h) * p.bias_stride + bi);
            }
          }
          ss[m * GK + i * KPC + jw] = vis ? sv : -INFINITY;
        }
    }
    __syncthreads();
    if (!ok) break;
    // 2. per row (one warp each): running max and sum over the group, exponentials in place
    for (int m = w; m < M; m += kAttnWarps) {
      float* sr = ss + m * GK;
      const int nkg = gn * KPC;
      float v[G::KPL];
      float gm = -INFINITY;
#pragma unroll
      for (int t = 0; t < G::KPL; ++t) {
        const int idx = lane + 32 * t;
        v[t] = idx < nkg ? sr[idx] : -INFINITY;
        gm = fmaxf(gm, v[t]);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) gm = fmaxf(gm, __shfl_xor_sync(0xffffffffu, gm, off));
      const float rm = rowst[4 * m], nm = fmaxf(rm, gm);
      float ls = 0.f;
#pragma unroll
      for (int t = 0; t < G::KPL; ++t) {
        const int idx = lane + 32 * t;
        const float pj = v[t] == -INFINITY ? 0.f : expf(v[t] - nm);
        if (idx < nkg) sr[idx] = pj;
        ls += pj;
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) ls += __shfl_xor_sync(0xffffffffu, ls, off);
      if (lane == 0) {
        const float so = rm == -INFINITY ? 0.f : expf(rm - nm);
        rowst[4 * m] = nm;
        rowst[4 * m + 1] = rowst[4 * m + 1] * so + ls;
        rowst[4 * m + 2] = so;
      }
    }
    __syncthreads();
    // 3. P.V over this warp's keys of the group, onto the rescaled accumulators
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const float so = rowst[4 * m + 2];
#pragma unroll
      for (int e = 0; e < DPL; ++e) acc[m][e] *= so;
    }
    for (int i = 0; i < gn; ++i) {
      const int nk = nkc[i];
      const float* vs = reinterpret_cast<const float*>(smem + S::kBuf0 + i * 2 * S::kKV + S::kKV);
      float pt[M][KPW];  // this warp's probabilities of the chunk, 16-byte broadcasts
#pragma unroll
      for (int m = 0; m < M; ++m)
#pragma unroll
        for (int t = 0; t < KPW; t += 4) {
          const float4 p4 = *reinterpret_cast<const float4*>(ss + m * GK + i * KPC + w * KPW + t);
          pt[m][t] = p4.x;
          pt[m][t + 1] = p4.y;
          pt[m][t + 2] = p4.z;
          pt[m][t + 3] = p4.w;
        }
#pragma unroll
      for (int t = 0; t < KPW; ++t) {
        const int jj = w * KPW + t;
        if (jj >= nk) break;  // rows past the chunk's keys hold stale shared memory
        const float* vr = vs + jj * DH + lane * DPL;
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
        for (int m = 0; m < M; ++m)
#pragma unroll
          for (int e = 0; e < DPL; ++e) acc[m][e] = fmaf(pt[m][t], vv[e], acc[m][e]);
      }
    }
    __syncthreads();  // buffers and scores are free again
    if (tid == 0)
      for (int i = 0; i < kAttnBufs && g0 + kAttnBufs + i < my_chunks; ++i)
        issue(i, rank + (g0 + kAttnBufs + i) * kAttnSplit);
  }
  if (!ok) set_error(p.st, DERR_TIMEOUT);

  // this CTA's state per row -- the warps' accumulators summed in warp order (the chunk buffers
  // are free: every chunk was waited for and folded before the last barrier) -- goes to part;
  // the CTA completing the head's ticket merges the kAttnSplit states in CTA order
#pragma unroll
  for (int m = 0; m < M; ++m)
#pragma unroll
    for (int e = 0; e < DPL; ++e) ws[(w * M + m) * DH + lane * DPL + e] = acc[m][e];
  __syncthreads();
  // one output element of row m, with its bf16 parts for a medium-M o projection when asked
  auto put = [&](int m, int d, float ov) {
    o_rows[m * p.o_stride + h * DH + d] = ov;
    if (p.xo_hi) {
      const size_t i = (static_cast<size_t>(z) * M + m) * p.xo_ld + h * DH + d;
      const __nv_bfloat16 oh = __float2bfloat16_rn(ov);
      p.xo_hi[i] = oh;
      p.xo_lo[i] = __float2bfloat16_rn(ov - __bfloat162float(oh));
    }
  };
  if (n_keys <= KPC) {
    // At most one chunk, CTA 0's: its state is the head's and the merge would return it unchanged
    // (weight exp(0) = 1 on it, 0 on the empty states), so CTA 0 writes O / L itself and no CTA
    // takes the ticket.
    if (rank == 0 && ok && !bad && !timed_out)
      for (int idx = tid; idx < M * DH; idx += kAttnThreads) {
        const int m = idx / DH, d = idx - m * DH;
        float O = 0.f;
#pragma unroll
        for (int q = 0; q < kAttnWarps; ++q) O += ws[(q * M + m) * DH + d];
        const float L = rowst[4 * m + 1];
        put(m, d, L > 0.f ? O / L : 0.f);
      }
    return;
  }
  constexpr int kSlot = kAttnMaxRows * E;  // one CTA state in part
  const int zh = z * p.n_heads + h;  // this request's head
  float* head_part = p.part + static_cast<size_t>(zh) * kAttnSplit * kSlot;
  float* mine = head_part + rank * kSlot;
  for (int idx = tid; idx < M * DH; idx += kAttnThreads) {
    const int m = idx / DH, d = idx - m * DH;
    float O = 0.f;
#pragma unroll
    for (int q = 0; q < kAttnWarps; ++q) O += ws[(q * M + m) * DH + d];
    __stcg(mine + m * E + d, O);
  }
  if (tid < M) {
    __stcg(mine + tid * E + DH, rowst[4 * tid]);
    __stcg(mine + tid * E + DH + 1, rowst[4 * tid + 1]);
  }
  int* last = reinterpret_cast<int*>(smem + S::kFlag);
  __syncthreads();
  if (tid == 0) *last = atom_add_acq_rel_gpu(&p.tickets[zh], 1u) == static_cast<unsigned>(kAttnSplit - 1);
  __syncthreads();
  if (*last) {
    if (!bad && !timed_out) {
      float* wq = reinterpret_cast<float*>(smem + S::kWq);  // [M][kAttnSplit] weights, then [M] totals
      constexpr int NE = (M * DH + kAttnThreads - 1) / kAttnThreads;
      float v[NE][kAttnSplit];  // the states' outputs, loaded before the weights are known
#pragma unroll
      for (int e = 0; e < NE; ++e) {
        const int idx = tid + e * kAttnThreads;
        if (idx >= M * DH) break;
        const int m = idx / DH, d = idx - m * DH;
#pragma unroll
        for (int q = 0; q < kAttnSplit; ++q) v[e][q] = __ldcg(head_part + q * kSlot + m * E + d);
      }
      if (tid < M) {
        float mq[kAttnSplit], lq[kAttnSplit];
#pragma unroll
        for (int q = 0; q < kAttnSplit; ++q) {
          mq[q] = __ldcg(head_part + q * kSlot + tid * E + DH);
          lq[q] = __ldcg(head_part + q * kSlot + tid * E + DH + 1);
        }
        float mt = -INFINITY;
#pragma unroll
        for (int q = 0; q < kAttnSplit; ++q) mt = fmaxf(mt, mq[q]);
        float L = 0.f;
#pragma unroll
        for (int q = 0; q < kAttnSplit; ++q) {
          const float gq = mq[q] == -INFINITY ? 0.f : expf(mq[q] - mt);
          wq[tid * kAttnSplit + q] = gq;
          L = fmaf(gq, lq[q], L);
        }
        wq[M * kAttnSplit + tid] = L;
      }
      __syncthreads();
#pragma unroll
      for (int e = 0; e < NE; ++e) {
        const int idx = tid + e * kAttnThreads;
        if (idx >= M * DH) break;
        const int m = idx / DH, d = idx - m * DH;
        float O = 0.f;
#pragma unroll
        for (int q = 0; q < kAttnSplit; ++q) O = fmaf(wq[m * kAttnSplit + q], v[e][q], O);
        const float L = wq[M * kAttnSplit + m];
        put(m, d, L > 0.f ? O / L : 0.f);
      }
    }
    if (tid == 0) p.tickets[zh] = 0u;
  }
}

}  // namespace ssd
