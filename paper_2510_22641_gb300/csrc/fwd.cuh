// Persistent forward kernel: one launch runs a whole forward pass of the
// decoder (Sec. "SSD Setup for VLMs": x_{l+1} = x_l + f_l(x_l), optionally the
// imitation network, then the LM head g and its argmax) for 1 .. 9 rows,
// i.e. a greedy step, the gamma passes of the drafting stage or the
// verification pass of Algorithm 1.
//
// Grid: one CTA per SM, resident for the whole launch (cooperative launch).
// Each CTA walks the same phase list.  Every phase but the embedding and the
// attention is a weight-streaming projection cut into units of 128 weight
// rows x 64 columns (16 KB); CTA c takes the contiguous unit range
// [c*U/G, (c+1)*U/G) of every phase (stream-K, so every SM moves the same
// number of weight bytes).  Roles inside a CTA (256 threads):
//  * warp 0 streams weight units -- and, in attention phases, K and V chunks
//    of the cache -- into an 8-stage ring with TMA.  Weights do not depend on
//    activations, so this warp runs ahead across phase boundaries: the next
//    phase's first units are in flight while the current one ends;
//  * warp 2 waits until the phase that produces a projection's input is
//    complete (per-phase tile counters in global memory) and copies each unit's
//    B operand -- prepared by
//    the epilogue that produced those activation columns: bf16 hi + lo of
//    gain * a (a to 2^-17 relative), 16 rows each, 128-byte swizzled K-major,
//    4 KB per 64 columns -- into shared memory with one bulk copy;
//  * one thread of warp 1 issues tcgen05.mma.kind::f16 (A = weight unit,
//    M = 128; B = the 16 hi rows and the 16 lo rows, N = 32: one MMA per
//    16-column K slice) into four 32-column TMEM accumulators;
//  * warps 4-7 drain the accumulators (tcgen05.ld; hi and lo halves added),
//    reduce row tiles split between CTAs (the last CTA to finish a tile sums
//    the partials in CTA order), run the fused epilogues (RMSNorm scale, RoPE
//    + KV-cache write, SiLU(gate) * up, scaled residual add, LM-head argmax),
//    write each finished tile's columns as the B operand of the projection
//    that reads them, publish the tile, and run the attention work items and
//    the embedding gather.
//
// Attention (Sec. "Methodology": drafting and verification read one KV cache):
// keys are cut into 16 KB chunks at absolute positions (32 keys for
// head_dim 128, 64 for 64); chunk c of a head belongs to split c mod S.  One
// work item = (head, split): a running softmax state per row over its chunks
// in increasing order, then the last split to finish merges the S states in
// split order.  Chunks wholly below kv_len were written by earlier launches
// and come through the TMA ring; the chunks holding this launch's rows are
// read with plain loads after the K/V tiles' ready flags.
//
// Batch invariance: the unit partition, the MMA shape (always N = 32), the K
// order, the split-tile reduction order, the attention chunk grid and the
// split merge order depend only on the grid size, the weight shapes and the
// key positions -- never on the number of rows -- and every output element is
// computed per row.  A row of the verification pass therefore equals the same
// row of a greedy step bitwise, which is what makes the verified output of
// Algorithm 1 identical to greedy decoding.
//
// Every wait is bounded (about 2 s): a wait that runs out sets DERR_TIMEOUT,
// after which every CTA stops issuing work, waits for its own copies and MMAs
// in flight, frees its TMEM and leaves.
#pragma once

#include "common.cuh"
#include "attn_warp.cuh"
#include "fwd_params.cuh"
#include "gemv.cuh"

namespace ssd {

template <int DH>
struct FwdSmem {
  static constexpr int kKPC = static_cast<int>(kFwdStageBytes) / (DH * 4);  // keys per K/V chunk
  static constexpr int kW = 0;                                              // [stages][16 KB]
  static constexpr int kB = kW + kFwdStages * static_cast<int>(kFwdStageBytes);  // [stages][hi 2 KB | lo 2 KB]
  static constexpr int kOut = kB + kFwdStages * kFwdBTile;                 // [rows][128] drained / final row tile
  static constexpr int kQ = kOut + kFwdRows * kTileN * 4;                   // [rows][DH] queries
  static constexpr int kS = kQ + kFwdRows * DH * 4;                         // [rows][KPC] scores / probabilities
  static constexpr int kGen = kS + kFwdRows * kKPC * 4;                     // K and V of one chunk read with plain loads
  static constexpr int kRs = kGen + 2 * static_cast<int>(kFwdStageBytes);   // [16] RMSNorm scales
  static constexpr int kCs = kRs + 16 * 4;                                  // [2][16] chunk max / sum
  static constexpr int kRed = kCs + 32 * 4;                                 // [4][16]
  static constexpr int kFlag = kRed + 64 * 4;                               // [4] ints
  static constexpr int kBar = kFlag + 16;
  static constexpr int kNBar = 2 * kFwdStages + 2 * kFwdAcc + 1;
  static constexpr int kTmemSlot = kBar + kNBar * 8;
  static constexpr int kTotal = kTmemSlot + 16 + 1024;  // + slack for the 1024-byte alignment
  static_assert(kB % 1024 == 0 && kOut % 16 == 0 && kGen % 16 == 0 && kBar % 8 == 0, "shared-memory alignment");
  static_assert(kKPC == AttnWarp<DH>::KPC && kFwdRows == kAttnMaxRows, "attention chunk shape");
};

// ------------------------------------------------------------------ synchronisation helpers

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned ld_relaxed_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void red_relaxed_add(unsigned* p, unsigned v) {
  asm volatile("red.relaxed.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void fence_proxy_async_global() { asm volatile("fence.proxy.async.global;" ::: "memory"); }

// AND of `ok` over the 128 drain threads (named barrier 1).
__device__ __forceinline__ bool drain_all(bool ok) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred q, 1, 128, p;\n selp.u32 %0, 1, 0, q;\n}"
      : "=r"(r)
      : "r"(ok ? 1u : 0u)
      : "memory");
  return r != 0;
}

struct FwdCtl {
  volatile int* abort;  // shared: this CTA has stopped
  DevState* st;
};

// Checked every 256 polls of a wait: this CTA's abort flag and the clock; once a
// wait has lasted 20 us, also the error word that other CTAs set.  (A global read
// on every few polls would put an L2 round trip into the wake-up of the streaming
// threads.)  A wait gives up after ~2 s.
__device__ __forceinline__ bool fwd_wait_check(const FwdCtl& k, uint64_t t0) {
  if (*k.abort) return false;
  const uint64_t el = globaltimer_ns() - t0;
  if (el > 20000ull && (*reinterpret_cast<volatile int*>(&k.st->error) & DERR_TIMEOUT)) {
    *k.abort = 1;
    return false;
  }
  if (el > 2000000000ull) {
    set_error(k.st, DERR_TIMEOUT);
    *k.abort = 1;
    return false;
  }
  return true;
}

// mbarrier phase wait; false once this CTA (or any CTA) has stopped or after ~2 s.
// Inlined: the streaming threads wait on every unit, and an out-of-line call from
// this register-heavy kernel costs more than the wait itself.
__device__ __forceinline__ bool fwd_mbar_wait(uint64_t* bar, uint32_t parity, const FwdCtl& k) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255u) == 0u && !fwd_wait_check(k, t0)) return false;
  }
}

// Waits until *f >= target; false once stopped or after ~2 s.  One acquire load
// when the flag is already set (the common case: one L2 round trip); otherwise
// relaxed polls (back-to-back for the first 20 us, then with a short sleep) and a
// final acquire load (an acquire also drops the SM's L1 lines, which the other
// roles keep hot, so it is not used for polling; a fence.acq_rel instead would also
// wait for the thread's bulk copies in flight).
__device__ __forceinline__ bool fwd_flag_wait(const unsigned* f, unsigned target, const FwdCtl& k) {
  if (ld_acquire_u32(f) >= target) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (ld_relaxed_u32(f) >= target) {
      ld_acquire_u32(f);
      return true;
    }
    if ((i & 15u) == 0u) {
      if (!fwd_wait_check(k, t0)) return false;
      if (globaltimer_ns() - t0 > 20000ull) __nanosleep(256);
    }
  }
}

// ------------------------------------------------------------------ optional timeline

__device__ __forceinline__ void fwd_put(const FwdParams& P, int c, int p, int e, unsigned long long v) {
  if (P.trace) P.trace[(static_cast<size_t>(c) * (P.n_phases + 1) + p) * 16 + e] = v;
}
__device__ __forceinline__ void fwd_stamp(const FwdParams& P, int c, int p, int e) {
  if (P.trace) fwd_put(P, c, p, e, globaltimer_ns());
}
__device__ __forceinline__ unsigned long long fwd_now(const FwdParams& P) { return P.trace ? globaltimer_ns() : 0ull; }
// per-slot stamps of CTAs 0..3 (after the per-phase block): [4][8192][4] = W issue, B issue, MMA issue
constexpr int kFwdSlotTrace = 8192;
__device__ __forceinline__ void fwd_slot_stamp(const FwdParams& P, int c, uint32_t i, int e) {
  if (P.trace && c < 4 && i < static_cast<uint32_t>(kFwdSlotTrace))
    P.trace[static_cast<size_t>(gridDim.x) * (P.n_phases + 1) * 16 + (static_cast<size_t>(c) * kFwdSlotTrace + i) * 4 + e] =
        globaltimer_ns();
}

// ------------------------------------------------------------------ schedule helpers

// Stream-K partition of a projection's units over min(G, units) CTAs, so that
// every participating CTA owns at least one unit and the owners of a row tile
// are consecutive CTAs.
__device__ __forceinline__ int gemv_ctas(int units, int G) { return units < G ? units : G; }
__device__ __forceinline__ int gemv_begin(int c, int units, int G) {
  const int ge = gemv_ctas(units, G);
  return c >= ge ? units : unit_begin(c, units, ge);
}

struct AttnGeom {
  int base, n_keys, n_chunks, n_ring;
  bool bad;
};

// Keys 0 .. base+M-1 exist for the last row; chunks wholly below kv_len come through the ring.
__device__ __forceinline__ AttnGeom attn_geom(const FwdPhase* ph, int kv_len, int max_seq, int kpc) {
  AttnGeom g;
  g.base = kv_len + ph->pos_off;
  g.bad = g.base < 0 || g.base + ph->M > max_seq;
  g.n_keys = g.bad ? 0 : g.base + ph->M;
  g.n_chunks = (g.n_keys + kpc - 1) / kpc;
  const int below = kv_len / kpc;
  g.n_ring = below < g.n_chunks ? below : g.n_chunks;
  return g;
}

__device__ __forceinline__ int ring_chunks_of(int n_ring, int r, int splits) {
  return n_ring > r ? (n_ring - r + splits - 1) / splits : 0;
}

// Ring slots (one K and one V chunk each) that CTA c consumes in an attention phase.
__device__ __forceinline__ int attn_ring_slots(const FwdParams& P, const AttnGeom& g, int c, int G) {
  const int I = P.n_heads * P.splits;
  int n = 0;
  for (int it = unit_begin(c, I, G); it < unit_begin(c + 1, I, G); ++it)
    n += 2 * ring_chunks_of(g.n_ring, it % P.splits, P.splits);
  return n;
}

// Publish finished tile t of phase p (drain threads, after their stores): every
// writer fences, the drain threads meet, then one relaxed add per counter -- the
// release pattern of fence + barrier + atomic.  (A red.release from the drain
// warps measurably slows the SM's concurrent TMA weight stream.)
__device__ __forceinline__ void fwd_release(const FwdParams& P, const FwdPhase* ph, int p, int t, int dt) {
  __threadfence();
  fence_proxy_async_global();
  drain_sync();
  if (dt == 0) {
    red_relaxed_add(P.flags + ph->flags + t, 1u);
    red_relaxed_add(P.done + p, 1u);
  }
}

// ------------------------------------------------------------------ epilogues (128 drain threads)

__device__ __forceinline__ void fwd_epilogue(const FwdParams& P, const FwdPhase* ph, int rt, float* out,
                                             const float* rs, int tid, int kv_len) {
  const int M = ph->M;
  const int kind = ph->kind;
  if (kind == FK_QKV) {
    const int r0 = rt * kTileN;
    const int mat = r0 / ph->seg_rows;  // 0 = q, 1 = k, 2 = v
    const int local0 = r0 - mat * ph->seg_rows;
    const int Dh = P.head_dim, half = Dh >> 1;
    const int base_pos = kv_len + ph->pos_off;
    if (mat < 2) {
      for (int idx = tid; idx < M * (kTileN / 2); idx += kDrainThreads) {
        const int m = idx / (kTileN / 2), pr = idx - m * (kTileN / 2);
        const int hh = pr / half, j = pr - hh * half;
        const int ra = hh * Dh + j, rb = ra + half;
        const int pos = base_pos + m;
        if (pos < 0 || pos >= P.max_seq) {
          set_error(P.st, DERR_POS);
          continue;
        }
        const float a = out[m * kTileN + ra] * rs[m];
        const float b = out[m * kTileN + rb] * rs[m];
        const float2 cs = P.rope[static_cast<size_t>(pos) * half + j];
        const float va = a * cs.x - b * cs.y;
        const float vb = a * cs.y + b * cs.x;
        if (mat == 0) {
          ph->q_out[m * ph->q_stride + local0 + ra] = va;
          ph->q_out[m * ph->q_stride + local0 + rb] = vb;
        } else {
          const int h = local0 / Dh + hh;
          float* kr = ph->k_cache + (static_cast<size_t>(h) * P.max_seq + pos) * Dh;
          kr[j] = va;
          kr[j + half] = vb;
        }
      }
    } else {
      for (int idx = tid; idx < M * kTileN; idx += kDrainThreads) {
        const int m = idx / kTileN, i = idx - m * kTileN;
        const int pos = base_pos + m;
        if (pos < 0 || pos >= P.max_seq) {
          set_error(P.st, DERR_POS);
          continue;
        }
        const int row = local0 + i, h = row / Dh, d = row - h * Dh;
        ph->v_cache[(static_cast<size_t>(h) * P.max_seq + pos) * Dh + d] = out[idx] * rs[m];
      }
    }
  } else if (kind == FK_GATE_SILU) {
    for (int idx = tid; idx < M * kHalfN; idx += kDrainThreads) {
      const int m = idx / kHalfN, j = idx - m * kHalfN;
      const int n = rt * kHalfN + j;
      if (n >= ph->N) continue;
      const float g = out[m * kTileN + j] * rs[m];
      const float u = out[m * kTileN + kHalfN + j] * rs[m];
      const float h = silu_f(g) * u;
      ph->h_out[m * ph->h_stride + n] = h;
      out[m * kTileN + j] = h;  // final value, for the B operand of the down projection
    }
  } else if (kind == FK_SILU) {
    for (int idx = tid; idx < M * kTileN; idx += kDrainThreads) {
      const int m = idx / kTileN, i = idx - m * kTileN;
      const int n = rt * kTileN + i;
      if (n >= ph->N) continue;
      const float h = silu_f(out[idx] * rs[m]);
      ph->h_out[m * ph->h_stride + n] = h;
      out[idx] = h;
    }
  } else if (kind == FK_RESID) {
    const float s = __ldg(ph->scale);
    for (int idx = tid; idx < M * kTileN; idx += kDrainThreads) {
      const int m = idx / kTileN, i = idx - m * kTileN;
      const int n = rt * kTileN + i;
      if (n >= ph->N) continue;
      const float b = __ldcg(ph->base + m * ph->base_stride + n);
      const float y = b + s * (out[idx] * rs[m]);
      ph->dst[m * ph->dst_stride + n] = y;
      out[idx] = y;
    }
  } else {  // FK_ARGMAX: argmax over the vocabulary, lowest index on ties
    const int lane = tid & 31;
    const int base_pos = kv_len + ph->pos_off;
    const int Pl = __ldcg(&P.st->prompt_len);
    const int n = rt * kTileN + tid;  // thread per tile row
    const bool valid = n < ph->N;
    for (int m = 0; m < M; ++m) {
      const float logit = out[m * kTileN + tid] * rs[m];
      if (ph->logits != nullptr && valid) {
        const int row = base_pos + m + 1 - Pl;
        if (row >= 0 && row < ph->logits_rows) ph->logits[static_cast<size_t>(row) * ph->N + n] = logit;
      }
      unsigned long long key = valid ? argmax_key(logit, static_cast<uint32_t>(n)) : 0ull;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const unsigned long long o = __shfl_xor_sync(0xffffffffu, key, off);
        key = o > key ? o : key;
      }
      if (lane == 0) atomicMax(&P.st->am_key[m], key);
    }
    __threadfence();
    drain_sync();
    if (tid == 0) {
      const unsigned prev = atomicAdd(&P.st->am_count, 1u);
      if (prev == static_cast<unsigned>(ph->n_rt - 1)) {
        __threadfence();
        for (int m = 0; m < M; ++m) {
          const unsigned long long key = atomicExch(&P.st->am_key[m], 0ull);
          ph->tok_dst[m] = static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull));
        }
        atomicExch(&P.st->am_count, 0u);
      }
    }
  }
}

// Columns [c0, c0 + nc) of this phase's output as the B operand of the projection
// that reads them: rows bt_row0 .. bt_row0 + M - 1 come from fin ([M][128], the
// values just written), the projection's other rows from its input rows in global
// memory; each value times the projection's RMSNorm gain, split into bf16 hi (row
// m) + lo (row 16 + m), rows beyond the projection's M zero, 128-byte swizzled.
// Gain slices of the (at most two) 8-column chunks thread dt writes, loaded ahead.
__device__ __forceinline__ void fwd_btile_gains(const FwdPhase* ph, int c0, int nc, int dt, uint4* g) {
  const int nch = nc >> 3, kmax = ph->bt_nkt * kTileK;
#pragma unroll
  for (int t = 0; t < 2; ++t) {
    const int task = dt + t * kDrainThreads;
    const int col = c0 + (task % nch) * 8;
    g[t] = (task < kNPad * nch && col < kmax) ? __ldg(reinterpret_cast<const uint4*>(ph->bt_gain + col))
                                              : make_uint4(0u, 0u, 0u, 0u);
  }
}

__device__ __forceinline__ void fwd_btile_write(const FwdParams& P, const FwdPhase* ph, const float* fin, int c0,
                                                int nc, int dt, const uint4* gpre = nullptr) {
  uint8_t* bt = P.btiles + ph->bt_dst_off;
  const float* xc = ph->bt_x;
  const int xs = ph->bt_x_stride, Mc = ph->bt_M, r0 = ph->bt_row0, Mown = ph->M;
  const __nv_bfloat16* gain = ph->bt_gain;
  const int kmax = ph->bt_nkt * kTileK;
  const int nch = nc >> 3;  // 8-column chunks (nc <= 128: at most two per thread)
#pragma unroll
  for (int t = 0; t < 2; ++t) {
    const int task = dt + t * kDrainThreads;
    if (task >= kNPad * nch) break;
    const int m = task / nch, c8 = task - m * nch;
    const int col = c0 + c8 * 8;
    if (col >= kmax) continue;
    uint32_t hw[4] = {0u, 0u, 0u, 0u}, lw[4] = {0u, 0u, 0u, 0u};
    if (m < Mc) {
      float v[8];
      if (m >= r0 && m < r0 + Mown) {
        const float* f = fin + (m - r0) * kTileN + (col - c0);
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = f[e];
      } else {
        const float4 a0 = __ldcg(reinterpret_cast<const float4*>(xc + static_cast<size_t>(m) * xs + col));
        const float4 a1 = __ldcg(reinterpret_cast<const float4*>(xc + static_cast<size_t>(m) * xs + col + 4));
        v[0] = a0.x; v[1] = a0.y; v[2] = a0.z; v[3] = a0.w;
        v[4] = a1.x; v[5] = a1.y; v[6] = a1.z; v[7] = a1.w;
      }
      if (gain) {
        const uint4 gv = gpre ? gpre[t] : __ldg(reinterpret_cast<const uint4*>(gain + col));
        const float2 g0 = bf16x2_to_float2(gv.x), g1 = bf16x2_to_float2(gv.y), g2 = bf16x2_to_float2(gv.z),
                     g3 = bf16x2_to_float2(gv.w);
        v[0] *= g0.x; v[1] *= g0.y; v[2] *= g1.x; v[3] *= g1.y;
        v[4] *= g2.x; v[5] *= g2.y; v[6] *= g3.x; v[7] *= g3.y;
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const __nv_bfloat16 h0 = __float2bfloat16_rn(v[2 * e]), h1 = __float2bfloat16_rn(v[2 * e + 1]);
        const __nv_bfloat16 l0 = __float2bfloat16_rn(v[2 * e] - __bfloat162float(h0));
        const __nv_bfloat16 l1 = __float2bfloat16_rn(v[2 * e + 1] - __bfloat162float(h1));
        hw[e] = pack_bf16x2(h0, h1);
        lw[e] = pack_bf16x2(l0, l1);
      }
    }
    uint8_t* tile = bt + static_cast<size_t>(col >> 6) * kFwdBTile;
    const int sw = (((col >> 3) & 7) ^ (m & 7)) << 4;  // 128-byte swizzle of row m (and of row 16 + m)
    __stcg(reinterpret_cast<uint4*>(tile + m * 128 + sw), make_uint4(hw[0], hw[1], hw[2], hw[3]));
    __stcg(reinterpret_cast<uint4*>(tile + (kNPad + m) * 128 + sw), make_uint4(lw[0], lw[1], lw[2], lw[3]));
  }
}

// ------------------------------------------------------------------ attention pieces (128 drain threads)

// Plain loads of one chunk's K or V rows (keys j0 .. j0+nk-1) into shared memory.
template <int DH>
__device__ __forceinline__ void attn_load_chunk(float* dst, const float* src, int nk, int dt) {
  const float4* s4 = reinterpret_cast<const float4*>(src);
  float4* d4 = reinterpret_cast<float4*>(dst);
  for (int i = dt; i < nk * DH / 4; i += kDrainThreads) d4[i] = __ldcg(s4 + i);
}

// The attention work items of CTA c in phase p (drain warps).  Advances the ring counter.
template <int DH>
__device__ bool fwd_attention(const FwdParams& P, const FwdPhase* ph, int p, int c, int G, int kv_len, uint32_t& i,
                              uint8_t* smem, uint64_t* full, uint64_t* empty, int dt, const FwdCtl& k) {
  using S = FwdSmem<DH>;
  using AW = AttnWarp<DH>;
  constexpr int KPC = S::kKPC, DPL = AW::DPL;
  float* fin = reinterpret_cast<float*>(smem + S::kOut);
  const AttnGeom ag = attn_geom(ph, kv_len, P.max_seq, KPC);
  const int M = ph->M, splits = P.splits, I = P.n_heads * splits, nsub = 4 * splits;
  const int it0 = unit_begin(c, I, G), it1 = unit_begin(c + 1, I, G);
  if (ag.bad && dt == 0 && it0 < it1) set_error(P.st, DERR_POS);
  const FwdPhase* qk = P.phases + ph->dep;  // the QKV phase of this layer
  const float* qsrc = ph->x;
  const int q_stride = ph->x_stride;
  const float* kc = ph->k_cache;
  const float* vc = ph->v_cache;
  float* o = ph->dst;
  const int o_stride = ph->dst_stride;
  float* Qs = reinterpret_cast<float*>(smem + S::kQ);
  float* Gk = reinterpret_cast<float*>(smem + S::kGen);
  float* Gv = Gk + kFwdStageBytes / 4;
  constexpr int kEnt = DH + 2;  // o[DH], max, sum
  float* part = P.attn_part + static_cast<size_t>(p % kFwdWindow) * P.n_heads * nsub * kFwdRows * kEnt;
  const int w = dt >> 5, lane = dt & 31;

  for (int it = it0; it < it1; ++it) {
    const int h = it / splits, r = it - h * splits;
    // q, k and v of every head come from one QKV phase whose row tiles finish within a
    // microsecond of each other: one wait on the phase instead of three flag round trips
    bool ok = true;
    if (!ag.bad) ok = fwd_flag_wait(P.done + ph->dep, static_cast<unsigned>(qk->n_tiles), k);
    if (!drain_all(ok)) return false;
    if (dt == 0) fwd_stamp(P, c, p, 8);
    for (int idx = dt; idx < M * DH; idx += kDrainThreads) {
      const int m = idx / DH, e = idx - m * DH;
      Qs[idx] = __ldcg(qsrc + static_cast<size_t>(m) * q_stride + h * DH + e);
    }
    AW st;
    st.init();
    // the first chunk holding keys at or above kv_len (written this launch) is fetched now,
    // behind the ring chunks
    const int nr = ring_chunks_of(ag.n_ring, r, splits);
    const int ck_gen = r + nr * splits;
    if (ck_gen < ag.n_chunks) {
      const int j0 = ck_gen * KPC, nk = min(KPC, ag.n_keys - j0);
      const size_t off = (static_cast<size_t>(h) * P.max_seq + j0) * DH;
      for (int e = dt; e < nk * DH / 4; e += kDrainThreads) {
        cp_async16(Gk + 4 * e, kc + off + 4 * e);
        cp_async16(Gv + 4 * e, vc + off + 4 * e);
      }
      cp_async_commit();
    }
    drain_sync();
    if (dt == 0) fwd_stamp(P, c, p, 9);
    for (int q = 0; q < nr; ++q) {
      const int ck = r + q * splits;
      const int sK = static_cast<int>(i % kFwdStages), sV = static_cast<int>((i + 1) % kFwdStages);
      ok = fwd_mbar_wait(&full[sK], (i / kFwdStages) & 1u, k) &&
           fwd_mbar_wait(&full[sV], ((i + 1) / kFwdStages) & 1u, k);
      if (!drain_all(ok)) return false;
      st.chunk_rows(reinterpret_cast<const float*>(smem + S::kW + sK * kFwdStageBytes),
                    reinterpret_cast<const float*>(smem + S::kW + sV * kFwdStageBytes), Qs, M, ck * KPC, KPC, ag.base,
                    P.attn_scale, w, lane);
      drain_sync();  // every warp is done with both stages
      if (dt == 0) {
        mbar_arrive(&empty[sK]);
        mbar_arrive(&empty[sV]);
      }
      i += 2;
    }
    if (dt == 0) fwd_stamp(P, c, p, 10);
    for (int ck = ck_gen; ck < ag.n_chunks; ck += splits) {
      const int j0 = ck * KPC, nk = min(KPC, ag.n_keys - j0);
      if (ck == ck_gen) {
        cp_async_wait_all();
      } else {
        const size_t off = (static_cast<size_t>(h) * P.max_seq + j0) * DH;
        attn_load_chunk<DH>(Gk, kc + off, nk, dt);
        attn_load_chunk<DH>(Gv, vc + off, nk, dt);
      }
      drain_sync();
      st.chunk_rows(Gk, Gv, Qs, M, j0, nk, ag.base, P.attn_scale, w, lane);
      drain_sync();
    }
    if (dt == 0) fwd_stamp(P, c, p, 11);
    // publish this warp's state as sub-split 4 r + w; the last split of the head merges
    // all 4 * splits states in order
#pragma unroll
    for (int m = 0; m < kFwdRows; ++m) {
      if (m >= M) break;
      float* e = part + ((static_cast<size_t>(h) * nsub + 4 * r + w) * kFwdRows + m) * kEnt;
#pragma unroll
      for (int d = 0; d < DPL; ++d) __stcg(e + lane * DPL + d, st.o[m][d]);
      if (lane == 0) {
        __stcg(e + DH, st.mx[m]);
        __stcg(e + DH + 1, st.l[m]);
      }
    }
    // The split holding the newest chunk (always the one with the most work) merges: it
    // waits for the other splits' tickets and reads its own states without a fence.
    const int r_merge = ag.n_chunks > 0 ? (ag.n_chunks - 1) % splits : 0;
    const bool merger = r == r_merge;
    if (!merger) {
      __threadfence();
      drain_sync();
      if (dt == 0) red_relaxed_add(P.tickets + ph->flags + h, 1u);
    } else {
      drain_sync();
      if (!drain_all(fwd_flag_wait(P.tickets + ph->flags + h, static_cast<unsigned>(splits - 1), k))) return false;
    }
    if (dt == 0) fwd_stamp(P, c, p, 12);
    if (merger) {
      for (int idx = dt; idx < M * DH; idx += kDrainThreads) {
        const int m = idx / DH, d = idx - m * DH;
        const float* e0 = part + (static_cast<size_t>(h) * nsub * kFwdRows + m) * kEnt;
        const size_t sstride = static_cast<size_t>(kFwdRows) * kEnt;
        // sub-splits in groups of 16, each group's loads issued together (one round for 4 splits);
        // a running maximum carries the groups, in a fixed order
        float mt = -INFINITY, L = 0.f, O = 0.f;
        for (int q0 = 0; q0 < nsub; q0 += 16) {
          float mq[16], lq[16], oq[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const bool in = q0 + q < nsub;
            mq[q] = in ? __ldcg(e0 + (q0 + q) * sstride + DH) : -INFINITY;
            lq[q] = in ? __ldcg(e0 + (q0 + q) * sstride + DH + 1) : 0.f;
            oq[q] = in ? __ldcg(e0 + (q0 + q) * sstride + d) : 0.f;
          }
          float gm = mt;
#pragma unroll
          for (int q = 0; q < 16; ++q) gm = fmaxf(gm, mq[q]);
          if (gm == -INFINITY) continue;
          const float so = expf(mt - gm);  // 0 for the first group with a visible key
          L *= so;
          O *= so;
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            if (mq[q] == -INFINITY) continue;
            const float wq = expf(mq[q] - gm);
            L = fmaf(wq, lq[q], L);
            O = fmaf(wq, oq[q], O);
          }
          mt = gm;
        }
        const float ov = L > 0.f ? O / L : 0.f;
        o[m * o_stride + h * DH + d] = ov;
        fin[m * kTileN + d] = ov;
      }
      if (dt == 0) P.tickets[ph->flags + h] = 0u;
      if (ph->bt_dst_off >= 0) {
        drain_sync();
        fwd_btile_write(P, ph, fin, h * DH, DH, dt);
      }
      fwd_release(P, ph, p, h, dt);
      if (dt == 0) fwd_stamp(P, c, p, 13);
    }
    drain_sync();
  }
  return true;
}

// Embedding gather x[m][:] = E[tok[m]][:] for the 128-column tiles of CTA c (drain warps).
__device__ __forceinline__ bool fwd_embed(const FwdParams& P, const FwdPhase* ph, int p, int c, int G, int dt,
                                          float* fin, const FwdCtl& k) {
  const int n = ph->n_tiles, t0 = unit_begin(c, n, G), t1 = unit_begin(c + 1, n, G);
  if (t0 >= t1) return true;
  if (ph->epi_dep >= 0 && !drain_all(fwd_flag_wait(P.done + ph->epi_dep, P.phases[ph->epi_dep].n_tiles, k)))
    return false;
  for (int t = t0; t < t1; ++t) {
    const int col = t * kTileN + dt;
    for (int m = 0; m < ph->M; ++m) {
      int tok = __ldcg(ph->tok_src + m);
      if (tok < 0 || tok >= P.vocab) {
        if (dt == 0) set_error(P.st, DERR_TOKEN);
        tok = 0;
      }
      if (col < ph->dst_stride) {
        float v = 0.f;
        if (col < P.d_model) v = __bfloat162float(__ldg(P.embed + static_cast<size_t>(tok) * P.d_model + col));
        ph->dst[static_cast<size_t>(m) * ph->dst_stride + col] = v;
        fin[m * kTileN + dt] = v;
      }
    }
    if (ph->bt_dst_off >= 0) {
      drain_sync();
      fwd_btile_write(P, ph, fin, t * kTileN, kTileN, dt);
    }
    fwd_release(P, ph, p, t, dt);
  }
  return true;
}

// ------------------------------------------------------------------ the kernel

template <int DH>
__global__ void __launch_bounds__(kFwdThreads, 1) fwd_kernel(const __grid_constant__ FwdParams P) {
  using S = FwdSmem<DH>;
  constexpr int KPC = S::kKPC;
  extern __shared__ __align__(1024) uint8_t fwd_smem_raw[];
  const uint32_t raw = smem_u32(fwd_smem_raw);
  uint8_t* smem = fwd_smem_raw + (((raw + 1023u) & ~1023u) - raw);
  // full[s]: both producers arrived and every byte of stage s (weight unit or K/V chunk, B operand) landed;
  // empty[s]: stage s consumed (MMA commit or attention), both producers may refill it
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBar);
  uint64_t* empty = full + kFwdStages;
  uint64_t* accf = empty + kFwdStages;                            // accumulator complete
  uint64_t* acce = accf + kFwdAcc;                                // accumulator drained
  uint64_t* mma_done = acce + kFwdAcc;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + S::kTmemSlot);
  volatile int* sflag = reinterpret_cast<volatile int*>(smem + S::kFlag);  // [0] abort, [1] merge, [2] last CTA

  const int G = gridDim.x, c = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    sflag[0] = (*reinterpret_cast<volatile int*>(&P.st->error) & DERR_TIMEOUT) ? 1 : 0;
    sflag[1] = 0;
    sflag[2] = 0;
    for (int s = 0; s < kFwdStages; ++s) {
      mbar_init(&full[s], 2);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < kFwdAcc; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 4);
    }
    mbar_init(mma_done, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kFwdTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tmem_fence_before();
  __syncthreads();
  tmem_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int kv_len = __ldcg(&P.st->kv_len);
  const FwdCtl k{sflag, P.st};
  if (tid == 0) fwd_stamp(P, c, P.n_phases, 0);

  if (warp == 0) {
    // ---------------------------------------------------------------- weights / K,V chunks (TMA)
    if (lane == 0) {
      uint32_t i = 0;
      bool ok = !sflag[0];
      for (int p = 0; ok && p < P.n_phases; ++p) {
        const FwdPhase* ph = P.phases + p;
        const int kind = ph->kind;
        if (kind == FK_EMBED) continue;
        if (kind == FK_ATTN) {
          const AttnGeom ag = attn_geom(ph, kv_len, P.max_seq, KPC);
          const float* kc = ph->k_cache;
          const float* vc = ph->v_cache;
          const int splits = P.splits, I = P.n_heads * splits;
          const int it0 = unit_begin(c, I, G), it1 = unit_begin(c + 1, I, G);
          for (int it = it0; ok && it < it1; ++it) {
            const int h = it / splits, r = it - h * splits;
            const int nr = ring_chunks_of(ag.n_ring, r, splits);
            for (int q = 0; ok && q < nr; ++q) {
              const size_t off = (static_cast<size_t>(h) * P.max_seq + static_cast<size_t>(r + q * splits) * KPC) * DH;
              for (int kv = 0; kv < 2; ++kv) {
                const int s = static_cast<int>(i % kFwdStages);
                if (i >= kFwdStages && !fwd_mbar_wait(&empty[s], ((i / kFwdStages) - 1) & 1u, k)) {
                  ok = false;
                  break;
                }
                mbar_arrive_expect_tx(&full[s], kFwdStageBytes);
                bulk_load(smem + S::kW + s * kFwdStageBytes, (kv ? vc : kc) + off, kFwdStageBytes, &full[s]);
                if (it == it0 && q == 0 && kv == 0) fwd_stamp(P, c, p, 0);
                ++i;
              }
            }
          }
          continue;
        }
        // per-phase constants in registers: the unit loop touches no global memory
        const int n_kt = ph->n_kt, seg = ph->seg_rows, units = ph->units;
        const CUtensorMap* m0 = P.maps + ph->map0;
        const CUtensorMap* m1 = P.maps + ph->map1;
        const CUtensorMap* m2 = P.maps + ph->map2;
        prefetch_tensormap(m0);
        if (kind == FK_GATE_SILU || kind == FK_QKV) prefetch_tensormap(m1);
        if (kind == FK_QKV) prefetch_tensormap(m2);
        const int ub = gemv_begin(c, units, G), u1 = gemv_begin(c + 1, units, G);
        int rt = ub / n_kt, kt = ub - rt * n_kt;
        unsigned long long w_empty = 0;
        for (int u = ub; u < u1; ++u) {
          const int s = static_cast<int>(i % kFwdStages);
          const unsigned long long tw = fwd_now(P);
          if (i >= kFwdStages && !fwd_mbar_wait(&empty[s], ((i / kFwdStages) - 1) & 1u, k)) {
            ok = false;
            break;
          }
          w_empty += fwd_now(P) - tw;
          uint8_t* wdst = smem + S::kW + s * kFwdStageBytes;
          const int x = kt * kTileK;
          mbar_arrive_expect_tx(&full[s], kFwdStageBytes);
          if (kind == FK_GATE_SILU) {
            tma_load_2d(wdst, m0, &full[s], x, rt * kHalfN);
            tma_load_2d(wdst + kFwdStageBytes / 2, m1, &full[s], x, rt * kHalfN);
          } else if (kind == FK_QKV) {
            const int r0 = rt * kTileN, mat = r0 / seg;
            tma_load_2d(wdst, mat == 0 ? m0 : (mat == 1 ? m1 : m2), &full[s], x, r0 - mat * seg);
          } else {
            tma_load_2d(wdst, m0, &full[s], x, rt * kTileN);
          }
          if (u == ub) fwd_stamp(P, c, p, 0);
          fwd_slot_stamp(P, c, i, 0);
          ++i;
          if (++kt == n_kt) {
            kt = 0;
            ++rt;
          }
        }
        fwd_stamp(P, c, p, 1);
        fwd_put(P, c, p, 8, w_empty);
      }
      // no copy may land after the CTA has left: wait for the last use of every stage
      for (uint32_t j = i > kFwdStages ? i - kFwdStages : 0; j < i; ++j)
        mbar_wait(&full[j % kFwdStages], (j / kFwdStages) & 1u);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      // B = 32 rows: the hi parts of the activation rows in 0..15, the lo parts in 16..31
      constexpr uint32_t idesc = umma_idesc_bf16(kTileN, kFwdAccCols);
      uint32_t i = 0, sg = 0;
      bool ok = !sflag[0];
      for (int p = 0; ok && p < P.n_phases; ++p) {
        const FwdPhase* ph = P.phases + p;
        const int kind = ph->kind;
        if (kind == FK_EMBED) continue;
        if (kind == FK_ATTN) {
          // The drain warps consume these stages; this thread still waits out each one's
          // full phase, so that the parity it tests on the stage's next use refers to that
          // use and not to the one before it.
          const int n = attn_ring_slots(P, attn_geom(ph, kv_len, P.max_seq, KPC), c, G);
          for (int q = 0; q < n; ++q) {
            if (!fwd_mbar_wait(&full[i % kFwdStages], (i / kFwdStages) & 1u, k)) {
              ok = false;
              break;
            }
            ++i;
          }
          continue;
        }
        const int n_kt = ph->n_kt, units = ph->units;
        const int ub = gemv_begin(c, units, G), u1 = gemv_begin(c + 1, units, G);
        int kt = ub % n_kt;
        bool seg_open = false;
        uint32_t d = tmem;
        unsigned long long w_acc = 0, w_f = 0;
        for (int u = ub; u < u1; ++u) {
          const int s = static_cast<int>(i % kFwdStages);
          unsigned long long t0 = fwd_now(P);
          if (!seg_open) {  // a new row-tile segment: take a free accumulator
            const uint32_t b = sg % kFwdAcc;
            if (!fwd_mbar_wait(&acce[b], ((sg / kFwdAcc) & 1u) ^ 1u, k)) {
              ok = false;
              break;
            }
            tmem_fence_after();
            d = tmem + b * kFwdAccCols;
          }
          const unsigned long long t1 = fwd_now(P);
          w_acc += t1 - t0;
          if (!fwd_mbar_wait(&full[s], (i / kFwdStages) & 1u, k)) {
            ok = false;
            break;
          }
          w_f += fwd_now(P) - t1;
          tmem_fence_after();
          const uint32_t wa = smem_u32(smem + S::kW + s * kFwdStageBytes);
          const uint32_t ba = smem_u32(smem + S::kB + s * kFwdBTile);
          const uint64_t adesc = umma_desc_sw128(wa), bdesc = umma_desc_sw128(ba);
#pragma unroll
          for (int kk = 0; kk < kTileK / 16; ++kk) {
            // +32 bytes (2 descriptor units) per 16-element K slice inside the swizzled row
            umma_f16(d, adesc + 2 * kk, bdesc + 2 * kk, idesc, (seg_open || kk > 0) ? 1u : 0u);
            seg_open = true;
          }
          if (u == ub) fwd_stamp(P, c, p, 4);
          fwd_slot_stamp(P, c, i, 2);
          umma_commit(&empty[s]);  // the weight unit and the B operand may be replaced
          if (kt == n_kt - 1 || u == u1 - 1) {
            umma_commit(&accf[sg % kFwdAcc]);
            ++sg;
            seg_open = false;
          }
          if (++kt == n_kt) kt = 0;
          ++i;
        }
        fwd_stamp(P, c, p, 5);
        fwd_put(P, c, p, 10, w_f);
        fwd_put(P, c, p, 11, w_acc);
      }
      umma_commit(mma_done);  // every MMA has finished before TMEM is released
      mbar_wait(mma_done, 0);
    }
  } else if (warp == 2) {
    // ---------------------------------------------------------------- B operands (bulk copies)
    if (lane == 0) {
      uint32_t i = 0;
      bool ok = !sflag[0];
      for (int p = 0; ok && p < P.n_phases; ++p) {
        const FwdPhase* ph = P.phases + p;
        const int kind = ph->kind;
        if (kind == FK_EMBED) continue;
        if (kind == FK_ATTN) {  // K/V stages: the second arrival on full[s] carries no bytes
          const int n = attn_ring_slots(P, attn_geom(ph, kv_len, P.max_seq, KPC), c, G);
          for (int q = 0; q < n; ++q) {
            const int s = static_cast<int>(i % kFwdStages);
            if (i >= kFwdStages && !fwd_mbar_wait(&empty[s], ((i / kFwdStages) - 1) & 1u, k)) {
              ok = false;
              break;
            }
            mbar_arrive(&full[s]);
            ++i;
          }
          continue;
        }
        const int dep = ph->dep, n_kt = ph->n_kt, units = ph->units;
        const uint8_t* bsrc = P.btiles + ph->bt_off;
        const int ub = gemv_begin(c, units, G), u1 = gemv_begin(c + 1, units, G);
        unsigned long long w_bf = 0, w_dep = 0;
        if (ub < u1 && dep >= 0) {
          // the producing phase's tiles finish within a few microseconds of each other
          // (stream-K), so wait for all of them once: one acquire and one proxy fence per
          // phase instead of a flag round trip per unit
          const unsigned long long t1 = fwd_now(P);
          if (!fwd_flag_wait(P.done + dep, static_cast<unsigned>(P.phases[dep].n_tiles), k)) {
            ok = false;
            break;
          }
          fence_proxy_async_global();  // the copies below read what the acquire made visible
          w_dep += fwd_now(P) - t1;
        }
        int kt = ub % n_kt;
        for (int u = ub; u < u1; ++u) {
          const int s = static_cast<int>(i % kFwdStages);
          const unsigned long long t0 = fwd_now(P);
          if (i >= kFwdStages && !fwd_mbar_wait(&empty[s], ((i / kFwdStages) - 1) & 1u, k)) {
            ok = false;
            break;
          }
          w_bf += fwd_now(P) - t0;
          mbar_arrive_expect_tx(&full[s], kFwdBTile);
          bulk_load(smem + S::kB + s * kFwdBTile, bsrc + static_cast<size_t>(kt) * kFwdBTile, kFwdBTile, &full[s]);
          if (u == ub) fwd_stamp(P, c, p, 2);
          fwd_slot_stamp(P, c, i, 1);
          if (++kt == n_kt) kt = 0;
          ++i;
        }
        fwd_stamp(P, c, p, 3);
        fwd_put(P, c, p, 14, w_bf);
        fwd_put(P, c, p, 15, w_dep);
      }
    }
  } else if (warp == 3) {
    // idle
  } else {
    // ---------------------------------------------------------------- drain, epilogues, attention, embedding
    const int dt = tid - 128;  // 0..127
    const int q4 = warp & 3;   // TMEM lane quadrant: tile rows 32 q4 .. 32 q4 + 31
    float* outb = reinterpret_cast<float*>(smem + S::kOut);
    float* rs = reinterpret_cast<float*>(smem + S::kRs);
    float* red = reinterpret_cast<float*>(smem + S::kRed);
    uint32_t i = 0, sg = 0;
    bool ok = !sflag[0];
    for (int p = 0; ok && p < P.n_phases; ++p) {
      const FwdPhase* ph = P.phases + p;
      const int kind = ph->kind;
      // the split scratch of phase p - window is reused by phase p
      if (p >= kFwdWindow) {
        if (!drain_all(fwd_flag_wait(P.done + (p - kFwdWindow), P.phases[p - kFwdWindow].n_tiles, k))) {
          ok = false;
          break;
        }
      }
      if (dt == 0) fwd_stamp(P, c, p, 6);
      if (kind == FK_EMBED) {
        ok = fwd_embed(P, ph, p, c, G, dt, outb, k);
        if (dt == 0) fwd_stamp(P, c, p, 7);
        continue;
      }
      if (kind == FK_ATTN) {
        ok = fwd_attention<DH>(P, ph, p, c, G, kv_len, i, smem, full, empty, dt, k);
        if (dt == 0) fwd_stamp(P, c, p, 7);
        continue;
      }
      const int M = ph->M, n_kt = ph->n_kt, units = ph->units;
      const int u0 = gemv_begin(c, units, G), u1 = gemv_begin(c + 1, units, G);
      const int ge = gemv_ctas(units, G);
      const int tcols = kind == FK_GATE_SILU ? kHalfN : kTileN;  // output columns per row tile
      i += static_cast<uint32_t>(u1 - u0);
      if (u0 >= u1) continue;
      if (ph->epi_dep >= 0 &&
          !drain_all(fwd_flag_wait(P.done + ph->epi_dep, P.phases[ph->epi_dep].n_tiles, k))) {
        ok = false;
        break;
      }
      // RMSNorm scale per row: rs[m] = 1/sqrt(mean(x^2) + eps), fixed reduction order
      if (ph->gain) {
        const int K4 = ph->K >> 2;
        const float* xrow = ph->x;
        const int xs = ph->x_stride;
        for (int m = 0; m < M; ++m) {
          const float4* xr = reinterpret_cast<const float4*>(xrow + static_cast<size_t>(m) * xs);
          float ss = 0.f;
          for (int e = dt; e < K4; e += kDrainThreads) {
            const float4 v = __ldcg(xr + e);
            ss = fmaf(v.x, v.x, ss);
            ss = fmaf(v.y, v.y, ss);
            ss = fmaf(v.z, v.z, ss);
            ss = fmaf(v.w, v.w, ss);
          }
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
          if (lane == 0) red[q4 * 16 + m] = ss;
        }
        drain_sync();
        if (dt < M) {
          float t = 0.f;
          for (int w = 0; w < 4; ++w) t += red[w * 16 + dt];
          rs[dt] = rsqrtf(t / static_cast<float>(ph->K) + P.eps);
        }
      } else if (dt < M) {
        rs[dt] = 1.0f;
      }
      drain_sync();

      // Split row tiles: the CTA holding a tile's first K slices (the end of its unit
      // range, so it reaches the tile last) sums its own accumulator and the other
      // holders' partials -- which they wrote at the start of their ranges -- in CTA
      // order, and runs the epilogue; the others write a partial and count a ticket.
      float* part = P.partials + static_cast<size_t>(p % kFwdWindow) * (G * kFwdRows * kTileN);
      const bool resid = kind == FK_RESID;
      const bool want_b = ph->bt_dst_off >= 0;
      const float rscale = resid ? __ldg(ph->scale) : 0.f;
      int seg_kt0 = u0 % n_kt;
      for (int u = u0; u < u1; ++u) {
        const int rt = u / n_kt, kt = u - rt * n_kt;
        if (!(kt == n_kt - 1 || u == u1 - 1)) continue;
        const bool whole = (seg_kt0 == 0) && (kt == n_kt - 1);
        const int c_first = unit_owner(rt * n_kt, units, ge);
        const int c_last = unit_owner(rt * n_kt + n_kt - 1, units, ge);
        const bool owner = whole || c == c_first;
        // epilogue inputs that do not depend on the accumulator, loaded before it is ready
        float bpre[kFwdRows];
        uint4 gpre[2];
        const int ncol = rt * kTileN + dt;
        if (owner && resid) {
#pragma unroll
          for (int m = 0; m < kFwdRows; ++m)
            bpre[m] = (m < M && ncol < ph->N) ? __ldcg(ph->base + m * ph->base_stride + ncol) : 0.f;
        }
        if (owner && want_b && ph->bt_gain) fwd_btile_gains(ph, rt * tcols, tcols, dt, gpre);
        const uint32_t b = sg % kFwdAcc;
        if (!drain_all(fwd_mbar_wait(&accf[b], (sg / kFwdAcc) & 1u, k))) {
          ok = false;
          break;
        }
        tmem_fence_after();
        float vh[kNPad], vl[kNPad];
        const uint32_t ta = tmem + (static_cast<uint32_t>(q4 * 32) << 16) + b * kFwdAccCols;
        tmem_ld16(ta, vh);
        tmem_ld16(ta + kNPad, vl);
        tmem_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acce[b]);  // the MMA warp may reuse accumulator b
#pragma unroll
        for (int m = 0; m < kFwdRows; ++m)
          if (m < M) outb[m * kTileN + q4 * 32 + lane] = vh[m] + vl[m];  // W a = W hi + W lo
        drain_sync();
        if (owner && !whole) {  // own accumulator, then the others' partials in CTA order
          const int nsp = c_last - c_first + 1;
          if (!drain_all(fwd_flag_wait(P.tickets + ph->flags + rt, static_cast<unsigned>(nsp - 1), k))) {
            ok = false;
            break;
          }
          for (int f = dt; f < M * (kTileN / 4); f += kDrainThreads) {
            float4 sum = reinterpret_cast<const float4*>(outb)[f];
            for (int b0 = 1; b0 < nsp; b0 += 8) {
              float4 pv[8];
#pragma unroll
              for (int j = 0; j < 8; ++j)
                pv[j] = (b0 + j < nsp) ? __ldcg(reinterpret_cast<const float4*>(
                                             part + static_cast<size_t>(c_first + b0 + j) * (kFwdRows * kTileN)) + f)
                                       : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                if (b0 + j >= nsp) continue;
                sum.x += pv[j].x;
                sum.y += pv[j].y;
                sum.z += pv[j].z;
                sum.w += pv[j].w;
              }
            }
            reinterpret_cast<float4*>(outb)[f] = sum;
          }
          if (dt == 0) P.tickets[ph->flags + rt] = 0u;
          drain_sync();
        }
        if (!owner) {
          float* dstp = part + static_cast<size_t>(c) * (kFwdRows * kTileN);
          for (int idx = dt; idx < M * kTileN; idx += kDrainThreads) __stcg(dstp + idx, outb[idx]);
          __threadfence();
          drain_sync();
          if (dt == 0) red_relaxed_add(P.tickets + ph->flags + rt, 1u);
        } else {
          if (resid) {  // dst = base + s * (W a), with the base loaded ahead
#pragma unroll
            for (int m = 0; m < kFwdRows; ++m) {
              if (m >= M || ncol >= ph->N) continue;
              const float y = bpre[m] + rscale * (outb[m * kTileN + dt] * rs[m]);
              ph->dst[m * ph->dst_stride + ncol] = y;
              outb[m * kTileN + dt] = y;
            }
          } else {
            fwd_epilogue(P, ph, rt, outb, rs, dt, kv_len);
          }
          if (want_b) {
            drain_sync();
            fwd_btile_write(P, ph, outb, rt * tcols, tcols, dt, ph->bt_gain ? gpre : nullptr);
          }
          fwd_release(P, ph, p, rt, dt);
        }
        drain_sync();
        seg_kt0 = 0;
        ++sg;
      }
      if (dt == 0) fwd_stamp(P, c, p, 7);
    }
  }

  // ---------------------------------------------------------------- teardown
  tmem_fence_before();
  __syncthreads();
  if (warp == 1) {
    tmem_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kFwdTmemCols) : "memory");
  }
  if (tid == 0) {
    fwd_stamp(P, c, P.n_phases, 1);
    __threadfence();
    sflag[2] = (atomicAdd(P.exit_count, 1u) == static_cast<unsigned>(G - 1)) ? 1 : 0;
  }
  __syncthreads();
  if (sflag[2]) {  // the last CTA out clears the flags, tickets and counters for the next launch
    __threadfence();
    for (int j = tid; j < P.n_flags; j += kFwdThreads) {
      P.flags[j] = 0u;
      P.tickets[j] = 0u;
    }
    for (int j = tid; j < P.n_phases; j += kFwdThreads) P.done[j] = 0u;
    __syncthreads();
    if (tid == 0) *P.exit_count = 0u;
  }
}

}  // namespace ssd
