// Phase table of the persistent forward kernel (one launch per greedy step,
// per drafting stage or per verification stage of Algorithm 1).
//
// A launch walks a list of phases -- embedding gather, the projections of
// x_{l+1} = x_l + f_l(x_l) (QKV, o, gate/up, down), split-KV attention, the
// imitation network and the LM head g with its argmax -- on a grid of one CTA
// per SM that stays resident for the whole list.  Phases hand tiles to each
// other through ready flags in global memory instead of kernel boundaries, so
// the weight stream of a phase starts while the previous phase is finishing.
#pragma once

#include "common.cuh"

namespace ssd {

constexpr int kFwdStages = 8;       // shared-memory ring: weight units and K/V chunks, 16 KB each
constexpr int kFwdThreads = 256;
constexpr int kFwdRows = 9;         // activation rows of one phase (gamma_max + 1)
constexpr int kFwdAcc = 4;          // TMEM accumulators of 32 fp32 columns (16 hi + 16 lo)
constexpr int kFwdAccCols = 32;
constexpr int kFwdTmemCols = 128;
constexpr int kFwdWindow = 4;       // phases sharing the split-tile scratch ring
constexpr int kFwdMaxSplits = 16;   // attention splits per head
constexpr uint32_t kFwdStageBytes = 16384;
constexpr int kFwdBTile = 4096;     // MMA B operand of one 64-column slice: 16 hi + 16 lo rows x 128 B
constexpr int kFwdBSlots = kFwdWindow + 1;  // B-operand buffers in flight (phase q uses slot q mod 5)

enum FwdKind : int {
  FK_QKV = 0,        // q/k/v projection + RoPE + KV-cache write
  FK_GATE_SILU = 1,  // gate/up pair + SiLU(gate) * up
  FK_SILU = 2,       // imitation-network FC1 + SiLU
  FK_RESID = 3,      // dst = base + scale * (W a)
  FK_ARGMAX = 4,     // LM head + argmax
  FK_ATTN = 5,       // causal split-KV attention over the cache
  FK_EMBED = 6,      // x = E[tok]
};

struct FwdPhase {
  int kind, M;                        // M activation rows (1 .. kFwdRows)
  int K, N, n_kt, n_rt, units, seg_rows;
  int map0, map1, map2;               // tensor maps (index into the map table)
  int dep;                            // phase whose tiles produce x (-1: x predates the launch)
  int dep_cols;                       // columns of x per tile of that phase
  int epi_dep;                        // phase that must be complete before this phase's epilogues
  int flags;                          // offset of this phase's tile flags and tickets
  int n_tiles;                        // tiles this phase reports
  int pos_off;                        // row m sits at position kv_len + pos_off + m
  // GEMV consumer side: byte offset of the B operands of this phase's 64-column slices in FwdParams::btiles
  long long bt_off;
  // producer side: where this phase's output columns go as the B operand of the projection that reads them
  long long bt_dst_off;               // -1: no projection reads this phase's output
  const float* bt_x;                  // that projection's input rows (fp32)
  int bt_x_stride, bt_M, bt_nkt;
  int bt_row0;                        // this phase's row 0 is row bt_row0 of that projection
  const __nv_bfloat16* bt_gain;       // its RMSNorm gain (folded into the operand), or null
  const float* x;                     // GEMV input rows / ATTN queries
  int x_stride;
  const __nv_bfloat16* gain;          // RMSNorm gain folded into the activations, or null
  float* q_out;
  int q_stride;
  float* k_cache;                     // this layer's [H][max_seq][head_dim] fp32
  float* v_cache;
  float* h_out;
  int h_stride;
  const float* base;
  int base_stride;
  float* dst;                         // RESID output, ATTN output o, EMBED rows
  int dst_stride;
  const float* scale;
  int* tok_dst;
  float* logits;
  int logits_rows;
  const int* tok_src;                 // EMBED token ids
};

struct FwdParams {
  const FwdPhase* phases;
  int n_phases;
  const CUtensorMap* maps;
  DevState* st;
  unsigned* flags;       // [n_flags] tile ready flags
  unsigned* tickets;     // [n_flags] split-tile / split-head tickets
  unsigned* done;        // [n_phases] finished tiles per phase
  unsigned* exit_count;  // CTAs that have left
  uint8_t* btiles;       // [kFwdBSlots][max n_kt][kFwdBTile] B operands, written by producer epilogues
  int n_flags;
  float* partials;       // [kFwdWindow][grid][kFwdRows][128]
  float* attn_part;      // [kFwdWindow][n_heads][4 * splits][kFwdRows][head_dim + 2] (one state per drain warp)
  int n_heads, head_dim, max_seq, splits;
  float attn_scale, eps;
  const float2* rope;    // [max_seq][head_dim / 2] (cos, sin)
  const __nv_bfloat16* embed;
  int vocab, d_model;
  // optional timeline: [grid][n_phases + 1][16] -- %globaltimer stamps of the first / last action
  // of each role in each phase (0..7) and the time each role spent waiting (8..15); row n_phases
  // holds the CTA's entry and exit.  Null when not tracing.
  unsigned long long* trace;
};

}  // namespace ssd
