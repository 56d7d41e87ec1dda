// Shape constants and parameters of the prefill (tcgen05) GEMM, shared by the
// kernels and the host engine.
#pragma once

#include "common.cuh"

namespace ssd {

constexpr int kTcM = 128;
constexpr int kTcN = 128;
constexpr int kTcK = 64;
constexpr int kTcStages = 4;
constexpr int kTcThreads = 192;
constexpr uint32_t kTcATile = kTcM * kTcK * 2;             // 16 KB
constexpr uint32_t kTcBTile = kTcN * kTcK * 2;             // 16 KB
constexpr uint32_t kTcStage = 2 * kTcATile + kTcBTile;     // 48 KB
constexpr int kTcTmemCols = 2 * kTcN;                      // double-buffered fp32 accumulator
constexpr int kTcSmem = kTcStages * kTcStage + 1024 + 256;  // + alignment slack + barriers

// The GEMM templated on its output tile width NT (128, or 256 = two 128-column sub-tiles sharing each
// A slice): ring stages, stage bytes, TMEM columns (double-buffered accumulator) and shared memory.
template <int NT>
struct TcShape {
  static constexpr int kSub = NT / kTcN;                              // 128-column sub-tiles
  static constexpr int kStages = NT == kTcN ? kTcStages : 3;
  static constexpr uint32_t kStage = 2 * kTcATile + kSub * kTcBTile;  // A hi, A lo, the sub-tiles' W
  static constexpr int kTmemCols = 2 * NT;
  static constexpr int kSmem = kStages * kStage + 1024 + 256;
};
constexpr int kFaQ = 128;  // prefill attention: query rows per CTA (the MMA's M)
constexpr int kFaK = 64;   // prefill attention: keys per block (the S MMA's N, the P.V MMA's K)

struct TcParams {
  int M, N, K;          // rows (tokens), output columns, reduction
  int tiles_m, tiles_n, k_steps;
  int seg_rows;         // QKV: rows per source matrix
  int seg_base;         // QKV: segment of the site's first matrix (0 = q; 1 = k, for a [k; v] site)
  int pos0;             // position of row 0
  DevState* st;
  // epilogues (same meaning as GemvParams)
  float* q_out;
  int q_stride;
  float* k_cache;
  float* v_cache;
  int head_dim, max_seq;
  const float2* rope_cs;  // null: no rotation (the encoder-decoder model)
  float* h_out;
  int h_stride;
  int act;                // GATE_SILU: 0 = SiLU(gate) * up, 1 = GELU_tanh(gate) * up
  const float* base;
  int base_stride;
  float* dst;
  int dst_stride;
  const float* scale;
};

}  // namespace ssd
