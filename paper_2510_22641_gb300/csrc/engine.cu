// Host engine and C ABI of the SSD library (see include/ssd.h).
//
// One ssd_ctx owns the KV cache, activation rows, workspaces, a private CUDA
// stream and the CUDA graphs that replay the decode loop.  Every projection is
// a ssd_wstream_kernel launch (stream-K weight streaming), attention is ssd_splitkv_attn_kernel
// (split-KV, causal over the query block), and the loop control of Algorithm 1
// runs in small device kernels; a decode is one graph launch whose WHILE node
// repeats draft + verify + accept on the device until the device state says
// done.
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <algorithm>
#include <atomic>
#include <cstdlib>
#include <cstring>
#include <map>
#include <string>
#include <utility>
#include <vector>

#include "attention.cuh"
#include "control.cuh"
#include "gemv.cuh"
#include "prefill_params.cuh"

namespace ssd {
cudaError_t gemv_launch_qkv(int M, const CUtensorMap*, const GemvParams&, int, cudaStream_t, bool);
cudaError_t gemv_launch_gate(int M, const CUtensorMap*, const GemvParams&, int, cudaStream_t, bool);
cudaError_t gemv_launch_silu(int M, const CUtensorMap*, const GemvParams&, int, cudaStream_t, bool);
cudaError_t gemv_launch_resid(int M, const CUtensorMap*, const GemvParams&, int, cudaStream_t, bool);
cudaError_t gemv_launch_head(int M, const CUtensorMap*, const GemvParams&, int, cudaStream_t, bool);
cudaError_t gemv_launch_xattn(int M, const CUtensorMap*, const GemvParams&, int, cudaStream_t, bool);
cudaError_t gemv_attrs_qkv();
cudaError_t gemv_attrs_gate();
cudaError_t gemv_attrs_silu();
cudaError_t gemv_attrs_resid();
cudaError_t gemv_attrs_head();
cudaError_t gemv_attrs_xattn();
cudaError_t prefill_attrs();
cudaError_t tc_gemm_launch(Epi e, int nt, const CUtensorMap* a, const CUtensorMap* b, const TcParams& p, int grid,
                           cudaStream_t s, bool pdl);
cudaError_t split_rows_launch(const float* x, int x_stride, int K, const __nv_bfloat16* gain, float eps,
                              __nv_bfloat16* hi, __nv_bfloat16* lo, int rows, cudaStream_t s, bool pdl);
cudaError_t prefill_attn_launch(int head_dim, const CUtensorMap* maps, float* o, int o_stride, int P, int n_heads,
                                int s_pad, float scale, DevState* st, cudaStream_t s, bool pdl);
cudaError_t attn_parts_launch(int head_dim, const float* q, int q_stride, const float* kc, const float* vc, int max_seq,
                              int P, int n_heads, __nv_bfloat16* parts, size_t q_elems, size_t kv_elems, int qs_stride,
                              int s_pad, cudaStream_t s, bool pdl);
cudaError_t mid_launch(Epi e, const CUtensorMap* wmaps, const CUtensorMap* amaps, const GemvParams& p, int M,
                       int num_sms, cudaStream_t s, bool pdl);
cudaError_t mid_attrs();
cudaError_t attn_launch(int M, int head_dim, const AttnParams& a, int nreq, cudaStream_t s, bool pdl);
cudaError_t attn_attrs();
int mid_max_ctas(int num_sms);
cudaError_t split_act_launch(const float* x, int x_stride, int K, const __nv_bfloat16* gain, float eps,
                             __nv_bfloat16* hi, __nv_bfloat16* lo, int ld, float* rs, int rows, cudaStream_t s,
                             bool pdl);
}  // namespace ssd

using namespace ssd;

namespace {

constexpr int kPrefillChunk = 8;  // prefill rows per pass through the layers
constexpr int kMaxVerifyRows = SSD_MAX_GAMMA + 1;  // rows of one request's verification pass
constexpr int kMidMinRows = kMaxRows + 1;  // projections over more rows use the medium-M kernel

struct Site {  // one projection: up to three weight matrices with a common K
  CUtensorMap maps[3];
  int N = 0, K = 0, n_rt = 0, n_kt = 0, units = 0, grid = 0, seg_rows = 0;
};

struct LayerSites {
  Site qkv, o, gateup, down;
};

// Weights of one projection for the prefill GEMM: 128-row (or 2 x 64-row) boxes
// of 64 columns, 128-byte swizzled.
struct TcSite {
  CUtensorMap maps[3];
  int N = 0, K = 0, tiles_n = 0, seg_rows = 0;
};

struct TcLayer {
  TcSite qkv, o, gateup, down;
};

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

// Host-side fault injection for tests of the error paths (ssd_set_fault_injection): the countdown-th
// device allocation or kernel launch after arming fails without reaching the GPU.
std::atomic<int> g_fault_kind{0};
std::atomic<int> g_fault_countdown{0};

bool injected_fault(int kind) {
  if (g_fault_kind.load() != kind) return false;
  if (g_fault_countdown.fetch_sub(1) != 1) return false;
  g_fault_kind.store(0);
  return true;
}

}  // namespace

struct ssd_ctx {
  ssd_config cfg{};
  int qdim = 0, num_sms = 0, device = 0;
  int dp = 0, qp = 0, fp = 0, ip = 0;  // activation row strides, padded to a multiple of kTileK
  // borrowed weights
  const __nv_bfloat16 *embed = nullptr, *lm_head = nullptr, *final_norm = nullptr;
  std::vector<const __nv_bfloat16*> attn_norm, ffn_norm;
  const __nv_bfloat16 *in_norm = nullptr;
  __nv_bfloat16* gains = nullptr;  // zero-padded copies of all RMSNorm gains
  const float *resid_scale = nullptr, *in_scale = nullptr;
  std::vector<LayerSites> layers;
  Site in1, in2, head;
  // prefill (tcgen05) state
  std::vector<TcLayer> tc_layers;
  std::vector<TcLayer> enc_tc_layers;  // encoder-decoder model: the encoder's layers
  std::vector<TcSite> cross_kv_tc;     // and every decoder layer's [ck; cv]
  CUtensorMap a_maps[3][2];  // activation splits (hi, lo) for K = d_model, n_heads*head_dim, d_ff
  __nv_bfloat16 *a_hi = nullptr, *a_lo = nullptr;
  float *x_pre = nullptr, *q_pre = nullptr, *o_pre = nullptr, *h_pre = nullptr;
  // the prefill attention's bf16 hi / lo operands, written by ssd_attn_parts_kernel: q rows
  // [Pm][qdim] x 2, K [H][fa_spad][Dh] x 2, V transposed [H][Dh][fa_spad] x 2; their tensor maps
  __nv_bfloat16* fa_parts = nullptr;
  CUtensorMap fa_maps[6];
  int fa_spad = 0;
  size_t fa_q_elems = 0, fa_kv_elems = 0;  // elements of one q part and of one K (or V^T) part
  bool prefill_rows = false;  // SSD_OPT_PREFILL_ROWS: prefill through the decode kernels in 8-row chunks
  // owned device memory
  DevState* st = nullptr;
  DevState* op_st = nullptr;  // state of standalone op calls (ssd_lm_head)
  int* out_int = nullptr;  // [max_seq] emitted tokens
  int2* step_log = nullptr;  // [max_seq] (accepted drafts a, gamma_eff) per step since the prefill
  float *xv = nullptr, *qb = nullptr, *ob = nullptr, *hb = nullptr, *hin = nullptr, *xt = nullptr;
  float *kc = nullptr, *vc = nullptr;  // KV cache [L][max_batch][H][max_seq][Dh], fp32
  size_t req_kv = 0;    // elements per request and layer in kc / vc
  size_t layer_kv = 0;  // elements per layer (max_batch * req_kv)
  size_t kv_slot = 0;   // request slot the single-request enqueue functions address (b * req_kv)
  // batched requests (the serving form of Algorithm 1; max_batch > 1)
  int max_batch = 1;
  int batch = 0;                 // requests of the last ssd_prefill_batch
  DevState* req = nullptr;       // [max_batch] per-request decode state
  int* bout = nullptr;           // [max_batch][max_seq] emitted tokens per request
  int2* blog = nullptr;          // [max_batch][max_seq] per-step (a, gamma_eff) per request
  __nv_bfloat16 *act_hi = nullptr, *act_lo = nullptr;  // split activations [kMaxMidRows][act_ld] (medium-M)
  float* act_rs = nullptr;       // [kMaxMidRows] RMSNorm scales of the split rows
  int act_ld = 0;
  // The next medium-M projection's operand as its producer left it in act_hi / act_lo (the attention
  // merge, or a medium-M reduction's epilogue), so that projection needs no split launch: valid
  // while act_ready, for the rows act_x (act_m of them), act_k columns, RMSNorm gain act_gain, with
  // the rows' sums of squares per producer tile in act_ssq[row][act_parts] (act_parts 0: none).
  float* act_ssq = nullptr;
  int act_ssq_ld = 0;
  bool act_ready = false;
  const float* act_x = nullptr;
  int act_m = 0, act_k = 0, act_parts = 0;
  const __nv_bfloat16* act_gain = nullptr;
  float* mid_partials = nullptr;  // [2 * grid][kMaxMidRows][kTileN]
  std::map<std::pair<int, int>, std::pair<CUtensorMap, CUtensorMap>> act_maps;  // (K, NP) -> hi, lo
  std::map<int, cudaGraphExec_t> batch_graphs;  // decode loops by gamma (0: greedy), for batch_graph_b requests
  std::map<int, int64_t> batch_body_launches;
  int batch_graph_b = 0;
  __nv_bfloat16* bvis = nullptr;  // batched prefill inputs: [max_batch * max_seq][d_model] rows, ids
  int* bprompt = nullptr;
  float2* rope = nullptr;
  float* partials = nullptr;
  unsigned* counters = nullptr;
  int n_counters = 0;
  float* attn_part = nullptr;       // split-KV attention: CTA states [H][kAttnSplit][kAttnMaxRows][Dh + 2]
  unsigned* attn_tickets = nullptr;  // [H]
  __nv_bfloat16* in_vis = nullptr;
  int* in_prompt = nullptr;
  // streams and graphs
  cudaStream_t us = nullptr, cs = nullptr;
  cudaEvent_t ev_in = nullptr, ev_out = nullptr;
  bool use_pdl = true;
  std::map<int, cudaGraphExec_t> decode_graphs, draft_graphs, verify_graphs, step_graphs;
  // dynamic draft length (Sec. "Choice of d"): d(p + 2) per kv_len p, step graphs by cap
  int* dyn_table = nullptr;   // device [max_seq + 1]
  int* dyn_launch = nullptr;  // device [SSD_MAX_GAMMA]: kernel launches of the step branch for gamma
  std::vector<int> dyn_table_h;
  int dyn_d0 = -1, dyn_n = -1, dyn_origin = -1;  // the tabulated schedule: d0, N, t's origin
  std::map<int, cudaGraphExec_t> dyn_graphs;
  int64_t dyn_host_launches = 0;
  // Diagnostic: drive the decode loop from the host with one plain graph per
  // step (ncu cannot profile kernels of graphs that hold conditional nodes).
  bool host_loop = false;
  std::map<std::pair<int, int>, cudaGraphExec_t> prefill_graphs;
  cudaGraphExec_t greedy_graph = nullptr;
  std::map<int, int64_t> decode_body_launches;
  std::map<std::pair<int, int>, int64_t> prefill_launch_count;
  int64_t greedy_body_launches = 0;
  int64_t launch_counter = 0;
  // host-side state machine
  bool prefilled = false;
  int drafted_gamma = 0;
  int prompt_len = 0;
  int64_t kv_upper = 0;  // upper bound on the device kv_len
  int last_decode_kind = 0;  // 0 none, 1 ssd, 2 greedy, 3 ssd with the dynamic draft length, 4 batched
  std::vector<int> batch_prompt;  // P_b of the prefilled batch
  int last_gamma = 0;
  std::pair<int, int> last_prefill_shape{0, 0};
  // encoder-decoder model (SSD_ARCH_T5)
  bool t5 = false;
  int max_enc = 0;
  std::vector<LayerSites> enc_layers;
  std::vector<const __nv_bfloat16*> enc_attn_norm, enc_ffn_norm, cross_norm;
  const __nv_bfloat16* enc_final = nullptr;
  std::vector<Site> cross_q, cross_o, cross_kv;      // per decoder layer: cq, co, [ck; cv]
  float *x_enc = nullptr, *enc_q = nullptr, *enc_o = nullptr;  // encoder rows [max_enc][dp or qp]
  float *enc_k = nullptr, *enc_v = nullptr;          // one encoder layer's K/V [H][max_enc][Dh]
  float *ckc = nullptr, *cvc = nullptr;              // cross-attention K/V [L][H][max_enc][Dh]
  size_t cross_layer_kv = 0;
  float *dec_bias = nullptr, *enc_bias = nullptr;    // [H][max_seq] and [H][2 max_enc - 1]
  float* one = nullptr;                              // device 1.0f: the encoder's residual scale
  int* start_tok = nullptr;                          // device copy of cfg.start_token
  // debug logits capture: full-model rows by predicted token index, draft rows by (step, j)
  float* logits_buf = nullptr;
  int logits_rows = 0;
  float* draft_logits_buf = nullptr;
  int draft_logits_steps = 0;
  std::string err;
};

// ------------------------------------------------------------------ helpers

// The kernel launches of launch_k and of the projection, attention and prefill wrappers go through
// here first: it counts the launch and reports an injected launch failure (the kernel is then not
// launched).
static cudaError_t count_launch(ssd_ctx* c) {
  ++c->launch_counter;
  return injected_fault(SSD_FAULT_LAUNCH) ? cudaErrorLaunchFailure : cudaSuccess;
}

// Layer l's K / V cache of the request slot the single-request path addresses.
static float* kv_k(ssd_ctx* c, int l) { return c->kc + l * c->layer_kv + c->kv_slot; }
static float* kv_v(ssd_ctx* c, int l) { return c->vc + l * c->layer_kv + c->kv_slot; }

static ssd_status fail(ssd_ctx* c, ssd_status s, const char* fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    c->err = buf;
  }
  return s;
}

#define CK(call)                                                                                          \
  do {                                                                                                    \
    cudaError_t e_ = (call);                                                                              \
    if (e_ != cudaSuccess) {                                                                              \
      return fail(c, e_ == cudaErrorMemoryAllocation ? SSD_ERR_OOM : SSD_ERR_CUDA, "%s failed: %s (%s:%d)", \
                  #call, cudaGetErrorString(e_), __FILE__, __LINE__);                                     \
    }                                                                                                     \
  } while (0)

#define CKS(expr)                      \
  do {                                 \
    ssd_status s_ = (expr);            \
    if (s_ != SSD_OK) return s_;       \
  } while (0)

template <typename Kern, typename... Args>
static cudaError_t launch_k(ssd_ctx* c, Kern kern, dim3 grid, dim3 block, size_t smem, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = c->cs;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = c->use_pdl ? 1 : 0;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  if (cudaError_t e = count_launch(c)) return e;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

static ssd_status encode_map_sw128(ssd_ctx* c, CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols,
                                   uint32_t box_rows) {
  if (reinterpret_cast<uintptr_t>(base) % 16 != 0)
    return fail(c, SSD_ERR_INVALID_ARG, "pointer %p is not 16-byte aligned", base);
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kTcK), box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(c, SSD_ERR_CUDA, "cuTensorMapEncodeTiled (swizzled) failed (%d)", static_cast<int>(r));
  return SSD_OK;
}

// GEMV weight boxes: box_rows x 64 columns, 128-byte swizzled (the MMA's A operand).
static ssd_status encode_map(ssd_ctx* c, CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols,
                             uint32_t box_rows) {
  return encode_map_sw128(c, m, base, rows, cols, box_rows);
}

// Site over 1..3 matrices [rows_each][K] stacked along N.  Units are 128 rows x
// 64 columns (a QKV unit holds whole heads, so RoPE pairs stay in one unit).
static ssd_status make_site(ssd_ctx* c, Site* s, const void* const* mats, int nmats, int rows_each, int K,
                            bool paired) {
  for (int i = 0; i < nmats; ++i)
    CKS(encode_map(c, &s->maps[i], mats[i], rows_each, K, kTileN));
  for (int i = nmats; i < 3; ++i) s->maps[i] = s->maps[0];
  s->N = rows_each * nmats;
  s->K = K;
  s->seg_rows = rows_each;
  s->n_rt = (s->N + kTileN - 1) / kTileN;
  s->n_kt = (K + kTileK - 1) / kTileK;
  s->units = s->n_rt * s->n_kt;
  s->grid = s->units < c->num_sms * kGemvCtasPerSm ? s->units : c->num_sms * kGemvCtasPerSm;
  return SSD_OK;
}

// gate/up pair: each unit holds 64 gate rows and the same 64 up rows.
static ssd_status make_pair_site(ssd_ctx* c, Site* s, const void* gate, const void* up, int rows, int K) {
  CKS(encode_map(c, &s->maps[0], gate, rows, K, kHalfN));
  CKS(encode_map(c, &s->maps[1], up, rows, K, kHalfN));
  s->maps[2] = s->maps[0];
  s->N = rows;
  s->K = K;
  s->seg_rows = rows;
  s->n_rt = (rows + kHalfN - 1) / kHalfN;
  s->n_kt = (K + kTileK - 1) / kTileK;
  s->units = s->n_rt * s->n_kt;
  s->grid = s->units < c->num_sms * kGemvCtasPerSm ? s->units : c->num_sms * kGemvCtasPerSm;
  return SSD_OK;
}

// One decoder (or encoder) layer's projections for the prefill GEMM: 128-row boxes (2 x 64 rows for
// the gate/up pair) of 64 columns.
static ssd_status make_tc_layer(ssd_ctx* c, TcLayer* t, const void* const qkv[3], const void* wo, const void* wg,
                                const void* wu, const void* wd, int qdim, int d_model, int d_ff) {
  for (int i = 0; i < 3; ++i) CKS(encode_map_sw128(c, &t->qkv.maps[i], qkv[i], qdim, d_model, kTcN));
  t->qkv.N = 3 * qdim;
  t->qkv.K = d_model;
  t->qkv.seg_rows = qdim;
  t->qkv.tiles_n = 3 * qdim / kTcN;
  CKS(encode_map_sw128(c, &t->o.maps[0], wo, d_model, qdim, kTcN));
  t->o.maps[1] = t->o.maps[2] = t->o.maps[0];
  t->o.N = d_model;
  t->o.K = qdim;
  t->o.seg_rows = d_model;
  t->o.tiles_n = (d_model + kTcN - 1) / kTcN;
  CKS(encode_map_sw128(c, &t->gateup.maps[0], wg, d_ff, d_model, kTcN / 2));
  CKS(encode_map_sw128(c, &t->gateup.maps[1], wu, d_ff, d_model, kTcN / 2));
  t->gateup.maps[2] = t->gateup.maps[0];
  t->gateup.N = d_ff;
  t->gateup.K = d_model;
  t->gateup.seg_rows = d_ff;
  t->gateup.tiles_n = (d_ff + kTcN / 2 - 1) / (kTcN / 2);
  CKS(encode_map_sw128(c, &t->down.maps[0], wd, d_model, d_ff, kTcN));
  t->down.maps[1] = t->down.maps[2] = t->down.maps[0];
  t->down.N = d_model;
  t->down.K = d_ff;
  t->down.seg_rows = d_model;
  t->down.tiles_n = (d_model + kTcN - 1) / kTcN;
  return SSD_OK;
}

static ssd_status gemv(ssd_ctx* c, Epi e, int M, const Site& s, GemvParams p) {
  p.K = s.K;
  p.n_kt = s.n_kt;
  p.n_rt = s.n_rt;
  p.units = s.units;
  p.N = s.N;
  p.seg_rows = s.seg_rows;
  p.partials = c->partials;
  p.counters = c->counters;
  p.st = c->st;
  p.eps = c->cfg.rms_eps;
  cudaError_t r;
  CK(count_launch(c));
  switch (e) {
    case Epi::QKV: r = gemv_launch_qkv(M, s.maps, p, s.grid, c->cs, c->use_pdl); break;
    case Epi::GATE_SILU: r = gemv_launch_gate(M, s.maps, p, s.grid, c->cs, c->use_pdl); break;
    case Epi::SILU: r = gemv_launch_silu(M, s.maps, p, s.grid, c->cs, c->use_pdl); break;
    case Epi::RESID: r = gemv_launch_resid(M, s.maps, p, s.grid, c->cs, c->use_pdl); break;
    case Epi::XATTN: r = gemv_launch_xattn(M, s.maps, p, s.grid, c->cs, c->use_pdl); break;
    default: r = gemv_launch_head(M, s.maps, p, s.grid, c->cs, c->use_pdl); break;
  }
  CK(r);
  return SSD_OK;
}

// One split-KV attention launch over M query rows per request for nreq requests (the ctx's
// scratch, state and head count filled in).
static ssd_status attn_run(ssd_ctx* c, int M, AttnParams a, int nreq = 1) {
  a.part = c->attn_part;
  a.tickets = c->attn_tickets;
  a.st = c->st;
  a.n_heads = c->cfg.n_heads;
  if (M < 1 || M > kAttnMaxRows) return fail(c, SSD_ERR_INVALID_ARG, "attention rows %d out of range", M);
  CK(count_launch(c));
  CK(attn_launch(M, c->cfg.head_dim, a, nreq, c->cs, c->use_pdl));
  return SSD_OK;
}

// Causal self-attention of layer l over the KV cache for the M rows at kv_len + pos_off + m.  The
// encoder-decoder model's decoder adds its relative-position bias and has no 1/sqrt(head_dim) factor.
// prefetch_old: the launch before is the layer's QKV projection with a late trigger.
static ssd_status attention(ssd_ctx* c, int l, int M, int pos_off, bool prefetch_old) {
  AttnParams a{};
  a.prefetch_old = prefetch_old ? 1 : 0;
  a.q = c->qb;
  a.q_stride = c->qp;
  a.k_cache = kv_k(c, l);
  a.v_cache = kv_v(c, l);
  a.o = c->ob;
  a.o_stride = c->qp;
  a.pos_off = pos_off;
  a.max_seq = c->cfg.max_seq;
  a.scale = c->t5 ? 1.0f : 1.0f / sqrtf(static_cast<float>(c->cfg.head_dim));
  if (c->t5) {
    a.bias = c->dec_bias;
    a.bias_stride = c->cfg.max_seq;
    a.bias_zero = c->cfg.max_seq - 1;
  }
  return attn_run(c, M, a);
}

// x = x + (*scale) * W in, on M rows (x: activation rows of stride dp).
static ssd_status resid_gemv(ssd_ctx* c, int M, const Site& s, const float* in, int in_stride, float* x,
                             const float* scale) {
  GemvParams p{};
  p.x = in;
  p.x_stride = in_stride;
  p.base = x;
  p.base_stride = c->dp;
  p.dst = x;
  p.dst_stride = c->dp;
  p.scale = scale;
  return gemv(c, Epi::RESID, M, s, p);
}

// One decoder layer x_{l+1} = x_l + f_l(x_l) on rows row0 .. row0+M-1 of xv at
// positions kv_len + pos_off + m.
// s_l of layer l; for l == n_layers (the IN_BLOCK imitation block) s_in.
static const float* resid_scale_of(const ssd_ctx* c, int l) {
  return l < c->cfg.n_layers ? c->resid_scale + l : c->in_scale;
}

// The QKV projection of block l on M rows x alone (RoPE + K/V writes at kv_len + pos_off + m):
// the IN_BLOCK block's cache rows of x_k rows whose block output is not needed.
static ssd_status enqueue_qkv_only(ssd_ctx* c, int l, const float* x, int M, int pos_off) {
  GemvParams p{};
  p.x = x;
  p.x_stride = c->dp;
  p.gain = c->attn_norm[l];
  p.pos_off = pos_off;
  p.q_out = c->qb;
  p.q_stride = c->qp;
  p.k_cache = kv_k(c, l);
  p.v_cache = kv_v(c, l);
  p.head_dim = c->cfg.head_dim;
  p.max_seq = c->cfg.max_seq;
  p.rope_cs = c->rope;
  return gemv(c, Epi::QKV, M, c->layers[l].qkv, p);
}

static ssd_status enqueue_layer_x(ssd_ctx* c, int l, float* x, int M, int pos_off);

static ssd_status enqueue_layer(ssd_ctx* c, int l, int row0, int M, int pos_off) {
  return enqueue_layer_x(c, l, c->xv + static_cast<size_t>(row0) * c->dp, M, pos_off);
}

// Decoder layer l of the encoder-decoder model on M rows x (positions kv_len + pos_off + m), in place:
//   x += s_l W_o Attn(RMSNorm_self(x))       causal, relative-position bias, no 1/sqrt(head_dim), no RoPE
//   x += s_l W_co CrossAttn(RMSNorm_cross(x))  over the encoder output's K/V (all st->enc_len keys)
//   x += s_l W_ff (GELU_tanh(W_i0 u) * W_i1 u), u = RMSNorm_ffn(x)
static ssd_status enqueue_t5_layer(ssd_ctx* c, int l, float* x, int M, int pos_off) {
  const int d = c->dp;
  const float* s_l = c->resid_scale + l;
  GemvParams p{};
  p.x = x;
  p.x_stride = d;
  p.gain = c->attn_norm[l];
  p.pos_off = pos_off;
  p.q_out = c->qb;
  p.q_stride = c->qp;
  p.k_cache = kv_k(c, l);
  p.v_cache = kv_v(c, l);
  p.head_dim = c->cfg.head_dim;
  p.max_seq = c->cfg.max_seq;
  p.late_trigger = 1;
  CKS(gemv(c, Epi::QKV, M, c->layers[l].qkv, p));
  CKS(attention(c, l, M, pos_off, true));
  CKS(resid_gemv(c, M, c->layers[l].o, c->ob, c->qp, x, s_l));
  p = GemvParams{};
  p.x = x;
  p.x_stride = d;
  p.gain = c->cross_norm[l];
  p.pos_off = pos_off;
  p.q_out = c->qb;
  p.q_stride = c->qp;
  p.head_dim = c->cfg.head_dim;
  p.max_seq = c->cfg.max_seq;
  if (c->max_enc <= kXattnKeys) {  // the cross-attention runs in the cross-q projection's epilogue
    p.xk = c->ckc + l * c->cross_layer_kv;
    p.xv = c->cvc + l * c->cross_layer_kv;
    p.x_max = c->max_enc;
    p.x_scale = 1.0f;
    p.xo = c->ob;
    p.xo_stride = c->qp;
    CKS(gemv(c, Epi::XATTN, M, c->cross_q[l], p));
  } else {
    CKS(gemv(c, Epi::QKV, M, c->cross_q[l], p));  // a one-matrix site: q only
    AttnParams a{};
    a.q = c->qb;
    a.q_stride = c->qp;
    a.k_cache = c->ckc + l * c->cross_layer_kv;
    a.v_cache = c->cvc + l * c->cross_layer_kv;
    a.o = c->ob;
    a.o_stride = c->qp;
    a.pos_off = pos_off;
    a.max_seq = c->max_enc;
    a.scale = 1.0f;
    a.fixed_keys = 1;
    CKS(attn_run(c, M, a));
  }
  CKS(resid_gemv(c, M, c->cross_o[l], c->ob, c->qp, x, s_l));
  p = GemvParams{};
  p.x = x;
  p.x_stride = d;
  p.gain = c->ffn_norm[l];
  p.h_out = c->hb;
  p.h_stride = c->fp;
  p.act = 1;
  CKS(gemv(c, Epi::GATE_SILU, M, c->layers[l].gateup, p));
  return resid_gemv(c, M, c->layers[l].down, c->hb, c->fp, x, s_l);
}

// Block l (a decoder layer, or the IN_BLOCK block for l == n_layers) on M rows x, in place.
static ssd_status enqueue_layer_x(ssd_ctx* c, int l, float* x, int M, int pos_off) {
  if (c->t5) return enqueue_t5_layer(c, l, x, M, pos_off);
  const int d = c->dp;
  GemvParams p{};
  p.x = x;
  p.x_stride = d;
  p.gain = c->attn_norm[l];
  p.pos_off = pos_off;
  p.q_out = c->qb;
  p.q_stride = c->qp;
  p.k_cache = kv_k(c, l);
  p.v_cache = kv_v(c, l);
  p.head_dim = c->cfg.head_dim;
  p.max_seq = c->cfg.max_seq;
  p.rope_cs = c->rope;
  p.late_trigger = 1;
  CKS(gemv(c, Epi::QKV, M, c->layers[l].qkv, p));
  CKS(attention(c, l, M, pos_off, true));
  p = GemvParams{};
  p.x = c->ob;
  p.x_stride = c->qp;
  p.base = x;
  p.base_stride = d;
  p.dst = x;
  p.dst_stride = d;
  p.scale = resid_scale_of(c, l);
  CKS(gemv(c, Epi::RESID, M, c->layers[l].o, p));
  p = GemvParams{};
  p.x = x;
  p.x_stride = d;
  p.gain = c->ffn_norm[l];
  p.h_out = c->hb;
  p.h_stride = c->fp;
  CKS(gemv(c, Epi::GATE_SILU, M, c->layers[l].gateup, p));
  p = GemvParams{};
  p.x = c->hb;
  p.x_stride = c->fp;
  p.base = x;
  p.base_stride = d;
  p.dst = x;
  p.dst_stride = d;
  p.scale = resid_scale_of(c, l);
  CKS(gemv(c, Epi::RESID, M, c->layers[l].down, p));
  return SSD_OK;
}

// LM head g(x) = W_lm RMSNorm_f(x) + greedy argmax on M rows of x.
static ssd_status enqueue_head(ssd_ctx* c, const float* x, int M, int pos_off, int* tok_dst, bool capture) {
  GemvParams p{};
  p.x = x;
  p.x_stride = c->dp;
  p.gain = c->final_norm;
  p.pos_off = pos_off;
  p.tok_dst = tok_dst;
  p.logits = capture ? c->logits_buf : nullptr;
  p.logits_rows = capture ? c->logits_rows : 0;
  return gemv(c, Epi::ARGMAX, M, c->head, p);
}

// LM head + argmax of draft row j (the token d_{j+1}); with a draft capture buffer its logits go
// to row st->steps * gamma_max + j.
static ssd_status enqueue_draft_head(ssd_ctx* c, const float* x, int j, int* tok_dst) {
  GemvParams p{};
  p.x = x;
  p.x_stride = c->dp;
  p.gain = c->final_norm;
  p.pos_off = j;
  p.tok_dst = tok_dst;
  p.logits = c->draft_logits_buf;
  p.logits_rows = c->draft_logits_buf ? c->draft_logits_steps * c->cfg.gamma_max : 0;
  p.logits_step_rows = c->cfg.gamma_max;
  return gemv(c, Epi::ARGMAX, 1, c->head, p);
}

static int* st_field(ssd_ctx* c, size_t off) {
  return reinterpret_cast<int*>(reinterpret_cast<char*>(c->st) + off);
}

// Drafting stage: gamma tokens from layers 0..k-1, the imitation network and g.
static ssd_status enqueue_draft(ssd_ctx* c, int gamma) {
  const int d = c->dp;
  int* tok_in = st_field(c, offsetof(DevState, tok_in));
  for (int j = 0; j < gamma; ++j) {
    float* xj = c->xv + static_cast<size_t>(j) * d;
    CK(launch_k(c, ssd_embed_kernel, dim3(1), dim3(256), 0, c->embed, static_cast<const int*>(tok_in + j), xj, d,
                c->cfg.d_model, c->cfg.vocab, c->st));
    for (int l = 0; l < c->cfg.draft_exit_k; ++l) CKS(enqueue_layer(c, l, j, 1, j));
    const float* hx = xj;
    if (c->cfg.in_kind == SSD_IN_BLOCK) {  // I(x_k): the imitation block on a copy (x_k stays for verification)
      CK(cudaMemcpyAsync(c->xt, xj, sizeof(float) * d, cudaMemcpyDeviceToDevice, c->cs));
      CKS(enqueue_layer_x(c, c->cfg.n_layers, c->xt, 1, j));
      hx = c->xt;
    }
    if (c->cfg.in_kind == SSD_IN_MLP2) {
      GemvParams p{};
      p.x = xj;
      p.x_stride = d;
      p.gain = c->in_norm;
      p.h_out = c->hin;
      p.h_stride = c->ip;
      CKS(gemv(c, Epi::SILU, 1, c->in1, p));
      p = GemvParams{};
      p.x = c->hin;
      p.x_stride = c->ip;
      p.base = xj;
      p.base_stride = d;
      p.dst = c->xt;
      p.dst_stride = d;
      p.scale = c->in_scale;
      CKS(gemv(c, Epi::RESID, 1, c->in2, p));
      hx = c->xt;
    }
    CKS(enqueue_draft_head(c, hx, j, tok_in + j + 1));
  }
  return SSD_OK;
}

// Verification stage + acceptance: row gamma through the shallow layers (rows
// 0..gamma-1 hold x_k from the draft), all gamma+1 rows through layers k..L-1,
// g + argmax per row, then the acceptance kernel.
static ssd_status enqueue_verify(ssd_ctx* c, int gamma, cudaGraphConditionalHandle cond, int has_cond) {
  const int d = c->dp;
  int* tok_in = st_field(c, offsetof(DevState, tok_in));
  int* full_tok = st_field(c, offsetof(DevState, full_tok));
  CK(launch_k(c, ssd_embed_kernel, dim3(1), dim3(256), 0, c->embed, static_cast<const int*>(tok_in + gamma),
              c->xv + static_cast<size_t>(gamma) * d, d, c->cfg.d_model, c->cfg.vocab, c->st));
  for (int l = 0; l < c->cfg.draft_exit_k; ++l) CKS(enqueue_layer(c, l, gamma, 1, gamma));
  if (c->cfg.in_kind == SSD_IN_BLOCK)  // the imitation block's cache row of d_gamma's x_k
    CKS(enqueue_qkv_only(c, c->cfg.n_layers, c->xv + static_cast<size_t>(gamma) * d, 1, gamma));
  for (int l = c->cfg.draft_exit_k; l < c->cfg.n_layers; ++l) CKS(enqueue_layer(c, l, 0, gamma + 1, 0));
  CKS(enqueue_head(c, c->xv, gamma + 1, 0, full_tok, true));
  CK(launch_k(c, ssd_accept_kernel, dim3(1), dim3(32), 0, c->st, gamma, c->out_int, c->cfg.max_seq, c->step_log,
              c->cfg.max_seq, cond,
              has_cond));
  return SSD_OK;
}

static ssd_status enqueue_greedy_step(ssd_ctx* c, cudaGraphConditionalHandle cond, int has_cond) {
  int* tok_in = st_field(c, offsetof(DevState, tok_in));
  int* full_tok = st_field(c, offsetof(DevState, full_tok));
  CK(launch_k(c, ssd_embed_kernel, dim3(1), dim3(256), 0, c->embed, static_cast<const int*>(tok_in), c->xv, c->dp,
              c->cfg.d_model, c->cfg.vocab, c->st));
  for (int l = 0; l < c->cfg.n_layers; ++l) CKS(enqueue_layer(c, l, 0, 1, 0));
  CKS(enqueue_head(c, c->xv, 1, 0, full_tok, true));
  CK(launch_k(c, ssd_greedy_accept_kernel, dim3(1), dim3(32), 0, c->st, c->out_int, c->cfg.max_seq, c->step_log,
              c->cfg.max_seq, cond, has_cond));
  return SSD_OK;
}

static ssd_status enqueue_prefill(ssd_ctx* c, int n_vis, int n_prompt) {
  const int d = c->dp, P = n_vis + n_prompt;
  int* full_tok = st_field(c, offsetof(DevState, full_tok));
  // tickets of the split-row reductions start from zero (a previous aborted run may have left some)
  CK(cudaMemsetAsync(c->counters, 0, sizeof(unsigned) * c->n_counters, c->cs));
  CK(cudaMemsetAsync(c->attn_tickets, 0, sizeof(unsigned) * c->max_batch * c->cfg.n_heads, c->cs));
  CK(launch_k(c, ssd_prefill_begin_kernel, dim3(1), dim3(32), 0, c->st, P, c->cfg.eos_id, 0));
  int r0 = 0;
  for (; r0 < P; r0 += kPrefillChunk) {
    const int Mc = P - r0 < kPrefillChunk ? P - r0 : kPrefillChunk;
    CK(launch_k(c, ssd_prefill_rows_kernel, dim3(Mc), dim3(256), 0, static_cast<const __nv_bfloat16*>(c->in_vis),
                static_cast<const int*>(c->in_prompt), n_vis, r0, c->embed, c->cfg.vocab, c->xv, d, c->cfg.d_model, c->st));
    for (int l = 0; l < c->cfg.n_layers; ++l) {
      if (l == c->cfg.draft_exit_k && c->cfg.in_kind == SSD_IN_BLOCK)  // the block's cache rows of x_k
        CKS(enqueue_qkv_only(c, c->cfg.n_layers, c->xv, Mc, r0));
      CKS(enqueue_layer(c, l, 0, Mc, r0));
    }
    if (c->cfg.draft_exit_k == c->cfg.n_layers && c->cfg.in_kind == SSD_IN_BLOCK)
      CKS(enqueue_qkv_only(c, c->cfg.n_layers, c->xv, Mc, r0));
  }
  r0 -= kPrefillChunk;
  CKS(enqueue_head(c, c->xv + static_cast<size_t>(P - 1 - r0) * d, 1, P - 1, full_tok, true));
  CK(launch_k(c, ssd_prefill_finish_kernel, dim3(1), dim3(32), 0, c->st, c->out_int, P));
  return SSD_OK;
}

// Prefill of the encoder-decoder model (Sec. "SSD Setup for VLMs" with the BLIP-2 FlanT5 language
// model): the encoder over the P rows [z; embed(prompt)] in chunks of kPrefillChunk rows through the
// decode kernels (bidirectional attention: every row sees all P keys, with the encoder's
// relative-position bias), the cross-attention K/V of every decoder layer from the encoder's normed
// output, then the decoder on start_token at position 0, whose greedy token is the first new token.
static ssd_status enqueue_prefill_t5(ssd_ctx* c, int n_vis, int n_prompt) {
  const int P = n_vis + n_prompt, dp = c->dp, qp = c->qp;
  int* full_tok = st_field(c, offsetof(DevState, full_tok));
  CK(cudaMemsetAsync(c->counters, 0, sizeof(unsigned) * c->n_counters, c->cs));
  CK(cudaMemsetAsync(c->attn_tickets, 0, sizeof(unsigned) * c->max_batch * c->cfg.n_heads, c->cs));
  CK(launch_k(c, ssd_prefill_begin_kernel, dim3(1), dim3(32), 0, c->st, 1, c->cfg.eos_id, P));
  CK(launch_k(c, ssd_prefill_rows_kernel, dim3(P), dim3(256), 0, static_cast<const __nv_bfloat16*>(c->in_vis),
              static_cast<const int*>(c->in_prompt), n_vis, 0, c->embed, c->cfg.vocab, c->x_enc, dp, c->cfg.d_model,
              c->st));
  for (int e = 0; e < c->cfg.n_enc_layers; ++e) {
    const LayerSites& S = c->enc_layers[e];
    for (int r0 = 0; r0 < P; r0 += kPrefillChunk) {
      const int Mc = std::min(kPrefillChunk, P - r0);
      GemvParams p{};
      p.x = c->x_enc + static_cast<size_t>(r0) * dp;
      p.x_stride = dp;
      p.gain = c->enc_attn_norm[e];
      p.pos_off = r0;
      p.abs_pos = 1;
      p.q_out = c->enc_q + static_cast<size_t>(r0) * qp;
      p.q_stride = qp;
      p.k_cache = c->enc_k;
      p.v_cache = c->enc_v;
      p.head_dim = c->cfg.head_dim;
      p.max_seq = c->max_enc;
      CKS(gemv(c, Epi::QKV, Mc, S.qkv, p));
    }
    for (int r0 = 0; r0 < P; r0 += kPrefillChunk) {
      const int Mc = std::min(kPrefillChunk, P - r0);
      AttnParams a{};
      a.q = c->enc_q + static_cast<size_t>(r0) * qp;
      a.q_stride = qp;
      a.k_cache = c->enc_k;
      a.v_cache = c->enc_v;
      a.o = c->enc_o + static_cast<size_t>(r0) * qp;
      a.o_stride = qp;
      a.pos_off = r0;
      a.abs_pos = 1;
      a.fixed_keys = 1;
      a.max_seq = c->max_enc;
      a.scale = 1.0f;
      a.bias = c->enc_bias;
      a.bias_stride = 2 * c->max_enc - 1;
      a.bias_zero = c->max_enc - 1;
      CKS(attn_run(c, Mc, a));
    }
    for (int r0 = 0; r0 < P; r0 += kPrefillChunk) {
      const int Mc = std::min(kPrefillChunk, P - r0);
      float* xr = c->x_enc + static_cast<size_t>(r0) * dp;
      CKS(resid_gemv(c, Mc, S.o, c->enc_o + static_cast<size_t>(r0) * qp, qp, xr, c->one));
      GemvParams p{};
      p.x = xr;
      p.x_stride = dp;
      p.gain = c->enc_ffn_norm[e];
      p.h_out = c->hb;
      p.h_stride = c->fp;
      p.act = 1;
      CKS(gemv(c, Epi::GATE_SILU, Mc, S.gateup, p));
      CKS(resid_gemv(c, Mc, S.down, c->hb, c->fp, xr, c->one));
    }
  }
  for (int l = 0; l < c->cfg.n_layers; ++l)
    for (int r0 = 0; r0 < P; r0 += kPrefillChunk) {
      const int Mc = std::min(kPrefillChunk, P - r0);
      GemvParams p{};
      p.x = c->x_enc + static_cast<size_t>(r0) * dp;
      p.x_stride = dp;
      p.gain = c->enc_final;  // cross K/V read the encoder's normed output
      p.pos_off = r0;
      p.abs_pos = 1;
      p.seg_base = 1;  // the [ck; cv] site's segments are k and v
      p.k_cache = c->ckc + l * c->cross_layer_kv;
      p.v_cache = c->cvc + l * c->cross_layer_kv;
      p.head_dim = c->cfg.head_dim;
      p.max_seq = c->max_enc;
      CKS(gemv(c, Epi::QKV, Mc, c->cross_kv[l], p));
    }
  CK(launch_k(c, ssd_embed_kernel, dim3(1), dim3(256), 0, c->embed, static_cast<const int*>(c->start_tok), c->xv, dp,
              c->cfg.d_model, c->cfg.vocab, c->st));
  for (int l = 0; l < c->cfg.n_layers; ++l) CKS(enqueue_layer(c, l, 0, 1, 0));
  CKS(enqueue_head(c, c->xv, 1, 0, full_tok, true));
  CK(launch_k(c, ssd_prefill_finish_kernel, dim3(1), dim3(32), 0, c->st, c->out_int, 1));
  return SSD_OK;
}

// Prefill over all P rows at once: activation splits + tcgen05 GEMMs with the
// fused epilogues, and causal attention over the prompt.
static ssd_status tc_gemm(ssd_ctx* c, Epi e, int kidx, const TcSite& site, int P, TcParams p) {
  p.M = P;
  p.N = site.N;
  p.K = site.K;
  p.tiles_m = (P + kTcM - 1) / kTcM;
  p.tiles_n = site.tiles_n;
  p.k_steps = site.K / kTcK;
  p.seg_rows = site.seg_rows;
  p.st = c->st;
  // 256-column tiles (each A slice feeds two 128-column weight tiles, halving the A traffic per flop)
  // where they still give every SM a tile
  const int wide_tiles = p.tiles_m * ((p.tiles_n + 1) / 2);
  const int nt = (e == Epi::QKV || e == Epi::GATE_SILU) && wide_tiles >= c->num_sms ? 256 : 128;
  const int tiles = nt == 256 ? wide_tiles : p.tiles_m * p.tiles_n;
  CK(count_launch(c));
  CK(tc_gemm_launch(e, nt, c->a_maps[kidx], site.maps, p, tiles < c->num_sms ? tiles : c->num_sms, c->cs,
                    c->use_pdl));
  return SSD_OK;
}

static ssd_status split(ssd_ctx* c, const float* x, int x_stride, int K, const __nv_bfloat16* gain, int P) {
  CK(count_launch(c));
  CK(split_rows_launch(x, x_stride, K, gain, c->cfg.rms_eps, c->a_hi, c->a_lo, P, c->cs, c->use_pdl));
  return SSD_OK;
}

static ssd_status enqueue_prefill_tc(ssd_ctx* c, int n_vis, int n_prompt) {
  const int P = n_vis + n_prompt, dp = c->dp;
  int* full_tok = st_field(c, offsetof(DevState, full_tok));
  CK(cudaMemsetAsync(c->counters, 0, sizeof(unsigned) * c->n_counters, c->cs));
  CK(cudaMemsetAsync(c->attn_tickets, 0, sizeof(unsigned) * c->max_batch * c->cfg.n_heads, c->cs));
  CK(launch_k(c, ssd_prefill_begin_kernel, dim3(1), dim3(32), 0, c->st, P, c->cfg.eos_id, 0));
  CK(launch_k(c, ssd_prefill_rows_kernel, dim3(P), dim3(256), 0, static_cast<const __nv_bfloat16*>(c->in_vis),
              static_cast<const int*>(c->in_prompt), n_vis, 0, c->embed, c->cfg.vocab, c->x_pre, dp, c->cfg.d_model,
              c->st));
  // the IN_BLOCK block's cache rows of every prompt row's x_k: its QKV GEMM alone
  auto block_kv = [&]() -> ssd_status {
    const int b = c->cfg.n_layers;
    TcParams p{};
    p.pos0 = 0;
    p.q_out = c->q_pre;
    p.q_stride = c->qp;
    p.k_cache = kv_k(c, b);
    p.v_cache = kv_v(c, b);
    p.head_dim = c->cfg.head_dim;
    p.max_seq = c->cfg.max_seq;
    p.rope_cs = c->rope;
    CKS(split(c, c->x_pre, dp, c->cfg.d_model, c->attn_norm[b], P));
    return tc_gemm(c, Epi::QKV, 0, c->tc_layers[b].qkv, P, p);
  };
  for (int l = 0; l < c->cfg.n_layers; ++l) {
    if (l == c->cfg.draft_exit_k && c->cfg.in_kind == SSD_IN_BLOCK) CKS(block_kv());
    const TcLayer& tl = c->tc_layers[l];
    TcParams p{};
    p.pos0 = 0;
    p.q_out = c->q_pre;
    p.q_stride = c->qp;
    p.k_cache = kv_k(c, l);
    p.v_cache = kv_v(c, l);
    p.head_dim = c->cfg.head_dim;
    p.max_seq = c->cfg.max_seq;
    p.rope_cs = c->rope;
    CKS(split(c, c->x_pre, dp, c->cfg.d_model, c->attn_norm[l], P));
    CKS(tc_gemm(c, Epi::QKV, 0, tl.qkv, P, p));
    CK(count_launch(c));
    CK(attn_parts_launch(c->cfg.head_dim, c->q_pre, c->qp, kv_k(c, l), kv_v(c, l), c->cfg.max_seq, P, c->cfg.n_heads,
                         c->fa_parts, c->fa_q_elems, c->fa_kv_elems, c->qdim, c->fa_spad, c->cs, c->use_pdl));
    CK(count_launch(c));
    CK(prefill_attn_launch(c->cfg.head_dim, c->fa_maps, c->o_pre, c->qp, P, c->cfg.n_heads, c->fa_spad,
                           1.0f / sqrtf(static_cast<float>(c->cfg.head_dim)), c->st, c->cs, c->use_pdl));
    CKS(split(c, c->o_pre, c->qp, c->qdim, nullptr, P));
    p = TcParams{};
    p.base = c->x_pre;
    p.base_stride = dp;
    p.dst = c->x_pre;
    p.dst_stride = dp;
    p.scale = resid_scale_of(c, l);
    CKS(tc_gemm(c, Epi::RESID, 1, tl.o, P, p));
    CKS(split(c, c->x_pre, dp, c->cfg.d_model, c->ffn_norm[l], P));
    p = TcParams{};
    p.h_out = c->h_pre;
    p.h_stride = c->fp;
    CKS(tc_gemm(c, Epi::GATE_SILU, 0, tl.gateup, P, p));
    CKS(split(c, c->h_pre, c->fp, c->cfg.d_ff, nullptr, P));
    p = TcParams{};
    p.base = c->x_pre;
    p.base_stride = dp;
    p.dst = c->x_pre;
    p.dst_stride = dp;
    p.scale = resid_scale_of(c, l);
    CKS(tc_gemm(c, Epi::RESID, 2, tl.down, P, p));
  }
  if (c->cfg.draft_exit_k == c->cfg.n_layers && c->cfg.in_kind == SSD_IN_BLOCK) CKS(block_kv());
  CKS(enqueue_head(c, c->x_pre + static_cast<size_t>(P - 1) * dp, 1, P - 1, full_tok, true));
  CK(launch_k(c, ssd_prefill_finish_kernel, dim3(1), dim3(32), 0, c->st, c->out_int, P));
  return SSD_OK;
}

// Prefill of the encoder-decoder model through the tensor-core GEMM (the same steps as
// enqueue_prefill_t5): each encoder projection runs once over all P rows -- activation split,
// tcgen05 GEMM with the fused epilogue (q/k/v without rotation into the encoder's K/V, scaled
// residual adds, gated GELU) -- the bidirectional attention with the encoder's relative-position
// bias in 16-row launches, then every decoder layer's cross K/V from one split of the encoder's
// normed output, and the decoder on start_token.
static ssd_status enqueue_prefill_t5_tc(ssd_ctx* c, int n_vis, int n_prompt) {
  const int P = n_vis + n_prompt, dp = c->dp, qp = c->qp;
  int* full_tok = st_field(c, offsetof(DevState, full_tok));
  CK(cudaMemsetAsync(c->counters, 0, sizeof(unsigned) * c->n_counters, c->cs));
  CK(cudaMemsetAsync(c->attn_tickets, 0, sizeof(unsigned) * c->max_batch * c->cfg.n_heads, c->cs));
  CK(launch_k(c, ssd_prefill_begin_kernel, dim3(1), dim3(32), 0, c->st, 1, c->cfg.eos_id, P));
  CK(launch_k(c, ssd_prefill_rows_kernel, dim3(P), dim3(256), 0, static_cast<const __nv_bfloat16*>(c->in_vis),
              static_cast<const int*>(c->in_prompt), n_vis, 0, c->embed, c->cfg.vocab, c->x_enc, dp, c->cfg.d_model,
              c->st));
  for (int e = 0; e < c->cfg.n_enc_layers; ++e) {
    const TcLayer& tl = c->enc_tc_layers[e];
    TcParams p{};
    p.pos0 = 0;
    p.q_out = c->enc_q;
    p.q_stride = qp;
    p.k_cache = c->enc_k;
    p.v_cache = c->enc_v;
    p.head_dim = c->cfg.head_dim;
    p.max_seq = c->max_enc;
    CKS(split(c, c->x_enc, dp, c->cfg.d_model, c->enc_attn_norm[e], P));
    CKS(tc_gemm(c, Epi::QKV, 0, tl.qkv, P, p));
    for (int r0 = 0; r0 < P; r0 += kAttnMaxRows) {
      const int Mc = std::min(kAttnMaxRows, P - r0);
      AttnParams a{};
      a.q = c->enc_q + static_cast<size_t>(r0) * qp;
      a.q_stride = qp;
      a.k_cache = c->enc_k;
      a.v_cache = c->enc_v;
      a.o = c->enc_o + static_cast<size_t>(r0) * qp;
      a.o_stride = qp;
      a.pos_off = r0;
      a.abs_pos = 1;
      a.fixed_keys = 1;
      a.max_seq = c->max_enc;
      a.scale = 1.0f;
      a.bias = c->enc_bias;
      a.bias_stride = 2 * c->max_enc - 1;
      a.bias_zero = c->max_enc - 1;
      CKS(attn_run(c, Mc, a));
    }
    CKS(split(c, c->enc_o, qp, c->qdim, nullptr, P));
    p = TcParams{};
    p.base = c->x_enc;
    p.base_stride = dp;
    p.dst = c->x_enc;
    p.dst_stride = dp;
    p.scale = c->one;
    CKS(tc_gemm(c, Epi::RESID, 1, tl.o, P, p));
    CKS(split(c, c->x_enc, dp, c->cfg.d_model, c->enc_ffn_norm[e], P));
    p = TcParams{};
    p.h_out = c->h_pre;
    p.h_stride = c->fp;
    p.act = 1;
    CKS(tc_gemm(c, Epi::GATE_SILU, 0, tl.gateup, P, p));
    CKS(split(c, c->h_pre, c->fp, c->cfg.d_ff, nullptr, P));
    p = TcParams{};
    p.base = c->x_enc;
    p.base_stride = dp;
    p.dst = c->x_enc;
    p.dst_stride = dp;
    p.scale = c->one;
    CKS(tc_gemm(c, Epi::RESID, 2, tl.down, P, p));
  }
  CKS(split(c, c->x_enc, dp, c->cfg.d_model, c->enc_final, P));  // cross K/V read the encoder's normed output
  for (int l = 0; l < c->cfg.n_layers; ++l) {
    TcParams p{};
    p.pos0 = 0;
    p.seg_base = 1;  // the [ck; cv] site's segments are k and v
    p.k_cache = c->ckc + l * c->cross_layer_kv;
    p.v_cache = c->cvc + l * c->cross_layer_kv;
    p.head_dim = c->cfg.head_dim;
    p.max_seq = c->max_enc;
    CKS(tc_gemm(c, Epi::QKV, 0, c->cross_kv_tc[l], P, p));
  }
  CK(launch_k(c, ssd_embed_kernel, dim3(1), dim3(256), 0, c->embed, static_cast<const int*>(c->start_tok), c->xv, dp,
              c->cfg.d_model, c->cfg.vocab, c->st));
  for (int l = 0; l < c->cfg.n_layers; ++l) CKS(enqueue_layer(c, l, 0, 1, 0));
  CKS(enqueue_head(c, c->xv, 1, 0, full_tok, true));
  CK(launch_k(c, ssd_prefill_finish_kernel, dim3(1), dim3(32), 0, c->st, c->out_int, 1));
  return SSD_OK;
}

// ------------------------------------------------------------------ batched requests
// The serving form of Algorithm 1: B requests, each with its own prompt, positions, cache slot
// and accept lengths, decode in lockstep.  Request b's row i (i = 0..g) of a step lives in row
// b * (g + 1) + i of xv, so drafting step j's rows (a stride of g + 1 rows) are exactly where the
// verification pass needs x_k (option B).  Every launch carries all B requests, finished ones
// too (their rows are computed and never used), so a step has one shape and one graph.

// The split activations' tensor maps for K columns and NP rows (built once per shape).
static ssd_status act_maps_for(ssd_ctx* c, int K, int NP, const CUtensorMap** out) {
  auto key = std::make_pair(K, NP);
  auto it = c->act_maps.find(key);
  if (it == c->act_maps.end()) {
    std::pair<CUtensorMap, CUtensorMap> m;
    CKS(encode_map_sw128(c, &m.first, c->act_hi, kMaxMidRows, K, NP));
    CKS(encode_map_sw128(c, &m.second, c->act_lo, kMaxMidRows, K, NP));
    it = c->act_maps.emplace(key, m).first;
  }
  *out = &it->second.first;  // hi, then lo (adjacent in the pair)
  return SSD_OK;
}

// The medium-M projection that reads the output of the one being enqueued: its rows x, columns K and
// RMSNorm gain, and whether it needs the rows' sums of squares (it has a gain).
struct NextSplit {
  const float* x;
  int K;
  const __nv_bfloat16* gain;
};

// Records that act_hi / act_lo now hold the operand of the projection nx describes over M rows.
static void set_act_ready(ssd_ctx* c, const NextSplit& nx, int M, int parts) {
  c->act_ready = true;
  c->act_x = nx.x;
  c->act_m = M;
  c->act_k = nx.K;
  c->act_gain = nx.gain;
  c->act_parts = parts;
}

// One projection over M > kMaxRows rows: the rows are split into bf16 hi / lo parts with their
// RMSNorm scales (gain folded in), then the medium-M tensor-core kernel streams the weights once.
// The split launch is skipped when the producing kernel already wrote this projection's parts
// (act_ready for the same rows, width and gain); with nx, this projection's reduction writes the
// next one's parts (and, when that one has a gain, the rows' sums of squares per output tile).
static ssd_status mid_gemm(ssd_ctx* c, Epi e, int M, const Site& s, GemvParams p, const NextSplit* nx = nullptr) {
  if (M > kMaxMidRows || !c->act_hi) return fail(c, SSD_ERR_INVALID_ARG, "%d rows exceed the medium-M kernel", M);
  const bool fused = c->act_ready && c->act_x == p.x && c->act_m == M && c->act_k == s.K && c->act_gain == p.gain &&
                     (p.gain == nullptr || c->act_parts > 0);
  c->act_ready = false;
  if (fused) {
    p.rs_parts = p.gain ? c->act_ssq : nullptr;
    p.rs_nparts = p.gain ? c->act_parts : 0;
  } else {
    CK(count_launch(c));
    CK(split_act_launch(p.x, p.x_stride, s.K, p.gain, c->cfg.rms_eps, c->act_hi, c->act_lo, s.K, c->act_rs, M, c->cs,
                        c->use_pdl));
    p.rs_in = c->act_rs;
  }
  if (nx) {
    if (nx->K > c->act_ld || (nx->gain && (e != Epi::RESID || s.n_rt > c->act_ssq_ld || p.rs_parts)))
      return fail(c, SSD_ERR_INVALID_ARG, "no fused split for this projection pair");
    p.nx_hi = c->act_hi;
    p.nx_lo = c->act_lo;
    p.nx_ld = nx->K;
    p.nx_gain = nx->gain;
    p.nx_ssq = nx->gain ? c->act_ssq : nullptr;
  }
  CUtensorMap amaps[2];
  const CUtensorMap* am = nullptr;
  CKS(act_maps_for(c, s.K, (M + 15) & ~15, &am));
  amaps[0] = am[0];
  amaps[1] = am[1];
  p.K = s.K;
  p.n_kt = s.n_kt;
  p.n_rt = s.n_rt;
  p.units = s.units;
  p.N = s.N;
  p.seg_rows = s.seg_rows;
  p.partials = c->mid_partials;
  p.counters = c->counters;
  p.st = c->st;
  p.eps = c->cfg.rms_eps;
  CK(count_launch(c));  // the stream
  CK(count_launch(c));  // the reduction + epilogue
  CK(mid_launch(e, s.maps, amaps, p, M, c->num_sms, c->cs, c->use_pdl));
  if (nx) set_act_ready(c, *nx, M, nx->gain ? s.n_rt : 0);
  return SSD_OK;
}

// A projection over M rows of the batch: the GEMV up to kMaxRows rows, the medium-M kernel beyond.
static ssd_status proj_rows(ssd_ctx* c, Epi e, int M, const Site& s, const GemvParams& p,
                            const NextSplit* nx = nullptr) {
  if (M <= kMaxRows) {
    c->act_ready = false;
    return gemv(c, e, M, s, p);
  }
  return mid_gemm(c, e, M, s, p, nx);
}

static void set_batch_rows(ssd_ctx* c, GemvParams& p, int R) {
  p.batch_rows = R;
  p.req_st = c->req;
  p.req_kv = static_cast<long long>(c->req_kv);
  p.tok_stride = static_cast<int>(sizeof(DevState) / sizeof(int));
}

// Decoder layer l on M = B * R rows x (row stride x_stride): request b's rows b * R .. b * R + R - 1
// at positions req[b].kv_len + pos_off + i, in place.
static ssd_status enqueue_layer_batch(ssd_ctx* c, int l, float* x, int x_stride, int M, int R, int pos_off) {
  GemvParams p{};
  p.x = x;
  p.x_stride = x_stride;
  p.gain = c->attn_norm[l];
  p.pos_off = pos_off;
  p.q_out = c->qb;
  p.q_stride = c->qp;
  p.k_cache = c->kc + l * c->layer_kv;
  p.v_cache = c->vc + l * c->layer_kv;
  p.head_dim = c->cfg.head_dim;
  p.max_seq = c->cfg.max_seq;
  p.rope_cs = c->rope;
  p.late_trigger = 1;
  set_batch_rows(c, p, R);
  CKS(proj_rows(c, Epi::QKV, M, c->layers[l].qkv, p));
  AttnParams a{};
  a.prefetch_old = 1;
  a.q = c->qb;
  a.q_stride = c->qp;
  a.k_cache = c->kc + l * c->layer_kv;
  a.v_cache = c->vc + l * c->layer_kv;
  a.o = c->ob;
  a.o_stride = c->qp;
  a.pos_off = pos_off;
  a.max_seq = c->cfg.max_seq;
  a.scale = 1.0f / sqrtf(static_cast<float>(c->cfg.head_dim));
  a.batch_rows = R;
  a.req_st = c->req;
  a.req_kv = static_cast<long long>(c->req_kv);
  // Medium-M rows: each kernel also writes the next projection's bf16 operand parts, so only the
  // first projection of a pass runs the split launch (o reads the attention's parts, gate/up the
  // o reduction's, down the gate/up reduction's, the next layer's q/k/v or the head the down's).
  const bool mid = M > kMaxRows && c->act_hi;
  const NextSplit o_in{c->ob, c->layers[l].o.K, nullptr};
  if (mid) {
    a.xo_hi = c->act_hi;
    a.xo_lo = c->act_lo;
    a.xo_ld = o_in.K;
  }
  c->act_ready = false;
  CKS(attn_run(c, R, a, M / R));
  if (mid) set_act_ready(c, o_in, M, 0);
  const NextSplit gate_in{x, c->layers[l].gateup.K, c->ffn_norm[l]};
  const NextSplit down_in{c->hb, c->layers[l].down.K, nullptr};
  const bool last = l + 1 >= c->cfg.n_layers;
  const NextSplit next_in{x, last ? c->head.K : c->layers[l + 1].qkv.K, last ? c->final_norm : c->attn_norm[l + 1]};
  p = GemvParams{};
  p.x = c->ob;
  p.x_stride = c->qp;
  p.base = x;
  p.base_stride = x_stride;
  p.dst = x;
  p.dst_stride = x_stride;
  p.scale = resid_scale_of(c, l);
  CKS(proj_rows(c, Epi::RESID, M, c->layers[l].o, p, &gate_in));
  p = GemvParams{};
  p.x = x;
  p.x_stride = x_stride;
  p.gain = c->ffn_norm[l];
  p.h_out = c->hb;
  p.h_stride = c->fp;
  CKS(proj_rows(c, Epi::GATE_SILU, M, c->layers[l].gateup, p, &down_in));
  p = GemvParams{};
  p.x = c->hb;
  p.x_stride = c->fp;
  p.base = x;
  p.base_stride = x_stride;
  p.dst = x;
  p.dst_stride = x_stride;
  p.scale = resid_scale_of(c, l);
  return proj_rows(c, Epi::RESID, M, c->layers[l].down, p, &next_in);
}

// LM head + argmax over M = B * R rows x: row (b, i) writes its token to tok0[b][i] (tok0 a field of
// req[0], indexed across requests by the DevState stride); draft heads (draft = true) capture their
// logits by (request, step, j = pos_off), full-model heads by (request, predicted token index).
static ssd_status enqueue_head_batch(ssd_ctx* c, const float* x, int x_stride, int M, int R, int pos_off, int* tok0,
                                     bool draft) {
  GemvParams p{};
  p.x = x;
  p.x_stride = x_stride;
  p.gain = c->final_norm;
  p.pos_off = pos_off;
  p.tok_dst = tok0;
  set_batch_rows(c, p, R);
  if (draft) {
    p.logits = c->draft_logits_buf;
    p.logits_rows = c->draft_logits_buf ? c->draft_logits_steps * c->cfg.gamma_max : 0;
    p.logits_step_rows = c->cfg.gamma_max;
  } else {
    p.logits = c->logits_buf;
    p.logits_rows = c->logits_buf ? c->logits_rows : 0;
  }
  return proj_rows(c, Epi::ARGMAX, M, c->head, p);
}

// Drafting stage of every request (gamma tokens each): layers 0..k-1 and the imitation network at
// M = B rows per token.
static ssd_status enqueue_draft_batch(ssd_ctx* c, int gamma) {
  const int B = c->batch, d = c->dp, rs = (gamma + 1) * c->dp;
  for (int j = 0; j < gamma; ++j) {
    float* xj = c->xv + static_cast<size_t>(j) * d;
    CK(launch_k(c, ssd_batch_embed_kernel, dim3(B), dim3(256), 0, c->embed, static_cast<const DevState*>(c->req), j,
                xj, rs, c->cfg.d_model, c->cfg.vocab, c->st));
    for (int l = 0; l < c->cfg.draft_exit_k; ++l) CKS(enqueue_layer_batch(c, l, xj, rs, B, 1, j));
    const float* hx = xj;
    int hx_stride = rs;
    if (c->cfg.in_kind == SSD_IN_MLP2) {
      GemvParams p{};
      p.x = xj;
      p.x_stride = rs;
      p.gain = c->in_norm;
      p.h_out = c->hin;
      p.h_stride = c->ip;
      CKS(gemv(c, Epi::SILU, B, c->in1, p));
      p = GemvParams{};
      p.x = c->hin;
      p.x_stride = c->ip;
      p.base = xj;
      p.base_stride = rs;
      p.dst = c->xt;
      p.dst_stride = d;
      p.scale = c->in_scale;
      CKS(gemv(c, Epi::RESID, B, c->in2, p));
      hx = c->xt;
      hx_stride = d;
    }
    CKS(enqueue_head_batch(c, hx, hx_stride, B, 1, j, &c->req[0].tok_in[j + 1], true));
  }
  return SSD_OK;
}

// Verification of every request's gamma + 1 rows and the acceptance: row gamma of each request
// through layers 0..k-1 (M = B), all B * (gamma + 1) rows through layers k..L-1 and the head.
static ssd_status enqueue_verify_batch(ssd_ctx* c, int gamma, cudaGraphConditionalHandle cond, int has_cond) {
  const int B = c->batch, d = c->dp, R = gamma + 1, rs = R * c->dp;
  float* xg = c->xv + static_cast<size_t>(gamma) * d;
  c->act_ready = false;
  CK(launch_k(c, ssd_batch_embed_kernel, dim3(B), dim3(256), 0, c->embed, static_cast<const DevState*>(c->req),
              gamma, xg, rs, c->cfg.d_model, c->cfg.vocab, c->st));
  for (int l = 0; l < c->cfg.draft_exit_k; ++l) CKS(enqueue_layer_batch(c, l, xg, rs, B, 1, gamma));
  for (int l = c->cfg.draft_exit_k; l < c->cfg.n_layers; ++l) CKS(enqueue_layer_batch(c, l, c->xv, d, B * R, R, 0));
  CKS(enqueue_head_batch(c, c->xv, d, B * R, R, 0, &c->req[0].full_tok[0], false));
  CK(launch_k(c, ssd_batch_accept_kernel, dim3(1), dim3(32 * ((B + 31) / 32)), 0, c->st, c->req, B, gamma, c->bout,
              c->cfg.max_seq, c->blog, c->cfg.max_seq, cond, has_cond));
  return SSD_OK;
}

// One greedy step of every request (the batched baseline): all L layers at M = B rows.
static ssd_status enqueue_greedy_batch(ssd_ctx* c, cudaGraphConditionalHandle cond, int has_cond) {
  const int B = c->batch, d = c->dp;
  CK(launch_k(c, ssd_batch_embed_kernel, dim3(B), dim3(256), 0, c->embed, static_cast<const DevState*>(c->req), 0,
              c->xv, d, c->cfg.d_model, c->cfg.vocab, c->st));
  for (int l = 0; l < c->cfg.n_layers; ++l) CKS(enqueue_layer_batch(c, l, c->xv, d, B, 1, 0));
  CKS(enqueue_head_batch(c, c->xv, d, B, 1, 0, &c->req[0].full_tok[0], false));
  CK(launch_k(c, ssd_batch_accept_kernel, dim3(1), dim3(32 * ((B + 31) / 32)), 0, c->st, c->req, B, 0, c->bout,
              c->cfg.max_seq, c->blog, c->cfg.max_seq, cond, has_cond));
  return SSD_OK;
}

static ssd_status enqueue_prefill_any(ssd_ctx* c, int n_vis, int n_prompt);

// Prefill of request b: the single-request prefill with its state, token row, inputs and cache
// slot swapped in (launched directly; every request has its own prompt length).
static ssd_status enqueue_prefill_slot(ssd_ctx* c, int b, const __nv_bfloat16* vis, const int* prompt, int n_vis,
                                       int n_prompt) {
  DevState* st = c->st;
  int* out = c->out_int;
  __nv_bfloat16* iv = c->in_vis;
  int* ip = c->in_prompt;
  c->st = c->req + b;
  c->out_int = c->bout + static_cast<size_t>(b) * c->cfg.max_seq;
  c->in_vis = const_cast<__nv_bfloat16*>(vis);
  c->in_prompt = const_cast<int*>(prompt);
  c->kv_slot = static_cast<size_t>(b) * c->req_kv;
  float* lg = c->logits_buf;  // request b's captured logits start at its own block of rows
  if (lg) c->logits_buf = lg + static_cast<size_t>(b) * c->logits_rows * c->cfg.vocab;
  const ssd_status r = enqueue_prefill_any(c, n_vis, n_prompt);
  c->logits_buf = lg;
  c->st = st;
  c->out_int = out;
  c->in_vis = iv;
  c->in_prompt = ip;
  c->kv_slot = 0;
  return r;
}

// ------------------------------------------------------------------ graphs

static ssd_status begin_capture(ssd_ctx* c, cudaGraph_t g) {
  CK(cudaStreamBeginCaptureToGraph(c->cs, g, nullptr, nullptr, 0, cudaStreamCaptureModeThreadLocal));
  return SSD_OK;
}

static ssd_status end_capture(ssd_ctx* c, cudaGraph_t g, ssd_status inner) {
  cudaGraph_t out = nullptr;
  cudaError_t e = cudaStreamEndCapture(c->cs, &out);
  if (inner != SSD_OK) return inner;
  if (e != cudaSuccess) return fail(c, SSD_ERR_CUDA, "stream capture failed: %s", cudaGetErrorString(e));
  (void)g;
  return SSD_OK;
}

// Graph = [loop_begin] -> WHILE(cond) { body }.  body is draft+verify+accept
// (gamma > 0) or one greedy step (gamma == 0), of one request or (batched) of every request.
static ssd_status build_loop_graph(ssd_ctx* c, int gamma, cudaGraphExec_t* exec, int64_t* body_launches,
                                   bool batched = false) {
  cudaGraph_t g = nullptr;
  CK(cudaGraphCreate(&g, 0));
  cudaGraphConditionalHandle cond;
  ssd_status s = SSD_OK;
  cudaError_t e = cudaGraphConditionalHandleCreate(&cond, g, 0, cudaGraphCondAssignDefault);
  if (e != cudaSuccess) {
    cudaGraphDestroy(g);
    CK(e);
  }
  s = begin_capture(c, g);
  if (s == SSD_OK) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1);
    cfg.blockDim = dim3(32);
    cfg.stream = c->cs;
    e = cudaLaunchKernelEx(&cfg, ssd_loop_begin_kernel, c->st, cond);
    s = end_capture(c, g, e == cudaSuccess ? SSD_OK : fail(c, SSD_ERR_CUDA, "loop_begin launch: %s",
                                                           cudaGetErrorString(e)));
  }
  cudaGraphNode_t begin = nullptr;
  size_t n = 1;
  if (s == SSD_OK && cudaGraphGetNodes(g, &begin, &n) != cudaSuccess) s = fail(c, SSD_ERR_CUDA, "graph nodes");
  cudaGraphNodeParams cp = {};
  cp.type = cudaGraphNodeTypeConditional;
  cp.conditional.handle = cond;
  cp.conditional.type = cudaGraphCondTypeWhile;
  cp.conditional.size = 1;
  cudaGraphNode_t cnode;
  if (s == SSD_OK) {
    e = cudaGraphAddNode(&cnode, g, &begin, nullptr, 1, &cp);
    if (e != cudaSuccess) s = fail(c, SSD_ERR_CUDA, "conditional node: %s", cudaGetErrorString(e));
  }
  if (s == SSD_OK) {
    cudaGraph_t body = cp.conditional.phGraph_out[0];
    s = begin_capture(c, body);
    if (s == SSD_OK) {
      const int64_t l0 = c->launch_counter;
      ssd_status inner = SSD_OK;
      if (batched) {
        inner = gamma > 0 ? enqueue_draft_batch(c, gamma) : SSD_OK;
        if (inner == SSD_OK) inner = gamma > 0 ? enqueue_verify_batch(c, gamma, cond, 1) : enqueue_greedy_batch(c, cond, 1);
      } else {
        inner = gamma > 0 ? enqueue_draft(c, gamma) : SSD_OK;
        if (inner == SSD_OK) inner = gamma > 0 ? enqueue_verify(c, gamma, cond, 1) : enqueue_greedy_step(c, cond, 1);
      }
      *body_launches = c->launch_counter - l0;
      s = end_capture(c, body, inner);
    }
  }
  if (s == SSD_OK) {
    e = cudaGraphInstantiate(exec, g, 0);
    if (e != cudaSuccess) s = fail(c, SSD_ERR_CUDA, "graph instantiate: %s", cudaGetErrorString(e));
  }
  cudaGraphDestroy(g);
  return s;
}

using EnqueueFn = ssd_status (*)(ssd_ctx*, int, int);

static ssd_status build_plain_graph(ssd_ctx* c, EnqueueFn fn, int a0, int a1, cudaGraphExec_t* exec,
                                    int64_t* launches) {
  cudaGraph_t g = nullptr;
  CK(cudaGraphCreate(&g, 0));
  ssd_status s = begin_capture(c, g);
  if (s == SSD_OK) {
    const int64_t l0 = c->launch_counter;
    ssd_status inner = fn(c, a0, a1);
    if (launches) *launches = c->launch_counter - l0;
    s = end_capture(c, g, inner);
  }
  if (s == SSD_OK) {
    cudaError_t e = cudaGraphInstantiate(exec, g, 0);
    if (e != cudaSuccess) s = fail(c, SSD_ERR_CUDA, "graph instantiate: %s", cudaGetErrorString(e));
  }
  cudaGraphDestroy(g);
  return s;
}

// d(t) of Sec. "Choice of d" in fp64: d0 + floor(10 / (1 + exp(-0.01 (t - N/2)))).
static int draft_length_fp64(int t, int d0, int n_max) {
  const double z = -0.01 * (static_cast<double>(t) - static_cast<double>(n_max) / 2.0);
  return d0 + static_cast<int>(std::floor(10.0 / (1.0 + std::exp(z))));
}

// Kernel launch without the programmatic-serialization attribute (graph nodes whose upstream is
// a conditional node, or that have none).
template <typename Kern, typename... Args>
static cudaError_t launch_plain(ssd_ctx* c, Kern kern, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(1);
  cfg.blockDim = dim3(32);
  cfg.stream = c->cs;
  if (cudaError_t e = count_launch(c)) return e;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

// Dynamic-length SSD graph = [loop_begin] -> WHILE(cond) { select -> SWITCH(sw) { branch g - 1:
// draft g + verify g + accept, g = 1..cap } -> loop test }.  The select kernel picks the branch
// from the d(t) table; the loop test (in the WHILE body itself) sets cond.
static ssd_status build_dyn_graph(ssd_ctx* c, int cap, cudaGraphExec_t* exec) {
  cudaGraph_t g = nullptr;
  CK(cudaGraphCreate(&g, 0));
  cudaGraphConditionalHandle cond;
  cudaError_t e = cudaGraphConditionalHandleCreate(&cond, g, 0, cudaGraphCondAssignDefault);
  if (e != cudaSuccess) {
    cudaGraphDestroy(g);
    CK(e);
  }
  ssd_status s = begin_capture(c, g);
  if (s == SSD_OK) {
    e = launch_plain(c, ssd_loop_begin_kernel, c->st, cond);
    s = end_capture(c, g, e == cudaSuccess ? SSD_OK : fail(c, SSD_ERR_CUDA, "loop_begin: %s", cudaGetErrorString(e)));
  }
  cudaGraphNode_t begin = nullptr;
  size_t n = 1;
  if (s == SSD_OK && cudaGraphGetNodes(g, &begin, &n) != cudaSuccess) s = fail(c, SSD_ERR_CUDA, "graph nodes");
  cudaGraphNodeParams wp = {};
  wp.type = cudaGraphNodeTypeConditional;
  wp.conditional.handle = cond;
  wp.conditional.type = cudaGraphCondTypeWhile;
  wp.conditional.size = 1;
  cudaGraphNode_t wnode;
  if (s == SSD_OK && (e = cudaGraphAddNode(&wnode, g, &begin, nullptr, 1, &wp)) != cudaSuccess)
    s = fail(c, SSD_ERR_CUDA, "WHILE node: %s", cudaGetErrorString(e));
  std::vector<int> launches(cap, 0);
  if (s == SSD_OK) {
    cudaGraph_t body = wp.conditional.phGraph_out[0];
    cudaGraphConditionalHandle sw;
    if ((e = cudaGraphConditionalHandleCreate(&sw, body, 0, 0)) != cudaSuccess)
      s = fail(c, SSD_ERR_CUDA, "switch handle: %s", cudaGetErrorString(e));
    if (s == SSD_OK) s = begin_capture(c, body);
    if (s == SSD_OK) {
      e = launch_plain(c, ssd_dyn_select_kernel, c->st, static_cast<const int*>(c->dyn_table),
                       static_cast<const int*>(c->dyn_launch), cap, sw);
      s = end_capture(c, body, e == cudaSuccess ? SSD_OK : fail(c, SSD_ERR_CUDA, "select: %s", cudaGetErrorString(e)));
    }
    cudaGraphNode_t sel = nullptr;
    size_t nb = 1;
    if (s == SSD_OK && cudaGraphGetNodes(body, &sel, &nb) != cudaSuccess) s = fail(c, SSD_ERR_CUDA, "body nodes");
    cudaGraphNodeParams sp = {};
    sp.type = cudaGraphNodeTypeConditional;
    sp.conditional.handle = sw;
    sp.conditional.type = cudaGraphCondTypeSwitch;
    sp.conditional.size = static_cast<unsigned>(cap);
    cudaGraphNode_t snode;
    if (s == SSD_OK && (e = cudaGraphAddNode(&snode, body, &sel, nullptr, 1, &sp)) != cudaSuccess)
      s = fail(c, SSD_ERR_CUDA, "SWITCH node: %s", cudaGetErrorString(e));
    for (int i = 0; s == SSD_OK && i < cap; ++i) {
      cudaGraph_t br = sp.conditional.phGraph_out[i];
      s = begin_capture(c, br);
      if (s == SSD_OK) {
        const int64_t l0 = c->launch_counter;
        ssd_status inner = enqueue_draft(c, i + 1);
        if (inner == SSD_OK) inner = enqueue_verify(c, i + 1, 0, 0);
        launches[i] = static_cast<int>(c->launch_counter - l0);
        s = end_capture(c, br, inner);
      }
    }
    if (s == SSD_OK) {
      if ((e = cudaStreamBeginCaptureToGraph(c->cs, body, &snode, nullptr, 1, cudaStreamCaptureModeThreadLocal)) !=
          cudaSuccess)
        s = fail(c, SSD_ERR_CUDA, "capture after SWITCH: %s", cudaGetErrorString(e));
      if (s == SSD_OK) {
        e = launch_plain(c, ssd_loop_continue_kernel, c->st, cond);
        s = end_capture(c, body, e == cudaSuccess ? SSD_OK : fail(c, SSD_ERR_CUDA, "loop test: %s", cudaGetErrorString(e)));
      }
    }
  }
  if (s == SSD_OK && (e = cudaMemcpy(c->dyn_launch, launches.data(), sizeof(int) * cap, cudaMemcpyHostToDevice)) !=
                         cudaSuccess)
    s = fail(c, SSD_ERR_CUDA, "launch counts: %s", cudaGetErrorString(e));
  if (s == SSD_OK && (e = cudaGraphInstantiate(exec, g, 0)) != cudaSuccess)
    s = fail(c, SSD_ERR_CUDA, "graph instantiate: %s", cudaGetErrorString(e));
  cudaGraphDestroy(g);
  return s;
}

static ssd_status enq_prefill_fn(ssd_ctx* c, int a, int b) {
  if (c->t5) return c->prefill_rows ? enqueue_prefill_t5(c, a, b) : enqueue_prefill_t5_tc(c, a, b);
  return c->prefill_rows ? enqueue_prefill(c, a, b) : enqueue_prefill_tc(c, a, b);
}
static ssd_status enqueue_prefill_any(ssd_ctx* c, int n_vis, int n_prompt) { return enq_prefill_fn(c, n_vis, n_prompt); }
static ssd_status enq_draft_fn(ssd_ctx* c, int g, int) { return enqueue_draft(c, g); }
static ssd_status enq_verify_fn(ssd_ctx* c, int g, int) { return enqueue_verify(c, g, 0, 0); }
// One decode step without a conditional node (host-driven loop, used for profiling).
static ssd_status enq_step_fn(ssd_ctx* c, int g, int) {
  if (g == 0) return enqueue_greedy_step(c, 0, 0);
  CKS(enqueue_draft(c, g));
  return enqueue_verify(c, g, 0, 0);
}

static void drop_graphs(ssd_ctx* c) {
  for (auto& kv : c->decode_graphs) cudaGraphExecDestroy(kv.second);
  for (auto& kv : c->draft_graphs) cudaGraphExecDestroy(kv.second);
  for (auto& kv : c->verify_graphs) cudaGraphExecDestroy(kv.second);
  for (auto& kv : c->step_graphs) cudaGraphExecDestroy(kv.second);
  c->step_graphs.clear();
  for (auto& kv : c->prefill_graphs) cudaGraphExecDestroy(kv.second);
  for (auto& kv : c->dyn_graphs) cudaGraphExecDestroy(kv.second);
  c->dyn_graphs.clear();
  if (c->greedy_graph) cudaGraphExecDestroy(c->greedy_graph);
  for (auto& kv : c->batch_graphs) cudaGraphExecDestroy(kv.second);
  c->batch_graphs.clear();
  c->decode_graphs.clear();
  c->draft_graphs.clear();
  c->verify_graphs.clear();
  c->prefill_graphs.clear();
  c->greedy_graph = nullptr;
}

// Order the private stream after the caller's stream, and back.
static ssd_status enter(ssd_ctx* c) {
  CK(cudaEventRecord(c->ev_in, c->us));
  CK(cudaStreamWaitEvent(c->cs, c->ev_in, 0));
  return SSD_OK;
}
static ssd_status leave(ssd_ctx* c) {
  CK(cudaEventRecord(c->ev_out, c->cs));
  CK(cudaStreamWaitEvent(c->us, c->ev_out, 0));
  return SSD_OK;
}

static ssd_status read_device_error(ssd_ctx* c) {
  int errw = 0;
  CK(cudaMemcpy(&errw, reinterpret_cast<char*>(c->st) + offsetof(DevState, error), sizeof(int),
                cudaMemcpyDeviceToHost));
  for (int b = 0; b < c->batch; ++b) {  // a batched prefill records faults in the request's state
    int e = 0;
    CK(cudaMemcpy(&e, reinterpret_cast<char*>(c->req + b) + offsetof(DevState, error), sizeof(int),
                  cudaMemcpyDeviceToHost));
    errw |= e;
  }
  if (errw & DERR_TIMEOUT) return fail(c, SSD_ERR_TIMEOUT, "a bounded device wait ran out (error word %d)", errw);
  if (errw) return fail(c, SSD_ERR_DEVICE, "device error word %d (1 = bad token id, 4 = position out of range)", errw);
  return SSD_OK;
}

// ------------------------------------------------------------------ C ABI

extern "C" {

const char* ssd_status_string(ssd_status s) {
  switch (s) {
    case SSD_OK: return "ok";
    case SSD_ERR_INVALID_ARG: return "invalid argument";
    case SSD_ERR_OOM: return "out of device memory";
    case SSD_ERR_CUDA: return "CUDA error";
    case SSD_ERR_CAPACITY: return "KV cache capacity exceeded";
    case SSD_ERR_STATE: return "call out of order";
    case SSD_ERR_TIMEOUT: return "device wait timed out";
    case SSD_ERR_DEVICE: return "device-side error";
    case SSD_ERR_UNSUPPORTED: return "unsupported device";
  }
  return "unknown status";
}

const char* ssd_last_error(const ssd_ctx* c) { return c ? c->err.c_str() : "null context"; }

static ssd_status alloc(ssd_ctx* c, void** p, size_t bytes) {
  cudaError_t e = injected_fault(SSD_FAULT_ALLOC) ? cudaErrorMemoryAllocation : cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    *p = nullptr;
    return fail(c, SSD_ERR_OOM, "cudaMalloc(%zu) failed: %s", bytes, cudaGetErrorString(e));
  }
  e = cudaMemset(*p, 0, bytes);
  if (e != cudaSuccess) return fail(c, SSD_ERR_CUDA, "cudaMemset failed: %s", cudaGetErrorString(e));
  return SSD_OK;
}

ssd_status ssd_destroy(ssd_ctx* c) {
  if (!c) return SSD_OK;
  if (c->cs) cudaStreamSynchronize(c->cs);
  drop_graphs(c);
  void* bufs[] = {c->fa_parts, c->a_hi, c->a_lo, c->x_pre, c->q_pre, c->o_pre, c->h_pre, c->st, c->op_st, c->out_int, c->step_log, c->xv, c->qb, c->ob, c->hb, c->hin, c->xt, c->kc, c->vc, c->rope, c->gains,
                  c->partials, c->counters, c->attn_part, c->attn_tickets, c->dyn_table, c->dyn_launch, c->in_vis, c->in_prompt,
                  c->x_enc, c->enc_q, c->enc_o, c->enc_k, c->enc_v, c->ckc, c->cvc, c->dec_bias, c->enc_bias, c->one,
                  c->start_tok, c->req, c->bout, c->blog, c->bvis, c->bprompt, c->act_hi, c->act_lo, c->act_rs,
                  c->mid_partials};
  for (void* b : bufs)
    if (b) cudaFree(b);
  if (c->ev_in) cudaEventDestroy(c->ev_in);
  if (c->ev_out) cudaEventDestroy(c->ev_out);
  if (c->cs) cudaStreamDestroy(c->cs);
  delete c;
  return SSD_OK;
}

// Relative-position bucket of the key-minus-query offset delta (T5 v1.1): bidirectional stacks split
// the buckets between earlier (and equal) and later keys, past-only stacks give all of them to
// earlier keys (later keys share bucket 0); within a half, offsets below n/2 get one bucket each and
// larger ones logarithmically spaced buckets up to max_distance, beyond which they share the last.
// The logarithmic index is computed in fp64 and floored after adding 1e-9, so that exact powers land
// on their bucket whatever the platform's log rounds to.
static int rel_bucket_host(int delta, bool bidirectional, int n_buckets, int max_distance) {
  int n = n_buckets, base = 0, dist;
  if (bidirectional) {
    n /= 2;
    if (delta > 0) base = n;
    dist = delta < 0 ? -delta : delta;
  } else {
    dist = delta < 0 ? -delta : 0;
  }
  const int exact = n / 2;
  if (dist < exact) return base + dist;
  const double f = std::log(static_cast<double>(dist) / exact) / std::log(static_cast<double>(max_distance) / exact) *
                       (n - exact) + 1e-9;
  const int far = exact + static_cast<int>(f);
  return base + (far < n - 1 ? far : n - 1);
}

// out[h][j] = rel[bucket(j - zero)][h] for j < n, on the ctx stream (bucket decided on the host).
static ssd_status build_bias_table(ssd_ctx* c, const void* rel, float* out, int n, int zero, bool bidirectional) {
  std::vector<int> b(n);
  for (int j = 0; j < n; ++j)
    b[j] = rel_bucket_host(j - zero, bidirectional, c->cfg.rel_buckets, c->cfg.rel_max_distance);
  int* db = nullptr;
  CK(cudaMalloc(&db, sizeof(int) * n));
  cudaError_t e = cudaMemcpy(db, b.data(), sizeof(int) * n, cudaMemcpyHostToDevice);
  const int H = c->cfg.n_heads;
  if (e == cudaSuccess) {
    ssd_bias_table_kernel<<<(n * H + 255) / 256, 256, 0, c->cs>>>(static_cast<const __nv_bfloat16*>(rel), db, n, H, out);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->cs);
  cudaFree(db);
  CK(e);
  return SSD_OK;
}

static ssd_status create_impl(ssd_ctx* c, const ssd_config* cfg, const ssd_weights* w) {
  const ssd_config& k = *cfg;
  const bool t5 = k.arch == SSD_ARCH_T5;
  if (k.arch != SSD_ARCH_LLAMA && !t5) return fail(c, SSD_ERR_INVALID_ARG, "arch %d", k.arch);
  if (k.n_layers < 1 || k.d_model < 64 || k.n_heads < 1 || k.vocab < 2 || k.d_ff < 64)
    return fail(c, SSD_ERR_INVALID_ARG, "bad model shape");
  if (k.head_dim != 64 && k.head_dim != 128) return fail(c, SSD_ERR_INVALID_ARG, "head_dim must be 64 or 128");
  const int qdim = k.n_heads * k.head_dim;
  constexpr int kAlign = 64;  // row strides stay 128-byte multiples for TMA
  if (k.d_model % kAlign || k.d_ff % kAlign || qdim % 128)
    return fail(c, SSD_ERR_INVALID_ARG, "d_model, d_ff must be multiples of 64 and n_heads*head_dim of 128");
  if (k.draft_exit_k < 1 || k.draft_exit_k > k.n_layers) return fail(c, SSD_ERR_INVALID_ARG, "draft_exit_k");
  if (k.in_kind != SSD_IN_IDENTITY && k.in_kind != SSD_IN_MLP2 && k.in_kind != SSD_IN_BLOCK)
    return fail(c, SSD_ERR_INVALID_ARG, "in_kind");
  if (k.in_kind == SSD_IN_MLP2 && (k.in_hidden < 64 || k.in_hidden % kAlign))
    return fail(c, SSD_ERR_INVALID_ARG, "in_hidden must be a positive multiple of 64");
  if (k.gamma_max < 1 || k.gamma_max > SSD_MAX_GAMMA || k.gamma_max + 1 > kMaxVerifyRows)
    return fail(c, SSD_ERR_INVALID_ARG, "gamma_max must be in [1, %d]", SSD_MAX_GAMMA);
  if (k.max_seq < 2) return fail(c, SSD_ERR_INVALID_ARG, "max_seq");
  const int max_batch = k.max_batch < 1 ? 1 : k.max_batch;
  if (max_batch > kMaxRows) return fail(c, SSD_ERR_INVALID_ARG, "max_batch %d > %d", k.max_batch, kMaxRows);
  if (max_batch > 1) {
    if (t5 || k.in_kind == SSD_IN_BLOCK)
      return fail(c, SSD_ERR_INVALID_ARG, "batched requests need SSD_ARCH_LLAMA with SSD_IN_IDENTITY or SSD_IN_MLP2");
    if (max_batch * (k.gamma_max + 1) > kMaxMidRows)
      return fail(c, SSD_ERR_INVALID_ARG, "max_batch * (gamma_max + 1) = %d > %d", max_batch * (k.gamma_max + 1),
                  kMaxMidRows);
  }
  if (!w || !w->embed || !w->lm_head || !w->final_norm || !w->wq || !w->wk || !w->wv || !w->wo || !w->w_gate ||
      !w->w_up || !w->w_down || !w->attn_norm || !w->ffn_norm || !w->resid_scale)
    return fail(c, SSD_ERR_INVALID_ARG, "null weight pointer");
  if (k.in_kind == SSD_IN_MLP2 && (!w->in_norm || !w->in_w1 || !w->in_w2 || !w->in_scale))
    return fail(c, SSD_ERR_INVALID_ARG, "null imitation-network weight pointer");
  if (k.in_kind == SSD_IN_BLOCK) {
    if (!w->in_block || !w->in_scale) return fail(c, SSD_ERR_INVALID_ARG, "null imitation-block weight pointer");
    for (int i = 0; i < 9; ++i)
      if (!w->in_block[i]) return fail(c, SSD_ERR_INVALID_ARG, "null imitation-block weight pointer %d", i);
  }
  for (int l = 0; l < k.n_layers; ++l)
    if (!w->wq[l] || !w->wk[l] || !w->wv[l] || !w->wo[l] || !w->w_gate[l] || !w->w_up[l] || !w->w_down[l] ||
        !w->attn_norm[l] || !w->ffn_norm[l])
      return fail(c, SSD_ERR_INVALID_ARG, "null weight pointer in layer %d", l);
  const ssd_encdec_weights* ed = t5 ? w->encdec : nullptr;
  if (t5) {
    if (k.in_kind == SSD_IN_BLOCK)
      return fail(c, SSD_ERR_INVALID_ARG, "the encoder-decoder model takes SSD_IN_IDENTITY or SSD_IN_MLP2");
    if (k.n_enc_layers < 1 || k.max_enc < 1) return fail(c, SSD_ERR_INVALID_ARG, "n_enc_layers / max_enc");
    if (k.rel_buckets < 4 || k.rel_buckets % 2 || k.rel_max_distance <= k.rel_buckets / 2)
      return fail(c, SSD_ERR_INVALID_ARG, "rel_buckets must be even and >= 4, rel_max_distance > rel_buckets / 2");
    if (k.start_token < 0 || k.start_token >= k.vocab) return fail(c, SSD_ERR_INVALID_ARG, "start_token");
    if (!ed || !ed->cq || !ed->ck || !ed->cv || !ed->co || !ed->cross_norm || !ed->enc_wq || !ed->enc_wk ||
        !ed->enc_wv || !ed->enc_wo || !ed->enc_wi0 || !ed->enc_wi1 || !ed->enc_wff || !ed->enc_attn_norm ||
        !ed->enc_ffn_norm || !ed->enc_final || !ed->enc_rel || !ed->dec_rel)
      return fail(c, SSD_ERR_INVALID_ARG, "null encoder-decoder weight pointer");
    for (int l = 0; l < k.n_layers; ++l)
      if (!ed->cq[l] || !ed->ck[l] || !ed->cv[l] || !ed->co[l] || !ed->cross_norm[l])
        return fail(c, SSD_ERR_INVALID_ARG, "null cross-attention weight pointer in layer %d", l);
    for (int e = 0; e < k.n_enc_layers; ++e)
      if (!ed->enc_wq[e] || !ed->enc_wk[e] || !ed->enc_wv[e] || !ed->enc_wo[e] || !ed->enc_wi0[e] ||
          !ed->enc_wi1[e] || !ed->enc_wff[e] || !ed->enc_attn_norm[e] || !ed->enc_ffn_norm[e])
        return fail(c, SSD_ERR_INVALID_ARG, "null weight pointer in encoder layer %d", e);
  }

  CK(cudaGetDevice(&c->device));
  cudaDeviceProp prop;
  CK(cudaGetDeviceProperties(&prop, c->device));
  if (prop.major != 10) return fail(c, SSD_ERR_UNSUPPORTED, "needs a Blackwell sm_103 device, got sm_%d%d",
                                    prop.major, prop.minor);
  c->num_sms = prop.multiProcessorCount;
  if (k.options & ~(SSD_OPT_HOST_LOOP | SSD_OPT_PREFILL_ROWS))
    return fail(c, SSD_ERR_INVALID_ARG, "unknown option bits 0x%x", k.options);
  c->host_loop = (k.options & SSD_OPT_HOST_LOOP) != 0;
  c->prefill_rows = (k.options & SSD_OPT_PREFILL_ROWS) != 0;
  if (!g_encode) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    CK(cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q));
    if (q != cudaDriverEntryPointSuccess || !fn) return fail(c, SSD_ERR_UNSUPPORTED, "cuTensorMapEncodeTiled");
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  CK(gemv_attrs_qkv());
  CK(gemv_attrs_gate());
  CK(gemv_attrs_silu());
  CK(gemv_attrs_resid());
  CK(gemv_attrs_head());
  CK(gemv_attrs_xattn());
  CK(attn_attrs());
  CK(prefill_attrs());
  CK(mid_attrs());

  c->cfg = k;
  c->max_batch = max_batch;
  c->qdim = qdim;
  c->t5 = t5;
  c->max_enc = t5 ? k.max_enc : 0;
  auto pad = [](int v) { return (v + kTileK - 1) / kTileK * kTileK; };
  c->dp = pad(k.d_model);
  c->qp = pad(qdim);
  c->fp = pad(k.d_ff);
  c->ip = pad(k.in_hidden > 0 ? k.in_hidden : 64);
  c->embed = static_cast<const __nv_bfloat16*>(w->embed);
  c->lm_head = static_cast<const __nv_bfloat16*>(w->lm_head);
  c->final_norm = static_cast<const __nv_bfloat16*>(w->final_norm);
  c->in_norm = static_cast<const __nv_bfloat16*>(w->in_norm);
  c->resid_scale = w->resid_scale;
  c->in_scale = w->in_scale;
  // layer l's weights; l == n_layers: the IN_BLOCK imitation block
  const int n_blocks = k.n_layers + (k.in_kind == SSD_IN_BLOCK ? 1 : 0);
  auto wt = [&](int l, int i) -> const void* {
    if (l == k.n_layers) return w->in_block[i];
    const void* const* a[9] = {w->wq, w->wk, w->wv, w->wo, w->w_gate, w->w_up, w->w_down, w->attn_norm, w->ffn_norm};
    return a[i][l];
  };
  c->layers.resize(n_blocks);
  for (int l = 0; l < n_blocks; ++l) {
    c->attn_norm.push_back(static_cast<const __nv_bfloat16*>(wt(l, 7)));
    c->ffn_norm.push_back(static_cast<const __nv_bfloat16*>(wt(l, 8)));
    const void* qkv[3] = {wt(l, 0), wt(l, 1), wt(l, 2)};
    const void* wo_l = wt(l, 3);
    const void* wd_l = wt(l, 6);
    CKS(make_site(c, &c->layers[l].qkv, qkv, 3, qdim, k.d_model, false));
    CKS(make_site(c, &c->layers[l].o, &wo_l, 1, k.d_model, qdim, false));
    CKS(make_pair_site(c, &c->layers[l].gateup, wt(l, 4), wt(l, 5), k.d_ff, k.d_model));
    CKS(make_site(c, &c->layers[l].down, &wd_l, 1, k.d_model, k.d_ff, false));
  }
  if (k.in_kind == SSD_IN_MLP2) {
    CKS(make_site(c, &c->in1, &w->in_w1, 1, k.in_hidden, k.d_model, false));
    CKS(make_site(c, &c->in2, &w->in_w2, 1, k.d_model, k.in_hidden, false));
  }
  CKS(make_site(c, &c->head, &w->lm_head, 1, k.vocab, k.d_model, false));
  if (t5) {
    c->cross_q.resize(k.n_layers);
    c->cross_o.resize(k.n_layers);
    c->cross_kv.resize(k.n_layers);
    for (int l = 0; l < k.n_layers; ++l) {
      const void* kv[2] = {ed->ck[l], ed->cv[l]};
      CKS(make_site(c, &c->cross_q[l], &ed->cq[l], 1, qdim, k.d_model, false));
      CKS(make_site(c, &c->cross_o[l], &ed->co[l], 1, k.d_model, qdim, false));
      CKS(make_site(c, &c->cross_kv[l], kv, 2, qdim, k.d_model, false));
    }
    c->enc_layers.resize(k.n_enc_layers);
    for (int e = 0; e < k.n_enc_layers; ++e) {
      LayerSites& S = c->enc_layers[e];
      const void* qkv[3] = {ed->enc_wq[e], ed->enc_wk[e], ed->enc_wv[e]};
      CKS(make_site(c, &S.qkv, qkv, 3, qdim, k.d_model, false));
      CKS(make_site(c, &S.o, &ed->enc_wo[e], 1, k.d_model, qdim, false));
      CKS(make_pair_site(c, &S.gateup, ed->enc_wi0[e], ed->enc_wi1[e], k.d_ff, k.d_model));
      CKS(make_site(c, &S.down, &ed->enc_wff[e], 1, k.d_model, k.d_ff, false));
    }
  }
  c->tc_layers.resize(n_blocks);
  for (int l = 0; l < n_blocks; ++l) {
    const void* qkv[3] = {wt(l, 0), wt(l, 1), wt(l, 2)};
    CKS(make_tc_layer(c, &c->tc_layers[l], qkv, wt(l, 3), wt(l, 4), wt(l, 5), wt(l, 6), qdim, k.d_model, k.d_ff));
  }
  if (t5) {  // the encoder's projections and every decoder layer's [ck; cv] for the prefill GEMM
    c->enc_tc_layers.resize(k.n_enc_layers);
    for (int e = 0; e < k.n_enc_layers; ++e) {
      const void* qkv[3] = {ed->enc_wq[e], ed->enc_wk[e], ed->enc_wv[e]};
      CKS(make_tc_layer(c, &c->enc_tc_layers[e], qkv, ed->enc_wo[e], ed->enc_wi0[e], ed->enc_wi1[e], ed->enc_wff[e],
                        qdim, k.d_model, k.d_ff));
    }
    c->cross_kv_tc.resize(k.n_layers);
    for (int l = 0; l < k.n_layers; ++l) {
      TcSite& t = c->cross_kv_tc[l];
      CKS(encode_map_sw128(c, &t.maps[0], ed->ck[l], qdim, k.d_model, kTcN));
      CKS(encode_map_sw128(c, &t.maps[1], ed->cv[l], qdim, k.d_model, kTcN));
      t.maps[2] = t.maps[0];
      t.N = 2 * qdim;
      t.K = k.d_model;
      t.seg_rows = qdim;
      t.tiles_n = 2 * qdim / kTcN;
    }
  }

  // owned memory (activation rows: one request's passes, or every request's verification rows)
  const int R = std::max(kMaxRows, max_batch * (k.gamma_max + 1));
  const size_t d = k.d_model;
  CKS(alloc(c, reinterpret_cast<void**>(&c->st), sizeof(DevState)));
  CKS(alloc(c, reinterpret_cast<void**>(&c->op_st), sizeof(DevState)));
  CKS(alloc(c, reinterpret_cast<void**>(&c->out_int), sizeof(int) * k.max_seq));
  CKS(alloc(c, reinterpret_cast<void**>(&c->step_log), sizeof(int2) * k.max_seq));
  CKS(alloc(c, reinterpret_cast<void**>(&c->xv), sizeof(float) * R * c->dp));
  CKS(alloc(c, reinterpret_cast<void**>(&c->xt), sizeof(float) * R * c->dp));
  CKS(alloc(c, reinterpret_cast<void**>(&c->qb), sizeof(float) * R * c->qp));
  CKS(alloc(c, reinterpret_cast<void**>(&c->ob), sizeof(float) * R * c->qp));
  CKS(alloc(c, reinterpret_cast<void**>(&c->hb), sizeof(float) * R * c->fp));
  CKS(alloc(c, reinterpret_cast<void**>(&c->hin), sizeof(float) * R * c->ip));
  // RMSNorm gains: zero-padded copies, so 256-column slices never read past a gain vector
  const int n_gains = 2 * n_blocks + 2 + (t5 ? 2 * k.n_enc_layers + k.n_layers + 1 : 0);
  CKS(alloc(c, reinterpret_cast<void**>(&c->gains), sizeof(__nv_bfloat16) * n_gains * c->dp));
  auto copy_gain = [&](int slot, const void* src) -> const __nv_bfloat16* {
    __nv_bfloat16* dst = c->gains + static_cast<size_t>(slot) * c->dp;
    if (src && cudaMemcpy(dst, src, sizeof(__nv_bfloat16) * k.d_model, cudaMemcpyDeviceToDevice) != cudaSuccess)
      return nullptr;
    return dst;
  };
  for (int l = 0; l < n_blocks; ++l) {
    c->attn_norm[l] = copy_gain(2 * l, wt(l, 7));
    c->ffn_norm[l] = copy_gain(2 * l + 1, wt(l, 8));
    if (!c->attn_norm[l] || !c->ffn_norm[l]) return fail(c, SSD_ERR_CUDA, "copying norm gains failed");
  }
  c->final_norm = copy_gain(2 * n_blocks, w->final_norm);
  c->in_norm = k.in_kind == SSD_IN_MLP2 ? copy_gain(2 * n_blocks + 1, w->in_norm) : nullptr;
  if (!c->final_norm || (k.in_kind == SSD_IN_MLP2 && !c->in_norm))
    return fail(c, SSD_ERR_CUDA, "copying norm gains failed");
  if (t5) {
    int slot = 2 * n_blocks + 2;
    for (int e = 0; e < k.n_enc_layers; ++e) {
      c->enc_attn_norm.push_back(copy_gain(slot++, ed->enc_attn_norm[e]));
      c->enc_ffn_norm.push_back(copy_gain(slot++, ed->enc_ffn_norm[e]));
      if (!c->enc_attn_norm.back() || !c->enc_ffn_norm.back()) return fail(c, SSD_ERR_CUDA, "copying norm gains failed");
    }
    for (int l = 0; l < k.n_layers; ++l) {
      c->cross_norm.push_back(copy_gain(slot++, ed->cross_norm[l]));
      if (!c->cross_norm.back()) return fail(c, SSD_ERR_CUDA, "copying norm gains failed");
    }
    c->enc_final = copy_gain(slot++, ed->enc_final);
    if (!c->enc_final) return fail(c, SSD_ERR_CUDA, "copying norm gains failed");
  }
  c->req_kv = static_cast<size_t>(k.n_heads) * k.max_seq * k.head_dim;
  c->layer_kv = c->req_kv * max_batch;
  CKS(alloc(c, reinterpret_cast<void**>(&c->kc), sizeof(float) * c->layer_kv * n_blocks));
  CKS(alloc(c, reinterpret_cast<void**>(&c->vc), sizeof(float) * c->layer_kv * n_blocks));
  CKS(alloc(c, reinterpret_cast<void**>(&c->rope), sizeof(float2) * k.max_seq * (k.head_dim / 2)));
  if (t5) {
    const size_t E = k.max_enc;
    c->cross_layer_kv = static_cast<size_t>(k.n_heads) * E * k.head_dim;
    CKS(alloc(c, reinterpret_cast<void**>(&c->x_enc), sizeof(float) * E * c->dp));
    CKS(alloc(c, reinterpret_cast<void**>(&c->enc_q), sizeof(float) * E * c->qp));
    CKS(alloc(c, reinterpret_cast<void**>(&c->enc_o), sizeof(float) * E * c->qp));
    CKS(alloc(c, reinterpret_cast<void**>(&c->enc_k), sizeof(float) * c->cross_layer_kv));
    CKS(alloc(c, reinterpret_cast<void**>(&c->enc_v), sizeof(float) * c->cross_layer_kv));
    CKS(alloc(c, reinterpret_cast<void**>(&c->ckc), sizeof(float) * c->cross_layer_kv * k.n_layers));
    CKS(alloc(c, reinterpret_cast<void**>(&c->cvc), sizeof(float) * c->cross_layer_kv * k.n_layers));
    CKS(alloc(c, reinterpret_cast<void**>(&c->dec_bias), sizeof(float) * k.n_heads * k.max_seq));
    CKS(alloc(c, reinterpret_cast<void**>(&c->enc_bias), sizeof(float) * k.n_heads * (2 * E - 1)));
    CKS(alloc(c, reinterpret_cast<void**>(&c->one), sizeof(float)));
    CKS(alloc(c, reinterpret_cast<void**>(&c->start_tok), sizeof(int)));
    const float one = 1.0f;
    CK(cudaMemcpy(c->one, &one, sizeof(float), cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->start_tok, &k.start_token, sizeof(int), cudaMemcpyHostToDevice));
  }
  CKS(alloc(c, reinterpret_cast<void**>(&c->partials), sizeof(float) * 2 * kGemvCtasPerSm * c->num_sms * R * kTileN));
  int max_rt = 1;
  for (const Site* s : {&c->layers[0].qkv, &c->layers[0].o, &c->layers[0].gateup, &c->layers[0].down, &c->head,
                        &c->in1, &c->in2})
    max_rt = s->n_rt > max_rt ? s->n_rt : max_rt;
  if (t5)
    for (const Site* s : {&c->cross_q[0], &c->cross_o[0], &c->cross_kv[0], &c->enc_layers[0].qkv, &c->enc_layers[0].o,
                          &c->enc_layers[0].gateup, &c->enc_layers[0].down})
      max_rt = s->n_rt > max_rt ? s->n_rt : max_rt;
  c->n_counters = max_rt;
  CKS(alloc(c, reinterpret_cast<void**>(&c->counters), sizeof(unsigned) * max_rt));

  CKS(alloc(c, reinterpret_cast<void**>(&c->attn_part),
            sizeof(float) * max_batch * k.n_heads * kAttnSplit * kAttnMaxRows * (k.head_dim + 2)));
  CKS(alloc(c, reinterpret_cast<void**>(&c->attn_tickets), sizeof(unsigned) * max_batch * k.n_heads));
  if (max_batch > 1) {
    const size_t S = k.max_seq;
    CKS(alloc(c, reinterpret_cast<void**>(&c->req), sizeof(DevState) * max_batch));
    CKS(alloc(c, reinterpret_cast<void**>(&c->bout), sizeof(int) * max_batch * S));
    CKS(alloc(c, reinterpret_cast<void**>(&c->blog), sizeof(int2) * max_batch * S));
    CKS(alloc(c, reinterpret_cast<void**>(&c->bvis), sizeof(__nv_bfloat16) * max_batch * S * d));
    CKS(alloc(c, reinterpret_cast<void**>(&c->bprompt), sizeof(int) * max_batch * S));
    if (R > kMaxRows) {  // verification rows beyond the GEMV: the medium-M kernel's buffers
      const size_t kmax = std::max(std::max(static_cast<size_t>(k.d_model), static_cast<size_t>(qdim)),
                                   static_cast<size_t>(k.d_ff));
      CKS(alloc(c, reinterpret_cast<void**>(&c->act_hi), sizeof(__nv_bfloat16) * kMaxMidRows * kmax));
      CKS(alloc(c, reinterpret_cast<void**>(&c->act_lo), sizeof(__nv_bfloat16) * kMaxMidRows * kmax));
      CKS(alloc(c, reinterpret_cast<void**>(&c->act_rs), sizeof(float) * kMaxMidRows));
      c->act_ld = static_cast<int>(kmax);
      c->act_ssq_ld = static_cast<int>((kmax + kTileN - 1) / kTileN);
      CKS(alloc(c, reinterpret_cast<void**>(&c->act_ssq), sizeof(float) * kMaxMidRows * c->act_ssq_ld));
      // partials: one slot per (streaming CTA, row tile) pair, c + rt
      CKS(alloc(c, reinterpret_cast<void**>(&c->mid_partials),
                sizeof(float) * (mid_max_ctas(c->num_sms) + c->n_counters) * kMaxMidRows * kTileN));
    }
  }
  CKS(alloc(c, reinterpret_cast<void**>(&c->dyn_table), sizeof(int) * (k.max_seq + 1)));
  CKS(alloc(c, reinterpret_cast<void**>(&c->dyn_launch), sizeof(int) * SSD_MAX_GAMMA));
  const size_t in_rows = std::max(static_cast<size_t>(k.max_seq), static_cast<size_t>(c->max_enc));
  CKS(alloc(c, reinterpret_cast<void**>(&c->in_vis), sizeof(__nv_bfloat16) * in_rows * d));
  {
    const size_t Pm = std::max(k.max_seq, c->max_enc);
    const size_t kmax = std::max(std::max(static_cast<size_t>(k.d_model), static_cast<size_t>(qdim)),
                                 static_cast<size_t>(k.d_ff));
    CKS(alloc(c, reinterpret_cast<void**>(&c->a_hi), sizeof(__nv_bfloat16) * Pm * kmax));
    CKS(alloc(c, reinterpret_cast<void**>(&c->a_lo), sizeof(__nv_bfloat16) * Pm * kmax));
    CKS(alloc(c, reinterpret_cast<void**>(&c->x_pre), sizeof(float) * Pm * c->dp));
    CKS(alloc(c, reinterpret_cast<void**>(&c->q_pre), sizeof(float) * Pm * c->qp));
    CKS(alloc(c, reinterpret_cast<void**>(&c->o_pre), sizeof(float) * Pm * c->qp));
    CKS(alloc(c, reinterpret_cast<void**>(&c->h_pre), sizeof(float) * Pm * c->fp));
    const int ks[3] = {k.d_model, qdim, k.d_ff};
    for (int i = 0; i < 3; ++i) {
      CKS(encode_map_sw128(c, &c->a_maps[i][0], c->a_hi, Pm, ks[i], kTcM));
      CKS(encode_map_sw128(c, &c->a_maps[i][1], c->a_lo, Pm, ks[i], kTcM));
    }
    if (!t5) {  // the prefill attention's operand parts (zeroed once: rows past a prompt stay finite)
      const int H = k.n_heads, Dh = k.head_dim;
      c->fa_spad = (k.max_seq + kFaK - 1) / kFaK * kFaK;
      c->fa_q_elems = Pm * static_cast<size_t>(qdim);
      c->fa_kv_elems = static_cast<size_t>(H) * c->fa_spad * Dh;
      const size_t n = 2 * c->fa_q_elems + 4 * c->fa_kv_elems;
      CKS(alloc(c, reinterpret_cast<void**>(&c->fa_parts), sizeof(__nv_bfloat16) * n));
      CK(cudaMemset(c->fa_parts, 0, sizeof(__nv_bfloat16) * n));
      __nv_bfloat16* base = c->fa_parts;
      const size_t qn = c->fa_q_elems, kn = c->fa_kv_elems;
      CKS(encode_map_sw128(c, &c->fa_maps[0], base, Pm, qdim, kFaQ));
      CKS(encode_map_sw128(c, &c->fa_maps[1], base + qn, Pm, qdim, kFaQ));
      CKS(encode_map_sw128(c, &c->fa_maps[2], base + 2 * qn, static_cast<uint64_t>(H) * c->fa_spad, Dh, kFaK));
      CKS(encode_map_sw128(c, &c->fa_maps[3], base + 2 * qn + kn, static_cast<uint64_t>(H) * c->fa_spad, Dh, kFaK));
      CKS(encode_map_sw128(c, &c->fa_maps[4], base + 2 * qn + 2 * kn, static_cast<uint64_t>(H) * Dh, c->fa_spad, Dh));
      CKS(encode_map_sw128(c, &c->fa_maps[5], base + 2 * qn + 3 * kn, static_cast<uint64_t>(H) * Dh, c->fa_spad, Dh));
    }
  }
  CKS(alloc(c, reinterpret_cast<void**>(&c->in_prompt), sizeof(int) * in_rows));
  CK(cudaStreamCreateWithFlags(&c->cs, cudaStreamNonBlocking));
  CK(cudaEventCreateWithFlags(&c->ev_in, cudaEventDisableTiming));
  CK(cudaEventCreateWithFlags(&c->ev_out, cudaEventDisableTiming));
  if (!t5) {  // the encoder-decoder model has no rotary embedding
    const int nrope = k.max_seq * (k.head_dim / 2);
    ssd_rope_table_kernel<<<(nrope + 255) / 256, 256, 0, c->cs>>>(c->rope, k.max_seq, k.head_dim,
                                                              static_cast<double>(k.rope_theta));
    CK(cudaGetLastError());
  }
  CK(cudaStreamSynchronize(c->cs));
  if (t5) {
    CKS(build_bias_table(c, ed->dec_rel, c->dec_bias, k.max_seq, k.max_seq - 1, false));
    CKS(build_bias_table(c, ed->enc_rel, c->enc_bias, 2 * k.max_enc - 1, k.max_enc - 1, true));
  }
  return SSD_OK;
}

ssd_status ssd_create(const ssd_config* cfg, const ssd_weights* w, void* cuda_stream, ssd_ctx** out) {
  if (!cfg || !out) return SSD_ERR_INVALID_ARG;
  *out = nullptr;
  ssd_ctx* c = new (std::nothrow) ssd_ctx();
  if (!c) return SSD_ERR_OOM;
  c->us = static_cast<cudaStream_t>(cuda_stream);
  ssd_status s = create_impl(c, cfg, w);
  if (s != SSD_OK) {
    fprintf(stderr, "ssd_create: %s\n", c->err.c_str());
    ssd_destroy(c);
    return s;
  }
  *out = c;
  return SSD_OK;
}

static ssd_status prefill_impl(ssd_ctx* c, int n_vis, int n_prompt) {
  const int P = n_vis + n_prompt;
  auto key = std::make_pair(n_vis, n_prompt);
  auto it = c->prefill_graphs.find(key);
  if (it == c->prefill_graphs.end()) {
    cudaGraphExec_t ge;
    int64_t nl = 0;
    CKS(build_plain_graph(c, enq_prefill_fn, n_vis, n_prompt, &ge, &nl));
    it = c->prefill_graphs.emplace(key, ge).first;
    c->prefill_launch_count[key] = nl;
  }
  CK(cudaGraphLaunch(it->second, c->cs));
  c->prefilled = true;
  c->batch = 0;  // slot 0 now holds this request: a batched decode needs a new batched prefill
  c->drafted_gamma = 0;
  c->prompt_len = c->t5 ? 1 : P;  // decoder positions before the first new token
  c->kv_upper = c->prompt_len;
  c->last_prefill_shape = key;
  return SSD_OK;
}

static ssd_status check_prefill_args(ssd_ctx* c, const void* vis, int n_vis, const int32_t* prompt, int n_prompt) {
  if (n_vis < 0 || n_prompt < 0 || n_vis + n_prompt < 1) return fail(c, SSD_ERR_INVALID_ARG, "empty prompt");
  if (n_vis > 0 && !vis) return fail(c, SSD_ERR_INVALID_ARG, "vis_emb is null");
  if (n_prompt > 0 && !prompt) return fail(c, SSD_ERR_INVALID_ARG, "prompt is null");
  if (c->t5) {
    if (n_vis + n_prompt > c->max_enc) return fail(c, SSD_ERR_CAPACITY, "encoder rows %d > max_enc %d",
                                                   n_vis + n_prompt, c->max_enc);
  } else if (n_vis + n_prompt + 1 > c->cfg.max_seq) {
    return fail(c, SSD_ERR_CAPACITY, "prompt longer than max_seq");
  }
  return SSD_OK;
}

ssd_status ssd_prefill(ssd_ctx* c, const void* vis, int n_vis, const int32_t* prompt, int n_prompt,
                       int32_t* first_tok) {
  if (!c) return SSD_ERR_INVALID_ARG;
  CKS(check_prefill_args(c, vis, n_vis, prompt, n_prompt));
  CKS(enter(c));
  if (n_vis > 0)
    CK(cudaMemcpyAsync(c->in_vis, vis, sizeof(__nv_bfloat16) * n_vis * c->cfg.d_model, cudaMemcpyDeviceToDevice,
                       c->cs));
  if (n_prompt > 0)
    CK(cudaMemcpyAsync(c->in_prompt, prompt, sizeof(int) * n_prompt, cudaMemcpyDeviceToDevice, c->cs));
  CKS(prefill_impl(c, n_vis, n_prompt));
  if (first_tok) ssd_first_token_kernel<<<1, 32, 0, c->cs>>>(c->st, first_tok);
  CK(cudaGetLastError());
  return leave(c);
}

ssd_status ssd_draft(ssd_ctx* c, int gamma, int32_t* draft_tok) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (!c->prefilled) return fail(c, SSD_ERR_STATE, "ssd_draft before ssd_prefill");
  if (gamma < 1 || gamma > c->cfg.gamma_max) return fail(c, SSD_ERR_INVALID_ARG, "gamma %d", gamma);
  if (c->kv_upper + gamma + 1 > c->cfg.max_seq) return fail(c, SSD_ERR_CAPACITY, "KV cache full");
  CKS(enter(c));
  auto it = c->draft_graphs.find(gamma);
  if (it == c->draft_graphs.end()) {
    cudaGraphExec_t ge;
    CKS(build_plain_graph(c, enq_draft_fn, gamma, 0, &ge, nullptr));
    it = c->draft_graphs.emplace(gamma, ge).first;
  }
  CK(cudaGraphLaunch(it->second, c->cs));
  if (draft_tok) ssd_copy_draft_kernel<<<1, 32, 0, c->cs>>>(c->st, gamma, draft_tok);
  CK(cudaGetLastError());
  c->drafted_gamma = gamma;
  return leave(c);
}

ssd_status ssd_verify(ssd_ctx* c, int gamma, int32_t* n_emitted, int32_t* emitted) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (!c->prefilled || c->drafted_gamma != gamma)
    return fail(c, SSD_ERR_STATE, "ssd_verify(gamma=%d) needs a preceding ssd_draft with the same gamma", gamma);
  CKS(enter(c));
  auto it = c->verify_graphs.find(gamma);
  if (it == c->verify_graphs.end()) {
    cudaGraphExec_t ge;
    CKS(build_plain_graph(c, enq_verify_fn, gamma, 0, &ge, nullptr));
    it = c->verify_graphs.emplace(gamma, ge).first;
  }
  CK(cudaGraphLaunch(it->second, c->cs));
  if (n_emitted || emitted) ssd_copy_emitted_kernel<<<1, 32, 0, c->cs>>>(c->st, n_emitted, emitted);
  CK(cudaGetLastError());
  c->drafted_gamma = 0;
  c->kv_upper += gamma + 1;
  return leave(c);
}

static ssd_status decode_impl(ssd_ctx* c, int max_new, int gamma, int32_t* out_tok, int32_t* n_out) {
  if (!c->prefilled) return fail(c, SSD_ERR_STATE, "decode before ssd_prefill");
  if (max_new < 1) return fail(c, SSD_ERR_INVALID_ARG, "max_new must be >= 1");
  if (gamma < 0 || gamma > c->cfg.gamma_max) return fail(c, SSD_ERR_INVALID_ARG, "gamma %d", gamma);
  if (static_cast<int64_t>(c->prompt_len) + max_new + gamma + 1 > c->cfg.max_seq)
    return fail(c, SSD_ERR_CAPACITY, "n_vis + n_prompt + max_new + gamma + 1 = %d > max_seq = %d",
                c->prompt_len + max_new + gamma + 1, c->cfg.max_seq);
  cudaGraphExec_t ge;
  if (c->host_loop) {
    auto it = c->step_graphs.find(gamma);
    if (it == c->step_graphs.end()) {
      int64_t nb = 0;
      CKS(build_plain_graph(c, enq_step_fn, gamma, 0, &ge, &nb));
      it = c->step_graphs.emplace(gamma, ge).first;
      if (gamma > 0) c->decode_body_launches[gamma] = nb; else c->greedy_body_launches = nb;
    }
    ssd_decode_setup_kernel<<<1, 32, 0, c->cs>>>(c->st, max_new, gamma);
    CK(cudaGetLastError());
    int done = 0;
    for (int it2 = 0; it2 < max_new && !done; ++it2) {
      CK(cudaGraphLaunch(it->second, c->cs));
      CK(cudaMemcpyAsync(&done, reinterpret_cast<char*>(c->st) + offsetof(DevState, done), sizeof(int),
                         cudaMemcpyDeviceToHost, c->cs));
      CK(cudaStreamSynchronize(c->cs));
    }
    if (out_tok || n_out) ssd_copy_out_kernel<<<1, 256, 0, c->cs>>>(c->st, c->out_int, out_tok, n_out, max_new);
    CK(cudaGetLastError());
    c->last_decode_kind = gamma > 0 ? 1 : 2;
    c->last_gamma = gamma;
    c->drafted_gamma = 0;
    c->kv_upper = c->prompt_len + max_new + gamma + 1;
    return SSD_OK;
  }
  if (gamma > 0) {
    auto it = c->decode_graphs.find(gamma);
    if (it == c->decode_graphs.end()) {
      int64_t nb = 0;
      CKS(build_loop_graph(c, gamma, &ge, &nb));
      it = c->decode_graphs.emplace(gamma, ge).first;
      c->decode_body_launches[gamma] = nb;
    }
    ge = it->second;
  } else {
    if (!c->greedy_graph) CKS(build_loop_graph(c, 0, &c->greedy_graph, &c->greedy_body_launches));
    ge = c->greedy_graph;
  }
  ssd_decode_setup_kernel<<<1, 32, 0, c->cs>>>(c->st, max_new, gamma);
  CK(cudaGetLastError());
  CK(cudaGraphLaunch(ge, c->cs));
  if (out_tok || n_out) ssd_copy_out_kernel<<<1, 256, 0, c->cs>>>(c->st, c->out_int, out_tok, n_out, max_new);
  CK(cudaGetLastError());
  c->last_decode_kind = gamma > 0 ? 1 : 2;
  c->last_gamma = gamma;
  c->drafted_gamma = 0;
  c->kv_upper = c->prompt_len + max_new + gamma + 1;
  return SSD_OK;
}

static ssd_status decode_dyn_impl(ssd_ctx* c, int max_new, int d0, int n_max, int t_from, int cap,
                                  int32_t* out_tok, int32_t* n_out) {
  if (!c->prefilled) return fail(c, SSD_ERR_STATE, "decode before ssd_prefill");
  if (max_new < 1) return fail(c, SSD_ERR_INVALID_ARG, "max_new must be >= 1");
  if (cap < 1 || cap > c->cfg.gamma_max) return fail(c, SSD_ERR_INVALID_ARG, "gamma cap %d", cap);
  if (d0 < 1 || n_max < 1) return fail(c, SSD_ERR_INVALID_ARG, "d0 %d, n_max %d", d0, n_max);
  if (t_from != SSD_DLEN_CONTEXT && t_from != SSD_DLEN_GENERATED)
    return fail(c, SSD_ERR_INVALID_ARG, "t_from %d", t_from);
  // t of the step whose last emitted token sits at position p: p + 2 over the whole context, or
  // p - P + 2 (= tokens emitted so far + 1) over the generated tokens
  const int origin = t_from == SSD_DLEN_CONTEXT ? 0 : c->prompt_len;
  if (static_cast<int64_t>(c->prompt_len) + max_new + cap + 1 > c->cfg.max_seq)
    return fail(c, SSD_ERR_CAPACITY, "n_vis + n_prompt + max_new + cap + 1 = %d > max_seq = %d",
                c->prompt_len + max_new + cap + 1, c->cfg.max_seq);
  if (d0 != c->dyn_d0 || n_max != c->dyn_n || origin != c->dyn_origin) {  // the old table may still be read
    CK(cudaStreamSynchronize(c->cs));
    c->dyn_table_h.resize(c->cfg.max_seq + 1);
    for (int p = 0; p <= c->cfg.max_seq; ++p) c->dyn_table_h[p] = draft_length_fp64(p - origin + 2, d0, n_max);
    CK(cudaMemcpy(c->dyn_table, c->dyn_table_h.data(), sizeof(int) * (c->cfg.max_seq + 1), cudaMemcpyHostToDevice));
    c->dyn_d0 = d0;
    c->dyn_n = n_max;
    c->dyn_origin = origin;
  }
  ssd_decode_setup_kernel<<<1, 32, 0, c->cs>>>(c->st, max_new, cap);
  CK(cudaGetLastError());
  if (c->host_loop) {  // one plain graph per step; the host reads kv_len and picks the step's gamma
    c->dyn_host_launches = 0;
    for (int it = 0; it < max_new; ++it) {
      DevState h;
      CK(cudaMemcpyAsync(&h, c->st, sizeof(int) * 8, cudaMemcpyDeviceToHost, c->cs));
      CK(cudaStreamSynchronize(c->cs));
      if (h.done) break;
      const int g = std::max(1, std::min(cap, c->dyn_table_h[h.kv_len]));
      auto sg = c->step_graphs.find(g);
      if (sg == c->step_graphs.end()) {
        cudaGraphExec_t ge;
        int64_t nb = 0;
        CKS(build_plain_graph(c, enq_step_fn, g, 0, &ge, &nb));
        sg = c->step_graphs.emplace(g, ge).first;
        c->decode_body_launches[g] = nb;
      }
      CK(cudaGraphLaunch(sg->second, c->cs));
      c->dyn_host_launches += c->decode_body_launches[g];
    }
  } else {
    auto it = c->dyn_graphs.find(cap);
    if (it == c->dyn_graphs.end()) {
      cudaGraphExec_t ge;
      CKS(build_dyn_graph(c, cap, &ge));
      it = c->dyn_graphs.emplace(cap, ge).first;
    }
    CK(cudaGraphLaunch(it->second, c->cs));
  }
  if (out_tok || n_out) ssd_copy_out_kernel<<<1, 256, 0, c->cs>>>(c->st, c->out_int, out_tok, n_out, max_new);
  CK(cudaGetLastError());
  c->last_decode_kind = 3;
  c->last_gamma = cap;
  c->drafted_gamma = 0;
  c->kv_upper = c->prompt_len + max_new + cap + 1;
  return SSD_OK;
}

int ssd_draft_length(int t, int d0, int n_max) { return draft_length_fp64(t, d0, n_max); }

int ssd_rel_bucket(int delta, int bidirectional, int n_buckets, int max_distance) {
  if (n_buckets < 4 || n_buckets % 2 || max_distance <= n_buckets / 2) return -1;
  return rel_bucket_host(delta, bidirectional != 0, n_buckets, max_distance);
}

ssd_status ssd_decode_dynamic(ssd_ctx* c, int max_new, int d0, int n_max, int t_from, int gamma_cap, int32_t* out_tok,
                              int32_t* n_out) {
  if (!c) return SSD_ERR_INVALID_ARG;
  CKS(enter(c));
  CKS(decode_dyn_impl(c, max_new, d0, n_max, t_from, gamma_cap, out_tok, n_out));
  return leave(c);
}

ssd_status ssd_decode(ssd_ctx* c, int max_new, int gamma, int32_t* out_tok, int32_t* n_out) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (gamma < 1) return fail(c, SSD_ERR_INVALID_ARG, "gamma must be >= 1");
  CKS(enter(c));
  CKS(decode_impl(c, max_new, gamma, out_tok, n_out));
  return leave(c);
}

ssd_status ssd_greedy_decode(ssd_ctx* c, int max_new, int32_t* out_tok, int32_t* n_out) {
  if (!c) return SSD_ERR_INVALID_ARG;
  CKS(enter(c));
  CKS(decode_impl(c, max_new, 0, out_tok, n_out));
  return leave(c);
}

ssd_status ssd_sync(ssd_ctx* c) {
  if (!c) return SSD_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(c->cs));
  CK(cudaStreamSynchronize(c->us));
  return read_device_error(c);
}

ssd_status ssd_get_stats(ssd_ctx* c, ssd_stats* out) {
  if (!c || !out) return SSD_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(c->cs));
  DevState h;
  CK(cudaMemcpy(&h, c->st, sizeof(DevState), cudaMemcpyDeviceToHost));
  memset(out, 0, sizeof(*out));
  out->steps = h.steps;
  out->drafted = h.drafted;
  out->accepted = h.accepted;
  out->emitted = h.n_out;
  for (int i = 0; i <= SSD_MAX_GAMMA; ++i) out->accept_hist[i] = h.hist[i];
  out->kv_len = h.kv_len;
  return SSD_OK;
}

static ssd_status generate_impl(ssd_ctx* c, const void* vis, int n_vis, const int32_t* prompt, int n_prompt,
                                int max_new, int gamma, int32_t* out, int* n_out, ssd_stats* stats) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (!out || !n_out) return fail(c, SSD_ERR_INVALID_ARG, "out / n_out is null");
  CKS(check_prefill_args(c, vis, n_vis, prompt, n_prompt));
  const int64_t dec_prompt = c->t5 ? 1 : static_cast<int64_t>(n_vis) + n_prompt;
  if (dec_prompt + max_new + gamma + 1 > c->cfg.max_seq)
    return fail(c, SSD_ERR_CAPACITY, "decoder prompt rows + max_new + gamma + 1 > max_seq");
  CKS(enter(c));
  if (n_vis > 0)
    CK(cudaMemcpyAsync(c->in_vis, vis, sizeof(__nv_bfloat16) * n_vis * c->cfg.d_model, cudaMemcpyHostToDevice,
                       c->cs));
  if (n_prompt > 0) CK(cudaMemcpyAsync(c->in_prompt, prompt, sizeof(int) * n_prompt, cudaMemcpyHostToDevice, c->cs));
  CKS(prefill_impl(c, n_vis, n_prompt));
  CKS(decode_impl(c, max_new, gamma, nullptr, nullptr));
  CK(cudaMemcpyAsync(out, c->out_int, sizeof(int) * max_new, cudaMemcpyDeviceToHost, c->cs));
  CK(cudaStreamSynchronize(c->cs));
  CKS(read_device_error(c));
  DevState h;
  CK(cudaMemcpy(&h, c->st, sizeof(DevState), cudaMemcpyDeviceToHost));
  *n_out = h.n_out < max_new ? h.n_out : max_new;
  if (stats) CKS(ssd_get_stats(c, stats));
  return leave(c);
}

ssd_status ssd_generate(ssd_ctx* c, const void* vis, int n_vis, const int32_t* prompt, int n_prompt, int max_new,
                        int gamma, int32_t* out, int* n_out, ssd_stats* stats) {
  if (c && gamma < 1) return fail(c, SSD_ERR_INVALID_ARG, "gamma must be >= 1");
  return generate_impl(c, vis, n_vis, prompt, n_prompt, max_new, gamma, out, n_out, stats);
}

ssd_status ssd_greedy_generate(ssd_ctx* c, const void* vis, int n_vis, const int32_t* prompt, int n_prompt,
                               int max_new, int32_t* out, int* n_out, ssd_stats* stats) {
  return generate_impl(c, vis, n_vis, prompt, n_prompt, max_new, 0, out, n_out, stats);
}

ssd_status ssd_set_logits_capture(ssd_ctx* c, float* buf, int max_rows) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (buf && max_rows < 1) return fail(c, SSD_ERR_INVALID_ARG, "max_rows");
  CK(cudaStreamSynchronize(c->cs));
  drop_graphs(c);
  c->logits_buf = buf;
  c->logits_rows = buf ? max_rows : 0;
  return SSD_OK;
}

ssd_status ssd_set_draft_logits_capture(ssd_ctx* c, float* buf, int max_steps) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (buf && max_steps < 1) return fail(c, SSD_ERR_INVALID_ARG, "max_steps %d", max_steps);
  CK(cudaStreamSynchronize(c->cs));
  drop_graphs(c);
  c->draft_logits_buf = buf;
  c->draft_logits_steps = buf ? max_steps : 0;
  return SSD_OK;
}

ssd_status ssd_get_step_log(ssd_ctx* c, int32_t* accepted, int32_t* drafted, int cap, int* n_steps) {
  if (!c || !n_steps || cap < 0 || (cap > 0 && !accepted && !drafted)) return SSD_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(c->cs));
  int steps = 0;
  CK(cudaMemcpy(&steps, reinterpret_cast<char*>(c->st) + offsetof(DevState, steps), sizeof(int),
                cudaMemcpyDeviceToHost));
  steps = std::min(steps, c->cfg.max_seq);
  const int n = std::min(steps, cap);
  if (n > 0) {
    std::vector<int2> h(n);
    CK(cudaMemcpy(h.data(), c->step_log, sizeof(int2) * n, cudaMemcpyDeviceToHost));
    for (int i = 0; i < n; ++i) {
      if (accepted) accepted[i] = h[i].x;
      if (drafted) drafted[i] = h[i].y;
    }
  }
  *n_steps = steps;
  return SSD_OK;
}

ssd_status ssd_get_kv(ssd_ctx* c, const void** k_cache, const void** v_cache, int* kv_len) {
  if (!c) return SSD_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(c->cs));
  if (k_cache) *k_cache = c->kc;
  if (v_cache) *v_cache = c->vc;
  if (kv_len) CK(cudaMemcpy(kv_len, c->st, sizeof(int), cudaMemcpyDeviceToHost));
  return SSD_OK;
}

ssd_status ssd_last_launch_count(ssd_ctx* c, int64_t* prefill_launches, int64_t* decode_launches) {
  if (!c) return SSD_ERR_INVALID_ARG;
  CK(cudaStreamSynchronize(c->cs));
  DevState h;
  CK(cudaMemcpy(&h, c->st, sizeof(DevState), cudaMemcpyDeviceToHost));
  if (prefill_launches) {
    auto it = c->prefill_launch_count.find(c->last_prefill_shape);
    *prefill_launches = it == c->prefill_launch_count.end() ? 0 : it->second;
  }
  if (decode_launches) {
    int64_t body = 0;
    if (c->last_decode_kind == 1) body = c->decode_body_launches[c->last_gamma];
    if (c->last_decode_kind == 2) body = c->greedy_body_launches;
    if (c->last_decode_kind == 4) body = c->batch_body_launches[c->last_gamma];
    // setup + loop_begin + steps x body + copy-out
    *decode_launches = c->last_decode_kind ? 2 + static_cast<int64_t>(h.steps) * body + 1 : 0;
    // dynamic draft length: setup + loop_begin + per step (select + branch + loop test) + copy-out,
    // or, host-driven, setup + the step graphs + copy-out
    if (c->last_decode_kind == 3)
      *decode_launches = c->host_loop ? 2 + c->dyn_host_launches : 3 + static_cast<int64_t>(h.dyn_launches);
  }
  return SSD_OK;
}

// ------------------------------------------------------------------ batched requests

static ssd_status check_batch_args(ssd_ctx* c, int B, const void* vis, const int32_t* n_vis, const int32_t* prompt,
                                   const int32_t* n_prompt) {
  if (c->max_batch < 2) return fail(c, SSD_ERR_INVALID_ARG, "batched calls need a ctx created with max_batch >= 2");
  if (B < 1 || B > c->max_batch) return fail(c, SSD_ERR_INVALID_ARG, "batch %d not in [1, %d]", B, c->max_batch);
  if (!n_vis || !n_prompt) return fail(c, SSD_ERR_INVALID_ARG, "n_vis / n_prompt is null");
  int64_t tv = 0, tp = 0;
  for (int b = 0; b < B; ++b) {
    if (n_vis[b] < 0 || n_prompt[b] < 0 || n_vis[b] + n_prompt[b] < 1)
      return fail(c, SSD_ERR_INVALID_ARG, "request %d has an empty prompt", b);
    if (n_vis[b] + n_prompt[b] + 1 > c->cfg.max_seq)
      return fail(c, SSD_ERR_CAPACITY, "request %d: prompt longer than max_seq", b);
    tv += n_vis[b];
    tp += n_prompt[b];
  }
  if (tv > 0 && !vis) return fail(c, SSD_ERR_INVALID_ARG, "vis_emb is null");
  if (tp > 0 && !prompt) return fail(c, SSD_ERR_INVALID_ARG, "prompt is null");
  return SSD_OK;
}

static ssd_status prefill_batch_impl(ssd_ctx* c, int B, const int32_t* n_vis, const int32_t* n_prompt) {
  size_t vo = 0, po = 0;
  c->batch = 0;  // the request errors are read only once the batch is complete
  for (int b = 0; b < B; ++b) {
    CKS(enqueue_prefill_slot(c, b, c->bvis + vo * c->cfg.d_model, c->bprompt + po, n_vis[b], n_prompt[b]));
    vo += n_vis[b];
    po += n_prompt[b];
  }
  // the batch's own launch state (error word, argmax keys, tickets) starts clean
  CK(launch_k(c, ssd_prefill_begin_kernel, dim3(1), dim3(32), 0, c->st, 0, c->cfg.eos_id, 0));
  c->batch = B;
  c->batch_prompt.assign(B, 0);
  for (int b = 0; b < B; ++b) c->batch_prompt[b] = n_vis[b] + n_prompt[b];
  c->prefilled = false;  // slot 0 now holds request 0 of the batch
  if (c->batch_graph_b != B) {
    for (auto& kv : c->batch_graphs) cudaGraphExecDestroy(kv.second);
    c->batch_graphs.clear();
    c->batch_graph_b = B;
  }
  return SSD_OK;
}

ssd_status ssd_prefill_batch(ssd_ctx* c, int B, const void* vis, const int32_t* n_vis, const int32_t* prompt,
                             const int32_t* n_prompt, int32_t* first_tok) {
  if (!c) return SSD_ERR_INVALID_ARG;
  CKS(check_batch_args(c, B, vis, n_vis, prompt, n_prompt));
  CKS(enter(c));
  int64_t tv = 0, tp = 0;
  for (int b = 0; b < B; ++b) {
    tv += n_vis[b];
    tp += n_prompt[b];
  }
  if (tv > 0)
    CK(cudaMemcpyAsync(c->bvis, vis, sizeof(__nv_bfloat16) * tv * c->cfg.d_model, cudaMemcpyDeviceToDevice, c->cs));
  if (tp > 0) CK(cudaMemcpyAsync(c->bprompt, prompt, sizeof(int) * tp, cudaMemcpyDeviceToDevice, c->cs));
  CKS(prefill_batch_impl(c, B, n_vis, n_prompt));
  if (first_tok) ssd_batch_first_tokens_kernel<<<1, 32 * ((B + 31) / 32), 0, c->cs>>>(c->req, B, first_tok);
  CK(cudaGetLastError());
  return leave(c);
}

static ssd_status enq_batch_step_fn(ssd_ctx* c, int g, int) {
  if (g == 0) return enqueue_greedy_batch(c, 0, 0);
  CKS(enqueue_draft_batch(c, g));
  return enqueue_verify_batch(c, g, 0, 0);
}

static ssd_status decode_batch_impl(ssd_ctx* c, int max_new, int gamma, int32_t* out_tok, int32_t* n_out) {
  const int B = c->batch;
  if (B < 1) return fail(c, SSD_ERR_STATE, "batched decode before ssd_prefill_batch");
  if (max_new < 1) return fail(c, SSD_ERR_INVALID_ARG, "max_new must be >= 1");
  if (gamma < 0 || gamma > c->cfg.gamma_max) return fail(c, SSD_ERR_INVALID_ARG, "gamma %d", gamma);
  for (int b = 0; b < B; ++b)
    if (static_cast<int64_t>(c->batch_prompt[b]) + max_new + gamma + 1 > c->cfg.max_seq)
      return fail(c, SSD_ERR_CAPACITY, "request %d: prompt + max_new + gamma + 1 = %d > max_seq = %d", b,
                  c->batch_prompt[b] + max_new + gamma + 1, c->cfg.max_seq);
  auto it = c->batch_graphs.find(gamma);
  if (it == c->batch_graphs.end()) {
    cudaGraphExec_t ge;
    int64_t nb = 0;
    if (c->host_loop) CKS(build_plain_graph(c, enq_batch_step_fn, gamma, 0, &ge, &nb));
    else CKS(build_loop_graph(c, gamma, &ge, &nb, true));
    it = c->batch_graphs.emplace(gamma, ge).first;
    c->batch_body_launches[gamma] = nb;
  }
  ssd_batch_setup_kernel<<<1, 32 * ((B + 31) / 32), 0, c->cs>>>(c->st, c->req, B, max_new, gamma);
  CK(cudaGetLastError());
  if (c->host_loop) {  // one plain graph per step; the host reads the batch's done flag
    for (int i = 0; i < max_new; ++i) {
      int done = 0;
      CK(cudaMemcpyAsync(&done, reinterpret_cast<char*>(c->st) + offsetof(DevState, done), sizeof(int),
                         cudaMemcpyDeviceToHost, c->cs));
      CK(cudaStreamSynchronize(c->cs));
      if (done) break;
      CK(cudaGraphLaunch(it->second, c->cs));
    }
  } else {
    CK(cudaGraphLaunch(it->second, c->cs));
  }
  if (out_tok || n_out)
    ssd_batch_copy_out_kernel<<<B, 256, 0, c->cs>>>(c->req, c->bout, c->cfg.max_seq, out_tok, n_out, max_new);
  CK(cudaGetLastError());
  c->last_decode_kind = 4;
  c->last_gamma = gamma;
  return SSD_OK;
}

ssd_status ssd_decode_batch(ssd_ctx* c, int max_new, int gamma, int32_t* out_tok, int32_t* n_out) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (gamma < 1) return fail(c, SSD_ERR_INVALID_ARG, "gamma must be >= 1");
  CKS(enter(c));
  CKS(decode_batch_impl(c, max_new, gamma, out_tok, n_out));
  return leave(c);
}

ssd_status ssd_greedy_decode_batch(ssd_ctx* c, int max_new, int32_t* out_tok, int32_t* n_out) {
  if (!c) return SSD_ERR_INVALID_ARG;
  CKS(enter(c));
  CKS(decode_batch_impl(c, max_new, 0, out_tok, n_out));
  return leave(c);
}

ssd_status ssd_generate_batch(ssd_ctx* c, int B, const void* vis, const int32_t* n_vis, const int32_t* prompt,
                              const int32_t* n_prompt, int max_new, int gamma, int32_t* out, int32_t* n_out) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (!out || !n_out) return fail(c, SSD_ERR_INVALID_ARG, "out / n_out is null");
  CKS(check_batch_args(c, B, vis, n_vis, prompt, n_prompt));
  if (max_new < 1) return fail(c, SSD_ERR_INVALID_ARG, "max_new must be >= 1");
  int64_t tv = 0, tp = 0;
  for (int b = 0; b < B; ++b) {
    tv += n_vis[b];
    tp += n_prompt[b];
    if (static_cast<int64_t>(n_vis[b]) + n_prompt[b] + max_new + gamma + 1 > c->cfg.max_seq)
      return fail(c, SSD_ERR_CAPACITY, "request %d: prompt + max_new + gamma + 1 > max_seq", b);
  }
  CKS(enter(c));
  if (tv > 0)
    CK(cudaMemcpyAsync(c->bvis, vis, sizeof(__nv_bfloat16) * tv * c->cfg.d_model, cudaMemcpyHostToDevice, c->cs));
  if (tp > 0) CK(cudaMemcpyAsync(c->bprompt, prompt, sizeof(int) * tp, cudaMemcpyHostToDevice, c->cs));
  CKS(prefill_batch_impl(c, B, n_vis, n_prompt));
  CKS(decode_batch_impl(c, max_new, gamma, nullptr, nullptr));
  CK(cudaMemcpy2DAsync(out, sizeof(int) * max_new, c->bout, sizeof(int) * c->cfg.max_seq, sizeof(int) * max_new, B,
                       cudaMemcpyDeviceToHost, c->cs));
  std::vector<DevState> h(B);
  CK(cudaMemcpyAsync(h.data(), c->req, sizeof(DevState) * B, cudaMemcpyDeviceToHost, c->cs));
  CK(cudaStreamSynchronize(c->cs));
  CKS(read_device_error(c));
  for (int b = 0; b < B; ++b) n_out[b] = h[b].n_out < max_new ? h[b].n_out : max_new;
  return leave(c);
}

ssd_status ssd_get_batch_stats(ssd_ctx* c, int b, ssd_stats* out) {
  if (!c || !out) return SSD_ERR_INVALID_ARG;
  if (b < 0 || b >= c->batch) return fail(c, SSD_ERR_INVALID_ARG, "request %d of a batch of %d", b, c->batch);
  CK(cudaStreamSynchronize(c->cs));
  DevState h;
  CK(cudaMemcpy(&h, c->req + b, sizeof(DevState), cudaMemcpyDeviceToHost));
  memset(out, 0, sizeof(*out));
  out->steps = h.steps;
  out->drafted = h.drafted;
  out->accepted = h.accepted;
  out->emitted = h.n_out;
  for (int i = 0; i <= SSD_MAX_GAMMA; ++i) out->accept_hist[i] = h.hist[i];
  out->kv_len = h.kv_len;
  return SSD_OK;
}

ssd_status ssd_get_batch_step_log(ssd_ctx* c, int b, int32_t* accepted, int32_t* drafted, int cap, int* n_steps) {
  if (!c || !n_steps || cap < 0 || (cap > 0 && !accepted && !drafted)) return SSD_ERR_INVALID_ARG;
  if (b < 0 || b >= c->batch) return fail(c, SSD_ERR_INVALID_ARG, "request %d of a batch of %d", b, c->batch);
  CK(cudaStreamSynchronize(c->cs));
  int steps = 0;
  CK(cudaMemcpy(&steps, reinterpret_cast<char*>(c->req + b) + offsetof(DevState, steps), sizeof(int),
                cudaMemcpyDeviceToHost));
  steps = std::min(steps, c->cfg.max_seq);
  const int n = std::min(steps, cap);
  if (n > 0) {
    std::vector<int2> h(n);
    CK(cudaMemcpy(h.data(), c->blog + static_cast<size_t>(b) * c->cfg.max_seq, sizeof(int2) * n,
                  cudaMemcpyDeviceToHost));
    for (int i = 0; i < n; ++i) {
      if (accepted) accepted[i] = h[i].x;
      if (drafted) drafted[i] = h[i].y;
    }
  }
  *n_steps = steps;
  return SSD_OK;
}

void ssd_set_fault_injection(int kind, int countdown) {
  g_fault_kind.store(0);
  g_fault_countdown.store(countdown > 0 ? countdown : 0);
  if (countdown > 0 && (kind == SSD_FAULT_ALLOC || kind == SSD_FAULT_LAUNCH)) g_fault_kind.store(kind);
}

ssd_status ssd_probe_bounded_wait(ssd_ctx* c, int64_t limit_ns) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (limit_ns < 0 || limit_ns > 2000000000ll) return fail(c, SSD_ERR_INVALID_ARG, "limit_ns %lld", (long long)limit_ns);
  CKS(enter(c));
  ssd_wait_probe_kernel<<<1, 32, 0, c->cs>>>(c->st, static_cast<unsigned long long>(limit_ns));
  CK(cudaGetLastError());
  c->prefilled = false;  // later kernels skip their work until the next prefill clears the error
  c->batch = 0;
  return leave(c);
}

ssd_status ssd_lm_head(ssd_ctx* c, const float* x, int rows, int32_t* tok, float* logits) {
  if (!c) return SSD_ERR_INVALID_ARG;
  if (!x || !tok || rows < 1 || rows > kMaxVerifyRows) return fail(c, SSD_ERR_INVALID_ARG, "x / tok / rows");
  CKS(enter(c));
  // rows go through the ctx's zero-padded staging buffer (256-column slices never leave a row)
  CK(cudaMemcpy2DAsync(c->xt, sizeof(float) * c->dp, x, sizeof(float) * c->cfg.d_model,
                       sizeof(float) * c->cfg.d_model, rows, cudaMemcpyDeviceToDevice, c->cs));
  // op state: kv_len = 0, prompt_len = 1 -> logits row m lands in row m of the capture buffer
  DevState zero{};
  zero.prompt_len = 1;
  CK(cudaMemcpyAsync(c->op_st, &zero, sizeof(DevState), cudaMemcpyHostToDevice, c->cs));
  GemvParams p{};
  p.x = c->xt;
  p.x_stride = c->dp;
  p.gain = c->final_norm;
  p.pos_off = 0;
  p.tok_dst = tok;
  p.logits = logits;
  p.logits_rows = logits ? rows : 0;
  p.K = c->head.K;
  p.n_kt = c->head.n_kt;
  p.n_rt = c->head.n_rt;
  p.units = c->head.units;
  p.N = c->head.N;
  p.seg_rows = c->head.seg_rows;
  p.partials = c->partials;
  p.counters = c->counters;
  p.st = c->op_st;
  p.eps = c->cfg.rms_eps;
  CK(count_launch(c));
  CK(gemv_launch_head(rows, c->head.maps, p, c->head.grid, c->cs, false));
  CKS(leave(c));
  // the host-side DevState must outlive the async copy
  CK(cudaStreamSynchronize(c->cs));
  return SSD_OK;
}

ssd_status ssd_profile_projection(ssd_ctx* c, int which, int layer, int rows, int reps, int64_t* bytes) {
  if (!c) return SSD_ERR_INVALID_ARG;
  // projections: up to kMaxRows rows through the GEMV, beyond that (a ctx with batched verification
  // rows) through the medium-M kernel; attention up to one request's verification rows
  const int max_rows = which == 7 ? kMaxVerifyRows : (c->act_hi ? std::min(kMaxMidRows, c->cfg.max_seq) : kMaxRows);
  if (rows < 1 || rows > max_rows || reps < 1) return fail(c, SSD_ERR_INVALID_ARG, "rows / reps");
  if (which < 0 || which > 7 || layer < 0 || layer >= c->cfg.n_layers)
    return fail(c, SSD_ERR_INVALID_ARG, "which / layer");
  if (which == 7) {  // split-KV attention of `layer` for rows kv_len .. kv_len+rows-1
    CK(cudaStreamSynchronize(c->cs));
    int kv = 0;
    CK(cudaMemcpy(&kv, reinterpret_cast<char*>(c->st) + offsetof(DevState, kv_len), sizeof(int),
                  cudaMemcpyDeviceToHost));
    if (kv < 0 || kv + rows > c->cfg.max_seq) return fail(c, SSD_ERR_INVALID_ARG, "kv_len %d + rows past max_seq", kv);
    const int64_t qd = static_cast<int64_t>(c->cfg.n_heads) * c->cfg.head_dim;
    if (bytes) *bytes = 2 * (kv + rows) * qd * 4 + 2 * static_cast<int64_t>(rows) * qd * 4;  // K, V; q in, o out
    CKS(enter(c));
    for (int r = 0; r < reps; ++r) CKS(attention(c, layer, rows, 0, false));
    c->prefilled = false;
    return leave(c);
  }
  if ((which == 5 || which == 6) && (c->cfg.in_kind != SSD_IN_MLP2 || rows > kMaxRows))
    return fail(c, SSD_ERR_INVALID_ARG, "imitation projections need SSD_IN_MLP2 and rows <= %d", kMaxRows);
  const int d = c->dp;
  const Site* site = nullptr;
  Epi e = Epi::RESID;
  GemvParams p{};
  p.x = c->xv;
  p.x_stride = d;
  switch (which) {
    case 0:
      site = &c->layers[layer].qkv;
      e = Epi::QKV;
      p.gain = c->attn_norm[layer];
      p.q_out = c->qb;
      p.q_stride = c->qp;
      p.k_cache = kv_k(c, layer);
      p.v_cache = kv_v(c, layer);
      p.head_dim = c->cfg.head_dim;
      p.max_seq = c->cfg.max_seq;
      p.rope_cs = c->t5 ? nullptr : c->rope;
      break;
    case 1:
    case 3:
      site = which == 1 ? &c->layers[layer].o : &c->layers[layer].down;
      p.x = which == 1 ? c->ob : c->hb;
      p.x_stride = which == 1 ? c->qp : c->fp;
      p.base = c->xt;
      p.base_stride = d;
      p.dst = c->xt;
      p.dst_stride = d;
      p.scale = c->resid_scale + layer;
      break;
    case 2:
      site = &c->layers[layer].gateup;
      e = Epi::GATE_SILU;
      p.gain = c->ffn_norm[layer];
      p.h_out = c->hb;
      p.h_stride = c->fp;
      break;
    case 4:
      site = &c->head;
      e = Epi::ARGMAX;
      p.gain = c->final_norm;
      p.tok_dst = rows <= kMaxRows ? st_field(c, offsetof(DevState, full_tok)) : c->out_int;
      break;
    case 5:
      site = &c->in1;
      e = Epi::SILU;
      p.gain = c->in_norm;
      p.h_out = c->hin;
      p.h_stride = c->ip;
      break;
    default:
      site = &c->in2;
      p.x = c->hin;
      p.x_stride = c->ip;
      p.base = c->xt;
      p.base_stride = d;
      p.dst = c->xt;
      p.dst_stride = d;
      p.scale = c->in_scale;
      break;
  }
  const int64_t N = site->N * (e == Epi::GATE_SILU ? 2 : 1);
  const int64_t out_elems = e == Epi::GATE_SILU ? site->N : (e == Epi::ARGMAX ? 1 : site->N);
  const int64_t out_bytes = e == Epi::QKV ? rows * (c->qdim * 4 + 2 * c->qdim * 2) : rows * out_elems * 4;
  if (bytes)
    *bytes = N * site->K * 2 + static_cast<int64_t>(rows) * site->K * 4 + (p.gain ? site->K * 2 : 0) + out_bytes +
             (e == Epi::RESID ? static_cast<int64_t>(rows) * site->N * 4 : 0);
  CKS(enter(c));
  c->act_ready = false;
  for (int r = 0; r < reps; ++r) CKS(proj_rows(c, e, rows, *site, p));
  c->prefilled = false;
  c->batch = 0;
  return leave(c);
}

}  // extern "C"
