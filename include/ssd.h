/*
 * ssd.h -- C ABI of the GB300 (sm_103a) self-speculative decoding library.
 *
 * Method: FastVLM, "Self-Speculative Decoding for Fast Vision-Language Model
 * Inference" (arXiv 2510.22641).  Problem statement (Sec. "SSD Setup for
 * VLMs"): the encoder output z = E(I, T0) and the prompt enter the decoder,
 * which emits greedy tokens y^{t+1} .. y^T.  The decoder has L layers
 * x_{l+1} = x_l + f_l(x_l) and an LM head o = g(x_L); greedy decoding takes
 * argmax softmax(o).  Self-speculative decoding (Sec. 3.1 and Algorithm 1):
 * the first n layers (here k) plus the imitation network I form the draft
 * model, which proposes d (here gamma) tokens autoregressively with
 * argmax g(I(x_k)); the full decoder then verifies them in one
 * non-autoregressive pass, keeps the longest matching prefix and appends its
 * own token at the first mismatch.  Draft and full model share one KV cache
 * (Sec. "Methodology", KV cache).
 *
 * Conventions for every entry point:
 *  - Pointers documented "device" must be CUDA device pointers on the device
 *    that was current at ssd_create; "host" pointers are ordinary CPU memory.
 *  - Weights are BORROWED: the caller owns them and must keep them alive and
 *    unchanged (except resid_scale / in_scale, see below) until ssd_destroy.
 *    The RMSNorm gain vectors are the exception: ssd_create copies them
 *    (zero-padded) into library memory.
 *    Everything else (KV cache, workspaces, CUDA graphs) is owned by the ctx.
 *  - A ctx is bound to one CUDA stream and is not thread-safe.  Calls marked
 *    "async" only enqueue work on that stream; "sync" calls wait for it.
 *  - No C++ exception crosses this boundary.  Every call returns an
 *    ssd_status; on failure ssd_last_error(ctx) holds a message.  A device-side
 *    fault detected by the kernels (bad token id, a bounded wait that ran out)
 *    sets an error word that the next sync call reports as SSD_ERR_DEVICE or
 *    SSD_ERR_TIMEOUT.
 *  - Sizes: d_model, d_ff and in_hidden must be multiples of 64 and
 *    n_heads*head_dim a multiple of 128; head_dim must be 64 or 128;
 *    1 <= gamma <= gamma_max <= SSD_MAX_GAMMA.
 */
#ifndef SSD_H_
#define SSD_H_

#include <stdint.h>

#if defined(__GNUC__)
#define SSD_API __attribute__((visibility("default")))
#else
#define SSD_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SSD_OK = 0,
  SSD_ERR_INVALID_ARG = 1,  /* null pointer, bad size, unsupported shape */
  SSD_ERR_OOM = 2,          /* a device allocation failed */
  SSD_ERR_CUDA = 3,         /* a CUDA runtime call failed */
  SSD_ERR_CAPACITY = 4,     /* n_vis + n_prompt + max_new + gamma + 1 > max_seq (T5: encoder rows > max_enc) */
  SSD_ERR_STATE = 5,        /* call out of order (e.g. verify without a draft) */
  SSD_ERR_TIMEOUT = 6,      /* a bounded device wait ran out */
  SSD_ERR_DEVICE = 7,       /* the kernels flagged bad input (e.g. token id >= vocab) */
  SSD_ERR_UNSUPPORTED = 8   /* no sm_103a device / feature missing */
} ssd_status;

/* Imitation network variants (Sec. "Methodology", Deep Representation Imitation). */
enum {
  SSD_IN_IDENTITY = 0,  /* draft without imitation: g(x_k) ("Draft w/o Im", Table 1) */
  SSD_IN_MLP2 = 1,      /* x + s_in * W2 SiLU(W1 RMSNorm_in(x)): two FC layers + one norm */
  SSD_IN_BLOCK = 2      /* one decoder block of the model's shape with its own KV cache, residual
                         * writes scaled by s_in (the module read as a block; Sec. "Choice of n") */
};

/* Model families. */
enum {
  SSD_ARCH_LLAMA = 0,  /* decoder-only pre-norm LLaMA stack (LLaVA-1.5): RMSNorm, rotary attention, SwiGLU */
  SSD_ARCH_T5 = 1      /* encoder-decoder T5 v1.1 stack (BLIP-2 FlanT5-xl, Sec. "Experiments"): the encoder reads
                        * [vis_emb; embed(prompt)] once; the decoder, which drafts and verifies, starts
                        * from start_token at position 0 and has, per layer, self-attention with a
                        * learned relative-position bias and no 1/sqrt(head_dim) factor, cross-attention
                        * to the encoder's normed output, and a gated-GELU (tanh form) MLP; no RoPE */
};

/* ssd_config.options: alternative execution paths with identical results (diagnostics and
 * cross-checks; 0 selects the default path).  Unknown bits are SSD_ERR_INVALID_ARG. */
#define SSD_OPT_HOST_LOOP 1     /* decode loops driven from the host, one plain CUDA graph per step
                                 * (kernel profilers do not see kernels inside conditional graph nodes) */
#define SSD_OPT_PREFILL_ROWS 2  /* prefill through the decode kernels in 8-row chunks instead of the
                                 * tensor-core GEMMs */

#define SSD_MAX_GAMMA 15  /* the paper's d0 + 10 for d0 = 5 (Sec. "Choice of d") */
#define SSD_MAX_ROWS 16   /* rows one decode pass may carry (gamma + 1, prefill chunk) */

typedef struct ssd_ctx ssd_ctx;

/* Model shape and decoding limits.  The decoder is a pre-norm LLaMA block stack
 * (RMSNorm, rotary multi-head attention, SwiGLU MLP), or with arch = SSD_ARCH_T5
 * the decoder of a T5 v1.1 encoder-decoder.  The fields n_enc_layers ..
 * start_token are read only for SSD_ARCH_T5 (zero them otherwise). */
typedef struct {
  int n_layers;      /* L */
  int d_model;       /* hidden width */
  int n_heads;
  int head_dim;      /* 64 or 128 */
  int d_ff;          /* SwiGLU width */
  int vocab;         /* |V| */
  int draft_exit_k;  /* k (the paper's n): draft = layers 0..k-1, 1 <= k <= L */
  int in_kind;       /* SSD_IN_* */
  int in_hidden;     /* width of the imitation network's first FC layer */
  int gamma_max;     /* largest gamma (the paper's d) any call will use */
  int max_seq;       /* KV cache capacity in positions */
  float rms_eps;     /* RMSNorm epsilon */
  float rope_theta;  /* rotary base, rotate-half pairing (i, i + head_dim/2) */
  int eos_id;        /* end-of-sequence token, -1 = disabled */
  int arch;          /* SSD_ARCH_* (0 = LLaMA) */
  int n_enc_layers;  /* T5: encoder depth */
  int max_enc;       /* T5: encoder rows capacity, >= n_vis + n_prompt of every prefill */
  int rel_buckets;   /* T5: relative-position buckets (even, >= 4) */
  int rel_max_distance; /* T5: offsets at or beyond this share the last bucket */
  int start_token;   /* T5: the decoder's first input id */
  int options;       /* SSD_OPT_* bits, 0 = the default path */
  int max_batch;     /* requests one batched decode may carry (0 or 1: single requests only; at most
                      * SSD_MAX_ROWS, with max_batch * (gamma_max + 1) <= 128; SSD_ARCH_LLAMA with
                      * SSD_IN_IDENTITY or SSD_IN_MLP2).  The KV cache holds max_batch request slots. */
} ssd_config;

/* Extra weights of SSD_ARCH_T5, device bf16, [out][in], borrowed.  The
 * ssd_weights layer arrays hold the DECODER: wq/wk/wv/wo its self-attention,
 * w_gate/w_up/w_down the gated-GELU MLP (wi_0, wi_1, wo), attn_norm the
 * self-attention norm, ffn_norm the MLP norm, final_norm the decoder's final
 * norm; resid_scale[l] scales all three residual writes of decoder layer l. */
typedef struct {
  /* host arrays of n_layers device pointers: cross-attention of decoder layer l */
  const void* const* cq;          /* [n_heads*head_dim][d_model], applied to RMSNorm_cross(x) */
  const void* const* ck;          /* [n_heads*head_dim][d_model], applied to the encoder output */
  const void* const* cv;          /* [n_heads*head_dim][d_model] */
  const void* const* co;          /* [d_model][n_heads*head_dim] */
  const void* const* cross_norm;  /* [d_model] */
  /* host arrays of n_enc_layers device pointers: the encoder (bidirectional attention) */
  const void* const* enc_wq;
  const void* const* enc_wk;
  const void* const* enc_wv;
  const void* const* enc_wo;
  const void* const* enc_wi0;     /* [d_ff][d_model] gate */
  const void* const* enc_wi1;     /* [d_ff][d_model] up */
  const void* const* enc_wff;     /* [d_model][d_ff] */
  const void* const* enc_attn_norm;
  const void* const* enc_ffn_norm;
  const void* enc_final;          /* [d_model] the encoder's final norm */
  const void* enc_rel;            /* [rel_buckets][n_heads] encoder bias (bidirectional buckets) */
  const void* dec_rel;            /* [rel_buckets][n_heads] decoder self-attention bias (past-only buckets) */
} ssd_encdec_weights;

/* Model weights, all device pointers, bf16, nn.Linear layout [out][in], borrowed. */
typedef struct {
  const void* embed;       /* [vocab][d_model] */
  const void* lm_head;     /* [vocab][d_model], shared by draft and full model */
  const void* final_norm;  /* [d_model], RMSNorm gain inside g(.) */
  /* host arrays of n_layers device pointers each */
  const void* const* wq;        /* [n_heads*head_dim][d_model] */
  const void* const* wk;        /* [n_heads*head_dim][d_model] */
  const void* const* wv;        /* [n_heads*head_dim][d_model] */
  const void* const* wo;        /* [d_model][n_heads*head_dim] */
  const void* const* w_gate;    /* [d_ff][d_model] */
  const void* const* w_up;      /* [d_ff][d_model] */
  const void* const* w_down;    /* [d_model][d_ff] */
  const void* const* attn_norm; /* [d_model] */
  const void* const* ffn_norm;  /* [d_model] */
  /* imitation network (ignored for SSD_IN_IDENTITY) */
  const void* in_norm;     /* [d_model] */
  const void* in_w1;       /* [in_hidden][d_model] */
  const void* in_w2;       /* [d_model][in_hidden] */
  /* fp32 device scalars read at every launch, so they may be changed between
   * decode calls: s_l scales both residual writes of layer l, s_in the IN's. */
  const float* resid_scale; /* [n_layers] */
  const float* in_scale;    /* [1] */
  /* SSD_IN_BLOCK: host array of 9 device pointers, the block's wq, wk, wv, wo,
   * w_gate, w_up, w_down, attn_norm, ffn_norm (layouts as above); NULL otherwise.
   * Its cache rows hold the block's K/V of every position's x_k: the prefill
   * fills the prompt rows, each drafting step its row, the verification pass
   * row gamma. */
  const void* const* in_block;
  /* SSD_ARCH_T5: the encoder and cross-attention weights; NULL otherwise. */
  const ssd_encdec_weights* encdec;
} ssd_weights;

/* Counters of the last prefill+decode, read back by ssd_get_stats. */
typedef struct {
  int64_t steps;          /* verify passes (SSD) or tokens (greedy) after the prefill */
  int64_t drafted;        /* sum of gamma_eff over steps */
  int64_t accepted;       /* sum of accepted drafts a over steps */
  int64_t emitted;        /* tokens emitted, including the prefill's */
  int64_t accept_hist[SSD_MAX_GAMMA + 1]; /* steps with a = 0 .. SSD_MAX_GAMMA */
  int64_t kv_len;         /* valid cache length at the end */
} ssd_stats;

/* Create a context: checks the shape, builds TMA descriptors for the borrowed
 * weights, allocates the KV cache [L][max_batch][H][max_seq][head_dim] fp32 (K and V),
 * activations and workspaces on the current device.  cuda_stream is a
 * cudaStream_t (NULL = legacy default stream).  sync. */
SSD_API ssd_status ssd_create(const ssd_config* cfg, const ssd_weights* w, void* cuda_stream, ssd_ctx** out);

/* Free everything the ctx owns (not the weights).  sync.  NULL is accepted. */
SSD_API ssd_status ssd_destroy(ssd_ctx* ctx);

/* Prefill (Sec. "SSD Setup for VLMs": z is the decoder's input).  Rows
 * [vis_emb (n_vis rows); embed(prompt)] at positions 0..P-1, P = n_vis + n_prompt,
 * run through all L layers; K/V of every layer for positions 0..P-1 are
 * written; the greedy token of the last row is written to first_tok.
 * SSD_ARCH_T5: the P rows are the ENCODER's input (P <= max_enc); the encoder
 * runs, every decoder layer's cross-attention K/V of its output are written,
 * and the decoder runs once on start_token at position 0, whose greedy token
 * is the first new token (kv_len = 1 afterwards; decoder positions count from
 * 0, so the capacity rule below reads 1 + max_new + gamma + 1 <= max_seq).
 *   vis_emb:   device bf16 [n_vis][d_model] (may be NULL when n_vis == 0)
 *   prompt:    device int32 [n_prompt], each in [0, vocab)
 *   first_tok: device int32 [1] (may be NULL)
 * Resets the decode state: kv_len = P, one token emitted.  async. */
SSD_API ssd_status ssd_prefill(ssd_ctx* ctx, const void* vis_emb, int n_vis, const int32_t* prompt,
                       int n_prompt, int32_t* first_tok);

/* Drafting stage (Sec. 3.1; Algorithm 1, draft loop): gamma tokens
 * d_j = argmax g(I(x_k)) from the current token, each from layers 0..k-1 and
 * the imitation network, writing the shallow layers' K/V at positions
 * kv_len .. kv_len+gamma-1.  draft_tok: device int32 [gamma] (may be NULL).
 * Needs a prefill first.  async. */
SSD_API ssd_status ssd_draft(ssd_ctx* ctx, int gamma, int32_t* draft_tok);

/* Verification stage and acceptance (Algorithm 1, verify loop): the full
 * model runs once over the gamma+1 rows [y, d_1..d_gamma] at positions
 * kv_len..kv_len+gamma (shallow rows reused from the draft), f_i = argmax
 * g(x_L) per row; a = longest prefix with d_{i+1} == f_i; emits d_1..d_a and
 * f_a; kv_len += a + 1 (rollback by length).  gamma must equal the preceding
 * ssd_draft's.  n_emitted: device int32 [1], emitted: device int32
 * [gamma + 1] (each may be NULL).  async. */
SSD_API ssd_status ssd_verify(ssd_ctx* ctx, int gamma, int32_t* n_emitted, int32_t* emitted);

/* Whole SSD decode after ssd_prefill, as one CUDA-graph launch whose loop runs
 * on the device (a conditional WHILE node): steps of draft + verify + accept
 * until max_new tokens (counting the prefill's) are out or eos is emitted.
 * In the last steps gamma_eff = min(gamma, remaining - 1).
 *   out_tok: device int32 [max_new] (all tokens incl. the prefill's)
 *   n_out:   device int32 [1]
 * async. */
SSD_API ssd_status ssd_decode(ssd_ctx* ctx, int max_new, int gamma, int32_t* out_tok, int32_t* n_out);

/* SSD decode with the dynamic draft length of Sec. "Choice of d":
 *   d(t) = d0 + floor(10 / (1 + exp(-0.01 (t - n_max / 2))))   (fp64, host)
 * with t counted one of two ways (the paper does not say which):
 *   t_from = SSD_DLEN_CONTEXT:   over the whole context -- the t-th token is generated
 *     from t - 1 tokens, so a step whose last emitted token sits at position kv_len
 *     uses t = kv_len + 2 (n_max: the longest sequence, e.g. max_seq);
 *   t_from = SSD_DLEN_GENERATED: over the generated tokens -- t = tokens emitted so far
 *     + 1, the index of the next new token (n_max: the generation length, max_new).
 * Each step drafts min(d(t), gamma_cap) tokens (gamma_cap <= gamma_max; the paper's
 * range is d0 .. d0 + 10) and, in the last steps, accepts at most remaining - 1.
 * One CUDA-graph launch: a WHILE node whose body selects the step's branch of a
 * SWITCH node (one draft + verify + accept branch per gamma) from a device
 * table of d indexed by kv_len.  Same buffers, capacity rule (with gamma_cap) and
 * errors as ssd_decode.  async. */
enum { SSD_DLEN_CONTEXT = 0, SSD_DLEN_GENERATED = 1 };
SSD_API ssd_status ssd_decode_dynamic(ssd_ctx* ctx, int max_new, int d0, int n_max, int t_from, int gamma_cap,
                                      int32_t* out_tok, int32_t* n_out);

/* d(t) of Sec. "Choice of d", the value ssd_decode_dynamic tabulates (host
 * function; no context, no GPU). */
SSD_API int ssd_draft_length(int t, int d0, int n_max);

/* Relative-position bucket of the key-minus-query offset `delta` that the
 * SSD_ARCH_T5 model's bias tables use (host function; no context, no GPU):
 * bidirectional != 0 splits the n_buckets between earlier (and equal) and later
 * keys (the encoder), otherwise all go to earlier keys and later keys share
 * bucket 0 (the decoder's self-attention).  Within a half, offsets below n/2
 * get one bucket each and larger ones logarithmically spaced buckets up to
 * max_distance, past which they share the last.  The logarithmic index is
 * floored in fp64 after adding 1e-9.  Returns -1 for n_buckets < 4, odd
 * n_buckets or max_distance <= n_buckets / 2. */
SSD_API int ssd_rel_bucket(int delta, int bidirectional, int n_buckets, int max_distance);

/* Baseline: plain greedy decoding with the full model (same kernels, one
 * token per step, device-side loop).  Same buffers as ssd_decode.  async. */
SSD_API ssd_status ssd_greedy_decode(ssd_ctx* ctx, int max_new, int32_t* out_tok, int32_t* n_out);

/* End-to-end call with HOST buffers: copies vis_emb (bf16 [n_vis][d_model])
 * and prompt (int32 [n_prompt]) to the device, prefill, SSD decode, copies the
 * tokens back.  out: host int32 [max_new]; n_out: host; stats may be NULL.
 * sync. */
SSD_API ssd_status ssd_generate(ssd_ctx* ctx, const void* vis_emb, int n_vis, const int32_t* prompt,
                        int n_prompt, int max_new, int gamma, int32_t* out, int* n_out,
                        ssd_stats* stats);

/* Same as ssd_generate with greedy decoding of the full model. sync. */
SSD_API ssd_status ssd_greedy_generate(ssd_ctx* ctx, const void* vis_emb, int n_vis, const int32_t* prompt,
                               int n_prompt, int max_new, int32_t* out, int* n_out,
                               ssd_stats* stats);

/* Wait for the ctx stream and report device-side errors.  sync. */
SSD_API ssd_status ssd_sync(ssd_ctx* ctx);

/* Counters of the last decode (see ssd_stats).  sync. */
SSD_API ssd_status ssd_get_stats(ssd_ctx* ctx, ssd_stats* stats);

/* Debug capture of the full model's logits: when buf (device fp32
 * [max_rows][vocab]) is non-NULL, every full-model LM-head row writes its
 * logits to row (position + 1 - P) -- the index of the token it predicts --
 * if that index is < max_rows.  Rows of rejected drafts are overwritten by
 * later steps.  NULL disables.  Takes effect for graphs built afterwards
 * (the ctx rebuilds them).  sync. */
SSD_API ssd_status ssd_set_logits_capture(ssd_ctx* ctx, float* buf, int max_rows);

/* Debug capture of the drafting stage's logits g(I(x_k)) (Algorithm 1, draft loop): when buf
 * (device fp32 [max_steps][gamma_max][vocab]) is non-NULL, the LM-head row of draft j in step s
 * (steps counted from the last prefill; every step drafts gamma rows, of which the first
 * gamma_eff are used) writes its logits to buf[s][j] while s < max_steps.  NULL disables.  Takes
 * effect for graphs built afterwards (the ctx rebuilds them).  sync. */
SSD_API ssd_status ssd_set_draft_logits_capture(ssd_ctx* ctx, float* buf, int max_steps);

/* Per-step record of the last decode (Algorithm 1, acceptance): for each step s since the last
 * prefill, accepted[s] = a (drafts kept) and drafted[s] = gamma_eff (drafts that could be kept);
 * greedy steps record (0, 0).  Fills min(steps, cap) entries of the host arrays (either may be
 * NULL) and sets *n_steps to the number of steps.  sync. */
SSD_API ssd_status ssd_get_step_log(ssd_ctx* ctx, int32_t* accepted, int32_t* drafted, int cap, int* n_steps);

/* Device pointers to the KV cache, layout [L][max_batch][n_heads][max_seq][head_dim]
 * fp32 (with SSD_IN_BLOCK, [L + 1]: slot L is the imitation block's; the
 * single-request calls use request slot 0), and the single request's current
 * valid length (sync read).  Positions >= kv_len hold stale rows of rejected
 * drafts. */
SSD_API ssd_status ssd_get_kv(ssd_ctx* ctx, const void** k_cache, const void** v_cache, int* kv_len);

/* Number of kernel launches the last ssd_decode / ssd_greedy_decode /
 * ssd_prefill performed (from the device step counter).  sync. */
SSD_API ssd_status ssd_last_launch_count(ssd_ctx* ctx, int64_t* prefill_launches, int64_t* decode_launches);

/* ---- Batched requests: the serving form of Algorithm 1 ----
 * B <= max_batch independent requests, each with its own visual rows, prompt
 * length, positions, cache slot and accept lengths, decode in lockstep: each
 * step drafts gamma tokens for every request (layers 0..k-1 and the imitation
 * network over B rows per token), verifies all B * (gamma + 1) rows in one
 * full-depth pass (the medium-M tensor-core kernel beyond 16 rows), and
 * accepts / rolls back each request on its own.  A request that is done (max_new
 * tokens or eos) keeps its tokens; its rows ride along unused until every request
 * is done.  Every request's rows are computed independently of the other
 * requests', so its tokens and accept lengths are those of the same request
 * decoded alone; beyond 16 verification rows the medium-M kernel's own split
 * points round differently from the GEMV's, so there they agree up to logits
 * that tie within rounding.  The single-request calls (ssd_prefill .. ssd_verify)
 * and the batched calls share the cache: a prefill of one kind invalidates the
 * other kind's decode state. */

/* Prefill of B requests (each as ssd_prefill: rows [vis_b; embed(prompt_b)] at
 * positions 0..P_b-1 into request b's cache slot, first token from the last row).
 *   vis_emb:   device bf16 [sum_b n_vis[b]][d_model], request b's rows after those of 0..b-1
 *   n_vis, n_prompt: host int32 [B]
 *   prompt:    device int32 [sum_b n_prompt[b]], concatenated the same way
 *   first_tok: device int32 [B] (may be NULL)
 * 1 <= B <= max_batch; n_vis[b] + n_prompt[b] + 1 <= max_seq.  async. */
SSD_API ssd_status ssd_prefill_batch(ssd_ctx* ctx, int batch, const void* vis_emb, const int32_t* n_vis,
                                     const int32_t* prompt, const int32_t* n_prompt, int32_t* first_tok);

/* SSD decode of the prefilled batch, one CUDA-graph launch (a WHILE node over
 * draft + verify + accept of every request until all are done).  Request b
 * stops after max_new tokens (the prefill's included) or an eos; in its last
 * steps it accepts at most max_new - n_out - 1 drafts.  Capacity: for every
 * request P_b + max_new + gamma + 1 <= max_seq.
 *   out_tok: device int32 [B][max_new];  n_out: device int32 [B]
 * async. */
SSD_API ssd_status ssd_decode_batch(ssd_ctx* ctx, int max_new, int gamma, int32_t* out_tok, int32_t* n_out);

/* Baseline: greedy decoding of every request of the prefilled batch with the
 * full model (all L layers over B rows per token).  Same buffers.  async. */
SSD_API ssd_status ssd_greedy_decode_batch(ssd_ctx* ctx, int max_new, int32_t* out_tok, int32_t* n_out);

/* End-to-end batched call with HOST buffers: copies the inputs (laid out as for
 * ssd_prefill_batch) to the device, prefill, SSD decode (gamma >= 1) or greedy
 * decode (gamma == 0), copies the tokens back.  out: host int32 [B][max_new];
 * n_out: host int32 [B].  sync. */
SSD_API ssd_status ssd_generate_batch(ssd_ctx* ctx, int batch, const void* vis_emb, const int32_t* n_vis,
                                      const int32_t* prompt, const int32_t* n_prompt, int max_new, int gamma,
                                      int32_t* out, int32_t* n_out);

/* Counters (see ssd_stats) and per-step record (see ssd_get_step_log) of
 * request b of the last batched decode.  sync.  With a batch prefilled, the
 * logits captures address request b's rows at buf + b * max_rows * vocab
 * (ssd_set_logits_capture) and buf + b * max_steps * gamma_max * vocab
 * (ssd_set_draft_logits_capture). */
SSD_API ssd_status ssd_get_batch_stats(ssd_ctx* ctx, int b, ssd_stats* stats);
SSD_API ssd_status ssd_get_batch_step_log(ssd_ctx* ctx, int b, int32_t* accepted, int32_t* drafted, int cap,
                                          int* n_steps);

/* The LM head alone (Sec. "SSD Setup for VLMs": o = g(x), greedy argmax):
 * logits = W_lm RMSNorm_f(x) and the argmax of each row (lowest index on ties)
 * for `rows` caller rows, with this ctx's lm_head / final_norm weights and
 * workspace.  Does not touch the decode state.
 *   x:      device fp32 [rows][d_model], 1 <= rows <= 9
 *   tok:    device int32 [rows]
 *   logits: device fp32 [rows][vocab], or NULL
 * async. */
SSD_API ssd_status ssd_lm_head(ssd_ctx* ctx, const float* x, int rows, int32_t* tok, float* logits);

/* The same LM head + argmax as ssd_lm_head, for callers that cannot allocate
 * device memory: code running while a stream is captured into a CUDA graph,
 * serving loops whose device memory is owned by their own allocator, hosts
 * that must avoid the implicit synchronisation of cudaMalloc/cudaFree.  The
 * paper has no counterpart; this is a deployment variant.  It needs no ctx and
 * allocates nothing: its scratch is a fixed ~5.3 MB array in device memory that
 * every GPU loading the library holds until the process exits.
 *   lm_head:    device bf16 [vocab][d_model];  final_norm: device bf16 [d_model]
 *   x:          device fp32 [rows][d_model];  tok: device int32 [rows]
 *   logits:     device fp32 [rows][vocab] or NULL;  cuda_stream: cudaStream_t
 * Limits: 1 <= rows <= 9, vocab <= 262144, d_model a multiple of 64, 16-byte
 * aligned pointers, and cuda_stream (when not NULL) a stream of the current
 * device; SSD_ERR_INVALID_ARG otherwise.  The first call on a device (with that
 * device current) looks up the array's device address and sets kernel
 * attributes: make it before any stream capture (a failed first call is retried
 * by the next one).  tok is set to -1 before the kernel runs and stays -1 if a
 * bounded device wait gives up, so -1 marks a call that did not complete.  All
 * calls share the one array, so calls that overlap on the GPU (other streams,
 * other threads) race and must be serialised by the caller.  async. */
SSD_API ssd_status ssd_lm_head_static(const void* lm_head, const void* final_norm, const float* x, int rows,
                                      int vocab, int d_model, float rms_eps, int32_t* tok, float* logits,
                                      void* cuda_stream);

/* Diagnostic for timing one kernel alone: enqueue `reps` back-to-back launches
 * of one weight-streaming projection (the GEMV kernel with its fused
 * epilogue; beyond 16 rows, in a ctx with max_batch > 1, the activation split
 * + the medium-M kernel) over `rows` activation rows (at most 16, or 128 and
 * max_seq), with whatever activations the ctx holds.  which: 0 QKV, 1 o_proj, 2 gate/up, 3 down (of `layer`), 4 LM head,
 * 5 imitation FC1, 6 imitation FC2, 7 the split-KV attention of `layer` for
 * query rows kv_len .. kv_len+rows-1 over the cache as it stands (waits for
 * the stream once to read kv_len).  *bytes receives the algorithmic bytes one
 * launch moves (weights or K/V + activation rows in + results out).  Clobbers the
 * decode state (activations, cache rows at kv_len..kv_len+rows-1): call
 * ssd_prefill before decoding again.  async. */
SSD_API ssd_status ssd_profile_projection(ssd_ctx* ctx, int which, int layer, int rows, int reps, int64_t* bytes);

/* ---- Failure-path diagnostics (for tests of callers' error handling; no GPU fault is made) ---- */

/* Host-side fault injection: after this call, the countdown-th device allocation
 * (kind SSD_FAULT_ALLOC: reported as SSD_ERR_OOM) or the countdown-th kernel launch
 * through the library's launch wrappers (kind SSD_FAULT_LAUNCH: reported as
 * SSD_ERR_CUDA, the kernel is not launched) of any ctx fails once, without
 * reaching the GPU.  kind SSD_FAULT_NONE or countdown <= 0 disarms.  Process-wide;
 * not thread-safe against concurrent ssd_* calls. */
enum { SSD_FAULT_NONE = 0, SSD_FAULT_ALLOC = 1, SSD_FAULT_LAUNCH = 2 };
SSD_API void ssd_set_fault_injection(int kind, int countdown);

/* Runs out one bounded device wait on purpose: a kernel waits, with the same
 * bounded-wait helper every pipeline stage uses, on an mbarrier phase that never
 * completes, for limit_ns (0 .. 2e9) nanoseconds, then records the timeout in the
 * ctx's error word like any stage that gives up.  The next ssd_sync returns
 * SSD_ERR_TIMEOUT; decode kernels enqueued meanwhile skip their work; the next
 * ssd_prefill / ssd_prefill_batch clears the word and the ctx is usable again.  async. */
SSD_API ssd_status ssd_probe_bounded_wait(ssd_ctx* ctx, int64_t limit_ns);

SSD_API const char* ssd_status_string(ssd_status s);
SSD_API const char* ssd_last_error(const ssd_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* SSD_H_ */
