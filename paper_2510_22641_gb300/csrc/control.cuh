// Small kernels around the projections: embedding gather, prefill rows, the
// greedy acceptance / rollback of Algorithm 1, the greedy baseline's step, and
// the device-side loop control of the decode graphs.
#pragma once

#include "common.cuh"

namespace ssd {

// x[m][:] = fp32(E[tok[m]][:]) -- the embedding layer that maps token ids to x_0.
__global__ void ssd_embed_kernel(const __nv_bfloat16* __restrict__ E, const int* tok, float* x, int x_stride, int d,
                             int vocab, DevState* st) {
  pdl_trigger();
  pdl_wait();
  const int m = blockIdx.x;
  int t = __ldcg(tok + m);
  if (t < 0 || t >= vocab) {
    if (threadIdx.x == 0) set_error(st, DERR_TOKEN);
    t = 0;
  }
  const uint4* src = reinterpret_cast<const uint4*>(E + static_cast<size_t>(t) * d);
  float4* dst = reinterpret_cast<float4*>(x + static_cast<size_t>(m) * x_stride);
  for (int i = threadIdx.x; i < d / 8; i += blockDim.x) {
    const uint4 v = __ldg(src + i);
    const float2 a = bf16x2_to_float2(v.x), b = bf16x2_to_float2(v.y), c = bf16x2_to_float2(v.z),
                 e = bf16x2_to_float2(v.w);
    dst[2 * i] = make_float4(a.x, a.y, b.x, b.y);
    dst[2 * i + 1] = make_float4(c.x, c.y, e.x, e.y);
  }
}

// Prefill input rows r0 + m of [z (n_vis rows); embed(prompt)] (Sec. "SSD Setup for VLMs": z is fed
// to the decoder as its first input rows).
__global__ void ssd_prefill_rows_kernel(const __nv_bfloat16* __restrict__ vis, const int* __restrict__ prompt, int n_vis,
                                    int r0, const __nv_bfloat16* __restrict__ E, int vocab, float* x, int x_stride,
                                    int d, DevState* st) {
  pdl_trigger();
  pdl_wait();
  const int m = blockIdx.x, r = r0 + m;
  const __nv_bfloat16* row;
  if (r < n_vis) {
    row = vis + static_cast<size_t>(r) * d;
  } else {
    int t = __ldg(prompt + (r - n_vis));
    if (t < 0 || t >= vocab) {
      if (threadIdx.x == 0) set_error(st, DERR_TOKEN);
      t = 0;
    }
    row = E + static_cast<size_t>(t) * d;
  }
  const uint4* src = reinterpret_cast<const uint4*>(row);
  float4* dst = reinterpret_cast<float4*>(x + static_cast<size_t>(m) * x_stride);
  for (int i = threadIdx.x; i < d / 8; i += blockDim.x) {
    const uint4 v = __ldg(src + i);
    const float2 a = bf16x2_to_float2(v.x), b = bf16x2_to_float2(v.y), c = bf16x2_to_float2(v.z),
                 e = bf16x2_to_float2(v.w);
    dst[2 * i] = make_float4(a.x, a.y, b.x, b.y);
    dst[2 * i + 1] = make_float4(c.x, c.y, e.x, e.y);
  }
}

// P: decoder rows of the prompt (the position of the first new token + 1); enc_len: encoder rows
// (encoder-decoder model; 0 otherwise).
__global__ void ssd_prefill_begin_kernel(DevState* st, int P, int eos_id, int enc_len) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x != 0) return;
  st->kv_len = 0;
  st->prompt_len = P;
  st->enc_len = enc_len;
  st->n_out = 0;
  st->done = 0;
  st->error = 0;
  st->eos_id = eos_id;
  st->steps = st->drafted = st->accepted = 0;
  for (int i = 0; i <= SSD_MAX_GAMMA; ++i) st->hist[i] = 0;
  for (int i = 0; i < kMaxMidRows; ++i) st->am_key[i * kAmKeyStride] = 0ull;
  for (int i = 0; i < kAmChunks; ++i) st->am_count[i * kAmCountStride] = 0u;
}

// The last prompt row's greedy token is the first new token; the cache now holds positions 0..P-1.
__global__ void ssd_prefill_finish_kernel(DevState* st, int* out_tok, int P) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x != 0) return;
  const int y = st->full_tok[0];
  st->cur_tok = y;
  st->tok_in[0] = y;
  st->kv_len = P;
  st->n_out = 1;
  st->max_new = 1 << 30;
  out_tok[0] = y;
  st->last_n = 1;
  st->last_emitted[0] = y;
  st->done = (st->eos_id >= 0 && y == st->eos_id) ? 1 : 0;
}

__global__ void ssd_decode_setup_kernel(DevState* st, int max_new, int gamma) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x != 0) return;
  st->max_new = max_new;
  st->gamma = gamma;
  st->steps = st->drafted = st->accepted = 0;
  st->dyn_launches = 0;
  for (int i = 0; i <= SSD_MAX_GAMMA; ++i) st->hist[i] = 0;
  if (st->n_out >= max_new || st->error) st->done = 1;
}

// Dynamic draft length (Sec. "Choice of d"): this step drafts gamma = table[kv_len] tokens,
// clamped to [1, cap] (table[p] = d(p + 2), evaluated on the host in fp64); the step's branch
// of the SWITCH node is gamma - 1.  launches[gamma - 1]: kernel launches of that branch.
__global__ void ssd_dyn_select_kernel(DevState* st, const int* table, const int* launches, int cap,
                                  cudaGraphConditionalHandle sw) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x != 0) return;
  int g = table[st->kv_len];
  g = g < 1 ? 1 : (g > cap ? cap : g);
  st->gamma = g;
  st->dyn_launches += launches[g - 1] + 2;  // + this kernel and the loop test
  cudaGraphSetConditional(sw, static_cast<unsigned>(g - 1));
}

// Loop test after a dynamic-length step: run the WHILE body again unless decoding is finished.
__global__ void ssd_loop_continue_kernel(DevState* st, cudaGraphConditionalHandle cond) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x == 0) cudaGraphSetConditional(cond, st->done ? 0u : 1u);
}

// First node of a decode graph: run the WHILE body only if decoding is not finished.
__global__ void ssd_loop_begin_kernel(DevState* st, cudaGraphConditionalHandle cond) {
  if (threadIdx.x == 0) cudaGraphSetConditional(cond, st->done ? 0u : 1u);
}

// Algorithm 1, acceptance: a = longest prefix with d_{i+1} == f_i (i < gamma_eff),
// emit d_1..d_a and f_a (the correction, or the bonus token when a = gamma_eff),
// roll the cache back by length: kv_len += a + 1.  step_log[steps] = (a, gamma_eff) while
// steps < log_cap.
__global__ void ssd_accept_kernel(DevState* st, int gamma, int* out_tok, int out_cap, int2* step_log, int log_cap,
                                  cudaGraphConditionalHandle cond, int has_cond) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x != 0) return;
  if (st->done) {
    st->last_n = 0;
    if (has_cond) cudaGraphSetConditional(cond, 0u);
    return;
  }
  const int remaining = st->max_new - st->n_out;
  const int g_eff = min(gamma, remaining - 1);
  int a = 0;
  while (a < g_eff && st->tok_in[a + 1] == st->full_tok[a]) ++a;
  int cnt = a + 1;
  bool eos = false;
  for (int i = 0; i < a + 1; ++i) {
    const int t = (i < a) ? st->tok_in[i + 1] : st->full_tok[a];
    st->last_emitted[i] = t;
    const int o = st->n_out + i;
    if (o < out_cap) out_tok[o] = t;
    if (st->eos_id >= 0 && t == st->eos_id) {
      cnt = i + 1;
      eos = true;
      break;
    }
  }
  st->last_n = cnt;
  st->n_out += cnt;
  st->kv_len += a + 1;
  if (st->steps < log_cap) step_log[st->steps] = make_int2(a, g_eff);
  const int y = st->full_tok[a];
  st->cur_tok = y;
  st->tok_in[0] = y;
  st->steps += 1;
  st->drafted += g_eff;
  st->accepted += a;
  st->hist[a] += 1;
  if (eos || st->n_out >= st->max_new || st->error) st->done = 1;
  if (has_cond) cudaGraphSetConditional(cond, st->done ? 0u : 1u);
}

// Greedy baseline step: emit f_0 of the single row, advance the cache by one.
__global__ void ssd_greedy_accept_kernel(DevState* st, int* out_tok, int out_cap, int2* step_log, int log_cap,
                                         cudaGraphConditionalHandle cond, int has_cond) {
  pdl_trigger();
  pdl_wait();
  if (threadIdx.x != 0) return;
  if (st->done) {
    if (has_cond) cudaGraphSetConditional(cond, 0u);
    return;
  }
  const int y = st->full_tok[0];
  if (st->n_out < out_cap) out_tok[st->n_out] = y;
  st->n_out += 1;
  st->kv_len += 1;
  st->cur_tok = y;
  st->tok_in[0] = y;
  if (st->steps < log_cap) step_log[st->steps] = make_int2(0, 0);
  st->steps += 1;
  st->last_n = 1;
  st->last_emitted[0] = y;
  if ((st->eos_id >= 0 && y == st->eos_id) || st->n_out >= st->max_new || st->error) st->done = 1;
  if (has_cond) cudaGraphSetConditional(cond, st->done ? 0u : 1u);
}

__global__ void ssd_copy_out_kernel(const DevState* st, const int* out_int, int* user_out, int* user_n, int max_new) {
  pdl_wait();
  const int n = min(st->n_out, max_new);
  for (int i = threadIdx.x; i < n; i += blockDim.x)
    if (user_out) user_out[i] = out_int[i];
  if (threadIdx.x == 0 && user_n) *user_n = n;
}

__global__ void ssd_copy_draft_kernel(const DevState* st, int gamma, int* draft_tok) {
  pdl_wait();
  if (threadIdx.x < gamma) draft_tok[threadIdx.x] = st->tok_in[threadIdx.x + 1];
}

__global__ void ssd_copy_emitted_kernel(const DevState* st, int* n_emitted, int* emitted) {
  pdl_wait();
  const int n = st->last_n;
  if (threadIdx.x == 0 && n_emitted) *n_emitted = n;
  if (emitted && threadIdx.x < n) emitted[threadIdx.x] = st->last_emitted[threadIdx.x];
}

__global__ void ssd_first_token_kernel(const DevState* st, int* first_tok) {
  pdl_wait();
  if (threadIdx.x == 0) *first_tok = st->cur_tok;
}

// ------------------------------------------------------------------ batched requests
// B independent requests decode in lockstep (Algorithm 1 per request): req[b] is request b's
// state; st (the launch state of the projections) holds the error word, the argmax keys and the
// batch's done flag and step count.  Request b's tokens go to out + b * out_cap, its step record
// to step_log + b * log_cap.

// Row b of x (stride x_stride) = E[req[b].tok_in[j]]: the embedding of request b's j-th input.
__global__ void ssd_batch_embed_kernel(const __nv_bfloat16* __restrict__ E, const DevState* req, int j, float* x,
                                       int x_stride, int d, int vocab, DevState* st) {
  pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  int t = __ldcg(&req[b].tok_in[j]);
  if (t < 0 || t >= vocab) {
    if (threadIdx.x == 0) set_error(st, DERR_TOKEN);
    t = 0;
  }
  const uint4* src = reinterpret_cast<const uint4*>(E + static_cast<size_t>(t) * d);
  float4* dst = reinterpret_cast<float4*>(x + static_cast<size_t>(b) * x_stride);
  for (int i = threadIdx.x; i < d / 8; i += blockDim.x) {
    const uint4 v = __ldg(src + i);
    const float2 a = bf16x2_to_float2(v.x), c = bf16x2_to_float2(v.y), e = bf16x2_to_float2(v.z),
                 f = bf16x2_to_float2(v.w);
    dst[2 * i] = make_float4(a.x, a.y, c.x, c.y);
    dst[2 * i + 1] = make_float4(e.x, e.y, f.x, f.y);
  }
}

// Start of a batched decode: every request's limits and counters; st->done once all are done.
__global__ void ssd_batch_setup_kernel(DevState* st, DevState* req, int B, int max_new, int gamma) {
  pdl_trigger();
  pdl_wait();
  __shared__ int all_done;
  if (threadIdx.x == 0) all_done = 1;
  __syncthreads();
  const bool err = __ldcg(&st->error) != 0;
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    DevState* r = req + b;
    r->max_new = max_new;
    r->gamma = gamma;
    r->steps = r->drafted = r->accepted = 0;
    for (int i = 0; i <= SSD_MAX_GAMMA; ++i) r->hist[i] = 0;
    if (r->n_out >= max_new || r->error || err) r->done = 1;
    if (!r->done) atomicAnd(&all_done, 0);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    st->done = all_done;
    st->steps = 0;
    st->max_new = max_new;
    st->gamma = gamma;
  }
}

// One request's acceptance (the rule of ssd_accept_kernel on state r), g_max drafts per step.
__device__ __forceinline__ void accept_one(DevState* r, int gamma, int* out, int out_cap, int2* log, int log_cap,
                                           bool err) {
  if (r->done) {
    r->last_n = 0;
    return;
  }
  const int remaining = r->max_new - r->n_out;
  const int g_eff = min(gamma, remaining - 1);
  int a = 0;
  while (a < g_eff && r->tok_in[a + 1] == r->full_tok[a]) ++a;
  int cnt = a + 1;
  bool eos = false;
  for (int i = 0; i < a + 1; ++i) {
    const int t = (i < a) ? r->tok_in[i + 1] : r->full_tok[a];
    r->last_emitted[i] = t;
    const int o = r->n_out + i;
    if (o < out_cap) out[o] = t;
    if (r->eos_id >= 0 && t == r->eos_id) {
      cnt = i + 1;
      eos = true;
      break;
    }
  }
  r->last_n = cnt;
  r->n_out += cnt;
  r->kv_len += a + 1;
  if (r->steps < log_cap) log[r->steps] = make_int2(a, g_eff);
  const int y = r->full_tok[a];
  r->cur_tok = y;
  r->tok_in[0] = y;
  r->steps += 1;
  r->drafted += g_eff;
  r->accepted += a;
  r->hist[a] += 1;
  if (eos || r->n_out >= r->max_new || err) r->done = 1;
}

// Algorithm 1's acceptance for every request of the batch (gamma = 0: a greedy step, f_0
// emitted); st->done (and the WHILE condition) once every request is done.
__global__ void ssd_batch_accept_kernel(DevState* st, DevState* req, int B, int gamma, int* out, int out_cap,
                                        int2* step_log, int log_cap, cudaGraphConditionalHandle cond, int has_cond) {
  pdl_trigger();
  pdl_wait();
  __shared__ int all_done;
  if (threadIdx.x == 0) all_done = 1;
  __syncthreads();
  const bool err = __ldcg(&st->error) != 0;
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    accept_one(req + b, gamma, out + static_cast<size_t>(b) * out_cap, out_cap,
               step_log + static_cast<size_t>(b) * log_cap, log_cap, err);
    if (!req[b].done) atomicAnd(&all_done, 0);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    st->done = all_done;
    st->steps += 1;
    if (has_cond) cudaGraphSetConditional(cond, all_done ? 0u : 1u);
  }
}

// First tokens (after a batched prefill) and tokens out of a batched decode.
__global__ void ssd_batch_first_tokens_kernel(const DevState* req, int B, int* first) {
  pdl_wait();
  for (int b = threadIdx.x; b < B; b += blockDim.x) first[b] = req[b].cur_tok;
}

__global__ void ssd_batch_copy_out_kernel(const DevState* req, const int* out_int, int out_cap, int* user_out,
                                          int* user_n, int max_new) {
  pdl_wait();
  const int b = blockIdx.x;
  const int n = min(req[b].n_out, max_new);
  for (int i = threadIdx.x; i < n; i += blockDim.x)
    if (user_out) user_out[static_cast<size_t>(b) * max_new + i] = out_int[static_cast<size_t>(b) * out_cap + i];
  if (threadIdx.x == 0 && user_n) user_n[b] = n;
}

// Diagnostic of the failure path: one thread waits, with the kernels' bounded-wait helper and a
// limit of limit_ns, on the first phase of a fresh mbarrier that nothing ever completes, so the wait
// runs out and records DERR_TIMEOUT exactly as a stalled pipeline stage would.  No copy is in flight
// and no other thread waits.
__global__ void ssd_wait_probe_kernel(DevState* st, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
    if (!mbar_wait_for(&bar, 0u, limit_ns)) set_error(st, DERR_TIMEOUT);
  }
}

// cos/sin of pos * theta^(-2j/head_dim), computed in fp64 and rounded to fp32.
__global__ void ssd_rope_table_kernel(float2* cs, int max_seq, int head_dim, double theta) {
  const int half = head_dim / 2;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= max_seq * half) return;
  const int pos = idx / half, j = idx - pos * half;
  const double ang = static_cast<double>(pos) * pow(theta, -2.0 * j / head_dim);
  double s, c;
  sincos(ang, &s, &c);
  cs[idx] = make_float2(static_cast<float>(c), static_cast<float>(s));
}

// Relative-position bias table out[h][j] = rel[bucket[j]][h] (rel: the learned [buckets][n_heads]
// bf16 table of a T5-style stack; bucket[j]: the bucket of offset j - zero, decided on the host).
__global__ void ssd_bias_table_kernel(const __nv_bfloat16* __restrict__ rel, const int* __restrict__ bucket, int n,
                                  int n_heads, float* out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n * n_heads) return;
  const int h = i / n, j = i - h * n;
  out[i] = __bfloat162float(rel[static_cast<size_t>(bucket[j]) * n_heads + h]);
}

}  // namespace ssd
