// Shared device definitions of the SSD library: device state, PTX wrappers
// (mbarrier, TMA bulk/tensor copies, programmatic dependent launch) and
// bounded waits.  sm_103a only.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/ssd.h"

namespace ssd {

constexpr int kMaxRows = SSD_MAX_ROWS;
constexpr int kMaxMidRows = 128;  // rows of one medium-M projection (the verification of batched requests)
constexpr int kAmKeyStride = 16;    // 64-bit argmax keys per LM-head row slot (128 bytes)
constexpr int kAmChunks = kMaxMidRows / 16;  // 16-row chunks of a medium-M LM head
constexpr int kAmCountStride = 32;  // 32-bit tickets per chunk slot (128 bytes)

// Device error bits (DevState::error).
enum : int { DERR_TOKEN = 1, DERR_TIMEOUT = 2, DERR_POS = 4 };

// Decode state kept in device memory so that a captured graph replays the
// whole draft/verify/accept loop without host round trips.  16-byte aligned, so
// that whatever follows a DevState (an array of them, a scratch struct) keeps
// 16-byte alignment for vector and bulk copies.
struct alignas(16) DevState {
  int kv_len;      // valid cache length p == position of the current token y
  int cur_tok;     // y: last emitted token, not yet in the cache
  int n_out;       // tokens emitted so far (the prefill's first token included)
  int max_new;     // stop after this many tokens
  int gamma;       // draft length of the running decode
  int done;        // 1 once max_new tokens are out or eos was emitted
  int error;       // DERR_* bits
  int prompt_len;  // P
  int steps;       // verify passes / greedy steps since the prefill
  int drafted;     // sum of gamma_eff
  int accepted;    // sum of a
  int last_n;      // tokens emitted by the last accept
  int eos_id;
  int dyn_launches;  // kernel launches of the running dynamic-length decode's steps
  int enc_len;     // encoder rows = cross-attention keys (encoder-decoder model), else 0
  int pad1;
  int hist[SSD_MAX_GAMMA + 1];   // steps per accepted length a
  int tok_in[kMaxRows];          // verify rows t_0 = y, t_j = d_j
  int full_tok[kMaxRows];        // f_i = full-model argmax of row i
  int last_emitted[kMaxRows];
  // packed argmax accumulators of the LM head's rows, row r at am_key[r * kAmKeyStride] (one
  // 128-byte line per row: the tiles' atomics on different rows do not share a line)
  unsigned long long am_key[kMaxMidRows * kAmKeyStride];
  // LM-head row tiles finished, per 16-row chunk ch at am_count[ch * kAmCountStride]
  unsigned int am_count[kAmChunks * kAmCountStride];
};

// ------------------------------------------------------------------ PTX wrappers

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t) :: "memory");
  return t;
}

// Waits for the phase with the given parity; gives up after limit_ns and returns false.
__device__ __forceinline__ bool mbar_wait_for(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255u) == 0u && globaltimer_ns() - t0 > limit_ns) return false;
  }
}

// After a wait gave up: the copies a ring's producer issued for its last `issued` fills (stage
// i % stages, phase i / stages) may still be landing; a bounded wait for each before the CTA leaves.
__device__ __forceinline__ void drain_ring(uint64_t* full, int stages, int issued) {
  for (int i = issued > stages ? issued - stages : 0; i < issued; ++i)
    mbar_wait_for(&full[i % stages], static_cast<uint32_t>(i / stages) & 1u, 100000000ull);
}

// The library's bounded wait: gives up after ~2 s.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  return mbar_wait_for(bar, parity, 2000000000ull);
}

// 2D tiled TMA load of one box into shared memory, completing on `bar`.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      ::"r"(smem_u32(dst)), "l"(map), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// 16-byte asynchronous global -> shared copies (completion: cp_async_wait_all / _wait_group).
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
// Same, reading src_bytes (0 or 16) and filling the rest of the 16 bytes with zeros.
__device__ __forceinline__ void cp_async16_fill(void* dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_group() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Device-scope fetch-and-add with acquire and release semantics (a split tile's ticket).
__device__ __forceinline__ unsigned atom_add_acq_rel_gpu(unsigned* a, unsigned v) {
  unsigned old;
  asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], %2;" : "=r"(old) : "l"(a), "r"(v) : "memory");
  return old;
}

// Prefetch one box of a tensor map into L2 (no shared memory, no completion).
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap* map, int x, int y) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(map), "r"(x), "r"(y)
               : "memory");
}

// Untiled bulk copy global -> shared (16-byte aligned, size a multiple of 16).
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(map) : "memory");
}

// Programmatic dependent launch: wait for the upstream grid's memory, and let
// the downstream grid start its prologue early.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Named barrier among the first `nthreads` threads (consumer warps only).
__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}

__device__ __forceinline__ float silu_f(float v) { return v / (1.0f + expf(-v)); }
// GELU in its tanh form, 0.5 v (1 + tanh(sqrt(2/pi) (v + 0.044715 v^3))) (the gated-GELU MLP of T5 v1.1).
__device__ __forceinline__ float gelu_tanh_f(float v) {
  return 0.5f * v * (1.0f + tanhf(0.7978845608028654f * (v + 0.044715f * v * v * v)));
}

// Total order on floats as unsigned keys (larger float -> larger key).
__device__ __forceinline__ uint32_t orderable(float f) {
  uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Packed (logit, index) key: max picks the largest logit, ties the lowest index.
__device__ __forceinline__ unsigned long long argmax_key(float logit, uint32_t idx) {
  return (static_cast<unsigned long long>(orderable(logit)) << 32) | (0xFFFFFFFFu - idx);
}

__device__ __forceinline__ void set_error(DevState* st, int bits) { atomicOr(&st->error, bits); }

}  // namespace ssd
