// ssd_lm_head_static: the LM-head projection + argmax without any allocation.
//
// Some callers cannot call cudaMalloc: code that runs while a stream is being
// captured into a CUDA graph (an allocation there is illegal or forces a
// synchronisation), serving loops with a fixed device-memory budget owned by
// their own allocator, and hosts that forbid the implicit device-wide
// synchronisation of cudaMalloc/cudaFree.  This entry point therefore keeps
// its scratch -- the tickets and partial sums of row tiles split between CTAs
// and the argmax accumulators -- in one file-scope __device__ array of fixed
// size that every GPU loading the library holds until the process exits.
#include <cudaTypedefs.h>

#include <mutex>

#include "gemv.cuh"

namespace ssd {
cudaError_t gemv_launch_head(int M, const CUtensorMap*, const GemvParams&, int, cudaStream_t, bool);
cudaError_t gemv_attrs_head();
}  // namespace ssd

using namespace ssd;

namespace {

constexpr int kStaticMaxVocab = 262144;                   // vocab limit (2048 row tiles of 128)
constexpr int kStaticMaxCtas = 320;                       // GEMV CTAs (2 per SM, up to 160 SMs)
constexpr int kStaticMaxTiles = kStaticMaxVocab / kTileN;
constexpr int kStaticMaxDevices = 64;

struct StaticScratch {
  DevState st;                                             // argmax accumulators, error word
  unsigned counters[kStaticMaxTiles];                      // tickets of split row tiles
  // partial sums of split row tiles, read 16 bytes at a time
  alignas(16) float partials[2 * kStaticMaxCtas * kMaxRows * kTileN];
};

// About 5.3 MB of device memory per GPU, held from library load until exit.
static __device__ __align__(256) StaticScratch g_head_scratch;

struct DeviceSetup {
  bool done = false;
  StaticScratch* scratch = nullptr;  // device address of g_head_scratch on this device
  int num_sms = 0;
};

std::mutex g_setup_mu;
DeviceSetup g_setup[kStaticMaxDevices];
PFN_cuTensorMapEncodeTiled_v12000 g_encode_static = nullptr;

// Once per device, with that device current: the array's device address, the
// SM count, the tensor-map encoder and the kernel's shared-memory limit.
cudaError_t setup_device(int dev, DeviceSetup** out) {
  std::lock_guard<std::mutex> lk(g_setup_mu);
  DeviceSetup& s = g_setup[dev];
  *out = &s;
  if (s.done) return cudaSuccess;
  // a failed set-up is not cached: the next call on this device tries again
  cudaError_t e = cudaGetSymbolAddress(reinterpret_cast<void**>(&s.scratch), g_head_scratch);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&s.num_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = gemv_attrs_head();
  if (e == cudaSuccess && !g_encode_static) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e == cudaSuccess && (q != cudaDriverEntryPointSuccess || !fn)) e = cudaErrorNotSupported;
    if (e == cudaSuccess) g_encode_static = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  s.done = e == cudaSuccess;
  return e;
}

}  // namespace

extern "C" {

ssd_status ssd_lm_head_static(const void* lm_head, const void* final_norm, const float* x, int rows, int vocab,
                              int d_model, float rms_eps, int32_t* tok, float* logits, void* cuda_stream) {
  if (!lm_head || !final_norm || !x || !tok) return SSD_ERR_INVALID_ARG;
  if (rows < 1 || rows > 9 || vocab < 1 || vocab > kStaticMaxVocab) return SSD_ERR_INVALID_ARG;
  if (d_model < kTileK || d_model % kTileK != 0) return SSD_ERR_INVALID_ARG;  // 64-column slices stay in a row
  const uintptr_t al = reinterpret_cast<uintptr_t>(lm_head) | reinterpret_cast<uintptr_t>(final_norm) |
                       reinterpret_cast<uintptr_t>(x);
  if (al % 16 != 0) return SSD_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kStaticMaxDevices) return SSD_ERR_CUDA;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  if (stream) {  // the array's address below is the current device's: the stream must belong to it
    int sdev = -1;
    if (cudaStreamGetDevice(stream, &sdev) != cudaSuccess) return SSD_ERR_CUDA;
    if (sdev != dev) return SSD_ERR_INVALID_ARG;
  }
  DeviceSetup* ds = nullptr;
  if (setup_device(dev, &ds) != cudaSuccess) return SSD_ERR_CUDA;

  CUtensorMap maps[3];
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d_model), static_cast<cuuint64_t>(vocab)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d_model) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kTileK), static_cast<cuuint32_t>(kTileN)};
  cuuint32_t es[2] = {1, 1};
  if (g_encode_static(&maps[0], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(lm_head), dims, strides, box,
                      es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return SSD_ERR_CUDA;
  maps[1] = maps[2] = maps[0];

  GemvParams p{};
  p.K = d_model;
  p.n_kt = d_model / kTileK;
  p.n_rt = (vocab + kTileN - 1) / kTileN;
  p.units = p.n_rt * p.n_kt;
  p.N = vocab;
  p.seg_rows = vocab;
  p.x = x;
  p.x_stride = d_model;
  p.gain = static_cast<const __nv_bfloat16*>(final_norm);
  p.eps = rms_eps;
  StaticScratch* sc = ds->scratch;
  p.partials = sc->partials;
  p.counters = sc->counters;
  p.st = &sc->st;
  p.pos_off = -1;  // kv_len = prompt_len = 0 after the clear below: logits row m -> row m
  p.tok_dst = tok;
  p.logits = logits;
  p.logits_rows = logits ? rows : 0;
  int grid = 2 * ds->num_sms;
  if (grid > kStaticMaxCtas) grid = kStaticMaxCtas;
  if (grid > p.units) grid = p.units;

  // The array keeps the previous call's contents: clear the state and the
  // tickets this call uses (the kernel leaves them at zero, but a call that
  // stopped early might not have).  tok starts at -1, which a call whose
  // kernel gave up on a bounded wait leaves in place.
  if (cudaMemsetAsync(tok, 0xFF, sizeof(int32_t) * rows, stream) != cudaSuccess) return SSD_ERR_CUDA;
  if (cudaMemsetAsync(&sc->st, 0, sizeof(DevState), stream) != cudaSuccess) return SSD_ERR_CUDA;
  if (cudaMemsetAsync(sc->counters, 0, sizeof(unsigned) * p.n_rt, stream) != cudaSuccess) return SSD_ERR_CUDA;
  if (gemv_launch_head(rows, maps, p, grid, stream, false) != cudaSuccess) return SSD_ERR_CUDA;
  return SSD_OK;
}

}  // extern "C"
