// noalloc.cu -- gs_linear_noalloc: the projection GEMM of gs_linear, with its
// split-K scratch taken from a fixed array in device memory instead of from
// the caller.
//
// For callers that cannot allocate device memory at the point of the call and
// have no workspace to hand over: code that runs inside another framework's
// operator with no workspace argument, plugin hosts whose allocator owns all
// device memory, or real-time paths where cudaMalloc's implicit device
// synchronisation is not allowed.  This file calls no cudaMalloc, cudaFree or
// allocating library routine.
//
// The array is GS_NOALLOC_SCRATCH_BYTES per device; every GPU that loads the
// library keeps it until the process exits.  All calls share it, so two calls
// whose kernels overlap on the GPU (different streams, or different host
// threads on one device) race on it; serialise them.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "gemm_tc.cuh"
#include "internal.h"
#include "../../include/gs.h"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[GS_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device.  The host-side
// name is only a stand-in for the symbol, so the address is looked up once
// per device with that device current.
int scratch_for_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return GS_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr)
      return GS_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return GS_OK;
}

inline size_t up256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

extern "C" int gs_linear_noalloc(const void* x, const void* w, void* y, int M, int N, int K,
                                 int epilogue, int split_k, void* stream) {
  using namespace gs;
  if (!x || !w || !y || M < 1 || K < 64 || K % 64 || split_k < 1 || (K / 64) % split_k)
    return GS_ERR_INVALID_ARG;
  if (epilogue < 0 || epilogue > 3) return GS_ERR_INVALID_ARG;
  if (epilogue == kEpiSwiGLU ? (N % 64) : (N % 128)) return GS_ERR_INVALID_ARG;
  if (M > 65536) return GS_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(x) & 15) || (reinterpret_cast<uintptr_t>(w) & 15) ||
      (reinterpret_cast<uintptr_t>(y) & 15))
    return GS_ERR_INVALID_ARG;
  const int bn = gemm_bn_for(M);
  const int tok_tiles = (M + bn - 1) / bn;
  const int w_rows = epilogue == kEpiSwiGLU ? 2 * N : N;
  const int feat_tiles = w_rows / 128;
  // scratch layout: error word | per-tile counters | split-K partials
  const size_t err_bytes = up256(64 * sizeof(int));
  const size_t cnt_bytes = up256(static_cast<size_t>(tok_tiles) * feat_tiles * sizeof(int));
  const size_t part_bytes =
      split_k > 1 ? static_cast<size_t>(split_k) * tok_tiles * feat_tiles * bn * 128 * sizeof(float)
                  : 0;
  if (err_bytes + cnt_bytes + part_bytes > GS_NOALLOC_SCRATCH_BYTES) return GS_ERR_OOM;

  if (ensure_kernel_attributes() != cudaSuccess) return GS_ERR_CUDA;
  void* base = nullptr;
  int rc = scratch_for_current_device(&base);
  if (rc != GS_OK) return rc;
  CUtensorMap tw, tx;
  if (!make_map(&tw, w, w_rows, K, epilogue == kEpiSwiGLU ? 64 : 128)) return GS_ERR_INVALID_ARG;
  if (!make_map(&tx, x, M, K, bn)) return GS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* b = static_cast<uint8_t*>(base);
  // the split-K counters must start at zero; the array keeps the last call's contents
  if (cudaMemsetAsync(b, 0, err_bytes + cnt_bytes, s) != cudaSuccess) return GS_ERR_CUDA;
  GemmArgs a = {};
  a.err = reinterpret_cast<int*>(b);
  a.counters = reinterpret_cast<int*>(b + err_bytes);
  a.partial = split_k > 1 ? reinterpret_cast<float*>(b + err_bytes + cnt_bytes) : nullptr;
  a.M = M;
  a.N = N;
  a.K = K;
  a.splits = split_k;
  a.cluster = 0;
  a.kb_per_split = (K / 64) / split_k;
  a.y = y;
  a.ldy = N;
  a.logits = nullptr;
  a.w_scale = 1.f;
  return launch_gemm(bn, epilogue, tw, tx, a, feat_tiles, tok_tiles, s) == cudaSuccess ? GS_OK
                                                                                        : GS_ERR_CUDA;
}

extern "C" int gs_linear_noalloc_status(void* stream) {
  using namespace gs;
  void* base = nullptr;
  int rc = scratch_for_current_device(&base);
  if (rc != GS_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int word = 0;
  if (cudaMemcpyAsync(&word, base, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return GS_ERR_CUDA;
  if (word == kErrNone) return GS_OK;
  if (cudaMemsetAsync(base, 0, sizeof(int), s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
    return GS_ERR_CUDA;
  return word == kErrTimeout ? GS_ERR_TIMEOUT : GS_ERR_DEVICE_CHECK;
}
