// internal.h -- declarations shared by the library's translation units.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace gs {

struct GemmArgs;

// cudaLaunchKernelEx with optional programmatic stream serialisation (PDL) and
// an optional thread-block cluster shape.
template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                      cudaStream_t s, bool pdl, dim3 cluster, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attrs[2];
  int n = 0;
  if (pdl) {
    attrs[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attrs[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (cluster.x * cluster.y * cluster.z > 1) {
    attrs[n].id = cudaLaunchAttributeClusterDimension;
    attrs[n].val.clusterDim.x = cluster.x;
    attrs[n].val.clusterDim.y = cluster.y;
    attrs[n].val.clusterDim.z = cluster.z;
    ++n;
  }
  cfg.attrs = attrs;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Token tile for a GEMM over T token rows.
// SMs of one GB300 (two dies x 76).  Work decompositions that must not depend
// on the device (the split-K factors) use this constant, not a query.
constexpr int kNumSMs = 152;

inline int gemm_bn_for(int T) { return T <= 32 ? 32 : (T <= 64 ? 64 : (T <= 128 ? 128 : 256)); }

// Launch Y = epilogue(W . X^T) for one weight matrix.  grid = (feat_tiles,
// tok_tiles, splits).  Returns a cudaError_t.
// Split-K partials are reduced through distributed shared memory inside a
// cluster of the `splits` CTAs of a tile when splits <= kMaxClusterSplits,
// else through global scratch by the last CTA to arrive (same order, same bits).
constexpr int kMaxClusterSplits = 8;
// The cluster reduction gives split CTA q the tokens [q*per, (q+1)*per) of a
// BN-token tile, per = BN / splits, and its epilogue handles per <= 8 or a
// per that divides 32 (a slice never straddles a 32-token chunk).
inline bool gemm_cluster_ok(int bn, int splits) {
  if (splits < 2 || splits > kMaxClusterSplits || bn > 64 || bn % splits) return false;
  const int per = bn / splits;
  return per <= 8 || 32 % per == 0;
}
cudaError_t launch_gemm(int bn, int epi, const CUtensorMap& tmW, const CUtensorMap& tmX,
                        const GemmArgs& args, int feat_tiles, int tok_tiles, cudaStream_t s,
                        bool pdl = false);

// 2-D fp16 tensor map over a row-major [rows, cols] array, box {64 columns,
// box_rows rows}, 128-byte swizzle, zero fill out of bounds.  The driver's
// encoder is looked up once per process (thread-safe).  False if the lookup
// or the encode fails.
bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows);


// Sets the dynamic shared-memory limit of every GEMM instantiation once.
cudaError_t gemm_init_attributes();
// Every kernel's launch attributes on the current device, once per device
// (thread-safe); call before the first launch.
cudaError_t ensure_kernel_attributes();

}  // namespace gs
