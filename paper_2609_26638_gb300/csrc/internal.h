// internal.h -- declarations shared by the library's translation units.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace gs {

struct GemmArgs;

// Token tile for a GEMM over T token rows.
inline int gemm_bn_for(int T) { return T <= 32 ? 32 : (T <= 64 ? 64 : (T <= 128 ? 128 : 256)); }

// Launch Y = epilogue(W . X^T) for one weight matrix.  grid = (feat_tiles,
// tok_tiles, splits).  Returns a cudaError_t.
cudaError_t launch_gemm(int bn, int epi, const CUtensorMap& tmW, const CUtensorMap& tmX,
                        const GemmArgs& args, int feat_tiles, int tok_tiles, cudaStream_t s);

// Sets the dynamic shared-memory limit of every GEMM instantiation once.
cudaError_t gemm_init_attributes();

}  // namespace gs
