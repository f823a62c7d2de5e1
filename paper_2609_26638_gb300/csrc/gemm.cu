// gemm.cu -- instantiations and launcher of the tcgen05 GEMM.
#include "gemm_tc.cuh"
#include "internal.h"

namespace gs {

template <int BN, int EPI>
static cudaError_t launch_one(const CUtensorMap& tmW, const CUtensorMap& tmX, GemmArgs a,
                              int feat_tiles, int tok_tiles, cudaStream_t s, bool pdl) {
  using S = GemmShape<BN>;
  // Pipeline depth, never more than the k-blocks one CTA loads.  Decode
  // windows (up to 64 rows, unchunked): a fixed depth that leaves room for a
  // second resident CTA and for the neighbouring kernels' CTAs that overlap it
  // under programmatic dependent launch.  Wider launches stream K through
  // each CTA: the deepest pipeline that still fits the CTAs one SM holds
  // (one when the grid is at most one CTA per SM, else two), since bytes in
  // flight per SM set their load rate.
  const bool cl = a.splits > 1 && a.cluster;
  int want = S::kStagesDefault;
  if (a.chunks > 1 || a.M > 64)
    want = S::stages_fitting(static_cast<long>(feat_tiles) * tok_tiles * a.splits <= kNumSMs ? 1 : 2,
                             EPI, cl);
  const int kb = a.kb_per_split;
  a.stages = kb < S::kStagesMin ? S::kStagesMin : (kb > want ? want : kb);
  dim3 grid(tok_tiles, feat_tiles, a.splits);
  const int cz = cl ? a.splits : 1;
  return launch_ex(gemm_tc_kernel<BN, EPI>, grid, dim3(128), S::smem_bytes(a.stages, EPI, cl), s,
                   pdl, dim3(1, 1, cz), tmW, tmX, a);
}

// Chunked-K launches (wide decode windows): two CTAs per SM, the deepest
// pipeline that still fits them, never more stages than k-blocks.
template <int BN, int EPI>
static cudaError_t launch_chunk_one(const CUtensorMap& tmW, const CUtensorMap& tmX, GemmArgs a,
                                    int feat_tiles, int tok_tiles, cudaStream_t s, bool pdl) {
  using S = GemmShape<BN>;
  const int want = S::stages_fitting(2, EPI, false);
  const int kb = a.K / 64;
  a.stages = kb < S::kStagesMin ? S::kStagesMin : (kb > want ? want : kb);
  dim3 grid(tok_tiles, feat_tiles, 1);
  return launch_ex(gemm_chunk_kernel<BN, EPI>, grid, dim3(192), S::smem_bytes(a.stages, EPI, false),
                   s, pdl, dim3(1, 1, 1), tmW, tmX, a);
}

template <int BN, int EPI>
static cudaError_t launch_one_or_chunk(const CUtensorMap& tmW, const CUtensorMap& tmX,
                                       const GemmArgs& a, int ft, int tt, cudaStream_t s, bool pdl) {
  if constexpr (BN <= 128) {
    if (a.chunks > 1 && a.splits == 1) return launch_chunk_one<BN, EPI>(tmW, tmX, a, ft, tt, s, pdl);
  }
  return launch_one<BN, EPI>(tmW, tmX, a, ft, tt, s, pdl);
}

template <int BN>
static cudaError_t launch_bn(int epi, const CUtensorMap& tmW, const CUtensorMap& tmX,
                             const GemmArgs& a, int ft, int tt, cudaStream_t s, bool pdl) {
  switch (epi) {
    case kEpiStoreF16: return launch_one_or_chunk<BN, kEpiStoreF16>(tmW, tmX, a, ft, tt, s, pdl);
    case kEpiResidF32: return launch_one_or_chunk<BN, kEpiResidF32>(tmW, tmX, a, ft, tt, s, pdl);
    case kEpiSwiGLU: return launch_one_or_chunk<BN, kEpiSwiGLU>(tmW, tmX, a, ft, tt, s, pdl);
    case kEpiArgmax: return launch_one_or_chunk<BN, kEpiArgmax>(tmW, tmX, a, ft, tt, s, pdl);
    case kEpiQKV: return launch_one_or_chunk<BN, kEpiQKV>(tmW, tmX, a, ft, tt, s, pdl);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemm(int bn, int epi, const CUtensorMap& tmW, const CUtensorMap& tmX,
                        const GemmArgs& a, int feat_tiles, int tok_tiles, cudaStream_t s,
                        bool pdl) {
  switch (bn) {
    case 32: return launch_bn<32>(epi, tmW, tmX, a, feat_tiles, tok_tiles, s, pdl);
    case 64: return launch_bn<64>(epi, tmW, tmX, a, feat_tiles, tok_tiles, s, pdl);
    case 128: return launch_bn<128>(epi, tmW, tmX, a, feat_tiles, tok_tiles, s, pdl);
    case 256: return launch_bn<256>(epi, tmW, tmX, a, feat_tiles, tok_tiles, s, pdl);
  }
  return cudaErrorInvalidValue;
}

template <int BN>
static cudaError_t set_attr_chunk() {
  const int bytes = GemmShape<BN>::kSmemMax;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(gemm_chunk_kernel<BN, kEpiStoreF16>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(gemm_chunk_kernel<BN, kEpiResidF32>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(gemm_chunk_kernel<BN, kEpiSwiGLU>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(gemm_chunk_kernel<BN, kEpiArgmax>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  return cudaFuncSetAttribute(gemm_chunk_kernel<BN, kEpiQKV>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

template <int BN>
static cudaError_t set_attr_bn() {
  const int bytes = GemmShape<BN>::kSmemMax;
  cudaError_t e;
  if constexpr (BN <= 128) {
    if ((e = set_attr_chunk<BN>()) != cudaSuccess) return e;
  }
  if ((e = cudaFuncSetAttribute(gemm_tc_kernel<BN, kEpiStoreF16>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(gemm_tc_kernel<BN, kEpiResidF32>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(gemm_tc_kernel<BN, kEpiSwiGLU>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(gemm_tc_kernel<BN, kEpiArgmax>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  return cudaFuncSetAttribute(gemm_tc_kernel<BN, kEpiQKV>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t gemm_init_attributes() {
  cudaError_t e;
  if ((e = set_attr_bn<32>()) != cudaSuccess) return e;
  if ((e = set_attr_bn<64>()) != cudaSuccess) return e;
  if ((e = set_attr_bn<128>()) != cudaSuccess) return e;
  return set_attr_bn<256>();
}

}  // namespace gs
