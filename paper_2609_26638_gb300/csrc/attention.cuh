// attention.cuh -- hybrid-mask attention over the paged bf16 KV cache.
//
// One CTA = (KV split c, KV head h, query block b).  A query block is a run of
// tokens of one sequence (the K+1 window of a decode forward, or 64 tokens of
// a prefill chunk); its rows are (token, query head of the GQA group), so the
// query heads that share a KV head read each K/V page once.  Every query
// token carries its own inclusive key limit, which encodes the mask: draft
// boundary row n, draft mask rows n+K, verify row i n+1+i, prefill row p (paper
// Appendix steps Draft forward / Verify forward).
//
// K and V pages (64 tokens x 64 dims, 8 KB each) are staged by TMA with
// 128-byte swizzle into a ring of shared-memory stages.  Warps form NG groups
// of one warp per 16 rows; group g takes the split's pages g, g+NG, ... so NG
// pages are in work at once.  Each warp runs S = Q K^T and O += P V on
// mma.sync m16n8k16 (bf16 in, fp32 out) with the online softmax in registers
// (exp2 with the 1/sqrt(64) scale folded).  NG depends only on the row count
// (4 up to 64 rows, 2 up to 128, else 1), so windows with the same group
// count give bit-identical rows.
//
// Splits cover fixed absolute page ranges [c*SP, (c+1)*SP), so a row's result
// depends only on its own keys and not on the window it sits in; keys past a
// row's limit contribute exact zeros.  The warp groups of a CTA first merge
// their partials in shared memory (group order).  The splits of one (block,
// head) are one thread-block cluster (at most kAttnMaxSplits CTAs; 16-CTA
// clusters measured slower: they wait for 16 free SMs in one GPC).  Row r is owned by CTA r mod C: each CTA stages
// its (O, m, l) rows grouped by owner and one thread sends each owner its
// block with a bulk async copy completing on the owner's mbarrier; each owner
// merges its rows over the splits in order.  A block whose keys fit in one
// split runs in CTA 0 alone and writes after the group merge.
#pragma once
#include "ptx.cuh"

namespace gs {

constexpr int kAttnMaxSplits = 8;
constexpr int kAttnStages = 6;
constexpr int kAttnPageBytes = 64 * 128;  // 64 tokens x 64 bf16

struct AttnArgs {
  const __nv_bfloat16* q;     // [T, Hq, 64]
  const int32_t* lim;         // [T] inclusive key limit per query token
  __nv_bfloat16* out;         // [T, Hq, 64]
  const int32_t* page_table;  // [slots, pt_stride]
  int pt_stride;
  const int32_t* blk_slot;    // [n_blocks] page-table row per block, or null -> fixed_slot
  const int32_t* blk_active;  // [n_blocks] nonzero = run, or null
  int fixed_slot;
  int T, QB;                  // tokens; tokens per query block
  int Hq, Hkv, G;
  long long kv_row_base;      // first KV-map row of this layer
  int rows_per_page;          // 2 * Hkv * 64
  int split_pages;            // SP; gridDim.x (the cluster) * SP covers the block's pages
  int* err;
};

// Rows (16 per warp), warp groups and threads for a block of r_max rows.
__host__ __device__ inline int attn_mtiles(int r_max) { return (r_max + 15) / 16; }
__host__ __device__ inline int attn_groups(int r_max) {
  return attn_mtiles(r_max) <= 4 ? 4 : (attn_mtiles(r_max) <= 8 ? 2 : 1);
}
__host__ __device__ inline int attn_threads(int r_max) {
  return attn_mtiles(r_max) * attn_groups(r_max) * 32;
}
// receive buffer: per source split, ceil(rows / C) rows of kAttnRecvRow floats:
// O[64], m, l, 2 pad (272 B keeps every row 16-byte aligned for float4 reads)
constexpr int kAttnRecvRow = 68;
__host__ __device__ inline int attn_recv_floats(int r_max) {
  return (attn_mtiles(r_max) * 16 + kAttnMaxSplits) * kAttnRecvRow;
}
__host__ __device__ inline int attn_smem_bytes(int r_max) {
  return 1024 + kAttnStages * 2 * kAttnPageBytes + attn_mtiles(r_max) * 16 * 128 + 128 +
         attn_recv_floats(r_max) * 4;
}
static_assert(kAttnStages * 2 * kAttnPageBytes >= 4 * 64 * 68 * 4 &&
                  kAttnStages * 2 * kAttnPageBytes >= (256 + kAttnMaxSplits) * 68 * 4,
              "the K/V ring must hold the group partials and the merge staging");
// Pages per split so that a sequence of `pages` pages needs at most kAttnMaxSplits splits.
__host__ __device__ inline int attn_min_split_pages(int pages) {
  return (pages + kAttnMaxSplits - 1) / kAttnMaxSplits;
}

__device__ __forceinline__ uint32_t sw128(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__global__ void __launch_bounds__(512)
    attn_paged_kernel(const __grid_constant__ CUtensorMap tmKV, const AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sK = smem;                                     // [stages][64][128 B]
  uint8_t* sV = smem + kAttnStages * kAttnPageBytes;      // [stages][64][128 B]
  uint8_t* sQ = smem + 2 * kAttnStages * kAttnPageBytes;  // [rows][128 B]
  const int nthreads = blockDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mtiles = attn_mtiles(a.QB * a.G);
  const int NG = nthreads / 32 / mtiles;    // warp groups
  const int grp = warp / mtiles, mt = warp % mtiles;
  const int rows_alloc = mtiles * 16;
  uint64_t* full = reinterpret_cast<uint64_t*>(sQ + rows_alloc * 128);
  __shared__ int s_maxlim;

  const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int C = gridDim.x;                  // split slots = cluster size
  // Before griddepcontrol.wait this kernel reads only what the kernel right
  // before it (the QKV GEMM, which writes q and the window's K/V) does not
  // write: the window descriptors (key limits, block slots), the page table,
  // and cache pages wholly before the current window.  Every branch that
  // leaves early is uniform across the cluster.
  if (a.blk_active != nullptr && a.blk_active[b] == 0) return;
  const int tok0 = b * a.QB;
  const int ntok = min(a.QB, a.T - tok0);
  if (ntok <= 0) return;
  const int R = ntok * a.G;
  const int slot = a.blk_slot ? a.blk_slot[b] : a.fixed_slot;

  if (warp == 0) {
    int m = -1;
    for (int i = lane; i < ntok; i += 32) m = max(m, a.lim[tok0 + i]);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) m = max(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    if (lane == 0) s_maxlim = m;
  }
  __syncthreads();
  const int maxlim = s_maxlim;
  const int npages_blk = maxlim / 64 + 1;
  const int SP = a.split_pages;
  const int nsplit = (npages_blk + SP - 1) / SP;
  if (maxlim < 0 || npages_blk > a.pt_stride || slot < 0 || nsplit > C) {
    if (threadIdx.x == 0) atomicExch(a.err, kErrBounds);
    return;
  }
  if (nsplit == 1 && c > 0) return;         // direct path: CTA 0 alone
  if (nsplit > 1) cluster_arrive_relaxed();  // completed by cluster_wait() before the pushes
  const int p_begin = c * SP;
  const int np = c < nsplit ? min(npages_blk, p_begin + SP) - p_begin : 0;
  const int32_t* pt = a.page_table + static_cast<size_t>(slot) * a.pt_stride;

  const int Ceff = nsplit == 1 ? 1 : C;          // CTAs taking part in the merge
  const int rpo = (rows_alloc + Ceff - 1) / Ceff;  // rows per owner
  const int blk_floats = rpo * kAttnRecvRow;       // one source CTA's block for one owner
  uint64_t* recv_bar = full + kAttnStages;
  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmKV);
    for (int s = 0; s < kAttnStages; ++s) mbar_init(smem_u32(&full[s]), 1);
    if (Ceff > 1) {
      mbar_init(smem_u32(recv_bar), 1);
      mbar_arrive_expect_tx(smem_u32(recv_bar), static_cast<uint32_t>(Ceff * blk_floats * 4));
    }
    fence_mbar_init();
  }
  __syncthreads();
  // pages wholly before the block's first slot hold committed states only
  const int safe_pages = a.blk_slot ? a.lim[tok0] / 64 : 0;
  const uint64_t pol = l2_policy_evict_first();
  auto issue = [&](int i) {
    const int s = i % kAttnStages;
    int phys = pt[p_begin + i];
    if (phys < 0) {  // unmapped page: the TMA box lands out of bounds and reads zeros
      atomicExch(a.err, kErrBounds);
      phys = 0x3FFFFFFF / a.rows_per_page;
    }
    const long long row = a.kv_row_base + static_cast<long long>(phys) * a.rows_per_page;
    const uint32_t fb = smem_u32(&full[s]);
    mbar_arrive_expect_tx(fb, 2 * kAttnPageBytes);
    tma_load_2d(smem_u32(sK + s * kAttnPageBytes), &tmKV, 0, static_cast<int>(row + h * 64), fb, pol);
    tma_load_2d(smem_u32(sV + s * kAttnPageBytes), &tmKV, 0,
                static_cast<int>(row + (a.Hkv + h) * 64), fb, pol);
  };
  int issued = 0;
  if (threadIdx.x == 0) {
    while (issued < min(np, kAttnStages) && p_begin + issued < safe_pages) issue(issued++);
  }
  pdl_wait();
  pdl_trigger();
  if (threadIdx.x == 0) {
    while (issued < min(np, kAttnStages)) issue(issued++);
  }

  // Q rows -> swizzled smem (zero rows past R)
  for (int idx = threadIdx.x; idx < rows_alloc * 8; idx += nthreads) {
    const int r = idx >> 3, ch = idx & 7;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (r < R) {
      const int t = tok0 + r / a.G;
      const int hq = h * a.G + r % a.G;
      v = *reinterpret_cast<const uint4*>(a.q + (static_cast<size_t>(t) * a.Hq + hq) * 64 + ch * 8);
    }
    *reinterpret_cast<uint4*>(sQ + sw128(r, ch)) = v;
  }
  __syncthreads();

  const bool has_rows = mt * 16 < R;
  const int g = lane >> 2, tq = lane & 3;
  const int r0 = mt * 16 + g, r1 = r0 + 8;
  const int lim0 = r0 < R ? a.lim[tok0 + r0 / a.G] : -1;
  const int lim1 = r1 < R ? a.lim[tok0 + r1 / a.G] : -1;

  uint32_t qa[4][4];
  if (has_rows) {
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const int row = mt * 16 + (lane & 15);
      const int ch = 2 * kk + (lane >> 4);
      ldsm_x4(smem_u32(sQ) + sw128(row, ch), qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3]);
    }
  }

  const float kScaleLog2 = 0.125f * 1.4426950408889634f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[8][4];
#pragma unroll
  for (int j = 0; j < 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  bool ok = true;

  for (int it = 0; it * NG < np; ++it) {
    const int i = it * NG + grp;              // this group's page of the iteration
    const int s = i % kAttnStages;
    const bool mine = i < np;
    if (ok && mine && !mbar_wait(smem_u32(&full[s]), (i / kAttnStages) & 1, a.err)) ok = false;
    if (ok && mine && has_rows) {
      const uint32_t kbase = smem_u32(sK + s * kAttnPageBytes);
      const uint32_t vbase = smem_u32(sV + s * kAttnPageBytes);
      float sacc[8][4];
#pragma unroll
      for (int j = 0; j < 8; ++j) sacc[j][0] = sacc[j][1] = sacc[j][2] = sacc[j][3] = 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
#pragma unroll
        for (int kk = 0; kk < 4; kk += 2) {
          uint32_t b0, b1, b2, b3;
          const int row = 8 * j + (lane & 7);
          const int ch = 2 * kk + (lane >> 3);
          ldsm_x4(kbase + sw128(row, ch), b0, b1, b2, b3);
          mma_bf16_16816(sacc[j], qa[kk], b0, b1);
          mma_bf16_16816(sacc[j], qa[kk + 1], b2, b3);
        }
      }
      // mask + online softmax (rows r0: elements 0,1; r1: elements 2,3)
      const int kbase_abs = (p_begin + i) * 64;
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int key = kbase_abs + 8 * j + 2 * tq;
        sacc[j][0] = key <= lim0 ? sacc[j][0] * kScaleLog2 : -INFINITY;
        sacc[j][1] = key + 1 <= lim0 ? sacc[j][1] * kScaleLog2 : -INFINITY;
        sacc[j][2] = key <= lim1 ? sacc[j][2] * kScaleLog2 : -INFINITY;
        sacc[j][3] = key + 1 <= lim1 ? sacc[j][3] * kScaleLog2 : -INFINITY;
        mx0 = fmaxf(mx0, fmaxf(sacc[j][0], sacc[j][1]));
        mx1 = fmaxf(mx1, fmaxf(sacc[j][2], sacc[j][3]));
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xFFFFFFFFu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xFFFFFFFFu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xFFFFFFFFu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xFFFFFFFFu, mx1, 2));
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      const float al0 = (mn0 == -INFINITY) ? 1.f : exp2f(m0 - mn0);
      const float al1 = (mn1 == -INFINITY) ? 1.f : exp2f(m1 - mn1);
      const float sub0 = (mn0 == -INFINITY) ? 0.f : mn0;
      const float sub1 = (mn1 == -INFINITY) ? 0.f : mn1;
      m0 = mn0;
      m1 = mn1;
      float ps0 = 0.f, ps1 = 0.f;
      uint32_t pa[4][4];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float p0 = exp2f(sacc[j][0] - sub0), p1 = exp2f(sacc[j][1] - sub0);
        const float p2 = exp2f(sacc[j][2] - sub1), p3 = exp2f(sacc[j][3] - sub1);
        ps0 += p0 + p1;
        ps1 += p2 + p3;
        pa[j >> 1][(j & 1) * 2 + 0] = pack_bf16x2(p0, p1);
        pa[j >> 1][(j & 1) * 2 + 1] = pack_bf16x2(p2, p3);
      }
      l0 = l0 * al0 + ps0;
      l1 = l1 * al1 + ps1;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        o[j][0] *= al0;
        o[j][1] *= al0;
        o[j][2] *= al1;
        o[j][3] *= al1;
      }
      // O += P V ; V stored [key][dim] -> transposed ldmatrix
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
        for (int jn = 0; jn < 8; jn += 2) {
          uint32_t b0, b1, b2, b3;
          const int row = 16 * kk + (lane & 7) + ((lane >> 3) & 1) * 8;
          const int ch = jn + (lane >> 4);
          ldsm_x4_t(vbase + sw128(row, ch), b0, b1, b2, b3);
          mma_bf16_16816(o[jn], pa[kk], b0, b1);
          mma_bf16_16816(o[jn + 1], pa[kk], b2, b3);
        }
      }
    }
    __syncthreads();
    if (threadIdx.x == 0 && ok) {
      for (int q = it * NG; q < it * NG + NG; ++q)
        if (q + kAttnStages < np) issue(q + kAttnStages);
    }
  }
  const bool all_ok = __syncthreads_and(ok);

  // row sums across the quad
  l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, 1);
  l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, 2);
  l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, 1);
  l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, 2);

  // ---- 1. groups -> group 0 (shared memory, group order): O = sum w_g O_g,
  //         L = sum w_g l_g, w_g = exp2(m_g - M).  gp [g][row][68] in the idle K/V ring.
  float* ring = reinterpret_cast<float*>(sK);
  if (NG > 1) {
    if (grp > 0 && has_rows) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        float* dst = ring + (static_cast<size_t>(grp) * rows_alloc + (half ? r1 : r0)) * kAttnRecvRow;
#pragma unroll
        for (int j = 0; j < 8; ++j)
          *reinterpret_cast<float2*>(dst + 8 * j + 2 * tq) =
              make_float2(o[j][half * 2 + 0], o[j][half * 2 + 1]);
        if (tq == 0) {
          dst[64] = half ? m1 : m0;
          dst[65] = half ? l1 : l0;
        }
      }
    }
    __syncthreads();
    if (grp == 0 && has_rows) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int r = half ? r1 : r0;
        const float mself = half ? m1 : m0;
        float M = mself;
        for (int q = 1; q < NG; ++q)
          M = fmaxf(M, ring[(static_cast<size_t>(q) * rows_alloc + r) * kAttnRecvRow + 64]);
        const float w0 = (mself == -INFINITY) ? 0.f : exp2f(mself - M);
        float L = w0 * (half ? l1 : l0);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          o[j][half * 2 + 0] *= w0;
          o[j][half * 2 + 1] *= w0;
        }
        for (int q = 1; q < NG; ++q) {
          const float* src = ring + (static_cast<size_t>(q) * rows_alloc + r) * kAttnRecvRow;
          const float mq = src[64];
          const float wq = (mq == -INFINITY) ? 0.f : exp2f(mq - M);
          L += wq * src[65];
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float2 v = *reinterpret_cast<const float2*>(src + 8 * j + 2 * tq);
            o[j][half * 2 + 0] += wq * v.x;
            o[j][half * 2 + 1] += wq * v.y;
          }
        }
        if (half) { m1 = M; l1 = L; } else { m0 = M; l0 = L; }
      }
    }
    __syncthreads();   // group partials consumed; the ring is reused below
  }
  const bool lead = grp == 0 && has_rows;

  if (Ceff == 1) {   // one split: the CTA's merged rows are final
    if (lead && all_ok) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int r = half ? r1 : r0;
        if (r >= R) continue;
        const float inv = 1.0f / (half ? l1 : l0);
        const int t = tok0 + r / a.G;
        const int hq = h * a.G + r % a.G;
        __nv_bfloat16* dst = a.out + (static_cast<size_t>(t) * a.Hq + hq) * 64;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float x0 = o[j][half * 2 + 0] * inv, x1 = o[j][half * 2 + 1] * inv;
          *reinterpret_cast<__nv_bfloat162*>(dst + 8 * j + 2 * tq) = __floats2bfloat162_rn(x0, x1);
        }
      }
    }
    return;
  }

  // ---- 2. splits -> owners (cluster).  stage [owner][slot][68] in the ring,
  //         recv [source split][slot][68].
  float* recv = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(full) + 128);
  float* stage = ring;
  if (lead) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int r = half ? r1 : r0;
      if (r >= R) continue;
      float* dst = stage + static_cast<size_t>(r % Ceff) * blk_floats + (r / Ceff) * kAttnRecvRow;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        *reinterpret_cast<float2*>(dst + 8 * j + 2 * tq) =
            make_float2(o[j][half * 2 + 0], o[j][half * 2 + 1]);
      if (tq == 0) {
        dst[64] = half ? m1 : m0;
        dst[65] = half ? l1 : l0;
      }
    }
  }
  fence_proxy_async_smem();
  __syncthreads();
  cluster_wait();   // every CTA of the cluster runs: peers' buffers and barriers exist
  if (threadIdx.x == 0) {
    const uint32_t bytes = static_cast<uint32_t>(blk_floats * 4);
    const uint32_t dst_local = smem_u32(recv) + static_cast<uint32_t>(c) * bytes;
    for (int q = 0; q < Ceff; ++q)
      bulk_copy_to_peer(cluster_map(dst_local, static_cast<uint32_t>(q)),
                        smem_u32(stage) + static_cast<uint32_t>(q) * bytes, bytes,
                        cluster_map(smem_u32(recv_bar), static_cast<uint32_t>(q)));
    bulk_commit();
  }
  const bool got = mbar_wait(smem_u32(recv_bar), 0, a.err);

  // ---- 3. owner merge of rows r = c + k * C over the splits in order:
  //         per row the weights w_s = exp2(m_s - M) / L (one thread per row),
  //         then one thread per (row, 4 dims) sums w_s O_s.  With one split
  //         holding all of a row's keys this is O * (1 / l), the direct path.
  const int my_rows = (R - c + Ceff - 1) / Ceff;
  for (int k = threadIdx.x; k < my_rows; k += nthreads) {
    float M = -INFINITY;
    for (int sidx = 0; sidx < Ceff; ++sidx)
      M = fmaxf(M, recv[(sidx * rpo + k) * kAttnRecvRow + 64]);
    float L = 0.f;
    for (int sidx = 0; sidx < Ceff; ++sidx) {
      float* p = recv + (sidx * rpo + k) * kAttnRecvRow;
      const float w = (p[64] == -INFINITY) ? 0.f : exp2f(p[64] - M);
      p[66] = w;
      L += w * p[65];
    }
    const float inv = 1.0f / L;
    for (int sidx = 0; sidx < Ceff; ++sidx) {
      float* p = recv + (sidx * rpo + k) * kAttnRecvRow;
      p[66] = p[66] * inv;
    }
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < my_rows * 16; idx += nthreads) {
    const int k = idx >> 4, d4 = (idx & 15) * 4;
    const int r = c + k * Ceff;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int sidx = 0; sidx < Ceff; ++sidx) {
      const float* p = recv + (sidx * rpo + k) * kAttnRecvRow;
      const float w = p[66];
      const float4 v = *reinterpret_cast<const float4*>(p + d4);
      acc.x += w * v.x;
      acc.y += w * v.y;
      acc.z += w * v.z;
      acc.w += w * v.w;
    }
    if (all_ok && got) {
      const int t = tok0 + r / a.G;
      const int hq = h * a.G + r % a.G;
      __nv_bfloat16* dst = a.out + (static_cast<size_t>(t) * a.Hq + hq) * 64 + d4;
      *reinterpret_cast<__nv_bfloat162*>(dst) = __floats2bfloat162_rn(acc.x, acc.y);
      *reinterpret_cast<__nv_bfloat162*>(dst + 2) = __floats2bfloat162_rn(acc.z, acc.w);
    }
  }
  if (threadIdx.x == 0) bulk_wait_read_all();   // outgoing blocks have left `stage`
}

}  // namespace gs
