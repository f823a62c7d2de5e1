// attention.cuh -- hybrid-mask attention over the paged fp16 KV cache.
//
// A query block is a run of tokens of one sequence (the K+1 window of a decode
// forward, or 64 tokens of a prefill chunk); its rows are (token, query head
// of the GQA group), so the query heads that share a KV head read each K/V
// page once.  Every query token carries its own inclusive key limit, which
// encodes the mask: draft boundary row n, draft mask rows n+K, verify row i
// n+1+i, prefill row p (paper Appendix steps Draft forward / Verify forward).
//
// Work items.  The block's pages are cut into fixed absolute ranges of SP
// pages ("items"): item i covers pages [i*SP, (i+1)*SP).  One warp group (one
// warp per 16 rows) reduces one item: it streams the item's K and V pages
// (64 tokens x 64 dims, 8 KB each) through its own ring of TMA stages with
// 128-byte swizzle, and each warp runs S = Q K^T and O += P V on mma.sync
// m16n8k16 (fp16 in, fp32 out) with the online softmax in registers (exp2,
// the 1/sqrt(64) scale folded), pages in order.  A CTA = (item group, KV
// head, query block) holds NG warp groups on consecutive items and shares the
// block's Q tile among them.
//
// Merge.  A block with one item writes its rows directly.  Otherwise each item
// writes its rows' (O, m, l) to global scratch, and the last item to finish
// (atomic ticket per (block, head), no spinning) merges the items in order
// 0, 1, ...: M = max m_i, w_i = exp2(m_i - M), O = sum w_i O_i / sum w_i l_i.
//
// Invariance.  Item boundaries are absolute page numbers fixed by SP, each
// item is reduced page by page in one warp, and the merge runs in item order,
// so a row's result depends only on its own query, keys and limit: not on the
// other rows of its window, the window size, the batch, or how many groups a
// CTA holds.  Keys past a row's limit contribute exact zeros.
#pragma once
#include "ptx.cuh"

namespace gs {

constexpr int kAttnStages = 3;             // K/V pages in flight per warp group
constexpr int kAttnPageBytes = 64 * 128;  // 64 tokens x 64 fp16
constexpr int kAttnRow = 68;              // partial row: O[64], m, l, 2 pad (272 B)
constexpr int kAttnMaxGroups = 4;

struct AttnArgs {
  const __half* q;            // [T, Hq, 64]
  const int32_t* lim;         // [T] inclusive key limit per query token
  __half* out;                // [T, Hq, 64]
  const int32_t* page_table;  // [slots, pt_stride]
  int pt_stride;
  const int32_t* blk_slot;    // [n_blocks] page-table row per block, or null -> fixed_slot
  const int32_t* blk_active;  // [n_blocks] nonzero = run, or null
  int fixed_slot;
  int T, QB;                  // tokens; tokens per query block
  int Hq, Hkv, G;
  long long kv_row_base;      // first KV-map row of this layer
  int rows_per_page;          // 2 * Hkv * 64
  int split_pages;            // SP: pages per item
  int max_items;              // item slots per (block, head) in `part`
  int r_pad;                  // row slots per item in `part` (>= rows of a block)
  float* part;                // [n_blocks][Hkv][max_items][r_pad][kAttnRow]
  int* ticket;                // [n_blocks][Hkv], zero between launches
  int* err;
};

// Rows (16 per warp) and launch shape for a block of r_max rows and ng groups.
__host__ __device__ inline int attn_mtiles(int r_max) { return (r_max + 15) / 16; }
__host__ __device__ inline int attn_threads(int r_max, int ng) { return attn_mtiles(r_max) * ng * 32; }
__host__ __device__ inline int attn_smem_bytes(int r_max, int ng) {
  return 1024 + attn_mtiles(r_max) * 16 * 128 + ng * kAttnStages * 2 * kAttnPageBytes +
         ng * kAttnStages * 8 + 64;
}
// Warp groups per CTA: two when the launch has several waves of single-group
// CTAs and two groups fit in 512 threads, else one.  Does not change results.
__host__ __device__ inline int attn_groups_for(int r_max, int ctas_one_group) {
  return (ctas_one_group >= 4 * 152 && attn_threads(r_max, 2) <= 512) ? 2 : 1;
}
// Largest dynamic shared memory any launch asks for (rows <= 256).
__host__ __device__ inline int attn_max_smem_bytes() {
  const int a = attn_smem_bytes(256, 1), b = attn_smem_bytes(128, 2);
  return a > b ? a : b;
}
// The merge keeps one coefficient per (item, row) in the merging group's ring.
__host__ __device__ inline int attn_max_merge_items(int r_max) {
  return kAttnStages * 2 * kAttnPageBytes / 4 / (attn_mtiles(r_max) * 16);
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

__device__ __forceinline__ void mma_f16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                              uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Barrier over the warps of one group (ids 1..kAttnMaxGroups; 0 is __syncthreads).
__device__ __forceinline__ void group_sync(int grp, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(grp + 1), "r"(nthreads) : "memory");
}

__global__ void __launch_bounds__(512)
    attn_paged_kernel(const __grid_constant__ CUtensorMap tmKV, const AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mtiles = attn_mtiles(a.QB * a.G);
  const int NG = blockDim.x / 32 / mtiles;    // warp groups of this CTA
  const int grp = warp / mtiles, mt = warp % mtiles;
  const int gthreads = mtiles * 32;
  const int gtid = threadIdx.x - grp * gthreads;
  const int rows_alloc = mtiles * 16;
  uint8_t* sQ = smem;                                              // [rows][128 B]
  uint8_t* ring = smem + rows_alloc * 128;                         // [NG][stages][K | V]
  uint8_t* sK = ring + grp * kAttnStages * 2 * kAttnPageBytes;     // this group's stages
  uint8_t* sV = sK + kAttnStages * kAttnPageBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + NG * kAttnStages * 2 * kAttnPageBytes);
  uint64_t* gfull = full + grp * kAttnStages;
  int* s_int = reinterpret_cast<int*>(full + NG * kAttnStages);   // [0] max limit, [1+g] last flag

  const int h = blockIdx.y, b = blockIdx.z;
  // Before griddepcontrol.wait this kernel reads only what the kernel right
  // before it (the QKV GEMM, which writes q and the window's K/V) does not
  // write: the window descriptors (key limits, block slots), the page table,
  // and cache pages wholly before the current window.  Every early exit is
  // uniform across the CTA.
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
    if (lane == 0) s_int[0] = m;
  }
  __syncthreads();
  const int maxlim = s_int[0];
  const int npages_blk = maxlim / 64 + 1;
  const int SP = a.split_pages;
  const int nitems = (npages_blk + SP - 1) / SP;
  if (maxlim < 0 || npages_blk > a.pt_stride || slot < 0 || nitems > a.max_items ||
      R > a.r_pad) {
    if (threadIdx.x == 0) atomicExch(a.err, kErrBounds);
    return;
  }
  const int item0 = blockIdx.x * NG;
  if (item0 >= nitems) return;
  const int item = item0 + grp;
  const bool has_item = item < nitems;
  const int p_begin = item * SP;
  const int np = has_item ? min(npages_blk, p_begin + SP) - p_begin : 0;
  const int32_t* pt = a.page_table + static_cast<size_t>(slot) * a.pt_stride;

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmKV);
    for (int s = 0; s < NG * kAttnStages; ++s) mbar_init(smem_u32(&full[s]), 1);
    fence_mbar_init();
  }
  __syncthreads();
  const bool producer = gtid == 0;
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
    const uint32_t fb = smem_u32(&gfull[s]);
    mbar_arrive_expect_tx(fb, 2 * kAttnPageBytes);
    tma_load_2d(smem_u32(sK + s * kAttnPageBytes), &tmKV, 0, static_cast<int>(row + h * 64), fb, pol);
    tma_load_2d(smem_u32(sV + s * kAttnPageBytes), &tmKV, 0,
                static_cast<int>(row + (a.Hkv + h) * 64), fb, pol);
  };
  int issued = 0;
  if (producer) {
    while (issued < min(np, kAttnStages) && p_begin + issued < safe_pages) issue(issued++);
  }
  pdl_wait();
  pdl_trigger();
  if (producer) {
    while (issued < min(np, kAttnStages)) issue(issued++);
  }

  // Q rows -> swizzled smem (zero rows past R)
  for (int idx = threadIdx.x; idx < rows_alloc * 8; idx += blockDim.x) {
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
  if (!has_item) return;

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

  for (int i = 0; i < np; ++i) {
    const int s = i % kAttnStages;
    if (ok && !mbar_wait(smem_u32(&gfull[s]), (i / kAttnStages) & 1, a.err)) ok = false;
    if (ok && has_rows) {
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
          mma_f16_16816(sacc[j], qa[kk], b0, b1);
          mma_f16_16816(sacc[j], qa[kk + 1], b2, b3);
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
        pa[j >> 1][(j & 1) * 2 + 0] = pack_f16x2(p0, p1);
        pa[j >> 1][(j & 1) * 2 + 1] = pack_f16x2(p2, p3);
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
          mma_f16_16816(o[jn], pa[kk], b0, b1);
          mma_f16_16816(o[jn + 1], pa[kk], b2, b3);
        }
      }
    }
    group_sync(grp, gthreads);   // every warp of the group is done with stage s
    if (producer && ok && i + kAttnStages < np) issue(i + kAttnStages);
  }

  // row sums across the quad
  l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, 1);
  l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, 2);
  l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, 1);
  l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, 2);

  if (nitems == 1) {   // the block's only item: its rows are final
    if (has_rows && ok) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int r = half ? r1 : r0;
        if (r >= R) continue;
        const float inv = 1.0f / (half ? l1 : l0);
        const int t = tok0 + r / a.G;
        const int hq = h * a.G + r % a.G;
        __half* dst = a.out + (static_cast<size_t>(t) * a.Hq + hq) * 64;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float x0 = o[j][half * 2 + 0] * inv, x1 = o[j][half * 2 + 1] * inv;
          *reinterpret_cast<__half2*>(dst + 8 * j + 2 * tq) = __floats2half2_rn(x0, x1);
        }
      }
    }
    return;
  }

  // ---- partial rows of this item -> global scratch
  const size_t bh = static_cast<size_t>(b) * a.Hkv + h;
  float* part_bh = a.part + bh * a.max_items * a.r_pad * kAttnRow;
  if (has_rows) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int r = half ? r1 : r0;
      if (r >= R) continue;
      float* dst = part_bh + (static_cast<size_t>(item) * a.r_pad + r) * kAttnRow;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        *reinterpret_cast<float2*>(dst + 8 * j + 2 * tq) =
            make_float2(o[j][half * 2 + 0], o[j][half * 2 + 1]);
      if (tq == 0)
        *reinterpret_cast<float2*>(dst + 64) = half ? make_float2(m1, l1) : make_float2(m0, l0);
    }
  }
  __threadfence();
  group_sync(grp, gthreads);
  if (producer) s_int[1 + grp] = (atomicAdd(a.ticket + bh, 1) == nitems - 1) ? 1 : 0;
  group_sync(grp, gthreads);
  if (!s_int[1 + grp]) return;

  // ---- last item of (block, head): merge items 0..nitems-1 in order.
  //      coef[i][r] = w_i / L (one thread per row), then one thread per
  //      (row, 4 dims) sums coef * O_i.
  __threadfence();
  float* coef = reinterpret_cast<float*>(sK);   // [nitems][rows_alloc], the group's idle ring
  const bool fits = nitems <= attn_max_merge_items(a.QB * a.G);
  if (!fits && gtid == 0) atomicExch(a.err, kErrBounds);
  if (fits) {
    for (int r = gtid; r < R; r += gthreads) {
      float M = -INFINITY;
      for (int it = 0; it < nitems; ++it)
        M = fmaxf(M, __ldcg(part_bh + (static_cast<size_t>(it) * a.r_pad + r) * kAttnRow + 64));
      float L = 0.f;
      for (int it = 0; it < nitems; ++it) {
        const float2 ml = __ldcg(reinterpret_cast<const float2*>(
            part_bh + (static_cast<size_t>(it) * a.r_pad + r) * kAttnRow + 64));
        const float w = (ml.x == -INFINITY) ? 0.f : exp2f(ml.x - M);
        coef[it * rows_alloc + r] = w;
        L += w * ml.y;
      }
      const float inv = 1.0f / L;
      for (int it = 0; it < nitems; ++it) coef[it * rows_alloc + r] *= inv;
    }
  }
  group_sync(grp, gthreads);
  if (fits) {
    for (int idx = gtid; idx < R * 16; idx += gthreads) {
      const int r = idx >> 4, d4 = (idx & 15) * 4;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int it = 0; it < nitems; ++it) {
        const float w = coef[it * rows_alloc + r];
        const float4 v = __ldcg(reinterpret_cast<const float4*>(
            part_bh + (static_cast<size_t>(it) * a.r_pad + r) * kAttnRow + d4));
        acc.x += w * v.x;
        acc.y += w * v.y;
        acc.z += w * v.z;
        acc.w += w * v.w;
      }
      const int t = tok0 + r / a.G;
      const int hq = h * a.G + r % a.G;
      __half* dst = a.out + (static_cast<size_t>(t) * a.Hq + hq) * 64 + d4;
      *reinterpret_cast<__half2*>(dst) = __floats2half2_rn(acc.x, acc.y);
      *reinterpret_cast<__half2*>(dst + 2) = __floats2half2_rn(acc.z, acc.w);
    }
  }
  if (gtid == 0) a.ticket[bh] = 0;   // every item of this launch has arrived
}

}  // namespace gs
