// attention.cuh -- hybrid-mask attention over the paged fp16 KV cache.
//
// A query block is a run of at most kAttnMaxRows / G tokens of one sequence
// (a decode window, cut into sub-blocks when K+1 tokens carry more than 128
// rows, or a slice of a prefill chunk); its rows are (token, query head of the
// GQA group), so the query heads that share a KV head read each K/V page once.
// Every query token carries its own inclusive key limit, which encodes the
// mask: draft boundary row n, draft mask rows n+K, verify row i n+1+i, prefill
// row p (paper Appendix steps Draft forward / Verify forward).
//
// Work items.  The block's pages are cut into fixed absolute ranges of SP
// pages ("items"): item i covers pages [i*SP, (i+1)*SP); one CTA reduces one
// item.  Inside an item the pages are dealt to two lanes by parity (lane l
// takes the item's pages l, l+2, ...); each lane is a warp group (one warp per
// 16 rows) with its own ring of TMA stages (K and V pages, 64 tokens x 64
// dims, 8 KB each, 128-byte swizzle).  Each warp runs S = Q K^T and O += P V
// on mma.sync m16n8k16 (fp16 in, fp32 out) with the online softmax in
// registers (exp2, the 1/sqrt(64) scale folded), its lane's pages in order.
// The two lanes' (O, m, l) then merge in shared memory, lane 0 first.
//
// Merge over items, item order 0, 1, ...: M = max m_i, w_i = exp2(m_i - M),
// coef_i = w_i / sum_j w_j l_j, O = sum coef_i O_i.  A block with one item
// writes its rows directly.  With at most 8 items the items of a (block, head)
// form one thread-block cluster: each CTA sends the rows that CTA (r mod n)
// owns to it with one bulk async copy into its shared memory, completing on
// its mbarrier, and each owner merges its rows.  With more items every item
// writes its rows to global scratch and the last one to finish (atomic ticket
// per (block, head), no spinning) merges them.  Both paths run the same
// arithmetic in the same order.
//
// Invariance.  Item boundaries are absolute page numbers fixed by SP, the
// lanes deal pages by parity, and the merges run in fixed order, so a row's
// result depends only on its query, keys, limit and SP: not on the other rows
// of its block, the window size, the batch, or the merge path.  Keys past a
// row's limit contribute exact zeros.
#pragma once
#include "ptx.cuh"

namespace gs {

constexpr int kAttnStages = 2;             // K/V pages in flight per lane
constexpr int kAttnLanes = 2;
constexpr int kAttnPageBytes = 64 * 128;  // 64 tokens x 64 fp16
constexpr int kAttnRow = 68;              // partial row: O[64], m, l, 2 pad (272 B)
constexpr int kAttnMaxRows = 128;         // rows of one query block
constexpr int kAttnMaxCluster = 8;        // items merged inside a cluster
constexpr int kAttnRingBytes = kAttnLanes * kAttnStages * 2 * kAttnPageBytes;

struct AttnArgs {
  const __half* q;            // [T, Hq, 64]
  const int32_t* lim;         // [T] inclusive key limit per query token
  __half* out;                // [T, Hq, 64]
  const int32_t* page_table;  // [slots, pt_stride]
  int pt_stride;
  const int32_t* blk_slot;    // [n_seq] page-table row per sequence, or null -> fixed_slot
  const int32_t* blk_active;  // [n_seq] nonzero = run, or null
  int fixed_slot;
  int T;                      // tokens
  int QB;                     // tokens per sequence window (prefill: per block)
  int QS, n_sub;              // tokens per query block; blocks per window
  int Hq, Hkv, G;
  long long kv_row_base;      // first KV-map row of this layer
  int rows_per_page;          // 2 * Hkv * 64
  int split_pages;            // SP: pages per item
  int max_items;              // items per (block, head) the grid covers
  int cluster;                // 1: the grid's x dimension is one cluster (max_items <= 8)
  float* part;                // global merge: [n_blocks][Hkv][max_items][rows][kAttnRow]
  int* ticket;                // global merge: [n_blocks][Hkv], zero between launches
  int* err;
};

__host__ __device__ inline int attn_mtiles(int rows) { return (rows + 15) / 16; }
__host__ __device__ inline int attn_threads(int rows) {
  return kAttnLanes * attn_mtiles(rows) * 32;
}
// receive buffer of an owner: n sources x ceil(rows / n) rows, at most rows + 8
__host__ __device__ inline int attn_recv_floats(int rows) {
  return (attn_mtiles(rows) * 16 + kAttnMaxCluster) * kAttnRow;
}
__host__ __device__ inline int attn_smem_bytes(int rows) {
  return 1024 + attn_mtiles(rows) * 16 * 128 + kAttnRingBytes + attn_recv_floats(rows) * 4 + 128;
}
__host__ __device__ inline int attn_max_smem_bytes() { return attn_smem_bytes(kAttnMaxRows); }
// The merge keeps m and l of every (item, row) in the idle ring.
__host__ __device__ inline int attn_max_merge_items(int rows) {
  return kAttnRingBytes / 4 / (2 * attn_mtiles(rows) * 16);
}
static_assert(kAttnRingBytes >= kAttnMaxRows * kAttnRow * 4 &&
                  kAttnRingBytes >= (kAttnMaxRows + kAttnMaxCluster) * kAttnRow * 4,
              "the idle ring holds a lane's partial rows and the owner-grouped rows");

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

// Barrier over the warps of one lane (ids 1, 2; 0 is __syncthreads).
__device__ __forceinline__ void lane_sync(int lane_id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(lane_id + 1), "r"(nthreads) : "memory");
}

__global__ void __launch_bounds__(512)
    attn_paged_kernel(const __grid_constant__ CUtensorMap tmKV, const AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mtiles = attn_mtiles(a.QS * a.G);
  const int ln = warp / mtiles, mt = warp % mtiles;   // page lane, row tile
  const int lthreads = mtiles * 32;
  const int ltid = threadIdx.x - ln * lthreads;
  const int rows_alloc = mtiles * 16;
  uint8_t* sQ = smem;                                   // [rows][128 B]
  uint8_t* ring = smem + rows_alloc * 128;              // [lane][stage][K | V]
  uint8_t* sK = ring + ln * kAttnStages * 2 * kAttnPageBytes;
  uint8_t* sV = sK + kAttnStages * kAttnPageBytes;
  float* recv = reinterpret_cast<float*>(ring + kAttnRingBytes);   // [source][slot][kAttnRow]
  uint64_t* full = reinterpret_cast<uint64_t*>(recv + attn_recv_floats(rows_alloc));
  uint64_t* lfull = full + ln * kAttnStages;
  uint64_t* recv_bar = full + kAttnLanes * kAttnStages;
  int* s_int = reinterpret_cast<int*>(recv_bar + 1);    // [0] max limit, [1] last-item flag

  const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int seq = b / a.n_sub, sub = b % a.n_sub;
  // Before griddepcontrol.wait this kernel reads only what the kernel right
  // before it (the QKV GEMM, which writes q and the window's K/V) does not
  // write: the window descriptors (key limits, block slots), the page table,
  // and cache pages wholly before the current window.  Every early exit is
  // uniform across the CTA, and across the cluster before its barrier.
  if (a.blk_active != nullptr && a.blk_active[seq] == 0) return;
  const int tok0 = seq * a.QB + sub * a.QS;
  const int ntok = min(min(a.QS, a.QB - sub * a.QS), a.T - tok0);
  if (ntok <= 0) return;
  const int R = ntok * a.G;
  const int slot = a.blk_slot ? a.blk_slot[seq] : a.fixed_slot;

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
  if (maxlim < 0 || npages_blk > a.pt_stride || slot < 0 || nitems > a.max_items) {
    if (threadIdx.x == 0) atomicExch(a.err, kErrBounds);
    return;
  }
  if (c >= nitems && (nitems == 1 || !a.cluster)) return;
  const bool in_cluster = a.cluster && nitems > 1;

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmKV);
    for (int s = 0; s < kAttnLanes * kAttnStages; ++s) mbar_init(smem_u32(&full[s]), 1);
    if (in_cluster) {
      mbar_init(smem_u32(recv_bar), 1);
      // nitems sources, ceil(rows / nitems) rows each, arrive by bulk copy
      const int rpo = (rows_alloc + nitems - 1) / nitems;
      mbar_arrive_expect_tx(smem_u32(recv_bar), static_cast<uint32_t>(nitems * rpo * kAttnRow * 4));
    }
    fence_mbar_init();
  }
  __syncthreads();
  if (in_cluster) cluster_arrive_release();   // waited on before the first remote access
  if (c >= nitems) return;                     // idle cluster member: arrived, owns nothing

  const int p_begin = c * SP;
  const int np = min(npages_blk, p_begin + SP) - p_begin;
  const int npl = np > ln ? (np - ln + 1) / kAttnLanes : 0;   // this lane's pages
  const int32_t* pt = a.page_table + static_cast<size_t>(slot) * a.pt_stride;
  const bool producer = ltid == 0;
  // pages wholly before the block's first slot hold committed states only
  const int safe_pages = a.blk_slot ? a.lim[tok0] / 64 : 0;
  const uint64_t pol = l2_policy_evict_first();
  auto page_of = [&](int i) { return p_begin + ln + kAttnLanes * i; };
  auto issue = [&](int i) {
    const int s = i % kAttnStages;
    int phys = pt[page_of(i)];
    if (phys < 0) {  // unmapped page: the TMA box lands out of bounds and reads zeros
      atomicExch(a.err, kErrBounds);
      phys = 0x3FFFFFFF / a.rows_per_page;
    }
    const long long row = a.kv_row_base + static_cast<long long>(phys) * a.rows_per_page;
    const uint32_t fb = smem_u32(&lfull[s]);
    mbar_arrive_expect_tx(fb, 2 * kAttnPageBytes);
    tma_load_2d(smem_u32(sK + s * kAttnPageBytes), &tmKV, 0, static_cast<int>(row + h * 64), fb, pol);
    tma_load_2d(smem_u32(sV + s * kAttnPageBytes), &tmKV, 0,
                static_cast<int>(row + (a.Hkv + h) * 64), fb, pol);
  };
  int issued = 0;
  if (producer) {
    while (issued < min(npl, kAttnStages) && page_of(issued) < safe_pages) issue(issued++);
  }
  pdl_wait();
  pdl_trigger();
  if (producer) {
    while (issued < min(npl, kAttnStages)) issue(issued++);
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

  for (int i = 0; i < npl; ++i) {
    const int s = i % kAttnStages;
    if (ok && !mbar_wait(smem_u32(&lfull[s]), (i / kAttnStages) & 1, a.err)) ok = false;
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
      const int kbase_abs = page_of(i) * 64;
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
    lane_sync(ln, lthreads);   // every warp of the lane is done with stage s
    if (producer && ok && i + kAttnStages < npl) issue(i + kAttnStages);
  }
  const bool all_ok = __syncthreads_and(ok);   // both lanes done: the ring is idle

  // row sums across the quad
  l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, 1);
  l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, 2);
  l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, 1);
  l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, 2);

  // ---- lane 1 -> lane 0 (shared memory): M = max, w = exp2(m - M) per lane,
  //      O = w0 O0 + w1 O1, l = w0 l0 + w1 l1.  lp [row][kAttnRow] in the ring.
  float* lp = reinterpret_cast<float*>(ring);
  if (ln == 1 && has_rows) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      float* dst = lp + (half ? r1 : r0) * kAttnRow;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        *reinterpret_cast<float2*>(dst + 8 * j + 2 * tq) =
            make_float2(o[j][half * 2 + 0], o[j][half * 2 + 1]);
      if (tq == 0) *reinterpret_cast<float2*>(dst + 64) = half ? make_float2(m1, l1) : make_float2(m0, l0);
    }
  }
  __syncthreads();
  if (ln == 0 && has_rows) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const float* src = lp + (half ? r1 : r0) * kAttnRow;
      const float2 ml = *reinterpret_cast<const float2*>(src + 64);
      const float ma = half ? m1 : m0;
      const float M = fmaxf(ma, ml.x);
      const float wa = (ma == -INFINITY) ? 0.f : exp2f(ma - M);
      const float wb = (ml.x == -INFINITY) ? 0.f : exp2f(ml.x - M);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float2 v = *reinterpret_cast<const float2*>(src + 8 * j + 2 * tq);
        o[j][half * 2 + 0] = wa * o[j][half * 2 + 0] + wb * v.x;
        o[j][half * 2 + 1] = wa * o[j][half * 2 + 1] + wb * v.y;
      }
      if (half) { l1 = wa * l1 + wb * ml.y; m1 = M; } else { l0 = wa * l0 + wb * ml.y; m0 = M; }
    }
  }
  __syncthreads();   // lp consumed; the ring is reused below
  const bool lead = ln == 0 && has_rows;

  if (nitems == 1) {   // the block's only item: its rows are final
    if (lead && all_ok) {
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

  // Merged rows of one item: source `it`, row r -> float pointer (O[64], m, l).
  // Cluster: recv[it][k] with r = c + k * nitems.  Global: part[b][h][it][r].
  const size_t bh = static_cast<size_t>(b) * a.Hkv + h;
  float* part_bh = a.part + bh * a.max_items * rows_alloc * kAttnRow;
  const int rpo = (rows_alloc + nitems - 1) / nitems;   // cluster: rows per owner
  bool got = true;
  int my_rows;
  if (in_cluster) {
    // ---- items -> owners.  stage [owner][slot][kAttnRow] in the ring.
    float* stage = reinterpret_cast<float*>(ring);
    const int blk_floats = rpo * kAttnRow;
    if (lead) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int r = half ? r1 : r0;
        if (r >= R) continue;
        float* dst = stage + static_cast<size_t>(r % nitems) * blk_floats + (r / nitems) * kAttnRow;
#pragma unroll
        for (int j = 0; j < 8; ++j)
          *reinterpret_cast<float2*>(dst + 8 * j + 2 * tq) =
              make_float2(o[j][half * 2 + 0], o[j][half * 2 + 1]);
        if (tq == 0)
          *reinterpret_cast<float2*>(dst + 64) = half ? make_float2(m1, l1) : make_float2(m0, l0);
      }
    }
    fence_proxy_async_smem();
    __syncthreads();
    cluster_wait();   // every CTA of the cluster runs: peers' buffers and barriers exist
    if (threadIdx.x == 0) {
      const uint32_t bytes = static_cast<uint32_t>(blk_floats * 4);
      const uint32_t dst_local = smem_u32(recv) + static_cast<uint32_t>(c) * bytes;
      for (int q = 0; q < nitems; ++q)
        bulk_copy_to_peer(cluster_map(dst_local, static_cast<uint32_t>(q)),
                          smem_u32(stage) + static_cast<uint32_t>(q) * bytes, bytes,
                          cluster_map(smem_u32(recv_bar), static_cast<uint32_t>(q)));
      bulk_commit();
    }
    got = mbar_wait(smem_u32(recv_bar), 0, a.err);
    my_rows = (R - c + nitems - 1) / nitems;
  } else {
    // ---- item rows -> global scratch; the last item to arrive merges
    if (lead) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int r = half ? r1 : r0;
        if (r >= R) continue;
        float* dst = part_bh + (static_cast<size_t>(c) * rows_alloc + r) * kAttnRow;
#pragma unroll
        for (int j = 0; j < 8; ++j)
          *reinterpret_cast<float2*>(dst + 8 * j + 2 * tq) =
              make_float2(o[j][half * 2 + 0], o[j][half * 2 + 1]);
        if (tq == 0)
          *reinterpret_cast<float2*>(dst + 64) = half ? make_float2(m1, l1) : make_float2(m0, l0);
      }
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_int[1] = (atomicAdd(a.ticket + bh, 1) == nitems - 1) ? 1 : 0;
    __syncthreads();
    if (!s_int[1]) return;
    __threadfence();
    if (threadIdx.x == 0) a.ticket[bh] = 0;   // every item of this launch has arrived
    my_rows = R;
  }
  auto row_of = [&](int k) { return in_cluster ? c + k * nitems : k; };
  // source rows: the owner's receive buffer (shared) or the global scratch
  // (written by other SMs in this launch: read at L2, never from L1)
  auto src_of = [&](int it, int k) -> const float* {
    return in_cluster ? recv + (static_cast<size_t>(it) * rpo + k) * kAttnRow
                      : part_bh + (static_cast<size_t>(it) * rows_alloc + k) * kAttnRow;
  };
  auto ld2 = [&](const float* p) {
    return in_cluster ? *reinterpret_cast<const float2*>(p) : __ldcg(reinterpret_cast<const float2*>(p));
  };
  auto ld4 = [&](const float* p) {
    return in_cluster ? *reinterpret_cast<const float4*>(p) : __ldcg(reinterpret_cast<const float4*>(p));
  };

  // ---- merge of items 0..nitems-1 in order for rows row_of(k), k < my_rows.
  //      mb/lb [item][k] hold m and l, then mb the coefficients w_it / L (one
  //      thread per row); then one thread per (row, 4 dims) sums coef * O_it.
  //      Both live in the idle ring (in a cluster once this CTA's outgoing
  //      copies have read it).
  if (in_cluster && threadIdx.x == 0) bulk_wait_read_all();
  __syncthreads();
  float* mb = reinterpret_cast<float*>(ring);
  float* lb = mb + static_cast<size_t>(nitems) * rows_alloc;
  const bool fits = 2 * nitems * rows_alloc <= kAttnRingBytes / 4;
  if (!fits && threadIdx.x == 0) atomicExch(a.err, kErrBounds);
  if (fits) {
    for (int idx = threadIdx.x; idx < nitems * my_rows; idx += blockDim.x) {
      const int it = idx / my_rows, k = idx - it * my_rows;
      const float2 ml = ld2(src_of(it, k) + 64);
      mb[it * rows_alloc + k] = ml.x;
      lb[it * rows_alloc + k] = ml.y;
    }
  }
  __syncthreads();
  if (fits) {
    for (int k = threadIdx.x; k < my_rows; k += blockDim.x) {
      float M = -INFINITY;
      for (int it = 0; it < nitems; ++it) M = fmaxf(M, mb[it * rows_alloc + k]);
      float L = 0.f;
      for (int it = 0; it < nitems; ++it) {
        const float mi = mb[it * rows_alloc + k];
        const float w = (mi == -INFINITY) ? 0.f : exp2f(mi - M);
        mb[it * rows_alloc + k] = w;
        L += w * lb[it * rows_alloc + k];
      }
      const float inv = 1.0f / L;
      for (int it = 0; it < nitems; ++it) mb[it * rows_alloc + k] *= inv;
    }
  }
  __syncthreads();
  if (fits) {
    for (int idx = threadIdx.x; idx < my_rows * 16; idx += blockDim.x) {
      const int k = idx >> 4, d4 = (idx & 15) * 4;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int it0 = 0; it0 < nitems; it0 += 8) {   // 8 loads in flight, summed in order
        const int n8 = min(8, nitems - it0);
        float4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (u < n8) v[u] = ld4(src_of(it0 + u, k) + d4);
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (u < n8) {
            const float w = mb[(it0 + u) * rows_alloc + k];
            acc.x += w * v[u].x;
            acc.y += w * v[u].y;
            acc.z += w * v[u].z;
            acc.w += w * v[u].w;
          }
      }
      if (all_ok && got) {
        const int r = row_of(k);
        const int t = tok0 + r / a.G;
        const int hq = h * a.G + r % a.G;
        __half* dst = a.out + (static_cast<size_t>(t) * a.Hq + hq) * 64 + d4;
        *reinterpret_cast<__half2*>(dst) = __floats2half2_rn(acc.x, acc.y);
        *reinterpret_cast<__half2*>(dst + 2) = __floats2half2_rn(acc.z, acc.w);
      }
    }
  }
}

}  // namespace gs
