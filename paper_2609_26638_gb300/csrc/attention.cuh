// attention.cuh -- hybrid-mask attention over the paged fp16 KV cache, on
// the tcgen05 tensor cores.
//
// A query block is a run of at most 128 / G tokens of one sequence (a decode
// window, cut into sub-blocks when K+1 tokens carry more than 128 rows, or a
// slice of a prefill chunk); its rows are (token, query head of the GQA
// group), so the query heads that share a KV head read each K/V page once.
// Every query token carries its own inclusive key limit, which encodes the
// mask: draft boundary row n, draft mask rows n+K, verify row i n+1+i, prefill
// row p (paper Appendix steps Draft forward / Verify forward).
//
// Work items.  The block's pages are cut into fixed absolute ranges of SP
// pages ("items"): item i covers pages [i*SP, (i+1)*SP); one CTA reduces one
// item, pages in order.  A page holds K as [64 tokens][64 dims] and V
// transposed, [64 dims][64 tokens] (8 KB each), so both are K-major operands.
// Per page j:
//   S_j = Q K_j^T       tcgen05.mma M=128 (rows) N=64 (keys) K=64 into TMEM
//   softmax             per row: running max m (log2 units), P_j =
//                       exp2(s*scale - m) as fp16 into shared memory (the A
//                       operand of the next MMA)
//   O += P_j [V_j | 1]  tcgen05.mma M=128 N=80 K=64 (keys), O in TMEM: 64 dims
//                       and, from 16 rows of ones kept after every V^T page,
//                       the row sum l in O's column 64 (fp32 on the tensor core)
// The max only moves when a page raises it by more than 2^8: then the thread
// first rescales its O row in TMEM (and l with it) by exp2(m_old - m_new).  Smaller
// rises keep the old m, so P stays <= 2^8 (well inside fp16).  Either way
// O / l is the softmax-weighted sum.  Warps 0-3 own rows 0-127 (TMEM lanes;
// warps whose rows are all padding only keep the barriers' pace); warp 4
// streams K/V pages by TMA (128-byte swizzle) through a ring of stages; warp
// 5 issues the MMAs, S one page ahead of the softmax, S double-buffered.
//
// Merge over items, item order 0, 1, ...: M = max m_i, w_i = exp2(m_i - M),
// coef_i = w_i / sum_j w_j l_j, O = sum coef_i O_i.  A block with one item
// writes its rows directly.  A (block, head) with at most 16 items may form one
// thread-block cluster: once every CTA of the cluster has finished its pages,
// each sends the rows that CTA (r mod n) owns to it with one bulk async copy
// into its shared memory, completing on its mbarrier, and each owner merges
// its rows.  Otherwise every item writes its rows to global scratch and the
// last one to finish (atomic ticket per (block, head), no spinning) merges
// them.  Both paths run the same arithmetic in the same order.
//
// Invariance.  Item boundaries are absolute page numbers fixed by SP, pages
// are reduced in order, the MMA's arithmetic for a row does not depend on the
// other rows, and the merges run in fixed order, so a row's result depends
// only on its query, keys, limit and SP: not on the other rows of its block,
// the window size, the batch, or the merge path.  Keys past a row's limit
// contribute exact zeros.
#pragma once
#include "ptx.cuh"

namespace gs {

constexpr int kAttnStages = 3;             // K/V page pairs in flight
constexpr int kAttnPageBytes = 64 * 128;  // 64 x 64 fp16
constexpr int kAttnOnesBytes = 16 * 128;  // 16 rows of fp16 ones after each V^T page
constexpr int kAttnStageBytes = 2 * kAttnPageBytes + kAttnOnesBytes;
constexpr int kAttnRow = 68;              // partial row: O[64], m, l, 2 pad (272 B)
constexpr int kAttnMaxRows = 128;         // rows of one query block (the MMA's M)
constexpr int kAttnMaxCluster = 16;       // items merged inside a cluster (16: non-portable size)
constexpr int kAttnSoftWarps = 4;         // one warp per TMEM lane quarter
constexpr int kAttnSoftThreads = kAttnSoftWarps * 32;
constexpr int kAttnThreads = kAttnSoftThreads + 64;   // + TMA warp, MMA warp
constexpr int kAttnTmaWarp = kAttnSoftWarps, kAttnMmaWarp = kAttnSoftWarps + 1;
constexpr int kAttnTmemCols = 256;        // S[2] at columns 0, 64; O at 128
constexpr float kAttnRescale = 8.0f;      // log2 growth of the max that forces a rescale
constexpr int kAttnRingBytes = kAttnStages * kAttnStageBytes;
// Q [128][128 B] | P[2] [128][128 B] | ring | barriers.  After the pages are
// done, Q and P hold the owner-grouped rows (cluster) and the ring the
// received rows or the merge's (m, l) tables.
constexpr int kAttnQOff = 0;
constexpr int kAttnPOff = kAttnMaxRows * 128;
constexpr int kAttnRingOff = kAttnPOff + 2 * kAttnMaxRows * 128;
constexpr int kAttnBarOff = kAttnRingOff + kAttnRingBytes;
constexpr int kAttnSmemBytes = 1024 + kAttnBarOff + 256 + 2 * kAttnSoftThreads * 4;
constexpr int kAttnRowsFloats = (kAttnMaxRows + kAttnMaxCluster) * kAttnRow;
static_assert(kAttnRingOff >= kAttnRowsFloats * 4 && kAttnRingBytes >= kAttnRowsFloats * 4,
              "Q + P hold the owner-grouped rows, the ring the received rows");

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
  int cluster;                // 1: the grid's x dimension is one cluster (max_items <= 16)
  float* part;                // global merge: [n_blocks][Hkv][max_items][128][kAttnRow]
  int* ticket;                // global merge: [n_blocks][Hkv], zero between launches
  int* err;
};

__host__ __device__ inline int attn_max_smem_bytes() { return kAttnSmemBytes; }
// The merge keeps m and l of every (item, row) in the idle ring.
__host__ __device__ inline int attn_max_merge_items(int /*rows*/) {
  return kAttnRingBytes / 4 / (2 * kAttnMaxRows);
}

__device__ __forceinline__ uint32_t sw128(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

__device__ __forceinline__ void tmem_ld16_nowait(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ uint32_t tmem_ld1(uint32_t taddr) {
  uint32_t r;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(r) : "r"(taddr));
  return r;
}

__device__ __forceinline__ void tmem_st1(uint32_t taddr, uint32_t v) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};" ::"r"(taddr), "r"(v) : "memory");
}

// 2^x on the SFU (PTX ex2.approx.ftz.f32, one instruction): the P values are
// 2^(s - m) <= 2^8, and a result below the fp32 normal range is an fp16 zero.
__device__ __forceinline__ float ex2_sfu(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// max of three (PTX max.f32 with three sources, sm_100 and later)
__device__ __forceinline__ float fmax3(float x, float y, float z) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(x), "f"(y), "f"(z));
  return r;
}

// Barriers and buffers the softmax warps share with the MMA warp.
struct AttnSync {
  uint64_t *s_full, *s_free, *p_full;
  uint64_t* empty;   // [stages] O += P V of the stage's page retired
  uint8_t* sP;       // [2][128][128 B]
  float* red;        // [128] per-thread page maxima (exchanged only when a max rises)
};

// Named barriers of the softmax warps (barrier 0 is __syncthreads).
constexpr int kAttnBarVote = 1, kAttnBarMax = 2;

// OR of a predicate over the softmax threads: one hardware barrier.
__device__ __forceinline__ bool softmax_vote_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.or.pred p, %2, %3, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "n"(kAttnBarVote), "n"(kAttnSoftThreads)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ void softmax_bar_max() {
  asm volatile("bar.sync %0, %1;" ::"n"(kAttnBarMax), "n"(kAttnSoftThreads) : "memory");
}

// Online softmax over the item's pages, one thread per TMEM lane.  DUP copies
// of each block row sit in the MMA's 128 rows (copy k of row rr at MMA row
// k * 128 / DUP + rr, so every lane quarter -- and every SM sub-partition --
// holds rows); the thread of copy k takes the NC = 64 / DUP columns
// [k NC, (k + 1) NC) of every page.  Per page: S from TMEM, mask and scale,
// this thread's maximum; the row's running max m (log2 units) only moves when
// a page raises it by more than 2^8, so one vote over the softmax threads (a
// hardware barrier) decides whether any row of the block rises, and only then
// are the copies' page maxima exchanged through shared memory (always on the
// first page, rarely after).  A rise rescales O and the row sum in O's column
// 64 (the copy-0 thread of the row; the previous O += P V must have retired);
// then P_j = exp2(s - m) as fp16 into row rr of the P tile.  m, P and the
// rescale are the same for every DUP.  Waits are bounded; a warp whose wait ran out keeps passing the named
// barriers and arriving on the MMA warp's barriers to the last page, so no
// thread is left at a barrier.  Returns false if a wait ran out.
template <int DUP>
__device__ __forceinline__ bool attn_softmax(const AttnArgs& a, const AttnSync& y, uint32_t tmem,
                                             int np, int p_begin, int R, int tok0, float& m) {
  constexpr int RPC = kAttnMaxRows / DUP;   // MMA rows per copy
  constexpr int NC = 64 / DUP;              // columns per thread
  constexpr int NCH = NC / 8;               // 8-column chunks per thread
  const int mrow = threadIdx.x, warp = mrow >> 5, lane = mrow & 31;   // MMA row = TMEM lane
  const int cp = mrow / RPC, rr = mrow % RPC;
  const int col0 = cp * NC;
  const bool busy = ((warp * 32) % RPC) < R;   // the warp holds at least one real row
  const int lim_r = rr < R ? a.lim[tok0 + rr / a.G] : -1;
  const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
  const float kScaleLog2 = 0.125f * 1.4426950408889634f;   // 1/sqrt(64) in log2 units
  bool ok = true;
  // waits are warp-uniform; after a failure the warp stops waiting
  auto wwait = [&](uint64_t* bar, uint32_t parity) {
    if (ok) ok = __all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(bar), parity, a.err)) != 0;
    return ok;
  };
  for (int j = 0; j < np; ++j) {
    const int buf = j & 1;
    const bool have = wwait(&y.s_full[buf], (j >> 1) & 1) && busy;
    // 1. this thread's columns of S_j; the buffer is free once every warp has read
    float sv[NC];
    float pm = -INFINITY;
    if (have) {
      tc_fence_after();
      uint32_t sr[NC];
      if constexpr (NC == 16) {
        tmem_ld16_nowait(trow + buf * 64 + col0, *reinterpret_cast<uint32_t(*)[16]>(sr));
      } else if constexpr (NC == 32) {
        tmem_ld32_nowait(trow + buf * 64 + col0, *reinterpret_cast<uint32_t(*)[32]>(sr));
      } else {
        tmem_ld32_nowait(trow + buf * 64, *reinterpret_cast<uint32_t(*)[32]>(sr));
        tmem_ld32_nowait(trow + buf * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(sr + 32));
      }
      tmem_wait_ld();
      // 2. mask (keys past the row's limit: only on the window's last pages),
      //    this thread's maximum (of the unscaled scores; the scale is positive)
      const int key0 = (p_begin + j) * 64 + col0;
      if (__all_sync(0xFFFFFFFFu, rr >= R || key0 + NC - 1 <= lim_r)) {
#pragma unroll
        for (int k = 0; k < NC; ++k) sv[k] = __uint_as_float(sr[k]);
      } else {
#pragma unroll
        for (int k = 0; k < NC; ++k) sv[k] = key0 + k <= lim_r ? __uint_as_float(sr[k]) : -INFINITY;
      }
      // max as a tree of three-way maxima (a chain of NC dependent fmax
      // would dominate the page)
      float mt[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        mt[e] = sv[e];
        int k = e + 8;
#pragma unroll
        for (; k + 8 < NC; k += 16) mt[e] = fmax3(mt[e], sv[k], sv[k + 8]);
        if (k < NC) mt[e] = fmaxf(mt[e], sv[k]);
      }
      pm = fmax3(fmax3(mt[0], mt[1], mt[2]), fmax3(mt[3], mt[4], mt[5]), fmaxf(mt[6], mt[7])) *
           kScaleLog2;
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&y.s_free[buf]));
    // 3. does any row rise by more than 2^8?  Then the row's page max over its
    //    DUP copies (copy k at MMA row k * RPC + rr).
    const bool any = softmax_vote_or(pm > m + kAttnRescale);
    float mx = -INFINITY;
    if (any) {
      y.red[mrow] = pm;
      softmax_bar_max();
#pragma unroll
      for (int k = 0; k < DUP; ++k) mx = fmaxf(mx, y.red[k * RPC + rr]);
    }
    // 4. a rise rescales O and the row sum first.  tcgen05.ld / st are
    //    warp-collective: a warp with any rising row rescales all its rows,
    //    the others by exactly 1.
    const bool rise = any && mx > m + kAttnRescale;
    const float alpha = !rise ? 1.f : ((m == -INFINITY) ? 0.f : exp2f(m - mx));
    if (cp == 0 && j > 0 && __any_sync(0xFFFFFFFFu, rise) &&
        wwait(&y.empty[(j - 1) % kAttnStages], ((j - 1) / kAttnStages) & 1)) {
      tc_fence_after();
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        uint32_t o32[32];
        tmem_ld32_nowait(trow + 128 + hh * 32, o32);
        tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < 32; ++k) o32[k] = __float_as_uint(alpha * __uint_as_float(o32[k]));
        tmem_st32(trow + 128 + hh * 32, o32);
      }
      // and the row sum, O's column 64
      const uint32_t l1 = tmem_ld1(trow + 192);
      tmem_wait_ld();
      tmem_st1(trow + 192, __float_as_uint(alpha * __uint_as_float(l1)));
      tmem_wait_st();
    }
    if (rise) m = mx;
    // 5. P_j = exp2(s - m) (fp16) into row rr of the P tile
    if (have) {
      const float sub = (m == -INFINITY) ? 0.f : m;
      uint8_t* prow = y.sP + buf * kAttnMaxRows * 128;
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        float p[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) p[e] = ex2_sfu(fmaf(sv[8 * c + e], kScaleLog2, -sub));
        uint32_t w4[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          __half2 hv = __floats2half2_rn(p[2 * e], p[2 * e + 1]);
          w4[e] = *reinterpret_cast<uint32_t*>(&hv);
        }
        *reinterpret_cast<uint4*>(prow + sw128(rr, col0 / 8 + c)) =
            make_uint4(w4[0], w4[1], w4[2], w4[3]);
      }
      fence_proxy_async_smem();
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&y.p_full[buf]));
  }
  return ok;
}

__global__ void __launch_bounds__(kAttnThreads, 2)
    attn_paged_kernel(const __grid_constant__ CUtensorMap tmKV, const AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int rows_alloc = kAttnMaxRows;
  uint8_t* sQ = smem + kAttnQOff;
  uint8_t* sP = smem + kAttnPOff;                        // [2][128][128 B]
  uint8_t* ring = smem + kAttnRingOff;                   // [stage][K | V^T]
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kAttnBarOff);
  uint64_t* full = bars;                                 // [stages] TMA landed
  uint64_t* empty = bars + kAttnStages;                  // [stages] PV of the page done
  uint64_t* s_full = bars + 2 * kAttnStages;             // [2] S in TMEM
  uint64_t* s_free = s_full + 2;                         // [2] S read by the 4 softmax warps
  uint64_t* p_full = s_full + 4;                         // [2] P in smem (4 warp arrivals)
  uint64_t* mma_done = s_full + 7;                       // every MMA of this CTA retired
  uint64_t* recv_bar = s_full + 8;
  uint64_t* q_full = s_full + 9;                         // Q tile in smem (4 warp arrivals)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(s_full + 12);
  // [0] max limit, [1] last-item flag, [2] pages the MMA warp took, [3] pages issued
  int* s_int = reinterpret_cast<int*>(s_full + 13);

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
    int mxl = -1;
    for (int i = lane; i < ntok; i += 32) mxl = max(mxl, a.lim[tok0 + i]);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) mxl = max(mxl, __shfl_xor_sync(0xFFFFFFFFu, mxl, o));
    if (lane == 0) s_int[0] = mxl;
  }
  __syncthreads();
  const int maxlim = s_int[0];
  const int npages_blk = maxlim / 64 + 1;
  const int SP = a.split_pages;
  const int nitems = (npages_blk + SP - 1) / SP;
  if (maxlim < 0 || npages_blk > a.pt_stride || slot < 0 || nitems > a.max_items ||
      R > kAttnMaxRows) {
    if (threadIdx.x == 0) atomicExch(a.err, kErrBounds);
    return;
  }
  if (c >= nitems && (nitems == 1 || !a.cluster)) return;
  const bool in_cluster = a.cluster && nitems > 1;
  if (c >= nitems) {   // idle cluster member: counts in the cluster barrier, owns nothing
    cluster_arrive_release();
    return;
  }

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmKV);
    for (int s = 0; s < kAttnStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&s_free[i]), kAttnSoftWarps);   // one arrival per softmax warp
      mbar_init(smem_u32(&p_full[i]), kAttnSoftWarps);
    }
    mbar_init(smem_u32(mma_done), 1);
    mbar_init(smem_u32(q_full), kAttnSoftWarps);
    if (in_cluster) {
      mbar_init(smem_u32(recv_bar), 1);
      // nitems sources, ceil(128 / nitems) rows each, arrive by bulk copy
      const int rpo = (rows_alloc + nitems - 1) / nitems;
      mbar_arrive_expect_tx(smem_u32(recv_bar), static_cast<uint32_t>(nitems * rpo * kAttnRow * 4));
    }
    s_int[2] = 0;
    s_int[3] = 0;
    fence_mbar_init();
  }
  // the ones rows after every V^T page: O += P [V | 1] puts the row sum in O's column 64
  for (int i = threadIdx.x; i < kAttnStages * kAttnOnesBytes / 16; i += blockDim.x) {
    const int st = i / (kAttnOnesBytes / 16), off = i % (kAttnOnesBytes / 16);
    *reinterpret_cast<uint4*>(ring + st * kAttnStageBytes + 2 * kAttnPageBytes + off * 16) =
        make_uint4(0x3C003C00u, 0x3C003C00u, 0x3C003C00u, 0x3C003C00u);
  }
  fence_proxy_async_smem();
  if (warp == kAttnMmaWarp) tmem_alloc(smem_u32(tmem_slot), kAttnTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  const int p_begin = c * SP;
  const int np = min(npages_blk, p_begin + SP) - p_begin;
  const int32_t* pt = a.page_table + static_cast<size_t>(slot) * a.pt_stride;
  bool ok = true;
  float m = -INFINITY, l = 0.f;   // the row's running max (log2 units) and sum
  float* red = reinterpret_cast<float*>(s_int + 8);        // [softmax threads] page maxima

  if (warp == kAttnTmaWarp) {
    // ---- TMA producer: K and V^T pages of the item, in order
    if (lane == 0) {
      const int safe_pages = a.blk_slot ? a.lim[tok0] / 64 : 0;   // wholly committed pages
      const uint64_t pol = l2_policy_evict_first();
      int issued = 0;
      auto issue = [&](int i) {
        const int s = i % kAttnStages;
        int phys = pt[p_begin + i];
        if (phys < 0) {  // unmapped page: the TMA box lands out of bounds and reads zeros
          atomicExch(a.err, kErrBounds);
          phys = 0x3FFFFFFF / a.rows_per_page;
        }
        const long long row = a.kv_row_base + static_cast<long long>(phys) * a.rows_per_page;
        const uint32_t fb = smem_u32(&full[s]);
        mbar_arrive_expect_tx(fb, 2 * kAttnPageBytes);   // K and V^T (the ones rows stay)
        uint8_t* st = ring + s * kAttnStageBytes;
        tma_load_2d(smem_u32(st), &tmKV, 0, static_cast<int>(row + h * 64), fb, pol);
        tma_load_2d(smem_u32(st + kAttnPageBytes), &tmKV, 0, static_cast<int>(row + (a.Hkv + h) * 64),
                    fb, pol);
      };
      while (issued < min(np, kAttnStages) && p_begin + issued < safe_pages) issue(issued++);
      pdl_wait();
      pdl_trigger();
      while (issued < np && ok) {
        const int s = issued % kAttnStages;
        if (issued >= kAttnStages &&
            !mbar_wait(smem_u32(&empty[s]), ((issued / kAttnStages) + 1) & 1, a.err)) {
          ok = false;
          break;
        }
        issue(issued++);
      }
      s_int[3] = issued;
    } else {
      pdl_wait();
      pdl_trigger();
    }
  } else if (warp == kAttnMmaWarp) {
    // ---- MMA issuer: S one page ahead of the softmax, O += P V after each P
    pdl_wait();
    pdl_trigger();
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_f16(128, 64);
      constexpr uint32_t idesc_pv = umma_idesc_f16(128, 80);   // V^T page and its 16 ones rows
      const uint64_t qdesc = umma_desc_sw128(smem_u32(sQ));
      auto issue_s = [&](int j) -> bool {
        const int s = j % kAttnStages, buf = j & 1;
        if (!mbar_wait(smem_u32(&full[s]), (j / kAttnStages) & 1, a.err)) return false;
        s_int[2] = j + 1;
        if (j >= 2 && !mbar_wait(smem_u32(&s_free[buf]), ((j >> 1) + 1) & 1, a.err)) return false;
        tc_fence_after();
        const uint64_t kdesc = umma_desc_sw128(smem_u32(ring + s * kAttnStageBytes));
#pragma unroll
        for (int k = 0; k < 4; ++k)
          umma_f16(tmem + buf * 64, qdesc + 2 * k, kdesc + 2 * k, idesc, k > 0 ? 1u : 0u);
        umma_commit(smem_u32(&s_full[buf]));
        return true;
      };
      if (!mbar_wait(smem_u32(q_full), 0, a.err)) ok = false;   // Q tile written
      if (ok) ok = issue_s(0);
      for (int j = 0; j < np && ok; ++j) {
        if (j + 1 < np && !(ok = issue_s(j + 1))) break;
        const int s = j % kAttnStages, buf = j & 1;
        if (!mbar_wait(smem_u32(&p_full[buf]), (j >> 1) & 1, a.err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t pdesc = umma_desc_sw128(smem_u32(sP + buf * kAttnMaxRows * 128));
        const uint64_t vdesc = umma_desc_sw128(smem_u32(ring + s * kAttnStageBytes + kAttnPageBytes));
#pragma unroll
        for (int k = 0; k < 4; ++k)
          umma_f16(tmem + 128, pdesc + 2 * k, vdesc + 2 * k, idesc_pv, (j > 0 || k > 0) ? 1u : 0u);
        umma_commit(smem_u32(&empty[s]));
      }
      umma_commit(smem_u32(mma_done));   // retires once every MMA above has
    }
  } else {
    // ---- softmax warps: DUP copies of each row across the 128 MMA rows
    const int dup = R <= 32 ? 4 : (R <= 64 ? 2 : 1);
    const int rpc = kAttnMaxRows / dup;
    // Q rows -> swizzled smem: MMA row i holds block row i % rpc (zero past R)
    pdl_wait();
    pdl_trigger();
    for (int idx = threadIdx.x; idx < rows_alloc * 8; idx += kAttnSoftThreads) {
      const int i = idx >> 3, ch = idx & 7, rr = i % rpc;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (rr < R) {
        const int t = tok0 + rr / a.G;
        const int hq = h * a.G + rr % a.G;
        v = *reinterpret_cast<const uint4*>(a.q + (static_cast<size_t>(t) * a.Hq + hq) * 64 + ch * 8);
      }
      *reinterpret_cast<uint4*>(sQ + sw128(i, ch)) = v;
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(q_full));
    AttnSync y{s_full, s_free, p_full, empty, sP, red};
    if (dup == 4) ok = attn_softmax<4>(a, y, tmem, np, p_begin, R, tok0, m);
    else if (dup == 2) ok = attn_softmax<2>(a, y, tmem, np, p_begin, R, tok0, m);
    else ok = attn_softmax<1>(a, y, tmem, np, p_begin, R, tok0, m);
  }

  const bool all_ok = __syncthreads_and(ok);
  // every MMA retired and every TMA copy landed before TMEM and the ring are reused
  if (warp == kAttnMmaWarp && lane == 0) mbar_wait(smem_u32(mma_done), 0, a.err);
  if (warp == kAttnTmaWarp && lane == 0) {
    for (int i = s_int[2]; i < s_int[3]; ++i)
      mbar_wait(smem_u32(&full[i % kAttnStages]), (i / kAttnStages) & 1, a.err);
  }
  __syncthreads();
  // the row's O and its sum (O's column 64) from TMEM (rows < R)
  const int r = threadIdx.x;
  const bool row_thread = r < R;
  float o[64];
  if (warp < 4) {
    tc_fence_after();
    uint32_t o0[32], o1[32];
    tmem_ld32_nowait(tmem + (static_cast<uint32_t>(warp * 32) << 16) + 128, o0);
    tmem_ld32_nowait(tmem + (static_cast<uint32_t>(warp * 32) << 16) + 128 + 32, o1);
    const uint32_t l1 = tmem_ld1(tmem + (static_cast<uint32_t>(warp * 32) << 16) + 192);
    tmem_wait_ld();
    l = __uint_as_float(l1);
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      o[k] = __uint_as_float(o0[k]);
      o[32 + k] = __uint_as_float(o1[k]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kAttnMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kAttnTmemCols);
  }

  if (nitems == 1) {   // the block's only item: its rows are final
    if (row_thread && all_ok) {
      const float inv = 1.0f / l;
      const int t = tok0 + r / a.G;
      const int hq = h * a.G + r % a.G;
      __half* dst = a.out + (static_cast<size_t>(t) * a.Hq + hq) * 64;
#pragma unroll
      for (int cch = 0; cch < 8; ++cch) {
        uint32_t w4[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          __half2 hv = __floats2half2_rn(o[8 * cch + 2 * e] * inv, o[8 * cch + 2 * e + 1] * inv);
          w4[e] = *reinterpret_cast<uint32_t*>(&hv);
        }
        *reinterpret_cast<uint4*>(dst + 8 * cch) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
      }
    }
    return;
  }

  // this thread's row (O, m, l) -> a [kAttnRow] slot
  auto put_row = [&](float* dst) {
#pragma unroll
    for (int k = 0; k < 64; k += 4)
      *reinterpret_cast<float4*>(dst + k) = make_float4(o[k], o[k + 1], o[k + 2], o[k + 3]);
    *reinterpret_cast<float2*>(dst + 64) = make_float2(m, l);
  };

  // Merged rows of one item: source `it`, row r -> float pointer (O[64], m, l).
  // Cluster: recv[it][k] (in the ring) with r = c + k * nitems.  Global:
  // part[b][h][it][r].
  const size_t bh = static_cast<size_t>(b) * a.Hkv + h;
  float* part_bh = a.part + bh * a.max_items * rows_alloc * kAttnRow;
  float* recv = reinterpret_cast<float*>(ring);
  const int rpo = (rows_alloc + nitems - 1) / nitems;   // cluster: rows per owner
  bool got = true;
  int my_rows;
  if (in_cluster) {
    // ---- items -> owners.  stage [owner][slot][kAttnRow] over Q and P.
    float* stage = reinterpret_cast<float*>(sQ);
    const int blk_floats = rpo * kAttnRow;
    if (row_thread)
      put_row(stage + static_cast<size_t>(r % nitems) * blk_floats + (r / nitems) * kAttnRow);
    fence_proxy_async_smem();
    __syncthreads();
    cluster_arrive_release();
    cluster_wait();   // every CTA of the cluster is done with its pages: receive buffers idle
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
    if (row_thread) put_row(part_bh + (static_cast<size_t>(c) * rows_alloc + r) * kAttnRow);
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
  // cluster: the received rows fill the ring, the tables go over Q and P (the
  // outgoing copies have read them); global: the tables go in the ring
  float* mb = reinterpret_cast<float*>(in_cluster ? sQ : ring);
  float* lb = mb + static_cast<size_t>(nitems) * rows_alloc;
  const bool fits = 2 * nitems * rows_alloc * 4 <= (in_cluster ? kAttnRingOff : kAttnRingBytes);
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
        const int rr = row_of(k);
        const int t = tok0 + rr / a.G;
        const int hq = h * a.G + rr % a.G;
        __half* dst = a.out + (static_cast<size_t>(t) * a.Hq + hq) * 64 + d4;
        *reinterpret_cast<__half2*>(dst) = __floats2half2_rn(acc.x, acc.y);
        *reinterpret_cast<__half2*>(dst + 2) = __floats2half2_rn(acc.z, acc.w);
      }
    }
  }
}

}  // namespace gs
