// gemm_tc.cuh -- tcgen05/TMEM GEMM for the decoder's projections and LM head.
//
// Computes D[f, t] = sum_k W[f, k] X[t, k] with the weight rows on the MMA M
// side (128 rows per CTA, "swap-AB") and the token rows on the MMA N side
// (BN in {32, 64, 128, 256}), so a 17-token decode window and an 8192-token
// prefill chunk use the same kernel.  Operands are K-major fp16 tiles staged by
// TMA with 128-byte swizzle; one elected thread issues tcgen05.mma into a TMEM
// fp32 accumulator of 128 lanes x BN columns; four warps read it back with
// tcgen05.ld for the fused epilogue.
//
// Launch overlap: weight tiles do not depend on the previous kernel, so the
// producer issues the first stages' weight loads before griddepcontrol.wait
// (programmatic dependent launch); activation loads and every global write
// come after it.
//
// Split-K: the CTAs that own different K ranges of one output tile either
// form a thread-block cluster (decode tiles, BN <= 64) -- each CTA owns a
// slice of the tile's tokens; every CTA stages its fp32 partials slice by
// slice in its own shared memory and one thread sends each slice to its
// owner with a bulk async copy that completes on the owner's mbarrier; the
// owner then sums the received slices locally -- or
// write the partials to global scratch, where the last CTA to arrive (atomic
// ticket, no spinning) sums them.  Both sum the splits in order 0..S-1 from a
// zero start, so the result does not depend on the path or on arrival order.
//
// Weights arrive as fp16 copies scaled by a power of two 2^s per tensor (an
// exact re-encoding of the model's bf16 values); the epilogue multiplies the
// fp32 accumulator by w_scale = 2^-s, which is exact, so the result equals
// the product with the unscaled weights.
//
// Epilogues: fp16 store, fp32 residual add, SwiGLU (gate and up rows of the
// same features share a tile), LM-head argmax (packed 64-bit atomicMax, ties
// to the lowest index) with an optional fp32 logit dump, and the QKV epilogue
// (RoPE on q and k, q to its buffer, k and v into the paged KV cache).
//
// RMSNorm is folded into the GEMMs: a residual epilogue also writes
// hb = fp16(h * g) with the gain g of the norm that comes next, and the sum of
// h^2 over its 128 features (one partial per feature tile, "ssp"); the GEMM
// that consumes hb multiplies its accumulator by rsqrt(sum(ssp) / d + eps).
// Since that factor is one scalar per token, this equals normalising first.
#pragma once
#include "ptx.cuh"

namespace gs {

// Split-K factors up to this many reduce inside a cluster (portable cluster size).
constexpr int kGemmMaxClusterSplits = 8;

enum GemmEpilogue : int {
  kEpiStoreF16 = 0, kEpiResidF32 = 1, kEpiSwiGLU = 2, kEpiArgmax = 3, kEpiQKV = 4
};

struct GemmArgs {
  int M;            // token rows
  int N;            // output features (for SwiGLU: d_ffn, the weight has 2N rows)
  int K;            // reduction length, multiple of 64
  int splits;       // split-K factor (divides K / 64)
  int kb_per_split; // (K / 64) / splits
  int cluster;      // 1: split-K partials reduced inside a cluster of `splits` CTAs
  int chunks;       // splits == 1: K reduced in this many chunks inside the CTA (>= 1)
  int stages;       // pipeline stages (GemmShape::kStagesMin..kStagesMax)
  void* y;          // output: fp16 [M, ldy] | fp32 [M, ldy] | uint64 [M] (argmax)
  int ldy;
  float* partial;   // global split-K partials [splits][tiles][BN][128] fp32 (cluster == 0)
  int* counters;    // per output tile, zero between launches (cluster == 0)
  float* logits;    // argmax only: optional fp32 [M, N] dump
  // argmax only, optional: per token and 128-row feature tile, (tile max,
  // sum over the tile of exp(logit - tile max)) at [token][feature tile],
  // of the logits times inv_temp
  float2* lse_part;
  float inv_temp;   // 1 / temperature of the softmax partials and the samples
  // argmax only, optional: sample instead of argmax (Gumbel-max over
  // logit * inv_temp, Philox stream kStreamDraft); rng_row[token] =
  // (unused, window row, round, slot)
  const uint4* rng_row;
  uint32_t seed_lo, seed_hi;
  int* err;
  float w_scale;    // 2^-s of the weight copy (1 for unscaled weights)
  int x_row0;       // X (and ssp_in) row of token 0
  // folded RMSNorm on the input: scale = rsqrt(sum_p ssp_in[t][p] * inv_d + eps)
  const float* ssp_in;
  int n_ssp;        // d / 128 partials per token
  float inv_d, eps;
  // residual epilogue extras: hb_out[t][f] = fp16(h[t][f] * g_next[f]); ssp_out[t][tile] = sum h^2
  __half* hb_out;
  const __nv_bfloat16* g_next;
  float* ssp_out;
  // QKV epilogue
  __half* q_out;               // [M, Hq, 64]
  __half* kv_layer;            // this layer's page pool [pages][2][Hkv][64][64]
  const int32_t* pos;          // [M] absolute slot
  const int32_t* tok_slot;     // [M] page-table row, -1 = no KV write
  const int32_t* page_table;
  const float2* rope;          // [max_ctx][32] cos, sin
  int pt_stride, n_pages, max_ctx, Hq, Hkv;
};

template <int BN>
struct GemmShape {
  static constexpr int kABytes = 128 * 128;        // 128 rows x 64 fp16
  static constexpr int kBBytes = BN * 128;         // BN rows x 64 fp16
  static constexpr int kStageBytes = kABytes + kBBytes;
  // Pipeline depth is chosen per launch (GemmArgs::stages): two stages for a
  // split CTA that loads two k-blocks, up to kStagesMax (about 190 KB) for
  // CTAs that stream the whole K.
  static constexpr int kStagesMax = BN <= 32 ? 8 : (BN <= 128 ? 6 : 4);
  static constexpr int kStagesMin = 2;
  static constexpr int kStagesDefault = BN <= 64 ? 4 : (BN <= 128 ? 3 : 4);
  static constexpr int kTmemCols = BN < 32 ? 32 : BN;
  static constexpr int kRedBytes = BN * 128 * 4;   // cluster reduction tile [BN][128] fp32
  static constexpr int kXBufBytes = 32 * 128 * 4;  // epilogue exchange (SwiGLU, RoPE, sums)
  static_assert(!(BN <= 64) || kXBufBytes + kRedBytes <= kStagesMin * kStageBytes,
                "cluster staging smem");
  // transposed epilogue slice [32][132] fp32 and per-token partial sums [32][16]
  static_assert((32 * 132 + 32 * 16) * 4 <= kStagesMin * kStageBytes, "epilogue slice smem");
  // argmax epilogue: keys [128][33] and quarter maxima [4][32], 8 bytes each,
  // then the softmax partials' tile maxima [32] and warp maxima and sums
  // [2][4][32], 4 bytes each
  static_assert((128 * 33 + 4 * 32) * 8 + 9 * 32 * 4 <= kStagesMin * kStageBytes, "argmax smem");
  // RoPE cos/sin rows of the tile's tokens, staged while the mainloop runs
  // (QKV launches, decode tiles)
  static constexpr bool kStageRope = BN <= 64;
  __host__ __device__ static constexpr int rope_bytes(int epi) {
    return (kStageRope && epi == kEpiQKV) ? BN * 32 * 8 : 0;
  }
  // cluster split-K receive buffer [S][BN / S][128] fp32 (decode tiles only)
  static constexpr bool kClusterOk = BN <= 64;
  static constexpr int kRecvBytes = kClusterOk ? BN * 128 * 4 : 0;
  // pipeline | barriers (256 B) | per token: norm scale (4 B), KV destination (8 B), position (4 B)
  // | RoPE rows | receive buffer
  __host__ __device__ static constexpr int recv_offset(int stages, int epi) {
    return stages * kStageBytes + 256 + 16 * BN + rope_bytes(epi);
  }
  __host__ __device__ static constexpr int smem_bytes(int stages, int epi, bool cluster) {
    return recv_offset(stages, epi) + (cluster ? kRecvBytes : 0) + 1024 /*align*/;
  }
  static constexpr int kSmemMax = smem_bytes(kStagesMax, kEpiQKV, true);
  static_assert(kSmemMax <= 227 * 1024, "deepest pipeline fits one CTA's smem");
  // Deepest pipeline with which `per_sm` CTAs share one SM's 228 KB (each CTA
  // also holds 1 KB of system smem and 16 B of static smem).
  static int stages_fitting(int per_sm, int epi, bool cluster) {
    for (int st = kStagesMax; st > kStagesMin; --st)
      if ((smem_bytes(st, epi, cluster) + 1024 + 16) * per_sm <= 228 * 1024) return st;
    return kStagesMin;
  }
};

// Epilogue of 32 consecutive tokens (t0 .. t0+31) of feature row `row`;
// only tokens j in [jlo, jhi) with t0 + j < M are produced.

// Per-token data the epilogue needs, staged in shared memory while the
// mainloop runs: rs = folded-norm scale, kvdst = element offset of the token's
// row in its KV page (-1: no write), pos = absolute slot.
struct TokMeta {
  const float* rs;
  const long long* kvdst;
  const int* pos;
  const float2* cs;   // [32 tokens][32] cos/sin, or null: read the table
};

// Epilogue of EW consecutive token slots t0 .. t0+EW-1 of feature row `row`;
// slots q in [jlo, jhi) with t0 + q < M are produced.  Split CTAs own at most
// 8 tokens and use EW = 8; whole tiles use EW = 32.
// Eight fp32 values -> eight fp16 bit patterns in one 16-byte word; `bad` is
// raised for a value beyond the fp16 range or a NaN (no branch per value).
__device__ __forceinline__ uint4 pack8_f16(const float (&x)[8], bool& bad) {
  uint32_t w[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    bad |= !(fabsf(x[2 * e]) <= 65504.0f) || !(fabsf(x[2 * e + 1]) <= 65504.0f);
    __half2 h = __floats2half2_rn(x[2 * e], x[2 * e + 1]);
    w[e] = *reinterpret_cast<uint32_t*>(&h);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// Epilogue of EW consecutive token slots t0 .. t0+EW-1 of the 128 rows of one
// feature tile; thread `row` (0..127, the four epilogue warps) holds row
// `row` of those tokens in v.  Slots q in [jlo, jhi) with t0 + q < M are
// produced.  Split CTAs own at most 8 tokens and use EW = 8; whole tiles use
// EW = 32.  The slice is first transposed through shared memory (xs[token][row],
// row stride 132 floats), then each work item -- one token and 8 consecutive
// rows -- reads, computes and writes 16-byte vectors, so global traffic is
// contiguous.  A value's arithmetic is the same for every EW and every token
// tile.  Values beyond the fp16 range raise kErrRange once per thread.
template <int BN, int EPI, int EW>
__device__ __forceinline__ void gemm_epilogue_chunk(const GemmArgs& a, float (&v)[EW], int row,
                                                    int feat_tile, int t0, int jlo, int jhi,
                                                    float* xbuf, TokMeta tm) {
  const float* rs = tm.rs;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  jhi = min(jhi, a.M - t0);
  if (rs != nullptr) {
#pragma unroll
    for (int j = 0; j < EW; ++j) v[j] *= rs[j] * a.w_scale;
  } else {
#pragma unroll
    for (int j = 0; j < EW; ++j) v[j] *= a.w_scale;
  }
  if constexpr (EPI != kEpiArgmax) {
    constexpr int LDX = 132;
    float* xs = xbuf;   // [EW][LDX]
#pragma unroll
    for (int j = 0; j < EW; ++j) xs[j * LDX + row] = v[j];
    asm volatile("bar.sync 1, 128;" ::: "memory");
    bool bad = false;
    const int tid = row;
    if constexpr (EPI == kEpiStoreF16) {
      __half* y = static_cast<__half*>(a.y);
      for (int it = tid; it < EW * 16; it += 128) {
        const int j = it >> 4, g = it & 15;
        if (j < jlo || j >= jhi) continue;
        const float4 a0 = *reinterpret_cast<const float4*>(xs + j * LDX + 8 * g);
        const float4 a1 = *reinterpret_cast<const float4*>(xs + j * LDX + 8 * g + 4);
        const float x[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
        *reinterpret_cast<uint4*>(y + static_cast<size_t>(t0 + j) * a.ldy + feat_tile * 128 + 8 * g) =
            pack8_f16(x, bad);
      }
    } else if constexpr (EPI == kEpiResidF32) {
      // h = h + acc (fp32), the next norm's input hb = fp16(h * g), and the sum
      // of h^2 over the tile's 128 features per token: each item sums its 8
      // features in order, then the 16 items of a token in order
      float* y = static_cast<float*>(a.y);
      float* part = xs + EW * LDX;   // [EW][16]
      for (int it = tid; it < EW * 16; it += 128) {
        const int j = it >> 4, g = it & 15;
        if (j < jlo || j >= jhi) continue;
        const int f = feat_tile * 128 + 8 * g;
        float* yr = y + static_cast<size_t>(t0 + j) * a.ldy + f;
        const float4 h0 = *reinterpret_cast<const float4*>(yr);
        const float4 h1 = *reinterpret_cast<const float4*>(yr + 4);
        const float4 a0 = *reinterpret_cast<const float4*>(xs + j * LDX + 8 * g);
        const float4 a1 = *reinterpret_cast<const float4*>(xs + j * LDX + 8 * g + 4);
        const float hn[8] = {h0.x + a0.x, h0.y + a0.y, h0.z + a0.z, h0.w + a0.w,
                             h1.x + a1.x, h1.y + a1.y, h1.z + a1.z, h1.w + a1.w};
        *reinterpret_cast<float4*>(yr) = make_float4(hn[0], hn[1], hn[2], hn[3]);
        *reinterpret_cast<float4*>(yr + 4) = make_float4(hn[4], hn[5], hn[6], hn[7]);
        if (a.hb_out != nullptr) {
          const uint4 graw = *reinterpret_cast<const uint4*>(a.g_next + f);
          const __nv_bfloat162* gp = reinterpret_cast<const __nv_bfloat162*>(&graw);
          float x[8];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 gg = __bfloat1622float2(gp[e]);
            x[2 * e] = hn[2 * e] * gg.x;
            x[2 * e + 1] = hn[2 * e + 1] * gg.y;
          }
          *reinterpret_cast<uint4*>(a.hb_out + static_cast<size_t>(t0 + j) * a.ldy + f) =
              pack8_f16(x, bad);
        }
        float sq = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) sq += hn[e] * hn[e];
        part[j * 16 + g] = sq;
      }
      if (a.ssp_out != nullptr) {
        asm volatile("bar.sync 2, 128;" ::: "memory");
        if (tid < EW) {
          const int j = tid;
          if (j >= jlo && j < jhi) {
            const float* pp = part + j * 16;
            float t = 0.f;
#pragma unroll
            for (int g = 0; g < 16; ++g) t += pp[g];
            a.ssp_out[static_cast<size_t>(t0 + j) * a.n_ssp + feat_tile] = t;
          }
        }
      }
    } else if constexpr (EPI == kEpiSwiGLU) {
      // rows 0..63: gate of output features f0..f0+63; rows 64..127: up of the same
      __half* y = static_cast<__half*>(a.y);
      for (int it = tid; it < EW * 8; it += 128) {
        const int j = it >> 3, g = it & 7;
        if (j < jlo || j >= jhi) continue;
        float x[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float gt = xs[j * LDX + 8 * g + e];
          const float up = xs[j * LDX + 64 + 8 * g + e];
          x[e] = gt / (1.0f + __expf(-gt)) * up;
        }
        *reinterpret_cast<uint4*>(y + static_cast<size_t>(t0 + j) * a.ldy + feat_tile * 64 + 8 * g) =
            pack8_f16(x, bad);
      }
    } else {   // kEpiQKV
      // rows of this tile: two heads of 64; RoPE rotates dims d and d ^ 32
      // with angle index d & 31 at the token's position; q to its buffer, k
      // and v into the token's KV page (V stored transposed, [dim][token])
      const int rbase = feat_tile * 128;
      const int region = rbase < a.Hq * 64 ? 0 : (rbase < (a.Hq + a.Hkv) * 64 ? 1 : 2);
      const int head0 = rbase / 64 - (region == 0 ? 0 : (region == 1 ? a.Hq : a.Hq + a.Hkv));
      for (int it = tid; it < EW * 16; it += 128) {
        const int j = it >> 4, hh = (it >> 3) & 1, g = it & 7;
        if (j < jlo || j >= jhi) continue;
        const int head = head0 + hh;
        const float* xr = xs + j * LDX + hh * 64;
        float x[8];
        if (region < 2) {
          const int p = tm.pos[j];
          const bool okp = p >= 0 && p < a.max_ctx;
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int d = 8 * g + e;
            const float2 cs = !okp ? make_float2(1.f, 0.f)
                                   : (tm.cs ? tm.cs[j * 32 + (d & 31)]
                                            : a.rope[static_cast<size_t>(p) * 32 + (d & 31)]);
            const float pr = xr[d ^ 32];
            x[e] = d < 32 ? xr[d] * cs.x - pr * cs.y : xr[d] * cs.x + pr * cs.y;
          }
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) x[e] = xr[8 * g + e];
        }
        if (region == 0) {
          *reinterpret_cast<uint4*>(a.q_out + (static_cast<size_t>(t0 + j) * a.Hq + head) * 64 + 8 * g) =
              pack8_f16(x, bad);
        } else {
          const long long base = tm.kvdst[j];
          if (base < 0) continue;
          if (region == 1) {   // K: [token][dim]
            *reinterpret_cast<uint4*>(a.kv_layer + base + static_cast<long long>(head) * 4096 + 8 * g) =
                pack8_f16(x, bad);
          } else {             // V^T: [dim][token]
            const int tok = tm.pos[j] & 63;
            __half* vt = a.kv_layer + base - tok * 64 + (static_cast<long long>(a.Hkv) + head) * 4096 + tok;
            const uint4 w = pack8_f16(x, bad);
            const __half* hv = reinterpret_cast<const __half*>(&w);
#pragma unroll
            for (int e = 0; e < 8; ++e) vt[(8 * g + e) * 64] = hv[e];
          }
        }
      }
    }
    if (bad) atomicExch(a.err, kErrRange);
    asm volatile("bar.sync 1, 128;" ::: "memory");   // xs is reused by the next slice
    return;
  } else {  // argmax over the vocabulary rows of this tile, per token
    const uint32_t f = static_cast<uint32_t>(feat_tile * 128 + row);
    unsigned long long* out = static_cast<unsigned long long*>(a.y);
    if (a.logits != nullptr) {
#pragma unroll
      for (int j = 0; j < EW; ++j)
        if (j >= jlo && j < jhi) a.logits[static_cast<size_t>(t0 + j) * a.N + f] = v[j];
    }
    // keys [row][slot] in shared memory (row stride EW + 1 keys), then thread
    // (slot j, row quarter q) takes the max over its 32 rows, and the first
    // warp the max over the four quarters: one atomicMax per token per CTA
    unsigned long long* kb = reinterpret_cast<unsigned long long*>(xbuf);
    constexpr int LD = EW + 1;
    if (a.rng_row != nullptr) {
      // sample: argmax of logit / T + Gumbel noise of this (row, vocabulary entry)
#pragma unroll
      for (int j = 0; j < EW; ++j) {
        float sc = -INFINITY;
        if (j >= jlo && j < jhi) {
          const uint4 c = a.rng_row[t0 + j];
          sc = v[j] * a.inv_temp +
               gumbel_of(philox_uniform(a.seed_lo, a.seed_hi, c.w, c.z, kStreamDraft, c.y, f));
        }
        kb[row * LD + j] = argmax_key(sc, f);
      }
    } else {
#pragma unroll
      for (int j = 0; j < EW; ++j) kb[row * LD + j] = argmax_key(v[j], f);
    }
    asm volatile("bar.sync 2, 128;" ::: "memory");
    unsigned long long* qb = kb + 128 * LD;   // [4][EW] quarter maxima
    if (threadIdx.x < 4 * EW) {
      const int j = threadIdx.x % EW, q = threadIdx.x / EW;
      unsigned long long best = 0;
      for (int rr = 0; rr < 32; ++rr) {
        const unsigned long long k = kb[(q * 32 + rr) * LD + j];
        best = k > best ? k : best;
      }
      qb[q * EW + j] = best;
    }
    asm volatile("bar.sync 2, 128;" ::: "memory");
    if (threadIdx.x < EW) {
      const int j = threadIdx.x;
      unsigned long long best = qb[j];
#pragma unroll
      for (int q = 1; q < 4; ++q) best = qb[q * EW + j] > best ? qb[q * EW + j] : best;
      if (j >= jlo && j < jhi) atomicMax(out + t0 + j, best);
    }
    asm volatile("bar.sync 2, 128;" ::: "memory");
    if (a.lse_part != nullptr) {
      // softmax partials of this tile over logit / T: the tile max (warp tree,
      // then the four warps), then the sum over its 128 rows of exp(x - max),
      // a warp tree then the four warps in order (fixed order: the same bits
      // for a row whatever the batch)
      float* tmax = reinterpret_cast<float*>(qb + 4 * EW);   // [EW]
      float* wmax = tmax + EW;                               // [4][EW]
      float* wsum = wmax + 4 * EW;                           // [4][EW]
#pragma unroll
      for (int j = 0; j < EW; ++j) {
        float m = v[j] * a.inv_temp;
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
        if (lane == 0) wmax[warp * EW + j] = m;
      }
      asm volatile("bar.sync 2, 128;" ::: "memory");
      if (threadIdx.x < EW) {
        const int j = threadIdx.x;
        tmax[j] = fmaxf(fmaxf(wmax[j], wmax[EW + j]), fmaxf(wmax[2 * EW + j], wmax[3 * EW + j]));
      }
      asm volatile("bar.sync 2, 128;" ::: "memory");
#pragma unroll
      for (int j = 0; j < EW; ++j) {
        float e = expf(v[j] * a.inv_temp - tmax[j]);
#pragma unroll
        for (int m = 16; m >= 1; m >>= 1) e += __shfl_xor_sync(0xFFFFFFFFu, e, m);
        if (lane == 0) wsum[warp * EW + j] = e;
      }
      asm volatile("bar.sync 2, 128;" ::: "memory");
      if (threadIdx.x < EW) {
        const int j = threadIdx.x;
        if (j >= jlo && j < jhi)
          a.lse_part[static_cast<size_t>(t0 + j) * gridDim.y + feat_tile] = make_float2(
              tmax[j], ((wsum[j] + wsum[EW + j]) + wsum[2 * EW + j]) + wsum[3 * EW + j]);
      }
      asm volatile("bar.sync 2, 128;" ::: "memory");
    }
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(128, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                   const GemmArgs a) {
  using S = GemmShape<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* smA = smem;
  const int NS = a.stages;   // pipeline stages of this launch
  uint8_t* smB = smem + NS * S::kABytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NS * S::kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + NS;
  uint64_t* accum = bars + 2 * NS;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  volatile int* flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint64_t* recv_bar = accum + 3;   // cluster split-K: partial slices received

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // token tiles vary fastest, so the CTAs that share a weight tile run together
  // and read it from DRAM once
  const int tok_tile = blockIdx.x;
  const int feat_tile = blockIdx.y;
  const int split = blockIdx.z;
  const int kb0 = split * a.kb_per_split;
  const int nkb = a.kb_per_split;
  // Chunked K: step i works on k-block t of chunk c, c = i % nchunk and
  // t = i / nchunk, so consecutive MMAs go to different accumulators and do
  // not wait on each other; each chunk still sums its k-blocks in order.
  const int nchunk = a.chunks > 1 ? a.chunks : 1;
  const int kpc = nkb / nchunk;
  auto kblock = [&](int i) { return nchunk > 1 ? (i % nchunk) * kpc + i / nchunk : i; };

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
    for (int s = 0; s < NS; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    mbar_init(smem_u32(accum), 1);
    *flag = 0;
    if constexpr (S::kClusterOk) {
      if (a.cluster) {
        mbar_init(smem_u32(recv_bar), 1);
        // S slices of BN / S tokens x 128 rows of fp32 will arrive
        mbar_arrive_expect_tx(smem_u32(recv_bar), BN * 128 * 4);
      }
    }
    fence_mbar_init();
  }
  // chunked K: one TMEM accumulator of BN columns per chunk
  const uint32_t tmem_cols = static_cast<uint32_t>(S::kTmemCols * nchunk);
  if (warp == 2) tmem_alloc(smem_u32(tmem_slot), tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (a.cluster) cluster_arrive_relaxed();   // completed by cluster_wait() before the pushes

  if (warp == 0 && lane == 0) {
    // TMA producer.  Weight tiles of the first stages go out before the
    // dependency wait; activations only after it.
    const uint64_t pol_w = l2_policy_evict_first();
    const uint64_t pol_x = l2_policy_evict_last();
    auto load_w = [&](int i, int s) {
      const uint32_t fb = smem_u32(&full[s]);
      const int kx = (kb0 + kblock(i)) * 64;
      if constexpr (EPI == kEpiSwiGLU) {
        tma_load_2d(smem_u32(smA + s * S::kABytes), &tmW, kx, feat_tile * 64, fb, pol_w);
        tma_load_2d(smem_u32(smA + s * S::kABytes + 64 * 128), &tmW, kx, a.N + feat_tile * 64, fb,
                    pol_w);
      } else {
        tma_load_2d(smem_u32(smA + s * S::kABytes), &tmW, kx, feat_tile * 128, fb, pol_w);
      }
    };
    auto load_x = [&](int i, int s) {
      tma_load_2d(smem_u32(smB + s * S::kBBytes), &tmX, (kb0 + kblock(i)) * 64,
                  a.x_row0 + tok_tile * BN, smem_u32(&full[s]), pol_x);
    };
    const int npre = nkb < NS ? nkb : NS;
    for (int i = 0; i < npre; ++i) {          // fresh stages: no empty-barrier wait needed
      mbar_arrive_expect_tx(smem_u32(&full[i]), S::kStageBytes);
      load_w(i, i);
    }
    pdl_wait();
    pdl_trigger();
    for (int i = 0; i < npre; ++i) load_x(i, i);
    for (int i = npre; i < nkb; ++i) {
      const int s = i % NS;
      const uint32_t ph = (i / NS) & 1;
      if (!mbar_wait(smem_u32(&empty[s]), ph ^ 1, a.err)) { *flag = 1; break; }
      mbar_arrive_expect_tx(smem_u32(&full[s]), S::kStageBytes);
      load_w(i, s);
      load_x(i, s);
    }
  } else {
    float* rs_s = reinterpret_cast<float*>(smem + NS * S::kStageBytes + 256);
    long long* kvdst_s = reinterpret_cast<long long*>(rs_s + BN);
    int* pos_s = reinterpret_cast<int*>(kvdst_s + BN);
    const int tok0s = tok_tile * BN;
    if constexpr (EPI == kEpiQKV) {
      // Positions, page-table rows and the RoPE table are written by kernels
      // that completed before the previous one started: stage them before the
      // dependency wait.
      if (warp >= 2) {
        for (int t = threadIdx.x - 64; t < BN; t += 64) {
          long long dst = -1;
          int p = -1;
          if (tok0s + t < a.M) {
            p = a.pos[tok0s + t];
            const int slot = a.tok_slot[tok0s + t];
            if (slot >= 0) {
              const int lp = p >> 6;
              const int phys = (p >= 0 && p < a.max_ctx && lp < a.pt_stride)
                                   ? a.page_table[static_cast<size_t>(slot) * a.pt_stride + lp] : -1;
              if (phys < 0 || phys >= a.n_pages) atomicExch(a.err, kErrBounds);
              else dst = static_cast<long long>(phys) * 2 * a.Hkv * 4096 + (p & 63) * 64;
            }
          }
          kvdst_s[t] = dst;
          pos_s[t] = p;
          if constexpr (S::kStageRope) {
            float2* cs_s = reinterpret_cast<float2*>(pos_s + BN);
            if (p >= 0 && p < a.max_ctx) {
              const float4* src = reinterpret_cast<const float4*>(a.rope + static_cast<size_t>(p) * 32);
              float4* dstv = reinterpret_cast<float4*>(cs_s + t * 32);
              float4 buf[16];
#pragma unroll
              for (int q = 0; q < 16; ++q) buf[q] = src[q];
#pragma unroll
              for (int q = 0; q < 16; ++q) dstv[q] = buf[q];
            }
          }
        }
      }
    }
    pdl_wait();
    pdl_trigger();
    if (warp >= 2 && a.ssp_in != nullptr) {
      // folded-norm scale from the previous kernel's per-tile sums of h^2
      for (int t = threadIdx.x - 64; t < BN; t += 64) {
        float ss = 0.f;
        if (tok0s + t < a.M) {
          const float* sp = a.ssp_in + static_cast<size_t>(a.x_row0 + tok0s + t) * a.n_ssp;
          float part[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) part[q] = q < a.n_ssp ? sp[q] : 0.f;
#pragma unroll
          for (int q = 0; q < 16; ++q) ss += part[q];
          for (int q = 16; q < a.n_ssp; ++q) ss += sp[q];
        }
        rs_s[t] = rsqrtf(ss * a.inv_d + a.eps);
      }
    }
    if (warp == 1 && lane == 0) {
      // MMA issuer.  Chunked K: chunk c (k-blocks [c*kpc, (c+1)*kpc)) has its
      // accumulator at TMEM column c * BN, fresh at its first k-block.
      constexpr uint32_t idesc = umma_idesc_f16(128, BN);
      for (int i = 0; i < nkb; ++i) {
        const int s = i % NS;
        const uint32_t ph = (i / NS) & 1;
        if (!mbar_wait(smem_u32(&full[s]), ph, a.err)) { *flag = 1; break; }
        tc_fence_after();
        const uint64_t ad = umma_desc_sw128(smem_u32(smA + s * S::kABytes));
        const uint64_t bd = umma_desc_sw128(smem_u32(smB + s * S::kBBytes));
        const uint32_t dst = tmem + static_cast<uint32_t>((i % nchunk) * BN);
        const bool fresh = i < nchunk;
#pragma unroll
        for (int k = 0; k < 4; ++k)
          umma_f16(dst, ad + 2 * k, bd + 2 * k, idesc, (!fresh || k > 0) ? 1u : 0u);
        umma_commit(smem_u32(&empty[s]));
      }
      umma_commit(smem_u32(accum));
    }
  }
  __syncwarp();

  // All four warps: wait for the accumulator, then the epilogue.
  const bool acc_ok = mbar_wait(smem_u32(accum), 0, a.err);
  tc_fence_after();
  const int row = warp * 32 + lane;      // TMEM lane = weight row of the tile
  const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
  const int tok0 = tok_tile * BN;
  // per-token epilogue inputs staged by warps 2-3 during the mainloop; the
  // failure flag is made uniform so every barrier below is reached by all
  const bool failed = __syncthreads_or(!acc_ok || *flag) != 0;
  const float* rs_s = reinterpret_cast<const float*>(smem + NS * S::kStageBytes + 256);
  const long long* kvdst_s = reinterpret_cast<const long long*>(rs_s + BN);
  const int* pos_s = reinterpret_cast<const int*>(kvdst_s + BN);
  const float2* cs_s = S::kStageRope ? reinterpret_cast<const float2*>(pos_s + BN) : nullptr;
  auto rs_of = [&](int c) -> TokMeta {
    return TokMeta{a.ssp_in ? rs_s + c * 32 : nullptr, kvdst_s + c * 32, pos_s + c * 32,
                   cs_s ? cs_s + c * 32 * 32 : nullptr};
  };

  if (a.splits == 1) {
    float* xbuf = reinterpret_cast<float*>(smA);   // pipeline smem is free after the accumulator
    if (!failed) {
      for (int c = 0; c < BN / 32; ++c) {
        if (tok0 + c * 32 >= a.M) break;   // uniform across the CTA
        float v[32];
        if (nchunk == 1) {
          tmem_ld_32x32b_x32(trow + c * 32, v);
        } else {
          // the chunks' partial sums in chunk order from zero: the same sums,
          // in the same order, as split-K across CTAs
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = 0.0f;
          for (int ch = 0; ch < nchunk; ++ch) {
            float w[32];
            tmem_ld_32x32b_x32(trow + ch * BN + c * 32, w);
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] += w[j];
          }
        }
        gemm_epilogue_chunk<BN, EPI, 32>(a, v, row, feat_tile, tok0 + c * 32, 0, 32, xbuf, rs_of(c));
      }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 2) tmem_dealloc(tmem, tmem_cols);
    return;
  }

  if constexpr (S::kClusterOk) {
    if (a.cluster) {
      // Cluster split-K.  CTA q owns tokens [q*per, (q+1)*per) of the tile.
      // Stage this CTA's partials token-major in its own shared memory (slice
      // q contiguous), send slice q to CTA q's receive buffer at position
      // [split] with one bulk copy, and wait for the S slices of our own
      // tokens on recv_bar; then sum them over s = 0..S-1.
      float* recv = reinterpret_cast<float*>(smem + S::recv_offset(NS, EPI));   // [S][per][128]
      float* stage = reinterpret_cast<float*>(smA + S::kXBufBytes);   // [BN][128], after xbuf
      float* xbuf = reinterpret_cast<float*>(smA);
      const int per = BN / a.splits;
      const int ntok = min(BN, a.M - tok0);
      if (!failed) {
        for (int c = 0; c < BN / 32; ++c) {
          if (c * 32 >= ntok) break;
          float v[32];
          tmem_ld_32x32b_x32(trow + c * 32, v);
#pragma unroll
          for (int j = 0; j < 32; ++j) stage[(c * 32 + j) * 128 + row] = v[j];
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncthreads();
      if (warp == 2) tmem_dealloc(tmem, tmem_cols);
      const uint32_t slice_bytes = static_cast<uint32_t>(per * 128 * 4);
      cluster_wait();       // every CTA of the cluster runs: peers' buffers and barriers exist
      if (threadIdx.x == 0) {
        const uint32_t dst_local = smem_u32(recv) + static_cast<uint32_t>(split) * slice_bytes;
        for (int q = 0; q < a.splits; ++q)
          bulk_copy_to_peer(cluster_map(dst_local, static_cast<uint32_t>(q)),
                            smem_u32(stage) + static_cast<uint32_t>(q) * slice_bytes, slice_bytes,
                            cluster_map(smem_u32(recv_bar), static_cast<uint32_t>(q)));
        bulk_commit();
      }
      const bool got = __syncthreads_and(mbar_wait(smem_u32(recv_bar), 0, a.err)) != 0;
      // the epilogue's exchange buffer overlaps `stage`: our outgoing slices
      // must have left it
      if (threadIdx.x == 0) bulk_wait_read_all();
      __syncthreads();
      const int lo = split * per, hi = min(lo + per, ntok);
      if (hi > lo && !failed && got) {
        const int nq = hi - lo;
        if (per <= 8) {
          float v[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) v[q] = 0.0f;
          for (int sp = 0; sp < a.splits; ++sp)
#pragma unroll
            for (int q = 0; q < 8; ++q)
              if (q < nq) v[q] += recv[(sp * per + q) * 128 + row];
          const TokMeta m = rs_of(0);
          const TokMeta tm{m.rs ? m.rs + lo : nullptr, m.kvdst + lo, m.pos + lo,
                           m.cs ? m.cs + lo * 32 : nullptr};
          gemm_epilogue_chunk<BN, EPI, 8>(a, v, row, feat_tile, tok0 + lo, 0, nq, xbuf, tm);
        } else {   // per in {16, 32}: one 32-token chunk
          const int c = lo / 32, jlo = lo - c * 32;
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = 0.0f;
          for (int sp = 0; sp < a.splits; ++sp)
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j >= jlo && j < jlo + nq) v[j] += recv[(sp * per + (j - jlo)) * 128 + row];
          gemm_epilogue_chunk<BN, EPI, 32>(a, v, row, feat_tile, tok0 + c * 32, jlo, jlo + nq, xbuf,
                                           rs_of(c));
        }
      }
      return;
    }
  }

  // global split-K: write this split's partial tile, token-major [BN][128]
  const int tiles = gridDim.x * gridDim.y;
  const int tile = feat_tile * gridDim.x + tok_tile;
  float* mine = a.partial + (static_cast<size_t>(split) * tiles + tile) * (BN * 128);
  if (!failed) {
    for (int c = 0; c < BN / 32; ++c) {
      if (tok0 + c * 32 >= a.M) break;
      float v[32];
      tmem_ld_32x32b_x32(trow + c * 32, v);
#pragma unroll
      for (int j = 0; j < 32; ++j) mine[(c * 32 + j) * 128 + row] = v[j];
    }
  }
  __threadfence();
  tc_fence_before();
  __syncthreads();
  if (warp == 2) tmem_dealloc(tmem, tmem_cols);
  __shared__ int is_last;
  if (threadIdx.x == 0) {
    const int old = atomicAdd(a.counters + tile, 1);
    is_last = (old == a.splits - 1);
    if (is_last) a.counters[tile] = 0;
  }
  __syncthreads();
  if (!is_last || failed) return;
  __threadfence();
  float* xbuf = reinterpret_cast<float*>(smA);
  for (int c = 0; c < BN / 32; ++c) {
    if (tok0 + c * 32 >= a.M) break;
    float v[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = 0.0f;
    for (int s = 0; s < a.splits; ++s) {
      const float* p = a.partial + (static_cast<size_t>(s) * tiles + tile) * (BN * 128);
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] += __ldcg(p + (c * 32 + j) * 128 + row);
    }
    gemm_epilogue_chunk<BN, EPI, 32>(a, v, row, feat_tile, tok0 + c * 32, 0, 32, xbuf, rs_of(c));
  }
}

// ---------------------------------------------------------------------------
// Chunked-K GEMM for wide decode windows.  K is reduced as `chunks` chunks of
// kpc k-blocks, each summed from zero, then the chunks summed in order
// 0..chunks-1 -- the same sums, in the same order, as split-K across CTAs --
// but with one running sum instead of one accumulator per chunk, so the token
// tile can be wide: TMEM holds the running sum (BN columns) and NB = 256 / BN
// - 1 chunk buffers, 256 columns in all, so two CTAs share an SM.
//   warp 4 lane 0   TMA producer (k-blocks in chunk order through the ring)
//   warp 5 lane 0   MMA issuer: chunk c into buffer c % NB, fresh at its first
//                   k-block, then a commit on acc_full[buffer]; a buffer is
//                   reused once the epilogue warps have drained it
//   warps 0-3       drain each chunk as it completes: sum = sum + chunk (the
//                   first chunk: 0 + chunk) in TMEM, then release the buffer;
//                   the last chunk goes from registers to the fused epilogue
// The epilogue warps also stage the per-token epilogue data while the first
// chunk runs.  Every wait is bounded; a failure is made uniform across the
// epilogue warps before their first named barrier.
template <int BN, int EPI>
__global__ void __launch_bounds__(192, 2)
    gemm_chunk_kernel(const __grid_constant__ CUtensorMap tmW,
                      const __grid_constant__ CUtensorMap tmX, const GemmArgs a) {
  using S = GemmShape<BN>;
  constexpr int NB = 256 / BN - 1;            // chunk buffers
  constexpr uint32_t kCols = 256;             // sum at column 0, buffer b at (1 + b) * BN
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* smA = smem;
  const int NS = a.stages;
  uint8_t* smB = smem + NS * S::kABytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NS * S::kStageBytes);
  uint64_t* full = bars;                      // [NS]
  uint64_t* empty = bars + NS;                // [NS]
  uint64_t* acc_full = bars + 2 * NS;         // [NB] chunk in its buffer
  uint64_t* acc_free = acc_full + NB;         // [NB] buffer drained (4 warp arrivals)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_free + NB);
  int* fail_flag = reinterpret_cast<int*>(tmem_slot + 1);
  static_assert((2 * S::kStagesMax + 2 * NB) * 8 + 8 <= 256, "gemm_chunk barriers");

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int tok_tile = blockIdx.x;
  const int feat_tile = blockIdx.y;
  const int nkb = a.K / 64;
  const int nchunk = a.chunks;
  const int kpc = nkb / nchunk;

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
    for (int s = 0; s < NS; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int b = 0; b < NB; ++b) {
      mbar_init(smem_u32(&acc_full[b]), 1);
      mbar_init(smem_u32(&acc_free[b]), 4);
    }
    *fail_flag = 0;
    fence_mbar_init();
  }
  if (warp == 4) tmem_alloc(smem_u32(tmem_slot), kCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 4) {
    if (lane == 0) {
      // TMA producer: the first stages' weight tiles before the dependency wait
      const uint64_t pol_w = l2_policy_evict_first();
      const uint64_t pol_x = l2_policy_evict_last();
      auto load_w = [&](int i, int s) {
        const uint32_t fb = smem_u32(&full[s]);
        if constexpr (EPI == kEpiSwiGLU) {
          tma_load_2d(smem_u32(smA + s * S::kABytes), &tmW, i * 64, feat_tile * 64, fb, pol_w);
          tma_load_2d(smem_u32(smA + s * S::kABytes + 64 * 128), &tmW, i * 64, a.N + feat_tile * 64,
                      fb, pol_w);
        } else {
          tma_load_2d(smem_u32(smA + s * S::kABytes), &tmW, i * 64, feat_tile * 128, fb, pol_w);
        }
      };
      auto load_x = [&](int i, int s) {
        tma_load_2d(smem_u32(smB + s * S::kBBytes), &tmX, i * 64, a.x_row0 + tok_tile * BN,
                    smem_u32(&full[s]), pol_x);
      };
      const int npre = nkb < NS ? nkb : NS;
      for (int i = 0; i < npre; ++i) {
        mbar_arrive_expect_tx(smem_u32(&full[i]), S::kStageBytes);
        load_w(i, i);
      }
      pdl_wait();
      pdl_trigger();
      for (int i = 0; i < npre; ++i) load_x(i, i);
      for (int i = npre; i < nkb; ++i) {
        const int s = i % NS;
        if (!mbar_wait(smem_u32(&empty[s]), ((i / NS) & 1) ^ 1, a.err)) break;
        mbar_arrive_expect_tx(smem_u32(&full[s]), S::kStageBytes);
        load_w(i, s);
        load_x(i, s);
      }
    } else {
      pdl_wait();
      pdl_trigger();
    }
  } else if (warp == 5) {
    pdl_wait();
    pdl_trigger();
    if (lane == 0) {
      // MMA issuer, N = the tile's rows rounded up to 16 (a ragged last tile
      // issues narrower MMAs; its columns past M are never read)
      const int rows = min(BN, a.M - tok_tile * BN);
      const int n_mma = BN <= 16 ? BN : ((rows + 15) / 16) * 16;
      const uint32_t idesc = umma_idesc_f16(128, n_mma < 16 ? 16 : n_mma);
      bool ok = true;
      for (int c = 0; c < nchunk && ok; ++c) {
        const int b = c % NB, u = c / NB;
        if (c >= NB && !mbar_wait(smem_u32(&acc_free[b]), (u - 1) & 1, a.err)) break;
        tc_fence_after();
        const uint32_t dst = tmem + static_cast<uint32_t>((1 + b) * BN);
        for (int k = 0; k < kpc; ++k) {
          const int i = c * kpc + k;
          const int s = i % NS;
          if (!mbar_wait(smem_u32(&full[s]), (i / NS) & 1, a.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = umma_desc_sw128(smem_u32(smA + s * S::kABytes));
          const uint64_t bd = umma_desc_sw128(smem_u32(smB + s * S::kBBytes));
#pragma unroll
          for (int q = 0; q < 4; ++q)
            umma_f16(dst, ad + 2 * q, bd + 2 * q, idesc, (k > 0 || q > 0) ? 1u : 0u);
          umma_commit(smem_u32(&empty[s]));
        }
        if (ok) umma_commit(smem_u32(&acc_full[b]));
      }
    }
  } else {
    // ---- warps 0-3: per-token epilogue data, then drain the chunks
    float* rs_s = reinterpret_cast<float*>(smem + NS * S::kStageBytes + 256);
    long long* kvdst_s = reinterpret_cast<long long*>(rs_s + BN);
    int* pos_s = reinterpret_cast<int*>(kvdst_s + BN);
    float2* cs_s = S::kStageRope ? reinterpret_cast<float2*>(pos_s + BN) : nullptr;
    const int tok0 = tok_tile * BN;
    if constexpr (EPI == kEpiQKV) {
      for (int t = threadIdx.x; t < BN; t += 128) {
        long long dst = -1;
        int p = -1;
        if (tok0 + t < a.M) {
          p = a.pos[tok0 + t];
          const int slot = a.tok_slot[tok0 + t];
          if (slot >= 0) {
            const int lp = p >> 6;
            const int phys = (p >= 0 && p < a.max_ctx && lp < a.pt_stride)
                                 ? a.page_table[static_cast<size_t>(slot) * a.pt_stride + lp] : -1;
            if (phys < 0 || phys >= a.n_pages) atomicExch(a.err, kErrBounds);
            else dst = static_cast<long long>(phys) * 2 * a.Hkv * 4096 + (p & 63) * 64;
          }
        }
        kvdst_s[t] = dst;
        pos_s[t] = p;
        if constexpr (S::kStageRope) {
          if (p >= 0 && p < a.max_ctx) {
            const float4* src = reinterpret_cast<const float4*>(a.rope + static_cast<size_t>(p) * 32);
            float4* dstv = reinterpret_cast<float4*>(cs_s + t * 32);
#pragma unroll 4
            for (int q = 0; q < 16; ++q) dstv[q] = src[q];
          }
        }
      }
    }
    pdl_wait();
    pdl_trigger();
    if (a.ssp_in != nullptr) {
      for (int t = threadIdx.x; t < BN; t += 128) {
        float ss = 0.f;
        if (tok0 + t < a.M) {
          const float* sp = a.ssp_in + static_cast<size_t>(a.x_row0 + tok0 + t) * a.n_ssp;
          float part[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) part[q] = q < a.n_ssp ? sp[q] : 0.f;
#pragma unroll
          for (int q = 0; q < 16; ++q) ss += part[q];
          for (int q = 16; q < a.n_ssp; ++q) ss += sp[q];
        }
        rs_s[t] = rsqrtf(ss * a.inv_d + a.eps);
      }
    }
    const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    const int npiece = min(BN / 32, (a.M - tok0 + 31) / 32);   // 32-token pieces with rows
    bool ok = true;
    for (int c = 0; c + 1 < nchunk && ok; ++c) {
      const int b = c % NB, u = c / NB;
      ok = __all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(&acc_full[b]), u & 1, a.err)) != 0;
      if (!ok) break;
      tc_fence_after();
      const uint32_t buf = trow + static_cast<uint32_t>((1 + b) * BN);
      for (int pc = 0; pc < npiece; ++pc) {
        uint32_t ch[32], sm[32];
        tmem_ld32_nowait(buf + pc * 32, ch);
        if (c > 0) tmem_ld32_nowait(trow + pc * 32, sm);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j)
          sm[j] = __float_as_uint((c > 0 ? __uint_as_float(sm[j]) : 0.0f) + __uint_as_float(ch[j]));
        tmem_st32(trow + pc * 32, sm);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&acc_free[b]));
    }
    if (ok) {
      const int c = nchunk - 1, b = c % NB, u = c / NB;
      ok = __all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(&acc_full[b]), u & 1, a.err)) != 0;
    }
    if (!ok && lane == 0) atomicExch(fail_flag, 1);
    asm volatile("bar.sync 3, 128;" ::: "memory");
    const bool failed = *reinterpret_cast<volatile int*>(fail_flag) != 0;
    if (!failed) {
      tc_fence_after();
      const int c = nchunk - 1, b = c % NB;
      const uint32_t buf = trow + static_cast<uint32_t>((1 + b) * BN);
      float* xbuf = reinterpret_cast<float*>(smA);   // every MMA has retired: the ring is free
      const float* rs_c = a.ssp_in ? rs_s : nullptr;
      for (int pc = 0; pc < npiece; ++pc) {
        uint32_t ch[32], sm[32];
        tmem_ld32_nowait(buf + pc * 32, ch);
        if (c > 0) tmem_ld32_nowait(trow + pc * 32, sm);
        tmem_wait_ld();
        float v[32];
#pragma unroll
        for (int j = 0; j < 32; ++j)
          v[j] = (c > 0 ? __uint_as_float(sm[j]) : 0.0f) + __uint_as_float(ch[j]);
        const TokMeta tm{rs_c ? rs_c + pc * 32 : nullptr, kvdst_s + pc * 32, pos_s + pc * 32,
                         cs_s ? cs_s + pc * 32 * 32 : nullptr};
        gemm_epilogue_chunk<BN, EPI, 32>(a, v, warp * 32 + lane, feat_tile, tok0 + pc * 32, 0, 32,
                                         xbuf, tm);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 4) tmem_dealloc(tmem, kCols);
}

}  // namespace gs
