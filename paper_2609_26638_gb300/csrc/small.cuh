// small.cuh -- bandwidth-trivial kernels of the round: window build, forcing,
// embedding gather, RMSNorm, RoPE + paged KV write, accept/commit.
#pragma once
#include "ptx.cuh"

namespace gs {

// Per-sequence device state, struct of arrays indexed by slot.
struct SeqStateDev {
  int32_t* seq_len;  // cached slots (causal states of committed tokens except x0)
  int32_t* x0;       // boundary token
  int32_t* n_out;    // committed tokens, x0 included
  int32_t* max_new;  // cap on n_out
  int32_t* done;     // 1 once EOS / cap reached
  int32_t* rounds;   // rounds run since prefill
};

// Which window a decode forward builds (paper Appendix steps Draft / Verify forward).
struct WindowArgs {
  const int32_t* slots;  // [n_seq]
  int n_seq, K, W;       // W = K + 1
  int mask_id, vocab;
  SeqStateDev st;
  int32_t* tok;          // [n_seq * W] input token ids
  int32_t* pos;          // [n_seq * W] absolute slot / RoPE position
  int32_t* lim;          // [n_seq * W] inclusive key limit
  int32_t* tok_slot;     // [n_seq * W] page-table row, -1 = do not write KV
  int32_t* blk_slot;     // [n_seq]
  int32_t* blk_active;   // [n_seq]
  // verify only
  const unsigned long long* draft_packed;  // [n_seq * W] draft argmax keys
  int32_t* draft_tok;    // [n_seq * W] a0, d_1..d_K (draft argmax)
  int32_t* verify_in;    // [n_seq * W] a0, d_1..d_K after forcing
  const int32_t* teacher;
  long long teacher_stride;
  const int32_t* L_sched;
  long long L_stride;
  int* err;
};

// Draft window: [x0, [M] x K] at slots n..n+K; row 0 sees keys 0..n, mask rows 0..n+K.
__global__ void window_draft_kernel(WindowArgs a) {
  pdl_wait();
  pdl_trigger();
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= a.n_seq * a.W) return;
  const int b = idx / a.W, i = idx % a.W;
  const int slot = a.slots[b];
  const bool active = a.st.done[slot] == 0;
  const int n = a.st.seq_len[slot];
  a.tok[idx] = i == 0 ? a.st.x0[slot] : a.mask_id;
  a.pos[idx] = n + i;
  a.lim[idx] = i == 0 ? n : n + a.K;
  a.tok_slot[idx] = active ? slot : -1;
  if (i == 0) {
    a.blk_slot[b] = slot;
    a.blk_active[b] = active ? 1 : 0;
  }
}

// Verify window: [a0, d_1..d_K] at slots n+1..n+K+1, token-level causal.
// Applies the forcing hook to the drafts when a teacher is given.
__global__ void window_verify_kernel(WindowArgs a) {
  pdl_wait();
  pdl_trigger();
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= a.n_seq * a.W) return;
  const int b = idx / a.W, i = idx % a.W;
  const int slot = a.slots[b];
  const int n = a.st.seq_len[slot];
  int t = argmax_key_index(a.draft_packed[idx]);
  a.draft_tok[idx] = t;
  if (a.teacher != nullptr && i >= 1 && a.st.done[slot] == 0) {
    const int r = a.st.rounds[slot];
    int L = 0;
    if (r < a.L_stride) L = a.L_sched[b * a.L_stride + r];
    else atomicExch(a.err, kErrBounds);
    const long long base = static_cast<long long>(b) * a.teacher_stride;
    if (i <= L) {
      const long long p = n + 1 + i;
      if (p < a.teacher_stride) t = a.teacher[base + p];
      else atomicExch(a.err, kErrBounds);
    } else if (i == L + 1) {
      const long long p = n + 1 + i;
      if (p < a.teacher_stride) t = (a.teacher[base + p] + 1) % a.vocab;
      else atomicExch(a.err, kErrBounds);
    }
  }
  if (t < 0 || t >= a.vocab) {
    atomicExch(a.err, kErrBounds);
    t = 0;
  }
  a.verify_in[idx] = t;
  a.tok[idx] = t;
  a.pos[idx] = n + 1 + i;
  a.lim[idx] = n + 1 + i;
  a.tok_slot[idx] = a.st.done[slot] == 0 ? slot : -1;
}

// Accept + commit + rollback (paper Appendix steps Accept / Cache update /
// Next round): A = longest prefix with d_j == a_j; commit a0, d_1..d_A,
// a_{A+1}, cut at EOS / output cap; seq_len <- n + A + 2; x0 <- a_{A+1}.
struct AcceptArgs {
  const int32_t* slots;
  int n_seq, K, W, eos;
  SeqStateDev st;
  const int32_t* verify_in;                 // [n_seq * W]
  const unsigned long long* verify_packed;  // [n_seq * W]
  int32_t* verify_tok;                      // [n_seq * W] a_1..a_{K+1}
  int32_t* out_tok;                         // [n_seq, K+2]
  int32_t* out_cnt;
  int32_t* out_done;
};

__global__ void accept_commit_kernel(AcceptArgs a) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= a.n_seq) return;
  const int slot = a.slots[b];
  const int W = a.W;
  for (int i = 0; i < W; ++i) a.verify_tok[b * W + i] = argmax_key_index(a.verify_packed[b * W + i]);
  if (a.st.done[slot]) {
    a.out_cnt[b] = 0;
    a.out_done[b] = 1;
    return;
  }
  const int* vin = a.verify_in + b * W;   // a0, d_1..d_K
  const int* vt = a.verify_tok + b * W;   // a_1..a_{K+1}
  int A = 0;
  while (A < a.K && vin[1 + A] == vt[A]) ++A;
  int n_out = a.st.n_out[slot];
  const int cap = a.st.max_new[slot];
  int cnt = 0, done = 0;
  for (int j = 0; j < A + 2; ++j) {
    const int t = j == 0 ? vin[0] : (j <= A ? vin[j] : vt[A]);
    a.out_tok[b * (a.K + 2) + cnt++] = t;
    ++n_out;
    if (t == a.eos || n_out >= cap) {
      done = 1;
      break;
    }
  }
  a.st.seq_len[slot] = a.st.seq_len[slot] + A + 2;
  a.st.x0[slot] = vt[A];
  a.st.n_out[slot] = n_out;
  a.st.done[slot] = done;
  a.st.rounds[slot] = a.st.rounds[slot] + 1;
  a.out_cnt[b] = cnt;
  a.out_done[b] = done;
}

// After a prefill: x0 = argmax at the last prefix position (paper Appendix step State).
__global__ void prefill_finish_kernel(const unsigned long long* packed, SeqStateDev st, int slot,
                                      int P, int max_new, int eos, int32_t* x0_out) {
  pdl_wait();
  pdl_trigger();
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  const int x0 = argmax_key_index(packed[0]);
  st.seq_len[slot] = P;
  st.x0[slot] = x0;
  st.n_out[slot] = 1;
  st.max_new[slot] = max_new;
  st.done[slot] = (x0 == eos || max_new <= 1) ? 1 : 0;
  st.rounds[slot] = 0;
  if (x0_out) *x0_out = x0;
}

__global__ void seq_restore_kernel(SeqStateDev st, int slot, int seq_len, int x0, int n_out,
                                   int max_new, int done, int rounds) {
  pdl_wait();
  pdl_trigger();
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  st.seq_len[slot] = seq_len;
  st.x0[slot] = x0;
  st.n_out[slot] = n_out;
  st.max_new[slot] = max_new;
  st.done[slot] = done;
  st.rounds[slot] = rounds;
}

// Prefill chunk positions: token t at slot p0 + t, causal limit p0 + t.
__global__ void prefill_window_kernel(int T, int p0, int slot, int32_t* pos, int32_t* lim,
                                      int32_t* tok_slot) {
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  pos[t] = p0 + t;
  lim[t] = p0 + t;
  tok_slot[t] = slot;
}

// h[t] = E[tok[t]] (fp32), or the visual row for t < n_vis.  d % 8 == 0.
__global__ void embed_kernel(const int32_t* tok, const __nv_bfloat16* E, const __nv_bfloat16* vis,
                             int n_vis, int T, int d, int vocab, float* h, int* err) {
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x;
  if (t >= T) return;
  const __nv_bfloat16* src;
  if (t < n_vis) {
    src = vis + static_cast<size_t>(t) * d;
  } else {
    int id = tok[t - n_vis];
    if (id < 0 || id >= vocab) {
      if (threadIdx.x == 0) atomicExch(err, kErrBounds);
      id = 0;
    }
    src = E + static_cast<size_t>(id) * d;
  }
  for (int c = threadIdx.x * 8; c < d; c += blockDim.x * 8) {
    const uint4 raw = *reinterpret_cast<const uint4*>(src + c);
    const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&raw);
    float4 lo, hi;
    float2 f;
    f = __bfloat1622float2(p[0]); lo.x = f.x; lo.y = f.y;
    f = __bfloat1622float2(p[1]); lo.z = f.x; lo.w = f.y;
    f = __bfloat1622float2(p[2]); hi.x = f.x; hi.y = f.y;
    f = __bfloat1622float2(p[3]); hi.z = f.x; hi.w = f.y;
    float* dst = h + static_cast<size_t>(t) * d + c;
    *reinterpret_cast<float4*>(dst) = lo;
    *reinterpret_cast<float4*>(dst + 4) = hi;
  }
}

// RMSNorm, one warp per row: y = x / sqrt(mean(x^2) + eps) * gain -> bf16.
// Optionally zeroes argmax keys of the row (the LM-head argmax accumulator).
__global__ void rmsnorm_kernel(const float* x, const __nv_bfloat16* gain, __nv_bfloat16* y, int T,
                               int d, float eps, unsigned long long* reset_keys) {
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const float* xr = x + static_cast<size_t>(row) * d;
  float ss = 0.f;
  for (int c = lane * 4; c < d; c += 128) {
    const float4 v = *reinterpret_cast<const float4*>(xr + c);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
  const float r = rsqrtf(ss / static_cast<float>(d) + eps);
  __nv_bfloat16* yr = y + static_cast<size_t>(row) * d;
  for (int c = lane * 4; c < d; c += 128) {
    const float4 v = *reinterpret_cast<const float4*>(xr + c);
    const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(gain + c);
    const float2 ga = __bfloat1622float2(g2[0]), gb = __bfloat1622float2(g2[1]);
    __nv_bfloat162 o0 = __floats2bfloat162_rn(v.x * r * ga.x, v.y * r * ga.y);
    __nv_bfloat162 o1 = __floats2bfloat162_rn(v.z * r * gb.x, v.w * r * gb.y);
    uint2 pk;
    pk.x = *reinterpret_cast<uint32_t*>(&o0);
    pk.y = *reinterpret_cast<uint32_t*>(&o1);
    *reinterpret_cast<uint2*>(yr + c) = pk;
  }
  if (reset_keys != nullptr && lane == 0) reset_keys[row] = 0ull;
}

// RoPE (rotate-half, pairs (i, i+32)) on q and k at absolute positions, then
// k and v written into the paged cache at the token's slot.  One warp per
// (token, head) of the fused qkv row; lane i owns dims i and i+32.
struct RopeKvArgs {
  const __nv_bfloat16* qkv;   // [T, (Hq + 2 Hkv) * 64]
  const int32_t* pos;         // [T]
  const int32_t* tok_slot;    // [T] page-table row or -1
  const float2* rope;         // [max_ctx][32] (cos, sin)
  __nv_bfloat16* q_out;       // [T, Hq, 64]
  __nv_bfloat16* kv;          // page pool of this layer: [pages][2][Hkv][64][64]
  const int32_t* page_table;
  int pt_stride, n_pages, T, Hq, Hkv, max_ctx;
  int* err;
};

__global__ void rope_kv_kernel(RopeKvArgs a) {
  pdl_wait();
  pdl_trigger();
  const int warps_per_block = blockDim.x >> 5;
  const int gw = blockIdx.x * warps_per_block + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int nh = a.Hq + 2 * a.Hkv;
  if (gw >= a.T * nh) return;
  const int t = gw / nh, hh = gw % nh;
  const int p = a.pos[t];
  const __nv_bfloat16* src = a.qkv + static_cast<size_t>(t) * nh * 64 + hh * 64;
  const float x1 = __bfloat162float(src[lane]);
  const float x2 = __bfloat162float(src[lane + 32]);
  float y1 = x1, y2 = x2;
  if (hh < a.Hq + a.Hkv) {
    if (p < 0 || p >= a.max_ctx) {
      if (lane == 0) atomicExch(a.err, kErrBounds);
      return;
    }
    const float2 cs = a.rope[static_cast<size_t>(p) * 32 + lane];
    y1 = x1 * cs.x - x2 * cs.y;
    y2 = x2 * cs.x + x1 * cs.y;
  }
  if (hh < a.Hq) {
    __nv_bfloat16* dst = a.q_out + (static_cast<size_t>(t) * a.Hq + hh) * 64;
    dst[lane] = __float2bfloat16_rn(y1);
    dst[lane + 32] = __float2bfloat16_rn(y2);
    return;
  }
  const int slot = a.tok_slot[t];
  if (slot < 0) return;
  const int lp = p >> 6;
  if (lp >= a.pt_stride) {
    if (lane == 0) atomicExch(a.err, kErrBounds);
    return;
  }
  const int phys = a.page_table[static_cast<size_t>(slot) * a.pt_stride + lp];
  if (phys < 0 || phys >= a.n_pages) {
    if (lane == 0) atomicExch(a.err, kErrBounds);
    return;
  }
  const int is_v = hh >= a.Hq + a.Hkv;
  const int kh = is_v ? hh - a.Hq - a.Hkv : hh - a.Hq;
  __nv_bfloat16* dst = a.kv + ((((static_cast<size_t>(phys) * 2 + is_v) * a.Hkv + kh) * 64 +
                                (p & 63)) * 64);
  dst[lane] = __float2bfloat16_rn(y1);
  dst[lane + 32] = __float2bfloat16_rn(y2);
}

// cos/sin table: angle p * theta^(-2i/64), computed in double precision.
__global__ void rope_table_kernel(float2* tab, int max_ctx, double theta) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= max_ctx * 32) return;
  const int p = idx / 32, i = idx % 32;
  const double inv = pow(theta, -2.0 * i / 64.0);
  const double ang = static_cast<double>(p) * inv;
  tab[idx] = make_float2(static_cast<float>(cos(ang)), static_cast<float>(sin(ang)));
}

__global__ void copy_i32_kernel(const int32_t* src, int32_t* dst, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) dst[i] = src[i];
}

}  // namespace gs
