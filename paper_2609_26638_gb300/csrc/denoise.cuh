// denoise.cuh -- kernels of the confidence-thresholded denoising loop: direct
// block-diffusion decoding (paper Appendix "Direct Block-Diffusion Decoding")
// and multi-step drafting (Sec. 6 "Draft Schedule", Fig. "Multi-step drafting
// versus one-shot drafting").
//
// Both refine a window [x0, P_1 .. P_{W-1}] at slots n .. n+W-1 with the
// hybrid mask of the draft forward (the boundary row x0 causal to the cache,
// the placeholder rows bidirectional inside the window).  Under the shifted
// alignment, row i predicts position i+1 (slot n+1+i); placeholder P_i holds
// the token fixed for prediction i-1, or [M] while it is open.  n_pred
// predictions take part: W-1 = B for a diffusion block (row B's prediction
// points past the block), W = K+1 for a draft of K masks (prediction K has no
// placeholder).  Each step reveals every open prediction whose probability
// exceeds tau, or, if none does, the single most confident one (ties to the
// lowest position); the loop ends when no prediction is open.
//
// A step's confidence is the softmax probability of the row's argmax token,
// 1 / sum_v exp(logit_v - max), formed from the LM head's per-tile partials
// (tile max, sum of exp over the tile) in tile order, so a row's value does
// not depend on the batch.
#pragma once
#include "small.cuh"

namespace gs {

struct DenoiseArgs {
  const int32_t* slots;   // [n_seq]
  int n_seq, W, n_pred;   // window rows, predictions that take part (<= W)
  int mask_id, vocab, eos;
  float tau;              // reveal threshold (tau_c or tau_d)
  SeqStateDev st;
  // per slot, [slot * W_max + i]: token fixed for prediction i, -1 while open
  int32_t* fixed;
  int W_max;
  int32_t* live;          // [slot] 1 while the sequence still has open predictions
  int32_t* part;          // [slot] 1 if the sequence takes part in this call
  int32_t* steps;         // [slot] denoising steps of this call
  int32_t* iter;          // loop iterations run (device counter)
  // window descriptors (as WindowArgs)
  int32_t* tok;
  int32_t* pos;
  int32_t* lim;
  int32_t* tok_slot;
  int32_t* blk_slot;
  int32_t* blk_active;
  // the step's LM head: argmax keys [n_seq * W] and softmax partials
  const unsigned long long* packed;
  const float2* lse_part;
  int lse_tiles;
  int* err;
  cudaGraphConditionalHandle cond;
  // block diffusion commit
  int32_t* out_tok;       // [n_seq, n_pred]
  int32_t* out_cnt;
  int32_t* out_done;
  int32_t* out_steps;     // [n_seq] or null
};

// Opens every prediction of the sequences that take part (not done).
__global__ void denoise_init_kernel(DenoiseArgs a) {
  const int b = blockIdx.x;
  if (b >= a.n_seq) return;
  const int slot = a.slots[b];
  const int take = a.st.done[slot] == 0;
  for (int i = threadIdx.x; i < a.W_max; i += blockDim.x)
    a.fixed[static_cast<size_t>(slot) * a.W_max + i] = -1;
  if (threadIdx.x == 0) {
    a.live[slot] = take;
    a.part[slot] = take;
    a.steps[slot] = 0;
    if (b == 0) *a.iter = 0;
  }
}

// Window of one denoising step: [x0, P_1..P_{W-1}] at slots n..n+W-1; row 0
// sees keys 0..n, placeholder rows 0..n+W-1.  Sequences with nothing open
// write no KV and their attention is skipped.
__global__ void denoise_window_kernel(DenoiseArgs a) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= a.n_seq * a.W) return;
  const int b = idx / a.W, i = idx % a.W;
  const int slot = a.slots[b];
  const int n = a.st.seq_len[slot];
  const int live = a.live[slot];
  int t = a.st.x0[slot];
  if (i > 0) {
    const int f = a.fixed[static_cast<size_t>(slot) * a.W_max + i - 1];
    t = f >= 0 ? f : a.mask_id;
  }
  a.tok[idx] = t;
  a.pos[idx] = n + i;
  a.lim[idx] = i == 0 ? n : n + a.W - 1;
  a.tok_slot[idx] = live ? slot : -1;
  if (i == 0) {
    a.blk_slot[b] = slot;
    a.blk_active[b] = live;
  }
}

// One CTA per sequence: the confidence of every open prediction, then the
// reveal rule.  Warp w takes the open rows w, w+4, ...; a row's partials are
// summed by its warp in a fixed lane-strided order.
__global__ void __launch_bounds__(128) denoise_reveal_kernel(DenoiseArgs a) {
  __shared__ float conf[256];
  __shared__ int tokv[256];
  const int b = blockIdx.x;
  if (b >= a.n_seq) return;
  const int slot = a.slots[b];
  if (a.live[slot] == 0) return;
  int32_t* fixed = a.fixed + static_cast<size_t>(slot) * a.W_max;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = warp; i < a.n_pred; i += 4) {
    if (fixed[i] >= 0) continue;   // uniform across the warp
    const int row = b * a.W + i;
    const unsigned long long key = a.packed[row];
    const float mx = argmax_key_value(key);
    const float2* lp = a.lse_part + static_cast<size_t>(row) * a.lse_tiles;
    float s = 0.f;
    for (int t = lane; t < a.lse_tiles; t += 32) {
      const float2 p = lp[t];
      s += p.y * expf(p.x - mx);
    }
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, m);
    if (lane == 0) {
      conf[i] = 1.0f / s;
      int tk = argmax_key_index(key);
      if (tk < 0 || tk >= a.vocab) {
        atomicExch(a.err, kErrBounds);
        tk = 0;
      }
      tokv[i] = tk;
    }
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  int n_above = 0, best = -1, open = 0;
  for (int i = 0; i < a.n_pred; ++i) {
    if (fixed[i] >= 0) continue;
    ++open;
    if (conf[i] > a.tau) ++n_above;
    if (best < 0 || conf[i] > conf[best]) best = i;
  }
  for (int i = 0; i < a.n_pred; ++i) {
    if (fixed[i] >= 0) continue;
    if (n_above > 0 ? conf[i] > a.tau : i == best) {
      fixed[i] = tokv[i];
      --open;
    }
  }
  a.steps[slot] += 1;
  if (open == 0) a.live[slot] = 0;
}

// Loop condition: another step while any sequence has open predictions.  A
// step reveals at least one prediction per live sequence, so n_pred steps
// finish every block; a sequence still open after that raises the error word
// and the loop ends (the iteration count is bounded whatever happens).
__global__ void denoise_cond_kernel(DenoiseArgs a) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  int any = 0;
  for (int b = 0; b < a.n_seq; ++b) any |= a.live[a.slots[b]];
  const int it = ++(*a.iter);
  if (any && it >= a.n_pred) {
    atomicExch(a.err, kErrBounds);
    any = 0;
  }
  cudaGraphSetConditional(a.cond, any ? 1u : 0u);
}

// Cache-write window of a completed block: [x0, y_1..y_B] at slots n..n+B,
// token-level causal (row i sees keys 0..n+i).  Only its KV writes matter.
__global__ void block_write_window_kernel(DenoiseArgs a) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= a.n_seq * a.W) return;
  const int b = idx / a.W, i = idx % a.W;
  const int slot = a.slots[b];
  const int n = a.st.seq_len[slot];
  const int take = a.part[slot];
  a.tok[idx] = i == 0 ? a.st.x0[slot] : a.fixed[static_cast<size_t>(slot) * a.W_max + i - 1];
  a.pos[idx] = n + i;
  a.lim[idx] = n + i;
  a.tok_slot[idx] = take ? slot : -1;
  if (i == 0) {
    a.blk_slot[b] = slot;
    a.blk_active[b] = take;
  }
}

// Commit a completed block: y_1..y_B, cut at the first stop token or at the
// output cap; seq_len <- n + B (the causal states of x0, y_1..y_{B-1}),
// x0 <- y_B.
__global__ void block_commit_kernel(DenoiseArgs a) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= a.n_seq) return;
  const int slot = a.slots[b];
  if (a.out_steps) a.out_steps[b] = a.steps[slot];
  if (!a.part[slot]) {
    a.out_cnt[b] = 0;
    a.out_done[b] = 1;
    return;
  }
  const int32_t* y = a.fixed + static_cast<size_t>(slot) * a.W_max;
  const int B = a.n_pred;
  int n_out = a.st.n_out[slot];
  const int cap = a.st.max_new[slot];
  int cnt = 0, done = 0;
  for (int j = 0; j < B; ++j) {
    const int t = y[j];
    a.out_tok[b * B + cnt++] = t;
    ++n_out;
    if (t == a.eos || n_out >= cap) {
      done = 1;
      break;
    }
  }
  a.st.seq_len[slot] = a.st.seq_len[slot] + B;
  a.st.x0[slot] = y[B - 1];
  a.st.n_out[slot] = n_out;
  a.st.done[slot] = done;
  a.st.rounds[slot] = a.st.rounds[slot] + 1;
  a.out_cnt[b] = cnt;
  a.out_done[b] = done;
}

}  // namespace gs
