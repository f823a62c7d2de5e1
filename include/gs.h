/*
 * gs.h -- C ABI of libgs: greedy self-speculative draft/verify decoding with a
 * shared-parameter AR / block-diffusion decoder on one GB300 (sm_103a).
 *
 * The method (paper Sec. 4.3 "Self-Speculative Decoding", Fig. "Self-speculative
 * decoding", Appendix "Self-Speculative Decoding and KV-Cache Update"): every
 * round runs one DRAFT forward over [x0, [M] x K] with the hybrid mask (the
 * boundary row x0 causal to the cache, the K mask rows bidirectional inside
 * the window), then one VERIFY forward over [a0, d_1..d_K] with token-level
 * causal attention, accepts the longest prefix with d_j == a_j, commits
 * a0, d_1..d_A, a_{A+1} and rolls the KV cache back to the accepted prefix.
 * The first boundary x0 is the argmax at the prefill's last position.
 *
 * Conventions shared by every entry point
 *  - Device pointers are CUDA global-memory addresses on the current device;
 *    host pointers are ordinary process memory.  Each argument says which.
 *  - The caller owns every buffer it passes (weights, workspace, inputs,
 *    outputs) and the stream.  After gs_create the library allocates no
 *    device memory; it carves everything from the caller's workspace.
 *  - Work is enqueued asynchronously on the handle's stream unless stated.
 *  - bf16 tensors are bfloat16 bit patterns, fp16 tensors IEEE binary16
 *    bit patterns; all row-major.
 *  - Arithmetic: the model's weights arrive as bf16; gs_create re-encodes each
 *    matrix as an fp16 copy scaled by a power of two (exact for every weight
 *    whose magnitude is above 2^-31 of the tensor's largest).  Activations
 *    between kernels and the KV cache are fp16 (11 significant bits, against
 *    8 for bf16); every contraction accumulates in fp32; the residual stream
 *    and the softmax statistics are fp32.  A kernel that would store a value
 *    beyond the fp16 range raises the device error word (GS_ERR_DEVICE_CHECK).
 *  - Return value: GS_OK (0) or one of the GS_ERR_* codes below; the message
 *    of the last failure is available from gs_last_error().  Kernel-side
 *    checks (slot ids, token ids, bounded waits) raise a device error word
 *    that gs_sync_check() turns into GS_ERR_DEVICE_CHECK / GS_ERR_TIMEOUT.
 */
#ifndef GS_H_
#define GS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
  GS_OK = 0,
  GS_ERR_INVALID_ARG = 1,   /* bad pointer, size, slot or config value        */
  GS_ERR_OOM = 2,           /* workspace too small / KV page pool exhausted    */
  GS_ERR_UNSUPPORTED = 3,   /* valid request the library does not implement   */
  GS_ERR_CUDA = 4,          /* a CUDA runtime call failed                      */
  GS_ERR_DEVICE_CHECK = 5,  /* a kernel's bounds check fired                   */
  GS_ERR_TIMEOUT = 6        /* a kernel's bounded wait ran out                 */
};

/* Acceptance rule (paper Sec. 3 "Speculative Decoding"): greedy accepts drafts
 * while they equal the verifier's argmax; stochastic is the standard
 * acceptance-rejection rule of speculative sampling, which preserves the
 * target distribution (named by the paper, not used in its experiments):
 * a0 and the drafts are sampled at the handle's temperature (gs_set_sampling)
 * from the draft rows, d_j is accepted while r_j < P_j(d_j) / q_j(d_j), the
 * first rejected position takes a sample of max(0, P_j - q_j), a fully
 * accepted draft a bonus sample of P_{K+1}. */
typedef enum { GS_ACCEPT_GREEDY = 0, GS_ACCEPT_STOCHASTIC = 1 } gs_accept_rule;

/* Decoder shape and capacity.  The paper does not print the architecture; the
 * library implements a pre-norm decoder: RMSNorm (learned gain, eps) ->
 * grouped-query attention with rotate-half RoPE on all head dims at absolute
 * positions -> RMSNorm -> SwiGLU FFN; untied input/output embeddings, no
 * biases.  Requirements: head_dim 64, n_heads % n_kv_heads == 0, n_heads and
 * n_kv_heads even (a 128-row projection tile holds two whole heads),
 * d_model % 128 == 0, d_ffn % 64 == 0, vocab % 128 == 0. */
typedef struct {
  int n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ffn, vocab;
  float rope_theta, rms_eps;
  int mask_token_id;   /* the [M] embedding row (paper Sec. 4, "AR-to-Diffusion Conversion") */
  int eos_token_id;    /* stop token, -1 = none (Appendix step "Next round")              */
  int max_batch;       /* sequence slots                                                  */
  int max_ctx;         /* slots one sequence may reserve: prefix + max_new + max_K + 2   */
  int max_K;           /* largest block size a round may use                              */
  int max_prefill;     /* tokens per prefill chunk (longer prefixes run in chunks)        */
  int kv_pages;        /* 64-token pages in the KV pool; 0 = max_batch * ceil(max_ctx/64) */
  int split_pages;     /* attention pages per work item (decode); 0 = automatic           */
} gs_config;

/* Weights: device pointers to bf16 arrays owned by the caller, row-major
 * [out_features, in_features].  Per-layer fields are HOST arrays of n_layers
 * device pointers (copied by gs_create).
 *   embed [vocab, d]   lm_head [vocab, d]   final_norm [d]
 *   attn_norm [d]   w_qkv [(Hq + 2 Hkv) * 64, d]  (q heads, then k heads, then v heads)
 *   w_o [d, Hq * 64]   ffn_norm [d]   w_gate_up [2 d_ffn, d] (gate rows, then up rows)
 *   w_down [d, d_ffn]
 * Every pointer must be 16-byte aligned. */
typedef struct {
  const void *embed, *lm_head, *final_norm;
  const void *const *attn_norm, *const *w_qkv, *const *w_o,
             *const *ffn_norm, *const *w_gate_up, *const *w_down;
} gs_weights;

/* Forced acceptance (benchmark hook, not in the paper).  After the draft
 * argmax, for the sequence in slot s at round r with L = L_sched[row * L_stride + r]
 * (row = the sequence's index in this call's slot list, r = the number of
 * rounds the sequence has run since its prefill):
 *   d_j := teacher[row * teacher_stride + n + 1 + j]    for 1 <= j <= L
 *   d_{L+1} := (teacher[row * teacher_stride + n + 2 + L] + 1) mod vocab  if L < K
 * where n is the sequence's cached length at the round's start and teacher[p]
 * is the greedy token at absolute slot p.  All pointers are device int32. */
typedef struct {
  const int32_t *teacher;
  int64_t teacher_stride;
  const int32_t *L_sched;
  int64_t L_stride;
} gs_force;

/* Optional per-round diagnostics (device pointers, any may be NULL).  A round
 * given a non-NULL gs_debug runs outside the CUDA-graph cache.
 *   draft_tok  int32 [n_seq, K+1]   argmax of the draft rows (a0, d_1..d_K)
 *   verify_in  int32 [n_seq, K+1]   verify inputs after forcing (a0, d_1..d_K)
 *   verify_tok int32 [n_seq, K+1]   argmax of the verify rows (a_1..a_{K+1})
 *   draft_logits / verify_logits fp32 [n_seq, K+1, vocab] */
typedef struct {
  int32_t *draft_tok, *verify_in, *verify_tok;
  float *draft_logits, *verify_logits;
} gs_debug;

typedef struct gs_handle gs_handle;

/* Bytes of device workspace gs_create needs for this config (fp16 weight
 * copies, KV page pool, page table, per-sequence state, activations, split
 * scratch).  0 if the config is invalid. */
size_t gs_workspace_bytes(const gs_config *cfg);

/* Build a handle.  cfg, w: host structs (copied).  workspace: device memory of
 * at least gs_workspace_bytes(cfg) bytes, 256-byte aligned, owned by the
 * caller and not touched by anyone else until gs_destroy.  stream: a
 * cudaStream_t (NULL = legacy default stream).  Zeroes the workspace, writes
 * the scaled fp16 copies of the weight matrices into it (the caller's bf16
 * matrices are not read again; embed and the norm gains are read at every
 * forward) and builds the TMA descriptors; synchronises the stream before
 * returning.
 * Errors: GS_ERR_INVALID_ARG, GS_ERR_UNSUPPORTED (shape), GS_ERR_OOM
 * (workspace too small), GS_ERR_CUDA. */
int gs_create(const gs_config *cfg, const gs_weights *w, void *workspace, size_t ws_bytes,
              void *stream, gs_handle **out);

/* Release the handle (graphs, host tables).  Frees no caller memory. */
int gs_destroy(gs_handle *h);

/* Message of the last failure on this handle ("" if none).  NULL handle gives
 * the last failure of gs_create in this thread. */
const char *gs_last_error(gs_handle *h);

/* Prefill (paper Appendix step "State"; Sec. 3 task formulation: image I and
 * prompt c).  Reserves KV pages for n_vis + n_text + max_new + max_K + 2
 * slots in sequence slot `slot` (freeing whatever the slot held), runs a
 * causal forward over the visual rows then the text tokens, sets the cached
 * length to P = n_vis + n_text and the boundary x0 to the argmax at position
 * P-1, which is the first committed output token.
 *   vis_emb  device bf16 [n_vis, d_model] (may be NULL when n_vis == 0)
 *   text     device int32 [n_text], ids in [0, vocab)
 *   max_new  cap on committed output tokens, x0 included (>= 1)
 *   x0_out   device int32 [1] or NULL
 * Errors: GS_ERR_INVALID_ARG, GS_ERR_OOM (pool exhausted or ctx too long). */
int gs_prefill(gs_handle *h, int slot, const void *vis_emb, int n_vis, const int32_t *text,
               int n_text, int max_new, int32_t *x0_out);

/* One self-speculative round for n_seq sequences (paper Appendix steps Draft
 * forward / Verify forward / Accept / Cache update / Next round).
 *   slots    device int32 [n_seq], distinct prefilled slots
 *   K        block size, 0 <= K <= max_K (K = 0 is two plain AR steps)
 *   rule     GS_ACCEPT_GREEDY, or GS_ACCEPT_STOCHASTIC (sampling at the
 *            handle's temperature and seed, see gs_set_sampling)
 *   force    NULL for natural drafting, else the forcing hook above (greedy only)
 *   out_tok  device int32 [n_seq, K+2]: committed tokens of this round
 *   out_cnt  device int32 [n_seq]: how many (0 for a sequence already done)
 *   out_done device int32 [n_seq]: 1 once the sequence hit EOS or max_new
 *   dbg      NULL, or diagnostics (see gs_debug)
 * Rounds with the same (n_seq, K, pointers) replay one cached CUDA graph; no
 * host synchronisation happens inside or between rounds. */
int gs_round(gs_handle *h, const int32_t *slots, int n_seq, int K, int rule, const gs_force *force,
             int32_t *out_tok, int32_t *out_cnt, int32_t *out_done, const gs_debug *dbg);

/* Sampling parameters of GS_ACCEPT_STOCHASTIC rounds (host values, kept by
 * the handle).  temperature > 0: tokens are sampled from softmax(logits / T).
 * seed: the 64-bit key of Philox4x32-10 (Salmon et al., SC 2011), whose
 * counter is (vocabulary entry / 4, window row, round of the sequence,
 * stream << 24 | slot); word (entry % 4) x gives the uniform
 * (2 * (x >> 9) + 1) * 2^-24 and token samples are Gumbel-max
 * (argmax of log-weight - log(-log u)).  Streams: 0 draft samples (a0, d_j),
 * 2 acceptance uniforms (row j, entry 0), 3 the replacement or bonus sample
 * (row j of the rejected position, K+1 for the bonus).  A round's draws thus
 * depend on the seed, the slot and the sequence's round count only.
 * Defaults: T = 1, seed = 0.  Errors: GS_ERR_INVALID_ARG. */
int gs_set_sampling(gs_handle *h, float temperature, uint64_t seed);

/* Direct block-diffusion decoding of one block per sequence (paper Appendix
 * "Direct Block-Diffusion Decoding"; Sec. 5 diffusion-vs-self-speculative
 * comparison).  From the same state as gs_round (the cache holds every
 * committed token but the boundary x0), a block of B [M] tokens at slots
 * n+1..n+B is denoised: each step is one forward over [x0, block] with the
 * draft's hybrid mask (x0 causal, block rows bidirectional in the window),
 * the prediction for position p read from the row at p-1; every still-masked
 * position whose argmax probability exceeds tau_c is revealed, or, if none
 * is, the single most confident one (ties to the lowest position); revealed
 * tokens stay fixed.  When every sequence's block is complete, one causal
 * forward over [x0, y_1..y_B] writes the cache (no LM head), and the block is
 * committed: y_1..y_B cut at the first EOS or at max_new, seq_len += B,
 * x0 = y_B.  All steps run inside one CUDA graph whose denoising loop is a
 * conditional (while) node: no host synchronisation; the loop is capped at B
 * steps (a sequence still open after B steps raises the device check).
 *   slots     device int32 [n_seq], distinct prefilled slots
 *   B         block size, 1 <= B <= max_K
 *   tau_c     confidence threshold (probabilities are in (0, 1]; tau_c >= 1
 *             reveals one position per step, tau_c < 0 the whole block at once)
 *   out_tok   device int32 [n_seq, B]: committed tokens of the block
 *   out_cnt   device int32 [n_seq]: how many (0 for a sequence already done)
 *   out_done  device int32 [n_seq]: 1 once the sequence hit EOS or max_new
 *   out_steps device int32 [n_seq] or NULL: denoising forwards of the block
 *             (the paper's TPF for this mode counts these, not the cache write)
 * Needs a handle created on a non-default stream.  Graphs are cached per
 * (n_seq, B, tau_c, pointers).  Errors: GS_ERR_INVALID_ARG, GS_ERR_CUDA. */
int gs_diffusion_block(gs_handle *h, const int32_t *slots, int n_seq, int B, float tau_c,
                       int32_t *out_tok, int32_t *out_cnt, int32_t *out_done, int32_t *out_steps);

/* A self-speculative round with multi-step drafting (paper Sec. 6 "Draft
 * Schedule", Fig. "Multi-step drafting versus one-shot drafting").  The draft
 * window [x0, [M] x K] is run repeatedly: prediction i (a0 for i = 0, d_i
 * otherwise, read from row i) is fixed once its argmax probability exceeds
 * tau_d, or, when no open prediction does, the single most confident one is;
 * a fixed prediction i < K is fed back at its own slot n+1+i in place of the
 * mask; after at most K+1 draft forwards the finished draft is verified,
 * accepted and committed exactly as by gs_round (GS_ACCEPT_GREEDY; the
 * forcing hook applies to the refined draft).  tau_d < 0 is the one-shot
 * round.  One graph launch with a conditional loop, no host synchronisation.
 *   out_tok [n_seq, K+2], out_cnt, out_done: as gs_round
 *   out_steps device int32 [n_seq] or NULL: draft forwards of the round
 * Needs a non-default stream.  Errors: GS_ERR_INVALID_ARG, GS_ERR_CUDA. */
int gs_round_refined(gs_handle *h, const int32_t *slots, int n_seq, int K, float tau_d,
                     const gs_force *force, int32_t *out_tok, int32_t *out_cnt, int32_t *out_done,
                     int32_t *out_steps);

/* Overwrite a sequence's per-slot state (resume/checkpoint: with the KV pages,
 * which keep their contents, the state is the cached length, the boundary
 * token, the output count and cap, the done flag and the round counter that
 * indexes a forcing schedule).  Rolling the cached length back to a value the
 * cache held before (e.g. the prefix length after a prefill) replays a decode.
 *   seq_len   1 <= seq_len and seq_len + max_K + 2 <= the slot's reservation
 *   x0        boundary token in [0, vocab); n_out >= 1 committed tokens (x0 included)
 *   max_new   output cap (>= n_out); done 0/1; rounds >= 0
 * Host values; enqueued on the stream.  Errors: GS_ERR_INVALID_ARG. */
int gs_seq_restore(gs_handle *h, int slot, int seq_len, int x0, int n_out, int max_new, int done,
                   int rounds);

/* Read one slot's state (synchronises the stream).  Any out pointer may be NULL. */
int gs_seq_state(gs_handle *h, int slot, int *seq_len, int *x0, int *n_out, int *done, int *rounds);

/* Number of kernel launches the most recent gs_round enqueued (or captured). */
int gs_round_launches(gs_handle *h);

/* Kinds of kernel reported by gs_round_profile (one per launch). */
enum {
  GS_KIND_WINDOW = 0,    /* draft window build or verify input build (Sec. 3.2) */
  GS_KIND_EMBED = 1,     /* token embedding + first RMSNorm input */
  GS_KIND_QKV = 2,       /* QKV projection + RoPE + KV-cache write */
  GS_KIND_ATTENTION = 3, /* hybrid-mask paged attention (Eq. 3 / Eq. 5 masks) */
  GS_KIND_O_PROJ = 4,    /* output projection + residual */
  GS_KIND_GATE_UP = 5,   /* gate/up projection + SwiGLU */
  GS_KIND_DOWN = 6,      /* down projection + residual */
  GS_KIND_LM_HEAD = 7,   /* LM head + greedy argmax */
  GS_KIND_ACCEPT = 8     /* longest-prefix acceptance and commit (Sec. 3.3) */
};

/* Measurement aid: one greedy round, with the same arguments and effects as
 * gs_round(h, slots, n_seq, K, GS_ACCEPT_GREEDY, force, out_tok, out_cnt,
 * out_done, NULL), captured (never from the graph cache) with a CUDA event
 * recorded after every kernel launch and replayed as one graph, so the host's
 * enqueue time never falls between two launches.  The paper has no
 * counterpart.
 *   ms[i]       device milliseconds between launch i-1's end event and launch
 *               i's end event (for i = 0, from an event recorded before the
 *               round).  An event between two kernels stops the second from
 *               starting early, so each figure is the kernel alone, from the
 *               front end starting it to its last CTA.
 *   kind[i]     GS_KIND_* of launch i.
 *   n_launches  number of launches written.
 * ms and kind are host arrays of max_launches entries.  Synchronises the
 * handle's stream (which must not be the default stream).
 * Errors: GS_ERR_INVALID_ARG (bad arguments, max_launches too small — the
 * round has then run), GS_ERR_CUDA. */
int gs_round_profile(gs_handle *h, const int32_t *slots, int n_seq, int K, const gs_force *force,
                     int32_t *out_tok, int32_t *out_cnt, int32_t *out_done, int max_launches,
                     float *ms, int *kind, int *n_launches);

/* Free the slot's KV pages (host bookkeeping only). */
int gs_release(gs_handle *h, int slot);

/* Synchronise the stream and report a kernel-side check or bounded-wait
 * failure raised since the last call (then clear it). */
int gs_sync_check(gs_handle *h);

/* Failure-detection self-test (the paper has no counterpart).  Enqueues on
 * the handle's stream one kernel that waits, through the same bounded
 * mbarrier wait every pipeline of the library uses, on a barrier nothing
 * arrives on; the wait gives up after limit_us microseconds of device time
 * (1 <= limit_us <= 2,000,000) and raises the timeout code in the handle's
 * error word, so the next gs_sync_check returns GS_ERR_TIMEOUT.  The context
 * stays usable: nothing else is in flight in the probe's CTA.
 * Errors: GS_ERR_INVALID_ARG, GS_ERR_CUDA. */
int gs_wait_probe(gs_handle *h, int limit_us);

/* ---------------------------------------------------------------------------
 * Sub-steps exposed for the attention-only sweep and kernel parity tests.
 * ------------------------------------------------------------------------ */

/* Hybrid-mask attention over a paged fp16 KV cache (paper Appendix steps
 * Draft forward / Verify forward; mask semantics Sec. 4.2).  Standalone form
 * of the kernel the rounds use.
 *   mode 0 DRAFT:  query row i of sequence s sits at slot n_s + i;
 *                  row 0 sees keys 0..n_s, rows i >= 1 see keys 0..n_s + W - 1
 *   mode 1 VERIFY: query row i sits at slot n_s + 1 + i and sees keys 0..n_s + 1 + i
 *   q        device fp16 [n_seq, W, n_heads, 64] (RoPE already applied)
 *   kv       device fp16 page pool [n_pages][2][n_kv_heads][64][64]: per page and
 *            KV head, K as [64 tokens][64 dims] and V transposed, [64 dims][64 tokens]
 *   page_table device int32 [n_seq, pt_stride]: logical page -> physical page
 *   n        device int32 [n_seq]: n_s
 *   out      device fp16 [n_seq, W, n_heads, 64]
 *   scratch  device, >= gs_attention_scratch_bytes(...) bytes: the kernel's
 *            error word (first int32: 0 = no failure, 1 = bounds check,
 *            2 = bounded wait ran out, 3 = fp16 range; cleared by each call),
 *            key limits, the block -> page-table map, merge tickets and the
 *            fp32 partial rows (O, m, l) of every work item
 *   split_pages pages per work item (>= 1): item i of a sequence covers its
 *            logical pages [i * split_pages, (i + 1) * split_pages); items are
 *            reduced independently and merged in item order, so results depend
 *            on split_pages but not on n_seq, W or the other sequences.
 *            GS_ERR_UNSUPPORTED if ceil(pt_stride / split_pages) > 54 (the
 *            merge keeps each item's running max and sum of every row in the
 *            kernel's idle page ring, 54 KB).
 *   stream   cudaStream_t */
size_t gs_attention_scratch_bytes(int n_seq, int W, int n_heads, int n_kv_heads, int max_pages,
                                  int split_pages);
int gs_attention(int mode, const void *q, const void *kv, int n_pages, const int32_t *page_table,
                 int pt_stride, const int32_t *n, int n_seq, int W, int n_heads, int n_kv_heads,
                 void *out, void *scratch, size_t scratch_bytes, int split_pages, void *stream);

/* Y = X . W^T on the tcgen05 GEMM the decoder uses.
 *   x device fp16 [M, K] (row stride K), w device fp16 [N, K], y device [M, N]
 *   epilogue 0: y fp16 = acc;  1: y fp32 += acc (residual);  2: SwiGLU: w is
 *   [2N, K] (gate rows then up rows), y fp16 [M, N] = silu(gate) * up;
 *   3: argmax: y is uint64 [M] packed (ordered fp32 bits << 32 | ~index),
 *   combined with atomicMax (caller zeroes it first).
 *   split_k S: 1 or a divisor of K/64.  K is reduced as S consecutive chunks,
 *   each summed from zero in k order, then the chunks summed in order
 *   0..S-1.  Where the chunks are reduced (across a cluster of CTAs, inside
 *   one CTA, or through the scratch) depends on M; the sums do not, so a row's
 *   result is the same for any M.  scratch device >= gs_linear_scratch_bytes,
 *   any contents: the call clears the parts that must start at zero.  Its
 *   first int32 is the kernel's error word after the stream reaches the end
 *   of the call (0 = no failure, 1 = bounds check, 2 = bounded wait ran out,
 *   3 = a value beyond the fp16 range).
 *   Requirements: K % 64 == 0, N % 128 == 0 (N % 64 for epilogue 2), M >= 1;
 *   x, w and y 16-byte aligned. */
size_t gs_linear_scratch_bytes(int M, int N, int split_k);
int gs_linear(const void *x, const void *w, void *y, int M, int N, int K, int epilogue, int split_k,
              void *scratch, size_t scratch_bytes, void *stream);

/* ---------------------------------------------------------------------------
 * Allocation-free variant of gs_linear.  The paper has no counterpart: this
 * entry point exists for callers that cannot allocate device memory at the
 * call and have no workspace to pass (an operator inside another framework
 * with no workspace argument, a plugin host whose allocator owns all device
 * memory, a real-time path where cudaMalloc's implicit synchronisation is not
 * allowed).
 *
 * Same arguments and results as gs_linear minus the scratch pointer: the
 * split-K scratch (error word, per-tile counters, fp32 partials) lives in a
 * fixed device array of GS_NOALLOC_SCRATCH_BYTES inside the library, which
 * every GPU that loads the library keeps until the process exits.  The call
 * makes no cudaMalloc / cudaFree and calls no allocating library routine.
 *   - The first call on a device looks up that array's device address (with
 *     the device current); make that first call before any stream capture.
 *   - Every call clears the counters it uses and the error word before its
 *     kernel runs.  gs_linear_noalloc_status reports that call's kernel-side
 *     checks.
 *   - All calls share the one array: calls whose kernels overlap on the GPU
 *     (two streams, or two host threads on one device) race; serialise them.
 * Errors: as gs_linear; GS_ERR_OOM when split_k x tiles of partials for
 * (M, N) do not fit in GS_NOALLOC_SCRATCH_BYTES (e.g. M <= 32 rows, N = 2048,
 * split_k = 8 needs 2 MiB). */
#define GS_NOALLOC_SCRATCH_BYTES (8u << 20)
int gs_linear_noalloc(const void *x, const void *w, void *y, int M, int N, int K, int epilogue,
                      int split_k, void *stream);

/* Kernel-side status of the most recent gs_linear_noalloc on the current
 * device: synchronises `stream` (the one that call used), then returns GS_OK,
 * GS_ERR_DEVICE_CHECK (a bounds check fired or a value left the fp16 range)
 * or GS_ERR_TIMEOUT (a bounded wait ran out), and clears the word.  Call it
 * before the next gs_linear_noalloc, which clears the word again.  Allocates
 * nothing.  Errors: GS_ERR_CUDA. */
int gs_linear_noalloc_status(void *stream);

#ifdef __cplusplus
}
#endif
#endif /* GS_H_ */
