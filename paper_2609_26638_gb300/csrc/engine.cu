// engine.cu -- libgs host side: workspace carving, paged-KV bookkeeping, the
// decoder forward as a launch sequence, the round (draft -> force -> verify ->
// accept) with a CUDA-graph cache, prefill, and the C ABI of include/gs.h.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <functional>
#include <map>
#include <mutex>
#include <string>
#include <tuple>
#include <vector>

#include "attention.cuh"
#include "denoise.cuh"
#include "gemm_tc.cuh"
#include "internal.h"
#include "small.cuh"
#include "../../include/gs.h"

using namespace gs;

namespace {

thread_local std::string g_create_error;

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// The driver's tensor-map encoder, looked up once per process.
EncodeTiledFn get_encode() {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}
}  // namespace

bool gs::make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols,
                  uint32_t box_rows) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides,
                   box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

namespace {

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
inline int cdiv(long long a, long long b) { return static_cast<int>((a + b - 1) / b); }
inline int round16(int x) { return (x + 15) / 16 * 16; }

// Sequential carving of the caller's workspace (also used to size it).
struct Carver {
  uint8_t* base;
  size_t off = 0;
  explicit Carver(void* b) : base(static_cast<uint8_t*>(b)) {}
  template <class T>
  T* take(size_t count) {
    off = align_up(off, 256);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
};

constexpr int kGemmCounters = 1 << 16;

// Query blocks of a window of W tokens: at most kAttnMaxRows rows (QS tokens
// of G rows) each, n_sub blocks per window, `rows` row slots per block.
struct AttnGeom {
  int QS, n_sub, rows;
};
AttnGeom attn_geom(int W, int G) {
  const int qs = std::min(W, kAttnMaxRows / G);
  return {qs, cdiv(W, qs), kAttnMaxRows};
}

// Items merge inside a cluster when there are at most 16 of them and the
// launch is about one wave (a cluster waits for free SMs of one GPC, and
// clusters fragment larger grids); otherwise through global scratch.  Both
// give the same bits.
}  // namespace

// Kernel attributes (dynamic shared memory above 48 KB, non-portable cluster
// sizes) are set once per device, under a lock, before the first launch.
cudaError_t gs::ensure_kernel_attributes() {
  static std::mutex mu;
  static uint64_t done = 0;   // bit d: device d configured
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  if (dev < 64 && ((done >> dev) & 1)) return cudaSuccess;
  e = gemm_init_attributes();
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_paged_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             attn_max_smem_bytes());
  if (e == cudaSuccess)   // clusters of up to 16 attention items
    e = cudaFuncSetAttribute(attn_paged_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess && dev < 64) done |= 1ull << dev;
  return e;
}

namespace {

bool attn_use_cluster(int items, int blocks_x_heads) {
  return items <= kAttnMaxCluster && items * blocks_x_heads <= 2 * kNumSMs;
}

cudaError_t launch_attention(const CUtensorMap& tm, const AttnArgs& a, int n_blocks,
                             cudaStream_t s, bool pdl) {
  dim3 grid(a.max_items, a.Hkv, n_blocks);
  return launch_ex(attn_paged_kernel, grid, dim3(kAttnThreads), kAttnSmemBytes, s, pdl,
                   dim3(a.cluster ? a.max_items : 1, 1, 1), tm, a);
}

struct GemmPlan {
  int bn, tok_tiles, feat_tiles, splits, chunks;
};

// Split-K factor of a weight matrix in decode rounds.  It depends on the
// weight's shape only, never on the token count: every split sums its K range
// from zero and the splits are added in order 0..S-1, and the MMA's per-column
// arithmetic does not depend on the tile width, so a token row gets the same
// bits in any window and any batch.  About one wave of CTAs for a one-tile
// window, at least 4 splits (cluster split CTAs own at most 8 of 32 tokens),
// at most one cluster; matrices with a wave of feature tiles are not split.
int decode_splits(int weight_rows, int K) {
  const int feat_tiles = weight_rows / 128;
  const int nkb = K / 64;
  if (feat_tiles >= kNumSMs) return 1;
  const int want = std::min(std::max(cdiv(kNumSMs, feat_tiles), 4), kMaxClusterSplits);
  int s = 1;
  for (int k = 1; k <= nkb; ++k)
    if (nkb % k == 0 && k <= want) s = k;
  return s;
}

// Decode windows of up to 64 tokens split K across the CTAs of a cluster.
// Wider decode launches with at least 8 k-blocks per split keep that (64-token
// tiles); the others reduce the same K chunks inside each CTA
// (gemm_chunk_kernel: each chunk summed from zero in a TMEM buffer, then added
// in chunk order to a running sum in TMEM), with the token tile the widest of
// 128 / 64 / 32 with the fewest waves x operand bytes per CTA.  All three
// give the same sums in the same order.  Prefill does not split K.
GemmPlan plan_split(int weight_rows, int T, int S, int nkb) {
  GemmPlan p;
  p.feat_tiles = weight_rows / 128;
  p.chunks = 1;
  p.splits = S;
  p.bn = gemm_bn_for(T);
  if (S > 1 && T > 64 && nkb / S >= 8 && gemm_cluster_ok(64, S)) {
    p.bn = 64;
  } else if (S > 1 && T > 64) {
    // chunked K inside each CTA (gemm_chunk_kernel, two CTAs per SM).  A CTA
    // streams K x (128 + BN) operand bytes, and the launch takes ceil(CTAs /
    // slots) rounds of them: pick the token tile of 128 / 64 / 32 with the
    // least waves x (128 + BN), the wider on a tie.
    p.chunks = S;
    p.splits = 1;
    long best = -1;
    for (int bn : {128, 64, 32}) {
      const long waves = cdiv(static_cast<long long>(p.feat_tiles) * cdiv(T, bn), 2 * kNumSMs);
      const long cost = waves * (128 + bn);
      if (best < 0 || cost < best) {
        best = cost;
        p.bn = bn;
      }
    }
  }
  p.tok_tiles = cdiv(T, p.bn);
  return p;
}

GemmPlan plan_gemm(int weight_rows, int K, int T, bool decode) {
  return plan_split(weight_rows, T, decode ? decode_splits(weight_rows, K) : 1, K / 64);
}

// fp32 partials the widest decode tiles (BN > 64, reduced through global
// scratch) need: splits x feature tiles x token columns (T + 255 bounds the
// padded token count) x 128, over the decoder's five weight shapes.
size_t gemm_partial_floats(const gs_config& c, int qkv_dim, int T_dec) {
  const int HD = c.n_heads * 64;
  const int shapes[5][2] = {{qkv_dim, c.d_model}, {c.d_model, HD}, {2 * c.d_ffn, c.d_model},
                            {c.d_model, c.d_ffn}, {c.vocab, c.d_model}};
  size_t need = 0;
  for (const auto& sh : shapes) {
    const int S = decode_splits(sh[0], sh[1]);
    if (S > 1)
      need = std::max(need, static_cast<size_t>(S) * (sh[0] / 128) * (T_dec + 255) * 128);
  }
  return need;
}

}  // namespace

struct gs_handle {
  gs_config cfg;
  cudaStream_t stream = nullptr;
  std::string err;

  // weights
  const __nv_bfloat16 *embed = nullptr, *final_norm = nullptr;
  std::vector<const __nv_bfloat16*> attn_norm, ffn_norm;
  // fp16 copies of the matrices, each scaled by 2^s (w_scale = 2^-s undoes it)
  std::vector<const __half*> w_qkv, w_o, w_gu, w_down;
  const __half* lm_head = nullptr;
  std::vector<float> sc_qkv, sc_o, sc_gu, sc_down;
  float sc_lm = 1.f;
  __half* wcopy = nullptr;
  std::vector<CUtensorMap> tm_qkv, tm_o, tm_gu, tm_down;
  CUtensorMap tm_lm;
  CUtensorMap tm_hb[4], tm_ao[4], tm_act[4];
  CUtensorMap tm_kv;

  // sizes
  int qkv_dim = 0, G = 1, T_max = 0, pt_stride = 0, n_pages = 0, W_max = 1;
  // attention work items: pages per item and item slots, decode and prefill
  int split_pages = 1, items_dec = 1, r_max_dec = 16;
  int split_pages_pf = 8, items_pf = 1, qb_pf = 64;
  float* attn_part = nullptr;
  size_t attn_part_floats = 0;
  int* attn_ticket = nullptr;

  // workspace
  int* err_word = nullptr;
  SeqStateDev st{};
  int32_t* page_table = nullptr;
  __half* kv = nullptr;
  float2* rope = nullptr;
  int32_t *tok = nullptr, *pos = nullptr, *lim = nullptr, *tok_slot = nullptr;
  int32_t *blk_slot = nullptr, *blk_active = nullptr;
  float* hbuf = nullptr;
  __half *hb = nullptr, *qr = nullptr, *ao = nullptr, *act = nullptr;
  float* ssp = nullptr;   // per-token sums of h^2 per 128-feature block [T_max][d/128]
  unsigned long long *packed_d = nullptr, *packed_v = nullptr;
  int32_t *draft_tok = nullptr, *verify_in = nullptr, *verify_tok = nullptr;
  float* gemm_partial = nullptr;
  size_t partial_floats = 0;
  int* gemm_counters = nullptr;

  // host page bookkeeping
  std::vector<int> free_pages;
  std::vector<std::vector<int>> slot_pages;
  std::vector<int> slot_reserved;  // slots (tokens) reserved per sequence slot
  std::vector<int32_t> pt_host;

  // graphs keyed by (n_seq, K, pointers)
  typedef std::tuple<int, int, const void*, const void*, long long, const void*, long long,
                     const void*, const void*, const void*, long long>
      GraphKey;
  std::map<GraphKey, cudaGraphExec_t> graphs;
  int launches = 0;             // kernel launches counted while enqueueing
  int last_round_launches = 0;

  // programmatic dependent launch on the decoder's launches (off while a
  // graph with a conditional loop is captured)
  bool pdl = true;
  // denoising loops (block diffusion, multi-step drafting): per-slot fixed
  // predictions, flags and step counts, the loop counter, the LM head's
  // softmax partials, a side stream for capturing loop bodies, their graphs
  int32_t *dn_fixed = nullptr, *dn_live = nullptr, *dn_part = nullptr, *dn_steps = nullptr;
  int32_t* dn_iter = nullptr;
  float2* lse_part = nullptr;
  int lse_tiles = 0;
  cudaStream_t side = nullptr;
  std::map<std::vector<uint64_t>, cudaGraphExec_t> loop_graphs;

  // stochastic rounds: temperature and seed (gs_set_sampling), the two LM
  // heads' logits and the verify head's softmax partials, the draft rows'
  // sampling counters
  float temperature = 1.f;
  uint64_t seed = 0;
  float *logits_d = nullptr, *logits_v = nullptr;
  float2* lse_v = nullptr;
  uint4* rng_row = nullptr;

  // gs_round_profile: an event after every launch and the launch's kind
  bool profiling = false;
  cudaError_t prof_err = cudaSuccess;
  std::vector<cudaEvent_t> prof_ev;
  std::vector<int> prof_kind;
};

namespace {

int fail(gs_handle* h, int code, const std::string& msg) {
  if (h) h->err = msg;
  else g_create_error = msg;
  return code;
}

#define GS_CUDA(h, call)                                                              \
  do {                                                                                \
    cudaError_t e_ = (call);                                                          \
    if (e_ != cudaSuccess)                                                            \
      return fail(h, GS_ERR_CUDA, std::string(#call " -> ") + cudaGetErrorString(e_)); \
  } while (0)

// Counts one kernel launch; under gs_round_profile also records an event
// behind it on the handle's stream and remembers what kind of kernel it was.
void note_launch(gs_handle* h, int kind) {
  ++h->launches;
  if (!h->profiling) return;
  const size_t i = h->prof_kind.size() + 1;  // event 0 marks the start of the round
  while (h->prof_ev.size() <= i) {
    cudaEvent_t e;
    cudaError_t r = cudaEventCreate(&e);
    if (r != cudaSuccess) {
      if (h->prof_err == cudaSuccess) h->prof_err = r;
      return;
    }
    h->prof_ev.push_back(e);
  }
  // an event-record node of the captured profiling graph
  cudaError_t r = cudaEventRecordWithFlags(h->prof_ev[i], h->stream, cudaEventRecordExternal);
  if (r != cudaSuccess && h->prof_err == cudaSuccess) h->prof_err = r;
  h->prof_kind.push_back(kind);
}

int bn_index(int bn) { return bn == 32 ? 0 : (bn == 64 ? 1 : (bn == 128 ? 2 : 3)); }

bool config_ok(const gs_config* c, std::string* why) {
  auto bad = [&](const char* m) { *why = m; return false; };
  if (!c) return bad("null config");
  if (c->n_layers < 1 || c->d_model < 128 || c->vocab < 128) return bad("bad sizes");
  if (c->head_dim != 64) return bad("head_dim must be 64");
  if (c->n_heads < 1 || c->n_kv_heads < 1 || c->n_heads % c->n_kv_heads) return bad("bad heads");
  if (c->n_heads / c->n_kv_heads > 8) return bad("GQA group > 8 unsupported");
  if (c->d_model % 128) return bad("d_model % 128");
  if (c->n_heads % 2 || c->n_kv_heads % 2) return bad("n_heads and n_kv_heads must be even");
  if ((c->n_heads * 64) % 64) return bad("attn dim % 64");
  if (c->d_ffn % 64 || c->d_ffn < 64) return bad("d_ffn % 64");
  if (c->vocab % 128) return bad("vocab % 128");
  if (c->mask_token_id < 0 || c->mask_token_id >= c->vocab) return bad("mask_token_id");
  if (c->eos_token_id >= c->vocab) return bad("eos_token_id");
  if (c->max_batch < 1 || c->max_ctx < 64 || c->max_K < 0 || c->max_prefill < 1)
    return bad("bad capacity");
  if ((c->max_K + 1) * (c->n_heads / c->n_kv_heads) > 256) return bad("window rows > 256");
  if (c->max_batch * (c->max_K + 1) > 65536) return bad("decode tokens > 65536");
  return true;
}

// Carve the workspace; with base == nullptr only sizes it.
size_t carve(gs_handle* h, const gs_config& c, void* base) {
  Carver cv(base);
  const int G = c.n_heads / c.n_kv_heads;
  const int qkv_dim = (c.n_heads + 2 * c.n_kv_heads) * 64;
  const int pt_stride = cdiv(c.max_ctx, 64);
  const int n_pages = c.kv_pages > 0 ? c.kv_pages : c.max_batch * pt_stride;
  const int W_max = c.max_K + 1;
  int T_max = std::max(c.max_batch * W_max, c.max_prefill);
  T_max = static_cast<int>(align_up(std::max(T_max, 256), 256));
  // attention work items (fixed absolute page ranges).  Decode: at most 16
  // items per sequence (one cluster) when a full batch of them still fits in
  // about one wave of CTAs, else at most 8, unless the config asks for
  // smaller items; prefill: at least 8 pages per item, at most 8 items.
  const int r_max = round16(W_max * G);
  const AttnGeom g_dec = attn_geom(W_max, G);
  const int qb_pf = std::max(1, kAttnMaxRows / G);
  const int items_target =
      attn_use_cluster(kAttnMaxCluster, c.max_batch * g_dec.n_sub * c.n_kv_heads) ? kAttnMaxCluster : 8;
  int sp = c.split_pages > 0 ? c.split_pages : std::max(2, cdiv(pt_stride, items_target));
  sp = std::max(sp, cdiv(pt_stride, attn_max_merge_items(g_dec.rows)));
  const int items_dec = cdiv(pt_stride, sp);
  const int sp_pf = std::max(8, cdiv(pt_stride, 8));
  const int items_pf = cdiv(pt_stride, sp_pf);
  const AttnGeom g_pf = attn_geom(qb_pf, G);
  const int blocks_pf = cdiv(std::min(c.max_prefill, T_max), qb_pf);
  const size_t attn_blocks = std::max(static_cast<size_t>(c.max_batch) * g_dec.n_sub,
                                      static_cast<size_t>(blocks_pf));
  // item rows of the global merge (used when a launch is too large for clusters)
  const size_t attn_part_floats =
      std::max(static_cast<size_t>(c.max_batch) * g_dec.n_sub * items_dec * g_dec.rows,
               static_cast<size_t>(blocks_pf) * items_pf * g_pf.rows) *
      c.n_kv_heads * kAttnRow;
  int* err_word = cv.take<int>(64);
  SeqStateDev st;
  st.seq_len = cv.take<int32_t>(c.max_batch);
  st.x0 = cv.take<int32_t>(c.max_batch);
  st.n_out = cv.take<int32_t>(c.max_batch);
  st.max_new = cv.take<int32_t>(c.max_batch);
  st.done = cv.take<int32_t>(c.max_batch);
  st.rounds = cv.take<int32_t>(c.max_batch);
  int32_t* page_table = cv.take<int32_t>(static_cast<size_t>(c.max_batch) * pt_stride);
  __half* kv = cv.take<__half>(static_cast<size_t>(c.n_layers) * n_pages * 2 * c.n_kv_heads * 64 *
                               64);
  float2* rope = cv.take<float2>(static_cast<size_t>(c.max_ctx) * 32);
  int32_t* tok = cv.take<int32_t>(T_max);
  int32_t* pos = cv.take<int32_t>(T_max);
  int32_t* lim = cv.take<int32_t>(T_max);
  int32_t* tok_slot = cv.take<int32_t>(T_max);
  int32_t* blk_slot = cv.take<int32_t>(std::max(c.max_batch, T_max / 64 + 1));
  int32_t* blk_active = cv.take<int32_t>(std::max(c.max_batch, T_max / 64 + 1));
  float* hbuf = cv.take<float>(static_cast<size_t>(T_max) * c.d_model);
  __half* hb = cv.take<__half>(static_cast<size_t>(T_max) * c.d_model);
  float* ssp = cv.take<float>(static_cast<size_t>(T_max) * (c.d_model / 128));
  __half* qr = cv.take<__half>(static_cast<size_t>(T_max) * c.n_heads * 64);
  __half* ao = cv.take<__half>(static_cast<size_t>(T_max) * c.n_heads * 64);
  __half* act = cv.take<__half>(static_cast<size_t>(T_max) * c.d_ffn);
  unsigned long long* packed_d = cv.take<unsigned long long>(T_max);
  unsigned long long* packed_v = cv.take<unsigned long long>(T_max);
  int32_t* draft_tok = cv.take<int32_t>(static_cast<size_t>(c.max_batch) * W_max);
  int32_t* verify_in = cv.take<int32_t>(static_cast<size_t>(c.max_batch) * W_max);
  int32_t* verify_tok = cv.take<int32_t>(static_cast<size_t>(c.max_batch) * W_max);
  const size_t partial_floats = gemm_partial_floats(c, qkv_dim, c.max_batch * W_max);
  float* gemm_partial = cv.take<float>(partial_floats);
  int* gemm_counters = cv.take<int>(kGemmCounters);
  float* attn_part = cv.take<float>(attn_part_floats);
  int* attn_ticket = cv.take<int>(attn_blocks * c.n_kv_heads);
  int32_t* dn_fixed = cv.take<int32_t>(static_cast<size_t>(c.max_batch) * W_max);
  int32_t* dn_live = cv.take<int32_t>(c.max_batch);
  int32_t* dn_part = cv.take<int32_t>(c.max_batch);
  int32_t* dn_steps = cv.take<int32_t>(c.max_batch);
  int32_t* dn_iter = cv.take<int32_t>(64);
  const int lse_tiles = c.vocab / 128;
  float2* lse_part = cv.take<float2>(static_cast<size_t>(c.max_batch) * W_max * lse_tiles);
  float2* lse_v = cv.take<float2>(static_cast<size_t>(c.max_batch) * W_max * lse_tiles);
  float* logits_d = cv.take<float>(static_cast<size_t>(c.max_batch) * W_max * c.vocab);
  float* logits_v = cv.take<float>(static_cast<size_t>(c.max_batch) * W_max * c.vocab);
  uint4* rng_row = cv.take<uint4>(static_cast<size_t>(c.max_batch) * W_max);
  // fp16 weight copies: per layer qkv | o | gate_up | down, then the LM head
  const size_t per_layer = static_cast<size_t>(qkv_dim) * c.d_model +
                           static_cast<size_t>(c.d_model) * c.n_heads * 64 +
                           2 * static_cast<size_t>(c.d_ffn) * c.d_model +
                           static_cast<size_t>(c.d_model) * c.d_ffn;
  // (every tensor's element count is a multiple of 64 * 64, so the copies pack without padding)
  __half* wcopy = cv.take<__half>(per_layer * c.n_layers + static_cast<size_t>(c.vocab) * c.d_model);

  if (h) {
    h->G = G;
    h->qkv_dim = qkv_dim;
    h->pt_stride = pt_stride;
    h->n_pages = n_pages;
    h->T_max = T_max;
    h->W_max = W_max;
    h->split_pages = sp;
    h->items_dec = items_dec;
    h->r_max_dec = r_max;
    h->split_pages_pf = sp_pf;
    h->items_pf = items_pf;
    h->qb_pf = qb_pf;
    h->attn_part = attn_part;
    h->attn_part_floats = attn_part_floats;
    h->attn_ticket = attn_ticket;
    h->err_word = err_word;
    h->wcopy = wcopy;
    h->partial_floats = partial_floats;
    h->st = st;
    h->page_table = page_table;
    h->kv = kv;
    h->rope = rope;
    h->tok = tok;
    h->pos = pos;
    h->lim = lim;
    h->tok_slot = tok_slot;
    h->blk_slot = blk_slot;
    h->blk_active = blk_active;
    h->hbuf = hbuf;
    h->hb = hb;
    h->ssp = ssp;
    h->qr = qr;
    h->ao = ao;
    h->act = act;
    h->packed_d = packed_d;
    h->packed_v = packed_v;
    h->draft_tok = draft_tok;
    h->verify_in = verify_in;
    h->verify_tok = verify_tok;
    h->gemm_partial = gemm_partial;
    h->gemm_counters = gemm_counters;
    h->dn_fixed = dn_fixed;
    h->dn_live = dn_live;
    h->dn_part = dn_part;
    h->dn_steps = dn_steps;
    h->dn_iter = dn_iter;
    h->lse_part = lse_part;
    h->lse_tiles = lse_tiles;
    h->lse_v = lse_v;
    h->logits_d = logits_d;
    h->logits_v = logits_v;
    h->rng_row = rng_row;
  }
  return align_up(cv.off, 256);
}

// ------------------------------------------------------------------ launches
// A GemmArgs with the fields every decoder GEMM shares; the caller adds the
// epilogue's outputs.
GemmArgs gemm_base(gs_handle* h) {
  GemmArgs a = {};
  a.partial = h->gemm_partial;
  a.counters = h->gemm_counters;
  a.err = h->err_word;
  a.n_ssp = h->cfg.d_model / 128;
  a.inv_d = 1.0f / static_cast<float>(h->cfg.d_model);
  a.eps = h->cfg.rms_eps;
  a.w_scale = 1.f;
  a.inv_temp = 1.f;
  return a;
}

int run_gemm(gs_handle* h, const CUtensorMap& tw, int weight_rows, const CUtensorMap* tx_set, int K,
             int T, int epi, GemmArgs a, bool decode, int kind) {
  const GemmPlan p = plan_gemm(weight_rows, K, T, decode);
  a.M = T;
  a.K = K;
  a.splits = p.splits;
  a.chunks = p.chunks;
  a.kb_per_split = (K / 64) / p.splits;
  a.cluster = gemm_cluster_ok(p.bn, p.splits) ? 1 : 0;
  if (p.splits > 1 && !a.cluster &&
      (static_cast<size_t>(p.splits) * p.feat_tiles * p.tok_tiles * p.bn * 128 > h->partial_floats ||
       p.feat_tiles * p.tok_tiles > kGemmCounters))
    return fail(h, GS_ERR_OOM, "split-K scratch too small");
  GS_CUDA(h, launch_gemm(p.bn, epi, tw, tx_set[bn_index(p.bn)], a, p.feat_tiles, p.tok_tiles,
                         h->stream, h->pdl));
  note_launch(h, kind);
  return GS_OK;
}

struct AttnLaunch {
  int n_seq, QB, split_pages, max_items;
  const int32_t* blk_slot;
  const int32_t* blk_active;
  int fixed_slot;
};

int run_attention(gs_handle* h, int layer, int T, const AttnLaunch& L) {
  const gs_config& c = h->cfg;
  const AttnGeom g = attn_geom(L.QB, h->G);
  AttnArgs a;
  a.q = h->qr;
  a.lim = h->lim;
  a.out = h->ao;
  a.page_table = h->page_table;
  a.pt_stride = h->pt_stride;
  a.blk_slot = L.blk_slot;
  a.blk_active = L.blk_active;
  a.fixed_slot = L.fixed_slot;
  a.T = T;
  a.QB = L.QB;
  a.QS = g.QS;
  a.n_sub = g.n_sub;
  a.Hq = c.n_heads;
  a.Hkv = c.n_kv_heads;
  a.G = h->G;
  a.rows_per_page = 2 * c.n_kv_heads * 64;
  a.kv_row_base = static_cast<long long>(layer) * h->n_pages * a.rows_per_page;
  a.split_pages = L.split_pages;
  a.max_items = L.max_items;
  a.cluster = attn_use_cluster(L.max_items, L.n_seq * g.n_sub * c.n_kv_heads) ? 1 : 0;
  a.part = h->attn_part;
  a.ticket = h->attn_ticket;
  a.err = h->err_word;
  const int n_blocks = L.n_seq * g.n_sub;
  if (!a.cluster &&
      (static_cast<size_t>(n_blocks) * c.n_kv_heads * L.max_items * g.rows * kAttnRow >
           h->attn_part_floats ||
       L.max_items > attn_max_merge_items(g.rows)))
    return fail(h, GS_ERR_OOM, "attention item scratch too small");
  GS_CUDA(h, launch_attention(h->tm_kv, a, n_blocks, h->stream, h->pdl));
  note_launch(h, GS_KIND_ATTENTION);
  return GS_OK;
}

// One decoder forward over T rows already described by tok/pos/lim/tok_slot.
// Visual rows (prefill) come first when n_vis > 0.  The LM head runs on rows
// [lm_row0, lm_row0 + n_lm) (none if n_lm == 0) and leaves argmax keys in
// `packed`.  Per layer: QKV (+norm scale, RoPE, KV write) -> attention ->
// O (+residual, next norm's input) -> gate/up (+norm scale, SwiGLU) -> down
// (+residual, next norm's input).
// LM-head options of a forward beyond the argmax: softmax partials at a
// temperature, and Gumbel-max sampling with per-row counters.
struct LmHeadOpts {
  float2* lse_part = nullptr;
  float inv_temp = 1.f;
  const uint4* rng_row = nullptr;
  uint64_t seed = 0;
};

int forward(gs_handle* h, int T, const int32_t* tok, const __nv_bfloat16* vis, int n_vis,
            const AttnLaunch& AL, int lm_row0, int n_lm, unsigned long long* packed,
            float* logits, bool decode, const LmHeadOpts& lmo = LmHeadOpts()) {
  const gs_config& c = h->cfg;
  const int d = c.d_model, F = c.d_ffn, HD = c.n_heads * 64, L = c.n_layers;
  GS_CUDA(h, launch_ex(embed_kernel, dim3(T), dim3(128), 0, h->stream, h->pdl, dim3(1), tok, h->embed, vis,
                       n_vis, T, d, c.vocab, h->hbuf, h->hb, h->attn_norm[0], h->ssp, packed,
                       h->err_word));
  note_launch(h, GS_KIND_EMBED);
  const size_t layer_kv = static_cast<size_t>(h->n_pages) * 2 * c.n_kv_heads * 64 * 64;
  int rc;
  for (int l = 0; l < L; ++l) {
    GemmArgs q = gemm_base(h);
    q.w_scale = h->sc_qkv[l];
    q.N = h->qkv_dim;
    q.ssp_in = h->ssp;
    q.q_out = h->qr;
    q.kv_layer = h->kv + l * layer_kv;
    q.pos = h->pos;
    q.tok_slot = h->tok_slot;
    q.page_table = h->page_table;
    q.rope = h->rope;
    q.pt_stride = h->pt_stride;
    q.n_pages = h->n_pages;
    q.max_ctx = c.max_ctx;
    q.Hq = c.n_heads;
    q.Hkv = c.n_kv_heads;
    if ((rc = run_gemm(h, h->tm_qkv[l], h->qkv_dim, h->tm_hb, d, T, kEpiQKV, q, decode,
                       GS_KIND_QKV)))
      return rc;
    if ((rc = run_attention(h, l, T, AL))) return rc;
    GemmArgs o = gemm_base(h);
    o.w_scale = h->sc_o[l];
    o.N = d;
    o.y = h->hbuf;
    o.ldy = d;
    o.hb_out = h->hb;
    o.g_next = h->ffn_norm[l];
    o.ssp_out = h->ssp;
    if ((rc = run_gemm(h, h->tm_o[l], d, h->tm_ao, HD, T, kEpiResidF32, o, decode,
                       GS_KIND_O_PROJ)))
      return rc;
    GemmArgs gu = gemm_base(h);
    gu.w_scale = h->sc_gu[l];
    gu.N = F;
    gu.y = h->act;
    gu.ldy = F;
    gu.ssp_in = h->ssp;
    if ((rc = run_gemm(h, h->tm_gu[l], 2 * F, h->tm_hb, d, T, kEpiSwiGLU, gu, decode,
                       GS_KIND_GATE_UP)))
      return rc;
    GemmArgs dn = gemm_base(h);
    dn.w_scale = h->sc_down[l];
    dn.N = d;
    dn.y = h->hbuf;
    dn.ldy = d;
    dn.hb_out = h->hb;
    dn.g_next = l + 1 < L ? h->attn_norm[l + 1] : h->final_norm;
    dn.ssp_out = h->ssp;
    if ((rc = run_gemm(h, h->tm_down[l], d, h->tm_act, F, T, kEpiResidF32, dn, decode,
                       GS_KIND_DOWN)))
      return rc;
  }
  if (n_lm == 0) return GS_OK;
  GemmArgs lm = gemm_base(h);
  lm.w_scale = h->sc_lm;
  lm.N = c.vocab;
  lm.y = packed;
  lm.logits = logits;
  lm.lse_part = lmo.lse_part;
  lm.inv_temp = lmo.inv_temp;
  lm.rng_row = lmo.rng_row;
  lm.seed_lo = static_cast<uint32_t>(lmo.seed);
  lm.seed_hi = static_cast<uint32_t>(lmo.seed >> 32);
  lm.ssp_in = h->ssp;
  lm.x_row0 = lm_row0;
  return run_gemm(h, h->tm_lm, c.vocab, h->tm_hb, d, n_lm, kEpiArgmax, lm, decode,
                  GS_KIND_LM_HEAD);
}

int enqueue_round(gs_handle* h, const int32_t* slots, int n_seq, int K, const gs_force* force,
                  int32_t* out_tok, int32_t* out_cnt, int32_t* out_done, const gs_debug* dbg,
                  int rule = GS_ACCEPT_GREEDY) {
  const bool stoch = rule == GS_ACCEPT_STOCHASTIC;
  const gs_config& c = h->cfg;
  const int W = K + 1, T = n_seq * W;
  WindowArgs w;
  memset(&w, 0, sizeof(w));
  w.slots = slots;
  w.n_seq = n_seq;
  w.K = K;
  w.W = W;
  w.mask_id = c.mask_token_id;
  w.vocab = c.vocab;
  w.st = h->st;
  w.tok = h->tok;
  w.pos = h->pos;
  w.lim = h->lim;
  w.tok_slot = h->tok_slot;
  w.blk_slot = h->blk_slot;
  w.blk_active = h->blk_active;
  w.draft_packed = h->packed_d;
  w.draft_tok = h->draft_tok;
  w.verify_in = h->verify_in;
  if (force) {
    w.teacher = force->teacher;
    w.teacher_stride = force->teacher_stride;
    w.L_sched = force->L_sched;
    w.L_stride = force->L_stride;
  }
  w.err = h->err_word;
  if (stoch) w.rng_row = h->rng_row;
  const int nb = cdiv(T, 128);
  AttnLaunch AL;
  AL.n_seq = n_seq;
  AL.QB = W;
  AL.split_pages = h->split_pages;
  AL.max_items = h->items_dec;
  AL.blk_slot = h->blk_slot;
  AL.blk_active = h->blk_active;
  AL.fixed_slot = -1;

  h->launches = 0;
  GS_CUDA(h, launch_ex(window_draft_kernel, dim3(nb), dim3(128), 0, h->stream, h->pdl, dim3(1), w));
  note_launch(h, GS_KIND_WINDOW);
  // stochastic rounds sample the draft rows and keep both heads' logits and
  // softmax partials at the temperature for the acceptance test
  LmHeadOpts lo_d, lo_v;
  if (stoch) {
    lo_d.lse_part = h->lse_part;
    lo_d.inv_temp = lo_v.inv_temp = 1.0f / h->temperature;
    lo_d.rng_row = h->rng_row;
    lo_d.seed = h->seed;
    lo_v.lse_part = h->lse_v;
  }
  int rc = forward(h, T, h->tok, nullptr, 0, AL, 0, T, h->packed_d,
                   stoch ? h->logits_d : (dbg ? dbg->draft_logits : nullptr), true, lo_d);
  if (rc) return rc;
  GS_CUDA(h, launch_ex(window_verify_kernel, dim3(nb), dim3(128), 0, h->stream, h->pdl, dim3(1), w));
  note_launch(h, GS_KIND_WINDOW);
  rc = forward(h, T, h->tok, nullptr, 0, AL, 0, T, h->packed_v,
               stoch ? h->logits_v : (dbg ? dbg->verify_logits : nullptr), true, lo_v);
  if (rc) return rc;
  if (stoch) {
    AcceptStochArgs as;
    memset(&as, 0, sizeof(as));
    as.slots = slots;
    as.n_seq = n_seq;
    as.K = K;
    as.W = W;
    as.eos = c.eos_token_id;
    as.vocab = c.vocab;
    as.lse_tiles = h->lse_tiles;
    as.st = h->st;
    as.verify_in = h->verify_in;
    as.logits_d = h->logits_d;
    as.logits_v = h->logits_v;
    as.lse_d = h->lse_part;
    as.lse_v = h->lse_v;
    as.inv_temp = 1.0f / h->temperature;
    as.seed_lo = static_cast<uint32_t>(h->seed);
    as.seed_hi = static_cast<uint32_t>(h->seed >> 32);
    as.verify_tok = h->verify_tok;
    as.out_tok = out_tok;
    as.out_cnt = out_cnt;
    as.out_done = out_done;
    as.err = h->err_word;
    GS_CUDA(h, launch_ex(accept_stochastic_kernel, dim3(n_seq), dim3(256), 0, h->stream, h->pdl,
                         dim3(1), as));
    note_launch(h, GS_KIND_ACCEPT);
    if (dbg) {
      const size_t bytes = static_cast<size_t>(T) * c.vocab * sizeof(float);
      if (dbg->draft_logits)
        GS_CUDA(h, cudaMemcpyAsync(dbg->draft_logits, h->logits_d, bytes, cudaMemcpyDeviceToDevice,
                                   h->stream));
      if (dbg->verify_logits)
        GS_CUDA(h, cudaMemcpyAsync(dbg->verify_logits, h->logits_v, bytes,
                                   cudaMemcpyDeviceToDevice, h->stream));
    }
  } else {
  AcceptArgs ac;
  ac.slots = slots;
  ac.n_seq = n_seq;
  ac.K = K;
  ac.W = W;
  ac.eos = c.eos_token_id;
  ac.st = h->st;
  ac.verify_in = h->verify_in;
  ac.verify_packed = h->packed_v;
  ac.verify_tok = h->verify_tok;
  ac.out_tok = out_tok;
  ac.out_cnt = out_cnt;
  ac.out_done = out_done;
  GS_CUDA(h, launch_ex(accept_commit_kernel, dim3(cdiv(n_seq, 64)), dim3(64), 0, h->stream, h->pdl, dim3(1),
                       ac));
  note_launch(h, GS_KIND_ACCEPT);
  }
  if (dbg) {
    if (dbg->draft_tok) copy_i32_kernel<<<nb, 128, 0, h->stream>>>(h->draft_tok, dbg->draft_tok, T);
    if (dbg->verify_in) copy_i32_kernel<<<nb, 128, 0, h->stream>>>(h->verify_in, dbg->verify_in, T);
    if (dbg->verify_tok)
      copy_i32_kernel<<<nb, 128, 0, h->stream>>>(h->verify_tok, dbg->verify_tok, T);
    GS_CUDA(h, cudaGetLastError());
    h->launches += (dbg->draft_tok != nullptr) + (dbg->verify_in != nullptr) +
                   (dbg->verify_tok != nullptr);
  }
  h->last_round_launches = h->launches;
  return GS_OK;
}

// Capture pre(), then a WHILE conditional node whose body is body(handle)
// (captured on the side stream), then post(), as one executable graph.  The
// loop runs while the handle's value is nonzero; it is 1 at every launch and
// the body's last kernel sets it.  Programmatic dependent launch is off for
// every launch of such a graph.
int capture_loop_graph(gs_handle* h, const std::function<int()>& pre,
                       const std::function<int(cudaGraphConditionalHandle)>& body,
                       const std::function<int()>& post, cudaGraphExec_t* out) {
  if (!h->side) GS_CUDA(h, cudaStreamCreateWithFlags(&h->side, cudaStreamNonBlocking));
  const bool pdl_was = h->pdl;
  h->pdl = false;
  cudaGraph_t g = nullptr;
  auto finish = [&](int code, const char* what, cudaError_t e) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(h->stream, &cs) == cudaSuccess && cs != cudaStreamCaptureStatusNone) {
      cudaGraph_t dead = nullptr;
      cudaStreamEndCapture(h->stream, &dead);
      if (dead) cudaGraphDestroy(dead);
    }
    h->pdl = pdl_was;
    if (code == GS_ERR_CUDA)
      return fail(h, code, std::string(what) + ": " + cudaGetErrorString(e));
    return code;
  };
  cudaError_t e = cudaStreamBeginCapture(h->stream, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) return finish(GS_ERR_CUDA, "loop capture", e);
  int rc = pre();
  if (rc) return finish(rc, "", cudaSuccess);
  cudaStreamCaptureStatus cs;
  cudaGraph_t cg = nullptr;
  const cudaGraphNode_t* deps = nullptr;
  const cudaGraphEdgeData* edata = nullptr;
  size_t ndeps = 0;
  e = cudaStreamGetCaptureInfo(h->stream, &cs, nullptr, &cg, &deps, &edata, &ndeps);
  if (e != cudaSuccess) return finish(GS_ERR_CUDA, "capture info", e);
  cudaGraphConditionalHandle hc;
  e = cudaGraphConditionalHandleCreate(&hc, cg, 1, cudaGraphCondAssignDefault);
  if (e != cudaSuccess) return finish(GS_ERR_CUDA, "conditional handle", e);
  cudaGraphNodeParams np = {};
  np.type = cudaGraphNodeTypeConditional;
  np.conditional.handle = hc;
  np.conditional.type = cudaGraphCondTypeWhile;
  np.conditional.size = 1;
  cudaGraphNode_t node;
  e = cudaGraphAddNode(&node, cg, deps, edata, ndeps, &np);
  if (e != cudaSuccess) return finish(GS_ERR_CUDA, "conditional node", e);
  cudaGraph_t body_graph = np.conditional.phGraph_out[0];
  e = cudaStreamUpdateCaptureDependencies(h->stream, &node, nullptr, 1,
                                          cudaStreamSetCaptureDependencies);
  if (e != cudaSuccess) return finish(GS_ERR_CUDA, "capture dependencies", e);
  e = cudaStreamBeginCaptureToGraph(h->side, body_graph, nullptr, nullptr, 0,
                                    cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) return finish(GS_ERR_CUDA, "body capture", e);
  std::swap(h->stream, h->side);
  rc = body(hc);
  std::swap(h->stream, h->side);
  cudaGraph_t captured_body = nullptr;
  e = cudaStreamEndCapture(h->side, &captured_body);
  if (rc) return finish(rc, "", cudaSuccess);
  if (e != cudaSuccess) return finish(GS_ERR_CUDA, "body capture end", e);
  rc = post();
  if (rc) return finish(rc, "", cudaSuccess);
  e = cudaStreamEndCapture(h->stream, &g);
  h->pdl = pdl_was;
  if (e != cudaSuccess) return fail(h, GS_ERR_CUDA, std::string("loop capture end: ") + cudaGetErrorString(e));
  e = cudaGraphInstantiate(out, g, 0);
  cudaGraphDestroy(g);
  if (e != cudaSuccess)
    return fail(h, GS_ERR_CUDA, std::string("loop graph instantiate: ") + cudaGetErrorString(e));
  return GS_OK;
}

DenoiseArgs denoise_args(gs_handle* h, const int32_t* slots, int n_seq, int W, int n_pred,
                         float tau) {
  DenoiseArgs d;
  memset(&d, 0, sizeof(d));
  d.slots = slots;
  d.n_seq = n_seq;
  d.W = W;
  d.n_pred = n_pred;
  d.mask_id = h->cfg.mask_token_id;
  d.vocab = h->cfg.vocab;
  d.eos = h->cfg.eos_token_id;
  d.tau = tau;
  d.st = h->st;
  d.fixed = h->dn_fixed;
  d.W_max = h->W_max;
  d.live = h->dn_live;
  d.part = h->dn_part;
  d.steps = h->dn_steps;
  d.iter = h->dn_iter;
  d.tok = h->tok;
  d.pos = h->pos;
  d.lim = h->lim;
  d.tok_slot = h->tok_slot;
  d.blk_slot = h->blk_slot;
  d.blk_active = h->blk_active;
  d.packed = h->packed_d;
  d.lse_part = h->lse_part;
  d.lse_tiles = h->lse_tiles;
  d.err = h->err_word;
  return d;
}

AttnLaunch decode_attention(gs_handle* h, int n_seq, int W) {
  AttnLaunch AL;
  AL.n_seq = n_seq;
  AL.QB = W;
  AL.split_pages = h->split_pages;
  AL.max_items = h->items_dec;
  AL.blk_slot = h->blk_slot;
  AL.blk_active = h->blk_active;
  AL.fixed_slot = -1;
  return AL;
}

// One denoising step (the body of the loop): window, forward with the LM
// head's argmax and softmax partials, reveal, loop condition.
int enqueue_denoise_step(gs_handle* h, DenoiseArgs d) {
  const int T = d.n_seq * d.W;
  GS_CUDA(h, launch_ex(denoise_window_kernel, dim3(cdiv(T, 128)), dim3(128), 0, h->stream, h->pdl,
                       dim3(1), d));
  note_launch(h, GS_KIND_WINDOW);
  LmHeadOpts lmo;
  lmo.lse_part = h->lse_part;
  int rc = forward(h, T, h->tok, nullptr, 0, decode_attention(h, d.n_seq, d.W), 0, T, h->packed_d,
                   nullptr, true, lmo);
  if (rc) return rc;
  GS_CUDA(h, launch_ex(denoise_reveal_kernel, dim3(d.n_seq), dim3(128), 0, h->stream, h->pdl,
                       dim3(1), d));
  note_launch(h, GS_KIND_ACCEPT);
  GS_CUDA(h, launch_ex(denoise_cond_kernel, dim3(1), dim3(32), 0, h->stream, h->pdl, dim3(1), d));
  note_launch(h, GS_KIND_ACCEPT);
  return GS_OK;
}

int launch_loop_graph(gs_handle* h, const std::vector<uint64_t>& key,
                      const std::function<int(cudaGraphExec_t*)>& build) {
  auto it = h->loop_graphs.find(key);
  if (it == h->loop_graphs.end()) {
    cudaGraphExec_t ge = nullptr;
    const int rc = build(&ge);
    if (rc) return rc;
    if (h->loop_graphs.size() >= 32) {
      cudaGraphExecDestroy(h->loop_graphs.begin()->second);
      h->loop_graphs.erase(h->loop_graphs.begin());
    }
    it = h->loop_graphs.emplace(key, ge).first;
  }
  GS_CUDA(h, cudaGraphLaunch(it->second, h->stream));
  return GS_OK;
}

uint64_t ptr_key(const void* p) { return static_cast<uint64_t>(reinterpret_cast<uintptr_t>(p)); }

uint32_t float_bits(float x) {
  uint32_t u;
  std::memcpy(&u, &x, 4);
  return u;
}

}  // namespace

// =================================================================== C ABI
extern "C" {

size_t gs_workspace_bytes(const gs_config* cfg) {
  std::string why;
  if (!config_ok(cfg, &why)) return 0;
  return carve(nullptr, *cfg, nullptr);
}

int gs_create(const gs_config* cfg, const gs_weights* w, void* workspace, size_t ws_bytes,
              void* stream, gs_handle** out) {
  if (!out) return fail(nullptr, GS_ERR_INVALID_ARG, "out is null");
  *out = nullptr;
  std::string why;
  if (!config_ok(cfg, &why)) return fail(nullptr, GS_ERR_INVALID_ARG, "config: " + why);
  if (!w || !w->embed || !w->lm_head || !w->final_norm || !w->attn_norm || !w->w_qkv || !w->w_o ||
      !w->ffn_norm || !w->w_gate_up || !w->w_down)
    return fail(nullptr, GS_ERR_INVALID_ARG, "null weight pointer");
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return fail(nullptr, GS_ERR_INVALID_ARG, "workspace null or not 256-byte aligned");
  const size_t need = carve(nullptr, *cfg, nullptr);
  if (ws_bytes < need)
    return fail(nullptr, GS_ERR_OOM, "workspace too small: need " + std::to_string(need));
  if (!get_encode()) return fail(nullptr, GS_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  if (const cudaError_t e = ensure_kernel_attributes(); e != cudaSuccess)
    return fail(nullptr, GS_ERR_CUDA, std::string("kernel attributes: ") + cudaGetErrorString(e));

  gs_handle* h = new gs_handle();
  h->cfg = *cfg;
  h->stream = static_cast<cudaStream_t>(stream);
  carve(h, *cfg, workspace);
  const gs_config& c = h->cfg;
  const int L = c.n_layers, d = c.d_model, F = c.d_ffn, HD = c.n_heads * 64;
  auto chk = [&](const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  bool ok = chk(w->embed) && chk(w->lm_head) && chk(w->final_norm);
  for (int l = 0; l < L && ok; ++l)
    ok = chk(w->attn_norm[l]) && chk(w->ffn_norm[l]) && chk(w->w_qkv[l]) && chk(w->w_o[l]) &&
         chk(w->w_gate_up[l]) && chk(w->w_down[l]);
  if (!ok) {
    delete h;
    return fail(nullptr, GS_ERR_INVALID_ARG, "null or misaligned weight pointer");
  }
  h->embed = static_cast<const __nv_bfloat16*>(w->embed);
  h->final_norm = static_cast<const __nv_bfloat16*>(w->final_norm);
  for (int l = 0; l < L; ++l) {
    h->attn_norm.push_back(static_cast<const __nv_bfloat16*>(w->attn_norm[l]));
    h->ffn_norm.push_back(static_cast<const __nv_bfloat16*>(w->ffn_norm[l]));
  }

  // zero the workspace, page table -> -1, rope table
  cudaError_t e = cudaMemsetAsync(workspace, 0, need, h->stream);
  h->pt_host.assign(static_cast<size_t>(c.max_batch) * h->pt_stride, -1);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h->page_table, h->pt_host.data(), h->pt_host.size() * 4,
                        cudaMemcpyHostToDevice, h->stream);
  if (e == cudaSuccess) {
    rope_table_kernel<<<cdiv(static_cast<long long>(c.max_ctx) * 32, 256), 256, 0, h->stream>>>(
        h->rope, c.max_ctx, static_cast<double>(c.rope_theta));
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) {
    // sequences start "done" so a round over an unprefilled slot commits nothing
    std::vector<int32_t> ones(c.max_batch, 1);
    e = cudaMemcpyAsync(h->st.done, ones.data(), ones.size() * 4, cudaMemcpyHostToDevice, h->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  }

  // fp16 weight copies.  Per tensor: the largest |w| (into the zeroed split-K
  // counters), then w * 2^s with 2^s putting that maximum just below 2^15.
  struct Src { const void* p; size_t n; };
  std::vector<Src> src;
  for (int l = 0; l < L; ++l) {
    src.push_back({w->w_qkv[l], static_cast<size_t>(h->qkv_dim) * d});
    src.push_back({w->w_o[l], static_cast<size_t>(d) * HD});
    src.push_back({w->w_gate_up[l], 2 * static_cast<size_t>(F) * d});
    src.push_back({w->w_down[l], static_cast<size_t>(d) * F});
  }
  src.push_back({w->lm_head, static_cast<size_t>(c.vocab) * d});
  unsigned int* amax = reinterpret_cast<unsigned int*>(h->gemm_counters);
  for (size_t t = 0; t < src.size() && e == cudaSuccess; ++t) {
    absmax_bf16_kernel<<<304, 256, 0, h->stream>>>(static_cast<const __nv_bfloat16*>(src[t].p),
                                                    src[t].n, amax + t);
    e = cudaGetLastError();
  }
  std::vector<unsigned int> amax_host(src.size(), 0);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(amax_host.data(), amax, src.size() * 4, cudaMemcpyDeviceToHost, h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  std::vector<float> scales(src.size(), 1.f);
  __half* dst = h->wcopy;
  std::vector<const __half*> copies(src.size());
  for (size_t t = 0; t < src.size() && e == cudaSuccess; ++t) {
    float m;
    std::memcpy(&m, &amax_host[t], 4);
    int s_exp = 0;
    if (m > 0.f && std::isfinite(m)) {
      int ex = 0;
      std::frexp(m, &ex);                // m = f * 2^ex, f in [0.5, 1)
      s_exp = std::min(100, std::max(-100, 15 - ex));
    }
    scales[t] = std::ldexp(1.f, -s_exp);
    scale_to_f16_kernel<<<304, 256, 0, h->stream>>>(static_cast<const __nv_bfloat16*>(src[t].p),
                                                     src[t].n, std::ldexp(1.f, s_exp), dst);
    e = cudaGetLastError();
    copies[t] = dst;
    dst += src[t].n;
  }
  if (e == cudaSuccess) e = cudaMemsetAsync(amax, 0, src.size() * 4, h->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) {
    delete h;
    return fail(nullptr, GS_ERR_CUDA, std::string("workspace init: ") + cudaGetErrorString(e));
  }
  for (int l = 0; l < L; ++l) {
    h->w_qkv.push_back(copies[4 * l + 0]);
    h->w_o.push_back(copies[4 * l + 1]);
    h->w_gu.push_back(copies[4 * l + 2]);
    h->w_down.push_back(copies[4 * l + 3]);
    h->sc_qkv.push_back(scales[4 * l + 0]);
    h->sc_o.push_back(scales[4 * l + 1]);
    h->sc_gu.push_back(scales[4 * l + 2]);
    h->sc_down.push_back(scales[4 * l + 3]);
  }
  h->lm_head = copies[4 * L];
  h->sc_lm = scales[4 * L];

  h->tm_qkv.resize(L);
  h->tm_o.resize(L);
  h->tm_gu.resize(L);
  h->tm_down.resize(L);
  for (int l = 0; l < L && ok; ++l)
    ok = make_map(&h->tm_qkv[l], h->w_qkv[l], h->qkv_dim, d, 128) &&
         make_map(&h->tm_o[l], h->w_o[l], d, HD, 128) &&
         make_map(&h->tm_gu[l], h->w_gu[l], 2 * F, d, 64) &&
         make_map(&h->tm_down[l], h->w_down[l], d, F, 128);
  ok = ok && make_map(&h->tm_lm, h->lm_head, c.vocab, d, 128);
  const int bns[4] = {32, 64, 128, 256};
  for (int i = 0; i < 4 && ok; ++i) {
    ok = make_map(&h->tm_hb[i], h->hb, h->T_max, d, bns[i]) &&
         make_map(&h->tm_ao[i], h->ao, h->T_max, HD, bns[i]) &&
         make_map(&h->tm_act[i], h->act, h->T_max, F, bns[i]);
  }
  const uint64_t kv_rows = static_cast<uint64_t>(L) * h->n_pages * 2 * c.n_kv_heads * 64;
  ok = ok && kv_rows < (1ull << 31) && make_map(&h->tm_kv, h->kv, kv_rows, 64, 64);
  if (!ok) {
    delete h;
    return fail(nullptr, GS_ERR_INVALID_ARG, "tensor-map encode failed");
  }
  h->free_pages.reserve(h->n_pages);
  for (int p = h->n_pages - 1; p >= 0; --p) h->free_pages.push_back(p);
  h->slot_pages.assign(c.max_batch, {});
  h->slot_reserved.assign(c.max_batch, 0);
  *out = h;
  return GS_OK;
}

int gs_destroy(gs_handle* h) {
  if (!h) return GS_ERR_INVALID_ARG;
  for (auto& kv : h->graphs) cudaGraphExecDestroy(kv.second);
  for (auto& kv : h->loop_graphs) cudaGraphExecDestroy(kv.second);
  if (h->side) cudaStreamDestroy(h->side);
  for (cudaEvent_t e : h->prof_ev) cudaEventDestroy(e);
  delete h;
  return GS_OK;
}

const char* gs_last_error(gs_handle* h) { return h ? h->err.c_str() : g_create_error.c_str(); }

int gs_release(gs_handle* h, int slot) {
  if (!h) return GS_ERR_INVALID_ARG;
  if (slot < 0 || slot >= h->cfg.max_batch) return fail(h, GS_ERR_INVALID_ARG, "slot out of range");
  for (int p : h->slot_pages[slot]) h->free_pages.push_back(p);
  h->slot_pages[slot].clear();
  h->slot_reserved[slot] = 0;
  std::fill(h->pt_host.begin() + static_cast<size_t>(slot) * h->pt_stride,
            h->pt_host.begin() + static_cast<size_t>(slot + 1) * h->pt_stride, -1);
  GS_CUDA(h, cudaMemcpyAsync(h->page_table + static_cast<size_t>(slot) * h->pt_stride,
                             h->pt_host.data() + static_cast<size_t>(slot) * h->pt_stride,
                             h->pt_stride * 4, cudaMemcpyHostToDevice, h->stream));
  const int one = 1;
  GS_CUDA(h, cudaMemcpyAsync(h->st.done + slot, &one, 4, cudaMemcpyHostToDevice, h->stream));
  GS_CUDA(h, cudaStreamSynchronize(h->stream));
  return GS_OK;
}

int gs_prefill(gs_handle* h, int slot, const void* vis_emb, int n_vis, const int32_t* text,
               int n_text, int max_new, int32_t* x0_out) {
  if (!h) return GS_ERR_INVALID_ARG;
  const gs_config& c = h->cfg;
  if (slot < 0 || slot >= c.max_batch) return fail(h, GS_ERR_INVALID_ARG, "slot out of range");
  if (n_vis < 0 || n_text < 0 || n_vis + n_text < 1 || max_new < 1)
    return fail(h, GS_ERR_INVALID_ARG, "bad prefix or max_new");
  if ((n_vis > 0 && !vis_emb) || (n_text > 0 && !text))
    return fail(h, GS_ERR_INVALID_ARG, "null prefix pointer");
  if (vis_emb && (reinterpret_cast<uintptr_t>(vis_emb) & 15))
    return fail(h, GS_ERR_INVALID_ARG, "vis_emb not 16-byte aligned");
  const long long P = static_cast<long long>(n_vis) + n_text;
  const long long reserve = P + max_new + c.max_K + 2;
  if (reserve > c.max_ctx) return fail(h, GS_ERR_OOM, "prefix + max_new + max_K + 2 > max_ctx");
  // (re)reserve pages
  int rc = gs_release(h, slot);
  if (rc) return rc;
  const int need = cdiv(reserve, 64);
  if (need > static_cast<int>(h->free_pages.size()))
    return fail(h, GS_ERR_OOM, "KV page pool exhausted");
  for (int i = 0; i < need; ++i) {
    const int p = h->free_pages.back();
    h->free_pages.pop_back();
    h->slot_pages[slot].push_back(p);
    h->pt_host[static_cast<size_t>(slot) * h->pt_stride + i] = p;
  }
  h->slot_reserved[slot] = static_cast<int>(reserve);
  GS_CUDA(h, cudaMemcpyAsync(h->page_table + static_cast<size_t>(slot) * h->pt_stride,
                             h->pt_host.data() + static_cast<size_t>(slot) * h->pt_stride,
                             h->pt_stride * 4, cudaMemcpyHostToDevice, h->stream));
  // causal forward in chunks of max_prefill tokens
  const int chunk = std::min(c.max_prefill, h->T_max);
  const __nv_bfloat16* vis = static_cast<const __nv_bfloat16*>(vis_emb);
  for (long long p0 = 0; p0 < P; p0 += chunk) {
    const int T = static_cast<int>(std::min<long long>(chunk, P - p0));
    const int vis_rows = static_cast<int>(std::max<long long>(0, std::min<long long>(n_vis - p0, T)));
    const long long text0 = std::max<long long>(0, p0 - n_vis);
    prefill_window_kernel<<<cdiv(T, 128), 128, 0, h->stream>>>(T, static_cast<int>(p0), slot,
                                                               h->pos, h->lim, h->tok_slot);
    GS_CUDA(h, cudaGetLastError());
    AttnLaunch AL;
    AL.QB = h->qb_pf;
    AL.n_seq = cdiv(T, h->qb_pf);   // prefill blocks (one per QB tokens)
    AL.split_pages = h->split_pages_pf;
    AL.max_items = h->items_pf;
    AL.blk_slot = nullptr;
    AL.blk_active = nullptr;
    AL.fixed_slot = slot;
    const bool last = p0 + T >= P;
    rc = forward(h, T, text ? text + text0 : nullptr, vis ? vis + p0 * c.d_model : nullptr,
                 vis_rows, AL, last ? T - 1 : 0, last ? 1 : 0, h->packed_d, nullptr, false);
    if (rc) return rc;
  }
  prefill_finish_kernel<<<1, 32, 0, h->stream>>>(h->packed_d, h->st, slot, static_cast<int>(P),
                                                 max_new, c.eos_token_id, x0_out);
  GS_CUDA(h, cudaGetLastError());
  return GS_OK;
}

int gs_round(gs_handle* h, const int32_t* slots, int n_seq, int K, int rule, const gs_force* force,
             int32_t* out_tok, int32_t* out_cnt, int32_t* out_done, const gs_debug* dbg) {
  if (!h) return GS_ERR_INVALID_ARG;
  const gs_config& c = h->cfg;
  if (rule != GS_ACCEPT_GREEDY && rule != GS_ACCEPT_STOCHASTIC)
    return fail(h, GS_ERR_INVALID_ARG, "unknown acceptance rule");
  if (rule == GS_ACCEPT_STOCHASTIC && force)
    return fail(h, GS_ERR_INVALID_ARG, "forcing applies to greedy rounds only");
  if (!slots || !out_tok || !out_cnt || !out_done)
    return fail(h, GS_ERR_INVALID_ARG, "null slots or output pointer");
  if (n_seq < 1 || n_seq > c.max_batch) return fail(h, GS_ERR_INVALID_ARG, "n_seq out of range");
  if (K < 0 || K > c.max_K) return fail(h, GS_ERR_INVALID_ARG, "K out of range");
  if (force && (!force->teacher || !force->L_sched || force->teacher_stride < 1))
    return fail(h, GS_ERR_INVALID_ARG, "incomplete force hook");
  if (dbg || h->stream == nullptr)
    return enqueue_round(h, slots, n_seq, K, force, out_tok, out_cnt, out_done, dbg, rule);
  // stochastic rounds are keyed by their temperature and seed as well (the
  // kernels take them as arguments)
  const long long samp = rule == GS_ACCEPT_STOCHASTIC
                             ? static_cast<long long>(float_bits(h->temperature)) ^
                                   static_cast<long long>(h->seed * 0x9E3779B97F4A7C15ull) ^ 1ll
                             : 0ll;
  gs_handle::GraphKey key(n_seq, K, slots, force ? force->teacher : nullptr,
                          force ? force->teacher_stride : 0, force ? force->L_sched : nullptr,
                          force ? force->L_stride : 0, out_tok, out_cnt, out_done, samp);
  auto it = h->graphs.find(key);
  if (it == h->graphs.end()) {
    cudaGraph_t g;
    GS_CUDA(h, cudaStreamBeginCapture(h->stream, cudaStreamCaptureModeThreadLocal));
    const int rc = enqueue_round(h, slots, n_seq, K, force, out_tok, out_cnt, out_done, nullptr, rule);
    cudaError_t e = cudaStreamEndCapture(h->stream, &g);
    if (rc) {
      if (e == cudaSuccess) cudaGraphDestroy(g);
      return rc;
    }
    if (e != cudaSuccess) return fail(h, GS_ERR_CUDA, std::string("capture: ") + cudaGetErrorString(e));
    cudaGraphExec_t ge;
    e = cudaGraphInstantiate(&ge, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess)
      return fail(h, GS_ERR_CUDA, std::string("instantiate: ") + cudaGetErrorString(e));
    if (h->graphs.size() >= 64) {
      cudaGraphExecDestroy(h->graphs.begin()->second);
      h->graphs.erase(h->graphs.begin());
    }
    it = h->graphs.emplace(key, ge).first;
  }
  GS_CUDA(h, cudaGraphLaunch(it->second, h->stream));
  return GS_OK;
}

int gs_diffusion_block(gs_handle* h, const int32_t* slots, int n_seq, int B, float tau_c,
                       int32_t* out_tok, int32_t* out_cnt, int32_t* out_done, int32_t* out_steps) {
  if (!h) return GS_ERR_INVALID_ARG;
  const gs_config& c = h->cfg;
  if (!slots || !out_tok || !out_cnt || !out_done)
    return fail(h, GS_ERR_INVALID_ARG, "null slots or output pointer");
  if (n_seq < 1 || n_seq > c.max_batch) return fail(h, GS_ERR_INVALID_ARG, "n_seq out of range");
  if (B < 1 || B > c.max_K) return fail(h, GS_ERR_INVALID_ARG, "B out of range (1..max_K)");
  if (!(tau_c == tau_c)) return fail(h, GS_ERR_INVALID_ARG, "tau_c is NaN");
  if (!h->stream) return fail(h, GS_ERR_INVALID_ARG, "block diffusion needs a non-default stream");
  const int W = B + 1, T = n_seq * W;
  const std::vector<uint64_t> key = {1, static_cast<uint64_t>(n_seq), static_cast<uint64_t>(B),
                                     float_bits(tau_c), ptr_key(slots), ptr_key(out_tok),
                                     ptr_key(out_cnt), ptr_key(out_done), ptr_key(out_steps)};
  return launch_loop_graph(h, key, [&](cudaGraphExec_t* ge) -> int {
    DenoiseArgs d = denoise_args(h, slots, n_seq, W, B, tau_c);
    d.out_tok = out_tok;
    d.out_cnt = out_cnt;
    d.out_done = out_done;
    d.out_steps = out_steps;
    h->launches = 0;
    return capture_loop_graph(
        h,
        [&]() -> int {
          GS_CUDA(h, launch_ex(denoise_init_kernel, dim3(n_seq), dim3(32), 0, h->stream, h->pdl,
                               dim3(1), d));
          note_launch(h, GS_KIND_WINDOW);
          return GS_OK;
        },
        [&](cudaGraphConditionalHandle hc) -> int {
          DenoiseArgs db = d;
          db.cond = hc;
          return enqueue_denoise_step(h, db);
        },
        [&]() -> int {
          // the cache-write pass of the completed blocks (no LM head), then commit
          GS_CUDA(h, launch_ex(block_write_window_kernel, dim3(cdiv(T, 128)), dim3(128), 0,
                               h->stream, h->pdl, dim3(1), d));
          note_launch(h, GS_KIND_WINDOW);
          int rc = forward(h, T, h->tok, nullptr, 0, decode_attention(h, n_seq, W), 0, 0,
                           h->packed_d, nullptr, true);
          if (rc) return rc;
          GS_CUDA(h, launch_ex(block_commit_kernel, dim3(cdiv(n_seq, 64)), dim3(64), 0, h->stream,
                               h->pdl, dim3(1), d));
          note_launch(h, GS_KIND_ACCEPT);
          return GS_OK;
        },
        ge);
  });
}

int gs_round_refined(gs_handle* h, const int32_t* slots, int n_seq, int K, float tau_d,
                     const gs_force* force, int32_t* out_tok, int32_t* out_cnt, int32_t* out_done,
                     int32_t* out_steps) {
  if (!h) return GS_ERR_INVALID_ARG;
  const gs_config& c = h->cfg;
  if (!slots || !out_tok || !out_cnt || !out_done)
    return fail(h, GS_ERR_INVALID_ARG, "null slots or output pointer");
  if (n_seq < 1 || n_seq > c.max_batch) return fail(h, GS_ERR_INVALID_ARG, "n_seq out of range");
  if (K < 0 || K > c.max_K) return fail(h, GS_ERR_INVALID_ARG, "K out of range");
  if (!(tau_d == tau_d)) return fail(h, GS_ERR_INVALID_ARG, "tau_d is NaN");
  if (force && (!force->teacher || !force->L_sched || force->teacher_stride < 1))
    return fail(h, GS_ERR_INVALID_ARG, "incomplete force hook");
  if (!h->stream) return fail(h, GS_ERR_INVALID_ARG, "multi-step drafting needs a non-default stream");
  const int W = K + 1, T = n_seq * W;
  const std::vector<uint64_t> key = {
      2, static_cast<uint64_t>(n_seq), static_cast<uint64_t>(K), float_bits(tau_d), ptr_key(slots),
      ptr_key(out_tok), ptr_key(out_cnt), ptr_key(out_done), ptr_key(out_steps),
      ptr_key(force ? force->teacher : nullptr),
      static_cast<uint64_t>(force ? force->teacher_stride : 0),
      ptr_key(force ? force->L_sched : nullptr), static_cast<uint64_t>(force ? force->L_stride : 0)};
  return launch_loop_graph(h, key, [&](cudaGraphExec_t* ge) -> int {
    DenoiseArgs d = denoise_args(h, slots, n_seq, W, W, tau_d);
    h->launches = 0;
    return capture_loop_graph(
        h,
        [&]() -> int {
          GS_CUDA(h, launch_ex(denoise_init_kernel, dim3(n_seq), dim3(32), 0, h->stream, h->pdl,
                               dim3(1), d));
          note_launch(h, GS_KIND_WINDOW);
          return GS_OK;
        },
        [&](cudaGraphConditionalHandle hc) -> int {
          DenoiseArgs db = d;
          db.cond = hc;
          return enqueue_denoise_step(h, db);
        },
        [&]() -> int {
          // verify the refined draft exactly as a one-shot draft, then accept
          WindowArgs w;
          memset(&w, 0, sizeof(w));
          w.slots = slots;
          w.n_seq = n_seq;
          w.K = K;
          w.W = W;
          w.mask_id = c.mask_token_id;
          w.vocab = c.vocab;
          w.st = h->st;
          w.tok = h->tok;
          w.pos = h->pos;
          w.lim = h->lim;
          w.tok_slot = h->tok_slot;
          w.blk_slot = h->blk_slot;
          w.blk_active = h->blk_active;
          w.draft_packed = h->packed_d;
          w.draft_tok = h->draft_tok;
          w.verify_in = h->verify_in;
          w.draft_fixed = h->dn_fixed;
          w.fixed_stride = h->W_max;
          w.steps_src = h->dn_steps;
          w.steps_out = out_steps;
          if (force) {
            w.teacher = force->teacher;
            w.teacher_stride = force->teacher_stride;
            w.L_sched = force->L_sched;
            w.L_stride = force->L_stride;
          }
          w.err = h->err_word;
          GS_CUDA(h, launch_ex(window_verify_kernel, dim3(cdiv(T, 128)), dim3(128), 0, h->stream,
                               h->pdl, dim3(1), w));
          note_launch(h, GS_KIND_WINDOW);
          int rc = forward(h, T, h->tok, nullptr, 0, decode_attention(h, n_seq, W), 0, T,
                           h->packed_v, nullptr, true);
          if (rc) return rc;
          AcceptArgs ac;
          ac.slots = slots;
          ac.n_seq = n_seq;
          ac.K = K;
          ac.W = W;
          ac.eos = c.eos_token_id;
          ac.st = h->st;
          ac.verify_in = h->verify_in;
          ac.verify_packed = h->packed_v;
          ac.verify_tok = h->verify_tok;
          ac.out_tok = out_tok;
          ac.out_cnt = out_cnt;
          ac.out_done = out_done;
          GS_CUDA(h, launch_ex(accept_commit_kernel, dim3(cdiv(n_seq, 64)), dim3(64), 0, h->stream,
                               h->pdl, dim3(1), ac));
          note_launch(h, GS_KIND_ACCEPT);
          return GS_OK;
        },
        ge);
  });
}

int gs_set_sampling(gs_handle* h, float temperature, uint64_t seed) {
  if (!h) return GS_ERR_INVALID_ARG;
  if (!(temperature > 0.f) || !std::isfinite(1.0f / temperature))
    return fail(h, GS_ERR_INVALID_ARG, "temperature must be positive and finite");
  h->temperature = temperature;
  h->seed = seed;
  return GS_OK;
}

int gs_seq_restore(gs_handle* h, int slot, int seq_len, int x0, int n_out, int max_new, int done,
                   int rounds) {
  if (!h) return GS_ERR_INVALID_ARG;
  const gs_config& c = h->cfg;
  if (slot < 0 || slot >= c.max_batch || h->slot_reserved[slot] == 0)
    return fail(h, GS_ERR_INVALID_ARG, "slot out of range or not prefilled");
  if (seq_len < 1 || seq_len + c.max_K + 2 > h->slot_reserved[slot])
    return fail(h, GS_ERR_INVALID_ARG, "seq_len outside the slot's reservation");
  if (x0 < 0 || x0 >= c.vocab || n_out < 1 || max_new < n_out || rounds < 0)
    return fail(h, GS_ERR_INVALID_ARG, "bad x0 / n_out / max_new / rounds");
  // the cap must keep every reachable round inside the reservation
  if (static_cast<long long>(seq_len) + (max_new - n_out) + c.max_K + 2 > h->slot_reserved[slot])
    return fail(h, GS_ERR_INVALID_ARG, "max_new reaches past the slot's reservation");
  seq_restore_kernel<<<1, 32, 0, h->stream>>>(h->st, slot, seq_len, x0, n_out, max_new,
                                              done ? 1 : 0, rounds);
  GS_CUDA(h, cudaGetLastError());
  return GS_OK;
}

int gs_round_launches(gs_handle* h) { return h ? h->last_round_launches : 0; }

int gs_round_profile(gs_handle* h, const int32_t* slots, int n_seq, int K, const gs_force* force,
                     int32_t* out_tok, int32_t* out_cnt, int32_t* out_done, int max_launches,
                     float* ms, int* kind, int* n_launches) {
  if (!h) return GS_ERR_INVALID_ARG;
  if (!ms || !kind || !n_launches || max_launches < 1)
    return fail(h, GS_ERR_INVALID_ARG, "null or empty profile output");
  if (!h->stream) return fail(h, GS_ERR_INVALID_ARG, "profiling needs a non-default stream");
  const gs_config& c = h->cfg;
  if (!slots || !out_tok || !out_cnt || !out_done)
    return fail(h, GS_ERR_INVALID_ARG, "null slots or output pointer");
  if (n_seq < 1 || n_seq > c.max_batch) return fail(h, GS_ERR_INVALID_ARG, "n_seq out of range");
  if (K < 0 || K > c.max_K) return fail(h, GS_ERR_INVALID_ARG, "K out of range");
  if (force && (!force->teacher || !force->L_sched || force->teacher_stride < 1))
    return fail(h, GS_ERR_INVALID_ARG, "incomplete force hook");
  *n_launches = 0;
  if (h->prof_ev.empty()) {
    cudaEvent_t e;
    GS_CUDA(h, cudaEventCreate(&e));
    h->prof_ev.push_back(e);
  }
  h->prof_kind.clear();
  h->prof_err = cudaSuccess;
  // The round with an event after every launch is captured and replayed as
  // one graph, so the host's enqueue time never separates two launches; an
  // event node between two kernels turns their programmatic overlap into a
  // plain dependency, so each interval is one kernel's whole duration.
  cudaGraph_t g = nullptr;
  GS_CUDA(h, cudaStreamBeginCapture(h->stream, cudaStreamCaptureModeThreadLocal));
  cudaError_t e0 = cudaEventRecordWithFlags(h->prof_ev[0], h->stream, cudaEventRecordExternal);
  h->profiling = true;
  const int rc = enqueue_round(h, slots, n_seq, K, force, out_tok, out_cnt, out_done, nullptr);
  h->profiling = false;
  cudaError_t e1 = cudaStreamEndCapture(h->stream, &g);
  if (rc) {
    if (e1 == cudaSuccess) cudaGraphDestroy(g);
    return rc;
  }
  if (e0 != cudaSuccess || e1 != cudaSuccess || h->prof_err != cudaSuccess) {
    if (e1 == cudaSuccess) cudaGraphDestroy(g);
    const cudaError_t e = e0 != cudaSuccess ? e0 : (e1 != cudaSuccess ? e1 : h->prof_err);
    return fail(h, GS_ERR_CUDA, std::string("profile capture: ") + cudaGetErrorString(e));
  }
  cudaGraphExec_t ge = nullptr;
  cudaError_t e2 = cudaGraphInstantiate(&ge, g, 0);
  cudaGraphDestroy(g);
  if (e2 != cudaSuccess) return fail(h, GS_ERR_CUDA, std::string("profile graph: ") + cudaGetErrorString(e2));
  e2 = cudaGraphLaunch(ge, h->stream);
  if (e2 == cudaSuccess) e2 = cudaStreamSynchronize(h->stream);
  cudaGraphExecDestroy(ge);
  if (e2 != cudaSuccess) return fail(h, GS_ERR_CUDA, std::string("profile replay: ") + cudaGetErrorString(e2));
  const int n = static_cast<int>(h->prof_kind.size());
  if (n > max_launches) return fail(h, GS_ERR_INVALID_ARG, "max_launches below the round's launches");
  for (int i = 0; i < n; ++i) {
    GS_CUDA(h, cudaEventElapsedTime(&ms[i], h->prof_ev[i], h->prof_ev[i + 1]));
    kind[i] = h->prof_kind[i];
  }
  *n_launches = n;
  return GS_OK;
}

int gs_seq_state(gs_handle* h, int slot, int* seq_len, int* x0, int* n_out, int* done, int* rounds) {
  if (!h) return GS_ERR_INVALID_ARG;
  if (slot < 0 || slot >= h->cfg.max_batch) return fail(h, GS_ERR_INVALID_ARG, "slot out of range");
  GS_CUDA(h, cudaStreamSynchronize(h->stream));
  int v[6];
  int32_t* src[6] = {h->st.seq_len, h->st.x0, h->st.n_out, h->st.done, h->st.rounds, h->st.max_new};
  for (int i = 0; i < 6; ++i) GS_CUDA(h, cudaMemcpy(&v[i], src[i] + slot, 4, cudaMemcpyDeviceToHost));
  if (seq_len) *seq_len = v[0];
  if (x0) *x0 = v[1];
  if (n_out) *n_out = v[2];
  if (done) *done = v[3];
  if (rounds) *rounds = v[4];
  return GS_OK;
}

int gs_wait_probe(gs_handle* h, int limit_us) {
  if (!h) return GS_ERR_INVALID_ARG;
  if (limit_us < 1 || limit_us > 2000000) return fail(h, GS_ERR_INVALID_ARG, "limit_us out of range");
  wait_probe_kernel<<<1, 32, 0, h->stream>>>(h->err_word, static_cast<uint64_t>(limit_us) * 1000u);
  GS_CUDA(h, cudaGetLastError());
  return GS_OK;
}

int gs_sync_check(gs_handle* h) {
  if (!h) return GS_ERR_INVALID_ARG;
  GS_CUDA(h, cudaStreamSynchronize(h->stream));
  int word = 0;
  GS_CUDA(h, cudaMemcpy(&word, h->err_word, 4, cudaMemcpyDeviceToHost));
  if (word == 0) return GS_OK;
  const int zero = 0;
  GS_CUDA(h, cudaMemcpy(h->err_word, &zero, 4, cudaMemcpyHostToDevice));
  if (word == kErrTimeout) return fail(h, GS_ERR_TIMEOUT, "a kernel's bounded wait ran out");
  return fail(h, GS_ERR_DEVICE_CHECK, "a kernel bounds check fired");
}

// ------------------------------------------------------------ sub-step entry points
size_t gs_attention_scratch_bytes(int n_seq, int W, int n_heads, int n_kv_heads, int max_pages,
                                  int split_pages) {
  if (n_seq < 1 || W < 1 || n_kv_heads < 1 || n_heads % n_kv_heads || max_pages < 1 ||
      split_pages < 1)
    return 0;
  const AttnGeom g = attn_geom(W, n_heads / n_kv_heads);
  const int items = cdiv(max_pages, split_pages);
  const size_t blocks = static_cast<size_t>(n_seq) * g.n_sub;
  Carver cv(nullptr);
  cv.take<int>(64);                                   // error word
  cv.take<int32_t>(static_cast<size_t>(n_seq) * W);  // key limits
  cv.take<int32_t>(n_seq);                            // sequence -> page-table row
  cv.take<int>(blocks * n_kv_heads);                  // merge tickets
  if (!attn_use_cluster(items, static_cast<int>(blocks) * n_kv_heads))   // global merge rows
    cv.take<float>(blocks * n_kv_heads * items * g.rows * kAttnRow);
  return align_up(cv.off, 256);
}

}  // extern "C"

namespace {
__global__ void attn_standalone_prep(int mode, const int32_t* n, int n_seq, int W, int32_t* lim,
                                     int32_t* blk_slot) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= n_seq * W) return;
  const int b = idx / W, i = idx % W;
  const int ns = n[b];
  lim[idx] = mode == 0 ? (i == 0 ? ns : ns + W - 1) : ns + 1 + i;
  if (i == 0) blk_slot[b] = b;
}
}  // namespace

extern "C" {

int gs_attention(int mode, const void* q, const void* kv, int n_pages, const int32_t* page_table,
                 int pt_stride, const int32_t* n, int n_seq, int W, int n_heads, int n_kv_heads,
                 void* out, void* scratch, size_t scratch_bytes, int split_pages, void* stream) {
  if ((mode != 0 && mode != 1) || !q || !kv || !page_table || !n || !out || !scratch ||
      n_pages < 1 || pt_stride < 1)
    return GS_ERR_INVALID_ARG;
  if (n_kv_heads < 1 || n_heads % n_kv_heads || W < 1 || n_seq < 1 || split_pages < 1)
    return GS_ERR_INVALID_ARG;
  const int G = n_heads / n_kv_heads;
  if (G > kAttnMaxRows) return GS_ERR_UNSUPPORTED;
  if (scratch_bytes < gs_attention_scratch_bytes(n_seq, W, n_heads, n_kv_heads, pt_stride, split_pages))
    return GS_ERR_OOM;
  if ((reinterpret_cast<uintptr_t>(kv) & 15) || (reinterpret_cast<uintptr_t>(q) & 15))
    return GS_ERR_INVALID_ARG;
  if (ensure_kernel_attributes() != cudaSuccess) return GS_ERR_CUDA;
  const AttnGeom g = attn_geom(W, G);
  const int items = cdiv(pt_stride, split_pages);
  if (items > attn_max_merge_items(g.rows)) return GS_ERR_UNSUPPORTED;
  const size_t blocks = static_cast<size_t>(n_seq) * g.n_sub;
  Carver cv(scratch);
  int* err = cv.take<int>(64);
  int32_t* lim = cv.take<int32_t>(static_cast<size_t>(n_seq) * W);
  int32_t* blk_slot = cv.take<int32_t>(n_seq);
  int* ticket = cv.take<int>(blocks * n_kv_heads);
  float* part = attn_use_cluster(items, static_cast<int>(blocks) * n_kv_heads)
                    ? nullptr
                    : cv.take<float>(blocks * n_kv_heads * items * g.rows * kAttnRow);
  CUtensorMap tm;
  const uint64_t rows = static_cast<uint64_t>(n_pages) * 2 * n_kv_heads * 64;
  if (rows >= (1ull << 31) || !make_map(&tm, kv, rows, 64, 64)) return GS_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the merge tickets start at zero (the kernel leaves them at zero)
  if (cudaMemsetAsync(ticket, 0, blocks * n_kv_heads * sizeof(int), s) != cudaSuccess)
    return GS_ERR_CUDA;
  attn_standalone_prep<<<cdiv(n_seq * W, 128), 128, 0, s>>>(mode, n, n_seq, W, lim, blk_slot);
  AttnArgs a;
  a.q = static_cast<const __half*>(q);
  a.lim = lim;
  a.out = static_cast<__half*>(out);
  a.page_table = page_table;
  a.pt_stride = pt_stride;
  a.blk_slot = blk_slot;
  a.blk_active = nullptr;
  a.fixed_slot = -1;
  a.T = n_seq * W;
  a.QB = W;
  a.QS = g.QS;
  a.n_sub = g.n_sub;
  a.Hq = n_heads;
  a.Hkv = n_kv_heads;
  a.G = G;
  a.rows_per_page = 2 * n_kv_heads * 64;
  a.kv_row_base = 0;
  a.split_pages = split_pages;
  a.max_items = items;
  a.cluster = attn_use_cluster(items, static_cast<int>(blocks) * n_kv_heads) ? 1 : 0;
  a.part = part;
  a.ticket = ticket;
  a.err = err;
  return launch_attention(tm, a, static_cast<int>(blocks), s, false) == cudaSuccess ? GS_OK
                                                                                   : GS_ERR_CUDA;
}

size_t gs_linear_scratch_bytes(int M, int N, int split_k) {
  if (M < 1 || N < 64 || split_k < 1) return 0;
  // the larger of the plans for an N-row and a 2N-row (SwiGLU) weight
  size_t counters = 0, partial = 0;
  for (int w_rows : {N, 2 * N}) {
    for (int nkb : {split_k, 8 * split_k}) {   // the plans for short and long K per split
      const GemmPlan p = plan_split(w_rows, M, split_k, nkb);
      counters = std::max(counters, static_cast<size_t>(p.tok_tiles) * p.feat_tiles);
      if (p.splits > 1 && !gemm_cluster_ok(p.bn, p.splits))
        partial = std::max(partial, static_cast<size_t>(p.splits) * p.tok_tiles * p.feat_tiles *
                                        p.bn * 128);
    }
  }
  Carver cv(nullptr);
  cv.take<int>(64);
  cv.take<int>(counters);
  if (partial) cv.take<float>(partial);
  return align_up(cv.off, 256);
}

int gs_linear(const void* x, const void* w, void* y, int M, int N, int K, int epilogue, int split_k,
              void* scratch, size_t scratch_bytes, void* stream) {
  if (!x || !w || !y || !scratch || M < 1 || K < 64 || K % 64 || split_k < 1 ||
      (K / 64) % split_k)
    return GS_ERR_INVALID_ARG;
  if (epilogue < 0 || epilogue > 3) return GS_ERR_INVALID_ARG;
  if (epilogue == kEpiSwiGLU ? (N % 64) : (N % 128)) return GS_ERR_INVALID_ARG;
  if (M > 65536) return GS_ERR_UNSUPPORTED;
  if (scratch_bytes < gs_linear_scratch_bytes(M, N, split_k)) return GS_ERR_OOM;
  if ((reinterpret_cast<uintptr_t>(x) & 15) || (reinterpret_cast<uintptr_t>(w) & 15) ||
      (reinterpret_cast<uintptr_t>(y) & 15))
    return GS_ERR_INVALID_ARG;
  if (ensure_kernel_attributes() != cudaSuccess) return GS_ERR_CUDA;
  // split-K as the decoder plans it: across the CTAs of a cluster (up to 64
  // rows), as chunks inside each CTA (wider), else through global scratch
  const int w_rows = epilogue == kEpiSwiGLU ? 2 * N : N;
  const GemmPlan p = plan_split(w_rows, M, split_k, K / 64);
  const int bn = p.bn, tok_tiles = p.tok_tiles, feat_tiles = p.feat_tiles;
  CUtensorMap tw, tx;
  if (!make_map(&tw, w, w_rows, K, epilogue == kEpiSwiGLU ? 64 : 128)) return GS_ERR_INVALID_ARG;
  if (!make_map(&tx, x, M, K, bn)) return GS_ERR_INVALID_ARG;
  Carver cv(scratch);
  GemmArgs a = {};
  a.err = cv.take<int>(64);
  a.counters = cv.take<int>(static_cast<size_t>(tok_tiles) * feat_tiles);
  // The error word and the per-tile arrival counters of the global split-K
  // path must start at zero, whatever the caller's scratch held before.
  const size_t head_bytes = cv.off;
  a.cluster = p.splits > 1 && gemm_cluster_ok(bn, p.splits) ? 1 : 0;
  a.partial = p.splits > 1 && !a.cluster
                  ? cv.take<float>(static_cast<size_t>(p.splits) * tok_tiles * feat_tiles * bn * 128)
                  : nullptr;
  a.M = M;
  a.N = N;
  a.K = K;
  a.splits = p.splits;
  a.chunks = p.chunks;
  a.kb_per_split = (K / 64) / a.splits;
  a.y = y;
  a.ldy = N;
  a.logits = nullptr;
  a.w_scale = 1.f;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(scratch, 0, head_bytes, s) != cudaSuccess) return GS_ERR_CUDA;
  return launch_gemm(bn, epilogue, tw, tx, a, feat_tiles, tok_tiles, s) == cudaSuccess
             ? GS_OK
             : GS_ERR_CUDA;
}

}  // extern "C"
