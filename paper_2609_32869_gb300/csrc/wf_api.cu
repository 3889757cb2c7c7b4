// Host orchestration of the Whisper-Flash decode step and the C ABI (wf.h).
//
// Per call the host enqueues kernels on the caller's stream; it never waits
// for the device except where an entry point says so (wf_compact,
// wf_get_state, wf_get_error).  All device memory is carved from the caller's
// workspace; the library allocates nothing on the device.
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <new>
#include <tuple>
#include <vector>

#include "wf_device.cuh"
#include "wf_internal.h"

using namespace wf;

struct wf_handle {
  wf_config cfg;
  int Bmax = 0, ctx = 0, Mmax = 0, d = 0, H = 0, F = 0, V = 0, K = 0, nl = 0, nd = 0;
  std::vector<wf_layer_weights> tl, dl;
  wf_target_weights tw;
  wf_drafter_weights dw;
  // per-slot state
  int32_t *L, *anchor, *remaining, *done, *step, *snap_L, *snap_anchor, *snap_rem;
  int32_t *active, *n_active_dev, *cand;
  uint32_t *err;
  // caches
  bf16 *self_k, *self_v, *cross_k, *cross_v, *hist_k, *hist_v;
  // activations
  float *x, *xd, *hproj;
  // per row and 128-feature tile (mean, M2) of x, xd, hproj for their LayerNorms
  float2 *st_x, *st_xd, *st_hp;
  bf16 *xn, *q, *att, *h1, *taps, *hn;
  // skinny passes: the next projection's folded LayerNorm operand (rows g, b,
  // then g . x of every token row) and the residual's partial row sums
  // (sum x, sum x^2), fold_np of them per row, written by the residual's
  // producer
  bf16 *xg;
  float2 *fpart;
  int fold_np = 0;
  // scratch
  float *apart;
  int32_t *attn_counters;
  size_t apart_floats;
  int attn_counter_cap;
  HeadRec *recs_t, *recs_d;
  HeadOut *hout_t, *hout_d;
  float *logits_t, *logits_d;
  float2 *rope;
  int n_vtiles = 0;
  int n_active = 0;
  long long spin = 0;  // bounded-wait limit in clock cycles (WF_OPT_SPIN_LIMIT; 0: default)
  int launches = 0;
  bool keep_logits = false;
  // skinny projections (wf_skinny.cu) for passes of at most kSkMaxRows rows;
  // used when every pass of the handle fits (max_batch * (K + 1) rows), so
  // speculative and plain greedy steps take the same arithmetic
  bool skinny = false;
  bool skinny_ok = false;  // the handle's shapes and max_batch allow it
  int sk_rows = 0;         // rows of its largest step pass (max_batch * (K + 1))
  // profiling (WF_OPT_PROFILE)
  bool profile = false;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_next = 0;
  struct Rec {
    int fam;
    cudaEvent_t a, b;
    double bytes;
  };
  std::vector<Rec> prof;
  cudaEvent_t pending = nullptr;
  // CUDA graphs of the hot entry points, keyed by what changes their launches
  struct GraphKey {
    int kind, n_active, forced;
    float temperature;
    uint64_t seed;
    const void *suppress;
    bool operator<(const GraphKey &o) const {
      return std::tie(kind, n_active, forced, temperature, seed, suppress) <
             std::tie(o.kind, o.n_active, o.forced, o.temperature, o.seed, o.suppress);
    }
  };
  struct GraphEntry {
    cudaGraphExec_t exec;
    int launches;
  };
  std::map<GraphKey, GraphEntry> graphs;
  bool use_graphs = true;
  cudaStream_t cap_stream = nullptr;
  int32_t *forced_buf = nullptr, *tok_buf = nullptr, *cnt_buf = nullptr;
  float *fq_buf = nullptr;  // forced proposal logits [Bmax][K][V] (wf_step copies them here)
  // persistent small-batch passes (wf_persist.cu)
  bool mk_ok = false;   // the shapes and limits allow it (fixed at create)
  bool mk_on = false;   // in use (WF_OPT_PERSIST)
  MkParams mkp = {};    // fields shared by every pass; the rest are set per launch
  MkLayer *mkl = nullptr;        // device [nl + nd]: target blocks, then drafter blocks
  char *mk_cnt_begin = nullptr;  // the persistent pass's counters, contiguous
  size_t mk_cnt_bytes = 0;
  CUtensorMap *tmaps = nullptr;  // device table
  int tm_self_k = 0, tm_hist_k = 0, tm_cross_k = 0;
};

namespace {

constexpr int kAlign = 256;

struct Carver {
  char *base;
  size_t off = 0;
  template <typename T>
  T *take(size_t count) {
    off = (off + kAlign - 1) / kAlign * kAlign;
    T *p = base ? reinterpret_cast<T *>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
};

bool cfg_ok(const wf_config *c) {
  if (!c) return false;
  if (c->d_model <= 0 || c->n_heads <= 0 || c->d_model != c->n_heads * 64) return false;
  if (c->d_model % 128 || c->d_ff % 64 || c->d_ff <= 0) return false;
  if (c->d_model > 1536) return false;
  if (c->n_layers <= 0 || c->n_layers > WF_MAX_LAYERS) return false;
  if (c->n_draft_layers <= 0 || c->n_draft_layers > 8) return false;
  if (c->vocab <= 0 || c->max_pos <= 0 || c->max_pos > 4096 || c->enc_frames <= 0) return false;
  if (c->block_k < 1 || c->block_k > 8) return false;
  if (c->n_taps < 1 || c->n_taps > WF_MAX_TAPS) return false;
  for (int i = 0; i < c->n_taps; ++i)
    if (c->taps[i] < 0 || c->taps[i] >= c->n_layers) return false;
  if (c->eos_id < 0 || c->eos_id >= c->vocab) return false;
  return true;
}

int rows_max(const wf_config *c, int Bmax, int ctx) {
  return std::max(Bmax * (c->block_k + 1), ctx);
}

// Lay the workspace out (base == nullptr: only measure).
size_t layout(wf_handle *h, const wf_config *c, int Bmax, int ctx, char *base) {
  Carver cv{base};
  const int d = c->d_model, H = c->n_heads, F = c->d_ff, V = c->vocab, K = c->block_k;
  const int nl = c->n_layers, nd = c->n_draft_layers, T = c->enc_frames;
  const int Mmax = rows_max(c, Bmax, ctx);
  const size_t sl = static_cast<size_t>(Bmax);
  wf_handle tmp;
  wf_handle *o = h ? h : &tmp;
  o->L = cv.take<int32_t>(sl);
  o->anchor = cv.take<int32_t>(sl);
  o->remaining = cv.take<int32_t>(sl);
  o->done = cv.take<int32_t>(sl);
  o->step = cv.take<int32_t>(sl);
  o->snap_L = cv.take<int32_t>(sl);
  o->snap_anchor = cv.take<int32_t>(sl);
  o->snap_rem = cv.take<int32_t>(sl);
  o->active = cv.take<int32_t>(sl);
  o->n_active_dev = cv.take<int32_t>(1);
  o->cand = cv.take<int32_t>(sl * K);
  o->err = cv.take<uint32_t>(1);
  o->forced_buf = cv.take<int32_t>(sl * K);
  o->tok_buf = cv.take<int32_t>(sl * (K + 1));
  o->cnt_buf = cv.take<int32_t>(sl);
  const size_t self_sz = static_cast<size_t>(nl) * sl * H * ctx * 64;
  o->self_k = cv.take<bf16>(self_sz);
  o->self_v = cv.take<bf16>(self_sz);
  const size_t cross_sz = static_cast<size_t>(nl + nd) * sl * H * T * 64;
  o->cross_k = cv.take<bf16>(cross_sz);
  o->cross_v = cv.take<bf16>(cross_sz);
  const size_t hist_sz = static_cast<size_t>(nd) * sl * H * ctx * 64;
  o->hist_k = cv.take<bf16>(hist_sz);
  o->hist_v = cv.take<bf16>(hist_sz);
  const size_t M = static_cast<size_t>(Mmax);
  o->x = cv.take<float>(M * d);
  o->xd = cv.take<float>(M * d);
  o->hproj = cv.take<float>(M * d);
  o->st_x = cv.take<float2>(M * (d / 128));
  o->st_xd = cv.take<float2>(M * (d / 128));
  o->st_hp = cv.take<float2>(M * (d / 128));
  o->xn = cv.take<bf16>(M * d);
  // the skinny passes' folded operand rows and partial sums: up to the
  // handle's largest step pass (or kSkMaxRows), plus the rows g and b
  const size_t xg_rows = static_cast<size_t>(std::max(kSkMaxRows, std::min(Bmax * (K + 1), kMtMaxRows)));
  o->xg = cv.take<bf16>((xg_rows + 2) * d);
  o->fpart = cv.take<float2>(xg_rows * kSkMaxParts);
  o->q = cv.take<bf16>(M * d);
  o->att = cv.take<bf16>(M * d);
  o->hn = cv.take<bf16>(M * d);
  o->h1 = cv.take<bf16>(M * F);
  o->taps = cv.take<bf16>(M * c->n_taps * d);
  const int groups = Bmax + Mmax / kAttnQGroup + 1;
  const int chunks = (std::max(ctx, T) + kAttnKeysPerCTA - 1) / kAttnKeysPerCTA;
  o->apart_floats = static_cast<size_t>(groups) * H * chunks * kAttnQGroup * 66;
  o->apart = cv.take<float>(o->apart_floats);
  o->attn_counter_cap = groups * H;
  o->attn_counters = cv.take<int32_t>(o->attn_counter_cap);
  const int vt = (V + 127) / 128;
  o->recs_t = cv.take<HeadRec>(M * vt);
  o->recs_d = cv.take<HeadRec>(M * vt);
  o->hout_t = cv.take<HeadOut>(M);
  o->hout_d = cv.take<HeadOut>(M);
  o->logits_t = cv.take<float>(M * V);
  o->logits_d = cv.take<float>(M * V);
  o->fq_buf = cv.take<float>(sl * K * V);
  o->rope = cv.take<float2>(static_cast<size_t>(c->max_pos) * 32);
  o->mk_ok = persist_supported(d, H, F, T, Bmax * (K + 1));
  if (o->mk_ok) {
    MkParams &p = o->mkp;
    const size_t R = kMkRows;
    p.x = cv.take<float>(R * d);
    p.q_x = cv.take<bf16>(R * d);
    p.att_x = cv.take<bf16>(R * d);
    p.xq_x = cv.take<bf16>(R * d);
    p.xatt_x = cv.take<bf16>(R * d);
    p.h_x = cv.take<bf16>(R * F);
    p.part2 = cv.take<float>(static_cast<size_t>(d / 8) * 3 * R * 8);
    p.xpart = cv.take<float>(mk_xpart_words(Bmax, H, T));
    p.cnt = cv.take<uint32_t>(kMkCounters);
    o->mk_cnt_begin = reinterpret_cast<char *>(p.cnt);
    p.cnt2 = cv.take<uint32_t>(d / 8);
    p.cntx = cv.take<uint32_t>(static_cast<size_t>(Bmax) * H);
    p.sync = cv.take<uint32_t>(2);
    o->mk_cnt_bytes = reinterpret_cast<char *>(p.sync + 2) - o->mk_cnt_begin;
    o->mkl = cv.take<MkLayer>(nl + nd);
    o->tmaps = cv.take<CUtensorMap>(static_cast<size_t>(6) * (nl + nd) + 6);
  }
  return cv.off + kAlign;
}

inline cudaStream_t S(void *s) { return static_cast<cudaStream_t>(s); }

// With WF_DEBUG set in the environment, failing CUDA calls are reported on
// stderr (the status code alone says only WF_ERR_CUDA).
void report_cuda(const char *what, cudaError_t e, int line) {
  static const bool on = getenv("WF_DEBUG") != nullptr;
  if (on) fprintf(stderr, "libwf: %s failed (wf_api.cu:%d): %s\n", what, line, cudaGetErrorString(e));
}
#define WF_TRY(expr)                                \
  do {                                              \
    cudaError_t _e = (expr);                        \
    if (_e != cudaSuccess) {                        \
      report_cuda(#expr, _e, __LINE__);             \
      return WF_ERR_CUDA;                           \
    }                                               \
  } while (0)

// Programmatic dependent launch for every kernel of a call (WF_OPT_PDL).
static bool g_pdl = true;
#define kPDL g_pdl

cudaEvent_t prof_event(wf_handle *h) {
  if (h->ev_next == h->ev_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    h->ev_pool.push_back(e);
  }
  return h->ev_pool[h->ev_next++];
}
// WF_DEBUG_SYNC in the environment: synchronise after every launch made
// outside graph capture and name the first that fails on stderr (debugging
// only: it serialises the launches).
void debug_sync(cudaStream_t s, const char *what, int M, int N, int K) {
  static const bool on = getenv("WF_DEBUG_SYNC") != nullptr;
  if (!on) return;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) return;
  const cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) fprintf(stderr, "libwf: %s (M=%d N=%d K=%d) failed: %s\n", what, M, N, K, cudaGetErrorString(e));
}
void prof_begin(wf_handle *h, cudaStream_t s) {
  if (!h->profile) return;
  h->pending = prof_event(h);
  if (h->pending) cudaEventRecord(h->pending, s);
}
void prof_end(wf_handle *h, cudaStream_t s, int fam, double bytes) {
  static const char *const kFam[] = {"gemm", "head", "attn_self", "attn_cross", "layernorm", "other", "persist"};
  debug_sync(s, fam >= 0 && fam < 7 ? kFam[fam] : "launch", -1, -1, -1);
  if (!h->profile || !h->pending) return;
  cudaEvent_t b = prof_event(h);
  if (!b) return;
  cudaEventRecord(b, s);
  h->prof.push_back({fam, h->pending, b, bytes});
  h->pending = nullptr;
}
// Algorithmic bytes of one projection: weights, token rows in, results out.
double gemm_bytes(const GemmParams &p) {
  double b = 2.0 * p.N * p.K + 2.0 * p.M * p.K + (p.bias ? 2.0 * p.N : 0.0);
  switch (p.epi) {
    case EPI_F32: b += 4.0 * p.M * p.N; break;
    case EPI_RESID:
      b += 8.0 * p.M * p.N + (p.tap0 ? 2.0 * p.M * p.N : 0.0) + (p.tap1 ? 2.0 * p.M * p.N : 0.0);
      break;
    case EPI_HEAD:
      b += 32.0 * p.M * ((p.N + 127) / 128) + (p.logits ? 4.0 * p.M * p.N : 0.0);
      break;
    default: b += 2.0 * p.M * p.N; break;
  }
  return b;
}

// ---------------------------------------------------------------- GEMMs --
// The skinny form of a projection's parameters (same epilogue fields).
SkinnyParams skinny_of(const GemmParams &g) {
  SkinnyParams p = {};
  p.M = g.M;
  p.N = g.N;
  p.K = g.K;
  p.epi = g.epi;
  p.bias = g.bias;
  p.out_f32 = g.out_f32;
  p.out_bf16 = g.out_bf16;
  p.ld_out = g.ld_out;
  p.resid = g.resid;
  p.ld_resid = g.ld_resid;
  p.tap0 = g.tap0;
  p.tap1 = g.tap1;
  p.ld_tap = g.ld_tap;
  p.q_cols = g.q_cols;
  p.d_model = g.d_model;
  p.n_heads = g.n_heads;
  p.ctx = g.ctx;
  p.rows_per_seq = g.rows_per_seq;
  p.kc = g.kc;
  p.vc = g.vc;
  p.seq_slot = g.seq_slot;
  p.pos_base = g.pos_base;
  p.err = g.err;
  p.spin = g.spin;
  return p;
}
GemmParams gemm_base(wf_handle *h, int M, int N, int K, int epi) {
  GemmParams p = {};
  p.M = M;
  p.N = N;
  p.K = K;
  p.epi = epi;
  p.splits = gemm_splits(N, K);
  p.err = h->err;
  p.spin = h->spin;
  p.d_model = h->d;
  p.n_heads = h->H;
  return p;
}

cudaError_t gemm(wf_handle *h, const void *X, const void *W, GemmParams p, cudaStream_t s) {
  h->launches++;
  prof_begin(h, s);
  cudaError_t e = launch_gemm(X, W, p, s, kPDL);
  prof_end(h, s, p.epi == EPI_HEAD ? WF_FAM_HEAD : WF_FAM_GEMM, gemm_bytes(p));
  return e;
}

// A skinny projection.  Operand: LN(ln_x) of fp32 rows with gain g and bias
// b when ln_x is given; the folded LayerNorm of the residual when only g is
// (rows h->xg and partial sums h->fpart left by the residual's producer; the
// gain and bias are in those rows); else the bf16 rows X.  An EPI_RESID
// projection followed by a LayerNorm with gain g_next and bias b_next writes
// that LayerNorm's folded operand.
cudaError_t skinny(wf_handle *h, const void *X, const float *ln_x, const void *g, const void *b,
                   const void *W, const GemmParams &gp, cudaStream_t s, const void *g_next = nullptr,
                   const void *b_next = nullptr) {
  SkinnyParams p = skinny_of(gp);
  // passes of more rows than one operand tile holds stream the operand (an
  // fp32 LayerNorm operand always fits one tile: it plans for its own rows)
  const bool mt = h->sk_rows > kSkMaxFoldRows && !ln_x;
  p.plan_M = (h->sk_rows > kSkMaxFoldRows && ln_x) ? gp.M : h->sk_rows;
  if (g_next) {
    p.xg_out = h->xg;
    p.g_next = static_cast<const bf16 *>(g_next);
    p.b_next = static_cast<const bf16 *>(b_next);
    p.part_out = h->fpart;
    p.part_stride = kSkMaxParts;
  }
  if (g && ln_x) {
    p.ln_x = ln_x;
    p.ln_ld = h->d;
    p.ln_g = static_cast<const bf16 *>(g);
    p.ln_b = static_cast<const bf16 *>(b);
    p.ln_eps = h->cfg.ln_eps;
  } else if (g) {
    p.fold = 1;
    p.x = h->xg;
    p.ld_x = h->d;
    p.fold_part = h->fpart;
    p.n_part = h->fold_np;
    p.part_stride = kSkMaxParts;
    p.ln_eps = h->cfg.ln_eps;
  } else {
    p.x = static_cast<const bf16 *>(X);
    p.ld_x = gp.K;
  }
  h->launches++;
  prof_begin(h, s);
  cudaError_t e = mt ? launch_skinny_mt(W, p, s, kPDL) : launch_skinny(W, p, s, kPDL);
  debug_sync(s, mt ? "skinny_mt" : "skinny", p.M, p.N, p.K);
  prof_end(h, s, WF_FAM_GEMM, gemm_bytes(gp));
  if (e == cudaSuccess && g_next) {  // partials per row: one per CTA column block of the plan
    int U = 0, S = 0, ns = 0;
    const bool planned = mt ? skinny_mt_plan(p.plan_M + (p.fold ? 2 : 0), p.N, p.K, p.fold != 0,
                                             p.epi == EPI_RESID, &U, &S, &ns)
                            : skinny_plan(p.plan_M, p.N, p.K, false, false, &U, &S);
    if (!planned) return cudaErrorInvalidValue;
    h->fold_np = p.N / 8 / U;
  }
  return e;
}

// Whether every projection of a pass of up to M rows has a skinny plan
// (one operand tile up to kSkMaxFoldRows rows, a streamed operand up to
// kMtMaxRows).
bool skinny_shapes_fit(int d, int F, int M) {
  // folded LayerNorm operands carry two more rows (g and b)
  int U = 0, S = 0, ns = 0;
  if (M > kSkMaxFoldRows)  // QKV, out (and cross out), cross query, fc1, fc2
    return M <= kMtMaxRows && skinny_mt_plan(M + 2, 3 * d, d, true, false, &U, &S, &ns) &&
           skinny_mt_plan(M, d, d, false, true, &U, &S, &ns) && skinny_mt_plan(M + 2, d, d, true, false, &U, &S, &ns) &&
           skinny_mt_plan(M + 2, F, d, true, false, &U, &S, &ns) && skinny_mt_plan(M, d, F, false, true, &U, &S, &ns);
  return M <= kSkMaxFoldRows && skinny_plan(M + 2, 3 * d, d, false, true, &U, &S) &&
         skinny_plan(M, d, d, false, false, &U, &S) && skinny_plan(M + 2, d, d, false, true, &U, &S) &&
         skinny_plan(M + 2, F, d, false, true, &U, &S) && skinny_plan(M, d, F, false, false, &U, &S) &&
         skinny_plan(M, 2 * d, d, true, false, &U, &S);
}

// Whether a pass of M rows takes the skinny projections.
bool use_skinny(const wf_handle *h, int M) { return h->skinny && M <= h->sk_rows; }

cudaError_t layernorm(wf_handle *h, const float *x, const float2 *st, int stride, int off,
                      const void *g, const void *b, bf16 *y, int rows, cudaStream_t s) {
  h->launches++;
  prof_begin(h, s);
  cudaError_t e = launch_layernorm(x, st, stride, off, static_cast<const bf16 *>(g),
                                   static_cast<const bf16 *>(b), y, rows, h->d, h->cfg.ln_eps, s,
                                   kPDL);
  prof_end(h, s, WF_FAM_LAYERNORM, 6.0 * rows * h->d);
  return e;
}

// A projection of LN(x): the GEMM normalises its own token operand from the
// fp32 rows and their tile statistics when its tiles fit in shared memory,
// otherwise a LayerNorm kernel writes the bf16 rows first.  Both forms give
// the same bits.
cudaError_t ln_gemm(wf_handle *h, const float *x, const float2 *st, const void *g, const void *b,
                    const void *W, GemmParams p, cudaStream_t s) {
  if (gemm_ln_fits(p.M, p.N, p.K, p.epi)) {
    p.ln_x = x;
    p.ln_ld = h->d;
    p.ln_tiles = h->d / 128;
    p.ln_stats = st;
    p.ln_g = static_cast<const bf16 *>(g);
    p.ln_b = static_cast<const bf16 *>(b);
    p.ln_eps = h->cfg.ln_eps;
    return gemm(h, nullptr, W, p, s);
  }
  cudaError_t e = layernorm(h, x, st, 1, 0, g, b, h->xn, p.M, s);
  if (e != cudaSuccess) return e;
  return gemm(h, h->xn, W, p, s);
}

cudaError_t attention(wf_handle *h, const bf16 *q, const bf16 *kc, const bf16 *vc,
                      const int32_t *slots, int n_seq, int rps, int ctx, int mode, bool rope,
                      cudaStream_t s) {
  AttnParams p = {};
  p.q = q;
  p.kc = kc;
  p.vc = vc;
  p.out = h->att;
  p.seq_slot = slots;
  p.pos_base = h->L;
  p.rope_tab = rope ? h->rope : nullptr;
  p.part = h->apart;
  p.counters = h->attn_counters;
  p.err = h->err;
  p.n_seq = n_seq;
  p.rps = rps;
  p.n_heads = h->H;
  p.ctx = ctx;
  p.mode = mode;
  p.spin = h->spin;
  p.outer = h->Bmax * h->H;
  if (attn_partial_floats(n_seq, rps, h->H, ctx) > h->apart_floats) return cudaErrorInvalidValue;
  if (attn_counter_slots(n_seq, rps, h->H) > h->attn_counter_cap) return cudaErrorInvalidValue;
  h->launches++;
  prof_begin(h, s);
  cudaError_t e = launch_attention(p, s, kPDL);
  prof_end(h, s, mode == 2 ? WF_FAM_ATTN_CROSS : WF_FAM_ATTN_SELF, 0.0);
  return e;
}

size_t layer_cache_off(wf_handle *h, int layer, int positions) {
  return static_cast<size_t>(layer) * h->Bmax * h->H * positions * 64;
}

struct Pass {
  int n_seq, rps;
  const int32_t *slots;
  bool drafter;
  float *x;
  float2 *st;  // LayerNorm statistics of x (tcgen05 path)
  bool taps;
  bool sk;     // skinny projections (no statistics travel)
};

// The cross-query projection (LN2 folded, one sequence) fused with the
// cross-attention of its queries over the acoustic memory xkc/xvc; the
// attention output lands in h->att for the cross-out projection.
cudaError_t skinny_xattn(wf_handle *h, const wf_layer_weights &lw, const bf16 *xkc, const bf16 *xvc,
                         const Pass &ps, cudaStream_t s) {
  const int M = ps.n_seq * ps.rps, d = h->d;
  SkinnyParams p = {};
  p.M = M;
  p.N = d;
  p.K = d;
  p.epi = EPI_BF16;
  p.fold = 1;
  p.x = h->xg;
  p.ld_x = d;
  p.fold_part = h->fpart;
  p.n_part = h->fold_np;
  p.part_stride = kSkMaxParts;
  p.ln_eps = h->cfg.ln_eps;
  p.bias = static_cast<const bf16 *>(lw.xq_b);
  p.out_bf16 = h->att;
  p.ld_out = d;
  p.kc = const_cast<bf16 *>(xkc);
  p.vc = const_cast<bf16 *>(xvc);
  p.ctx = h->cfg.enc_frames;
  p.seq_slot = ps.slots;
  p.n_heads = h->H;
  p.d_model = d;
  p.xa_outer = h->Bmax * h->H;
  p.err = h->err;
  p.spin = h->spin;
  h->launches++;
  prof_begin(h, s);
  cudaError_t e = launch_skinny_xattn(lw.xq_w, p, s, kPDL);
  // the projection's weights and operand plus the acoustic keys and values read
  const double kv = 2.0 * ps.n_seq * h->H * static_cast<double>(h->cfg.enc_frames) * 64 * sizeof(bf16);
  prof_end(h, s, WF_FAM_ATTN_CROSS, static_cast<double>(d) * d * sizeof(bf16) + kv);
  return e;
}

// The QKV projection (LN1 folded, one sequence) fused with the self-attention
// of its rows over the cache kc/vc (target: causal; drafter: the history
// memory and the block, with RoPE); the new keys and values are written to
// the cache at L + j and the attention output lands in h->att.
cudaError_t skinny_sattn(wf_handle *h, const wf_layer_weights &lw, bf16 *kc, bf16 *vc, const Pass &ps,
                         cudaStream_t s) {
  const int M = ps.n_seq * ps.rps, d = h->d;
  SkinnyParams p = {};
  p.M = M;
  p.N = 3 * d;
  p.K = d;
  p.epi = EPI_KV;
  p.fold = 1;
  p.x = h->xg;
  p.ld_x = d;
  p.fold_part = h->fpart;
  p.n_part = h->fold_np;
  p.part_stride = kSkMaxParts;
  p.ln_eps = h->cfg.ln_eps;
  p.bias = static_cast<const bf16 *>(lw.qkv_b);
  p.out_bf16 = h->att;
  p.ld_out = d;
  p.kc = kc;
  p.vc = vc;
  p.ctx = h->ctx;
  p.seq_slot = ps.slots;
  p.pos_base = h->L;
  p.n_heads = h->H;
  p.d_model = d;
  p.xa_outer = h->Bmax * h->H;
  p.xa_mode = ps.drafter ? 1 : 0;
  p.rope_tab = ps.drafter ? h->rope : nullptr;
  p.err = h->err;
  p.spin = h->spin;
  h->launches++;
  prof_begin(h, s);
  cudaError_t e = launch_skinny_sattn(lw.qkv_w, p, s, kPDL);
  prof_end(h, s, WF_FAM_ATTN_SELF, 3.0 * d * d * sizeof(bf16));
  return e;
}

// One pre-LayerNorm Whisper block over the pass's rows; next: the following
// block of the pass (whose first LayerNorm a skinny pass folds), or null.
cudaError_t run_block(wf_handle *h, const Pass &ps, const wf_layer_weights &lw, int layer,
                      const wf_layer_weights *next, cudaStream_t s) {
  const int M = ps.n_seq * ps.rps, d = h->d;
  cudaError_t e;
  bf16 *kc, *vc, *xkc, *xvc;
  if (ps.drafter) {
    kc = h->hist_k + layer_cache_off(h, layer, h->ctx);
    vc = h->hist_v + layer_cache_off(h, layer, h->ctx);
    xkc = h->cross_k + layer_cache_off(h, h->nl + layer, h->cfg.enc_frames);
    xvc = h->cross_v + layer_cache_off(h, h->nl + layer, h->cfg.enc_frames);
  } else {
    kc = h->self_k + layer_cache_off(h, layer, h->ctx);
    vc = h->self_v + layer_cache_off(h, layer, h->ctx);
    xkc = h->cross_k + layer_cache_off(h, layer, h->cfg.enc_frames);
    xvc = h->cross_v + layer_cache_off(h, layer, h->cfg.enc_frames);
  }
  // self-attention: for one sequence on a single-sequence handle's skinny
  // path, the QKV projection and the attention run as one kernel (a cluster
  // per head); a batched handle keeps its one projection form at any n_seq
  const bool one_tile = ps.sk && ps.n_seq == 1 && h->sk_rows <= kSkMaxFoldRows;
  if (one_tile && skinny_sattn_fits(M, d, h->H, h->ctx)) {
    if ((e = skinny_sattn(h, lw, kc, vc, ps, s)) != cudaSuccess) return e;
  } else {
  {
    GemmParams p = gemm_base(h, M, 3 * d, d, EPI_KV);
    p.bias = static_cast<const bf16 *>(lw.qkv_b);
    p.out_bf16 = h->q;
    p.ld_out = d;
    p.q_cols = d;
    p.kc = kc;
    p.vc = vc;
    p.ctx = h->ctx;
    p.rows_per_seq = ps.rps;
    p.seq_slot = ps.slots;
    p.pos_base = h->L;
    e = ps.sk ? skinny(h, nullptr, nullptr, lw.ln1_g, lw.ln1_b, lw.qkv_w, p, s)
              : ln_gemm(h, ps.x, ps.st, lw.ln1_g, lw.ln1_b, lw.qkv_w, p, s);
    if (e != cudaSuccess) return e;
  }
  if ((e = attention(h, h->q, kc, vc, ps.slots, ps.n_seq, ps.rps, h->ctx, ps.drafter ? 1 : 0,
                     ps.drafter, s)) != cudaSuccess)
    return e;
  }
  {
    GemmParams p = gemm_base(h, M, d, d, EPI_RESID);
    p.bias = static_cast<const bf16 *>(lw.out_b);
    p.resid = ps.x;
    p.ld_resid = d;
    p.stats_out = ps.st;
    e = ps.sk ? skinny(h, h->att, nullptr, nullptr, nullptr, lw.out_w, p, s, lw.ln2_g, lw.ln2_b)
              : gemm(h, h->att, lw.out_w, p, s);
    if (e != cudaSuccess) return e;
  }
  // cross-attention: likewise the query projection and the attention
  if (one_tile && skinny_xattn_fits(M, d, h->H, h->cfg.enc_frames)) {
    if ((e = skinny_xattn(h, lw, xkc, xvc, ps, s)) != cudaSuccess) return e;
  } else {
    {
      GemmParams p = gemm_base(h, M, d, d, EPI_BF16);
      p.bias = static_cast<const bf16 *>(lw.xq_b);
      p.out_bf16 = h->q;
      p.ld_out = d;
      e = ps.sk ? skinny(h, nullptr, nullptr, lw.ln2_g, lw.ln2_b, lw.xq_w, p, s)
                : ln_gemm(h, ps.x, ps.st, lw.ln2_g, lw.ln2_b, lw.xq_w, p, s);
      if (e != cudaSuccess) return e;
    }
    if ((e = attention(h, h->q, xkc, xvc, ps.slots, ps.n_seq, ps.rps, h->cfg.enc_frames, 2, false,
                       s)) != cudaSuccess)
      return e;
  }
  {
    GemmParams p = gemm_base(h, M, d, d, EPI_RESID);
    p.bias = static_cast<const bf16 *>(lw.xout_b);
    p.resid = ps.x;
    p.ld_resid = d;
    p.stats_out = ps.st;
    e = ps.sk ? skinny(h, h->att, nullptr, nullptr, nullptr, lw.xout_w, p, s, lw.ln3_g, lw.ln3_b)
              : gemm(h, h->att, lw.xout_w, p, s);
    if (e != cudaSuccess) return e;
  }
  // feed-forward
  {
    GemmParams p = gemm_base(h, M, h->F, d, EPI_GELU);
    p.bias = static_cast<const bf16 *>(lw.fc1_b);
    p.out_bf16 = h->h1;
    p.ld_out = h->F;
    e = ps.sk ? skinny(h, nullptr, nullptr, lw.ln3_g, lw.ln3_b, lw.fc1_w, p, s)
              : ln_gemm(h, ps.x, ps.st, lw.ln3_g, lw.ln3_b, lw.fc1_w, p, s);
    if (e != cudaSuccess) return e;
  }
  {
    GemmParams p = gemm_base(h, M, d, h->F, EPI_RESID);
    p.bias = static_cast<const bf16 *>(lw.fc2_b);
    p.resid = ps.x;
    p.ld_resid = d;
    p.stats_out = ps.st;
    if (ps.taps) {
      // the block's output residual stream, before the final LayerNorm (App. A.2)
      int found = 0;
      for (int t = 0; t < h->cfg.n_taps; ++t) {
        if (h->cfg.taps[t] != layer) continue;
        bf16 *dst = h->taps + static_cast<size_t>(t) * d;
        if (found == 0) p.tap0 = dst;
        else if (found == 1) p.tap1 = dst;
        ++found;
      }
      p.ld_tap = h->cfg.n_taps * d;
    }
    e = ps.sk ? skinny(h, h->h1, nullptr, nullptr, nullptr, lw.fc2_w, p, s, next ? next->ln1_g : nullptr,
                       next ? next->ln1_b : nullptr)
              : gemm(h, h->h1, lw.fc2_w, p, s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// Final LayerNorm (the target's, shared with the drafter) and the tied head.
// x == nullptr: h->xn already holds the normalised rows (persistent pass).
cudaError_t head(wf_handle *h, const float *x, const float2 *st, int stride, int off, int rows,
                 const int32_t *slots,
                 int rps, HeadRec *recs, HeadOut *out, float *logits, const wf_sample_params *sp,
                 uint32_t tag, int32_t *cand, cudaStream_t s) {
  cudaError_t e;
  if (x && (e = layernorm(h, x, st, stride, off, h->tw.lnf_g, h->tw.lnf_b, h->xn, rows, s)) != cudaSuccess)
    return e;
  const bool sampling = sp && sp->temperature > 0.f;
  GemmParams p = gemm_base(h, rows, h->V, h->d, EPI_HEAD);
  p.recs = recs;
  p.logits = (sampling || h->keep_logits) ? logits : nullptr;
  p.keep_logits = h->keep_logits ? 1 : 0;
  p.temperature = sampling ? sp->temperature : 0.f;
  p.seed = sp ? sp->seed : 0;
  p.suppress = sp ? sp->d_suppress : nullptr;
  p.step = h->step;
  p.tag = tag;
  p.rows_per_seq = rps;
  p.seq_slot = slots;
  if ((e = gemm(h, h->xn, h->tw.tok_emb, p, s)) != cudaSuccess) return e;
  HeadReduceParams r = {};
  r.recs = recs;
  r.out = out;
  r.rows = rows;
  r.n_tiles = h->n_vtiles;
  r.cand = cand;
  r.seq_slot = slots;
  r.rps = rps;
  r.K = h->K;
  r.sampling = sampling ? 1 : 0;
  h->launches++;
  prof_begin(h, s);
  e = launch_head_reduce(r, s, kPDL);
  prof_end(h, s, WF_FAM_OTHER, 0.0);
  return e;
}

// History memory (Sec. 3.2, App. A.2): project the tapped residual streams of
// the pass's rows, normalise, and write each drafter block's keys/values at
// the rows' text positions (L + j).
cudaError_t ingest(wf_handle *h, int n_seq, int rps, const int32_t *slots, cudaStream_t s) {
  const int M = n_seq * rps, d = h->d;
  cudaError_t e;
  {
    GemmParams p = gemm_base(h, M, d, h->cfg.n_taps * d, EPI_F32);
    p.bias = static_cast<const bf16 *>(h->dw.proj_b);
    p.out_f32 = h->hproj;
    p.ld_out = d;
    p.stats_out = h->st_hp;
    if ((e = gemm(h, h->taps, h->dw.proj_w, p, s)) != cudaSuccess) return e;
  }
  // LN_h is applied inside each drafter block's key/value projection (or by
  // one LayerNorm kernel ahead of them when their tiles do not fit)
  // LN_h over the fp32 projection in the skinny kernel only for one operand
  // tile that has a plan (whole K per CTA)
  int sk_u = 0, sk_s = 0;
  const bool sk = use_skinny(h, M) && M <= kSkMaxRows && skinny_plan(M, 2 * d, d, true, false, &sk_u, &sk_s);
  const bool fused = sk || gemm_ln_fits(M, 2 * d, d, EPI_KV);
  if (!fused &&
      (e = layernorm(h, h->hproj, h->st_hp, 1, 0, h->dw.hln_g, h->dw.hln_b, h->hn, M, s)) != cudaSuccess)
    return e;
  for (int l = 0; l < h->nd; ++l) {
    const wf_layer_weights &lw = h->dl[l];
    GemmParams p = gemm_base(h, M, 2 * d, d, EPI_KV);
    p.bias = static_cast<const bf16 *>(lw.qkv_b) + d;
    p.q_cols = 0;
    p.kc = h->hist_k + layer_cache_off(h, l, h->ctx);
    p.vc = h->hist_v + layer_cache_off(h, l, h->ctx);
    p.ctx = h->ctx;
    p.rows_per_seq = rps;
    p.seq_slot = slots;
    p.pos_base = h->L;
    const bf16 *wkv = static_cast<const bf16 *>(lw.qkv_w) + static_cast<size_t>(d) * d;
    if (sk) {
      if ((e = skinny(h, nullptr, h->hproj, h->dw.hln_g, h->dw.hln_b, wkv, p, s)) != cudaSuccess) return e;
    } else if (fused) {
      p.ln_x = h->hproj;
      p.ln_ld = d;
      p.ln_tiles = d / 128;
      p.ln_stats = h->st_hp;
      p.ln_g = static_cast<const bf16 *>(h->dw.hln_g);
      p.ln_b = static_cast<const bf16 *>(h->dw.hln_b);
      p.ln_eps = h->cfg.ln_eps;
      if ((e = gemm(h, nullptr, wkv, p, s)) != cudaSuccess) return e;
    } else if ((e = gemm(h, h->hn, wkv, p, s)) != cudaSuccess) {
      return e;
    }
  }
  return cudaSuccess;
}

cudaError_t target_pass(wf_handle *h, int n_seq, int rps, const int32_t *slots, int src,
                        const int32_t *prompt, int P, const int32_t *forced, bool taps,
                        cudaStream_t s) {
  EmbedParams ep = {};
  ep.tok_emb = static_cast<const bf16 *>(h->tw.tok_emb);
  ep.pos_emb = static_cast<const bf16 *>(h->tw.pos_emb);
  ep.seq_slot = slots;
  ep.L = h->L;
  ep.anchor = h->anchor;
  ep.cand_in = h->cand;
  ep.cand_out = h->cand;
  ep.forced = forced;
  ep.prompt = prompt;
  ep.x = h->x;
  if (use_skinny(h, n_seq * rps)) {  // the first block's folded LN1 operand
    ep.xg = h->xg;
    ep.g_next = static_cast<const bf16 *>(h->tl[0].ln1_g);
    ep.b_next = static_cast<const bf16 *>(h->tl[0].ln1_b);
    ep.part_out = h->fpart;
    ep.part_stride = kSkMaxParts;
    h->fold_np = 1;
  }
  ep.stats_out = h->st_x;
  ep.n_seq = n_seq;
  ep.rps = rps;
  ep.d = h->d;
  ep.K = h->K;
  ep.P = P;
  ep.vocab = h->V;
  ep.src = src;
  ep.drafter = 0;
  ep.err = h->err;
  h->launches++;
  prof_begin(h, s);
  cudaError_t e = launch_embed(ep, s, kPDL);
  prof_end(h, s, WF_FAM_OTHER, 0.0);
  if (e != cudaSuccess) return e;
  Pass ps{n_seq, rps, slots, false, h->x, h->st_x, taps, use_skinny(h, n_seq * rps)};
  for (int l = 0; l < h->nl; ++l)
    if ((e = run_block(h, ps, h->tl[l], l, l + 1 < h->nl ? &h->tl[l + 1] : nullptr, s)) != cudaSuccess)
      return e;
  return cudaSuccess;
}

// Tensor maps and per-block tables of the persistent passes: every weight
// matrix as [rows][cols] bf16 with [8][64] boxes (one unit of 8 output rows,
// one 128-byte swizzle atom), every cache as [rows][64] with [128][64] boxes.
cudaError_t persist_setup(wf_handle *h, cudaStream_t s) {
  int G = 0;
  cudaError_t e = persist_init(&G);
  if (e != cudaSuccess) return e;
  if (G > kMkMaxG) G = kMkMaxG;
  if (G < 4 * kMkRows) return cudaErrorInvalidConfiguration;
  const int d = h->d, F = h->F, H = h->H, T = h->cfg.enc_frames;
  if (!persist_grid_fits(d, F, G)) {  // too few SMs for these widths: launch by launch only
    h->mk_ok = false;
    return cudaSuccess;
  }
  const int nl = h->nl, nd = h->nd;
  std::vector<CUtensorMap> maps;
  std::vector<MkLayer> lys;
  auto add_map = [&](const void *ptr, uint64_t rows, uint64_t cols, uint32_t box) -> int {
    const CUtensorMap *m = tmap_bf16_2d(ptr, rows, cols, box);
    if (!m) return -1;
    maps.push_back(*m);
    return static_cast<int>(maps.size()) - 1;
  };
  // one copy per projection unit: 8 rows by the unit's whole K range
  auto add_units = [&](const void *ptr, uint64_t rows, uint64_t cols, uint32_t kblocks) -> int {
    CUtensorMap m;
    if (!tmap_bf16_units(&m, ptr, rows, cols, kblocks)) return -1;
    maps.push_back(m);
    return static_cast<int>(maps.size()) - 1;
  };
  for (int l = 0; l < nl + nd; ++l) {
    const wf_layer_weights &w = l < nl ? h->tl[l] : h->dl[l - nl];
    MkLayer ly = {};
    ly.ln1_g = static_cast<const bf16 *>(w.ln1_g);
    ly.ln1_b = static_cast<const bf16 *>(w.ln1_b);
    ly.qkv_b = static_cast<const bf16 *>(w.qkv_b);
    ly.out_b = static_cast<const bf16 *>(w.out_b);
    ly.ln2_g = static_cast<const bf16 *>(w.ln2_g);
    ly.ln2_b = static_cast<const bf16 *>(w.ln2_b);
    ly.xq_b = static_cast<const bf16 *>(w.xq_b);
    ly.xout_b = static_cast<const bf16 *>(w.xout_b);
    ly.ln3_g = static_cast<const bf16 *>(w.ln3_g);
    ly.ln3_b = static_cast<const bf16 *>(w.ln3_b);
    ly.fc1_b = static_cast<const bf16 *>(w.fc1_b);
    ly.fc2_b = static_cast<const bf16 *>(w.fc2_b);
    ly.tm[0] = add_units(w.qkv_w, 3 * d, d, d / 64);
    ly.tm[1] = add_units(w.out_w, d, d, d / 64);
    ly.tm[2] = add_units(w.xq_w, d, d, d / 64);
    ly.tm[3] = add_units(w.xout_w, d, d, d / 64);
    ly.tm[4] = add_units(w.fc1_w, F, d, d / 64);
    ly.tm[5] = add_units(w.fc2_w, d, F, F / 4 / 64);  // one quarter of K per copy
    for (int k = 0; k < 6; ++k)
      if (ly.tm[k] < 0) return cudaErrorInvalidValue;
    ly.self_layer = l < nl ? l : l - nl;
    ly.cross_layer = l;
    ly.tap[0] = ly.tap[1] = -1;
    if (l < nl) {
      int found = 0;
      for (int t = 0; t < h->cfg.n_taps && found < 2; ++t)
        if (h->cfg.taps[t] == l) ly.tap[found++] = t;
    }
    lys.push_back(ly);
  }
  const uint64_t self_rows = static_cast<uint64_t>(nl) * h->Bmax * H * h->ctx;
  const uint64_t hist_rows = static_cast<uint64_t>(nd) * h->Bmax * H * h->ctx;
  const uint64_t cross_rows = static_cast<uint64_t>(nl + nd) * h->Bmax * H * T;
  // one copy per 128 keys (or values) of one head
  h->tm_self_k = add_map(h->self_k, self_rows, 64, 128);
  const int sv = add_map(h->self_v, self_rows, 64, 128);
  h->tm_hist_k = add_map(h->hist_k, hist_rows, 64, 128);
  const int hv = add_map(h->hist_v, hist_rows, 64, 128);
  h->tm_cross_k = add_map(h->cross_k, cross_rows, 64, 128);
  const int cv2 = add_map(h->cross_v, cross_rows, 64, 128);
  if (h->tm_self_k < 0 || sv != h->tm_self_k + 1 || h->tm_hist_k < 0 || hv != h->tm_hist_k + 1 ||
      h->tm_cross_k < 0 || cv2 != h->tm_cross_k + 1)
    return cudaErrorInvalidValue;
  // synchronous copies: the host vectors die with this call
  if ((e = cudaMemcpy(h->tmaps, maps.data(), maps.size() * sizeof(CUtensorMap), cudaMemcpyHostToDevice)) !=
      cudaSuccess)
    return e;
  if ((e = cudaMemcpy(h->mkl, lys.data(), lys.size() * sizeof(MkLayer), cudaMemcpyHostToDevice)) != cudaSuccess)
    return e;
  // every counter starts at zero; each pass leaves them at zero
  if ((e = cudaMemsetAsync(h->mk_cnt_begin, 0, h->mk_cnt_bytes, s)) != cudaSuccess) return e;
  MkParams &p = h->mkp;
  p.tmaps = h->tmaps;
  p.G = G;
  p.d = d;
  p.H = H;
  p.F = F;
  p.T = T;
  p.ctx = h->ctx;
  p.Bmax = h->Bmax;
  p.K = h->K;
  p.vocab = h->V;
  p.tm_xk = h->tm_cross_k;
  p.tm_xv = h->tm_cross_k + 1;
  p.L = h->L;
  p.anchor = h->anchor;
  p.cand_in = h->cand;
  p.tok_emb = static_cast<const bf16 *>(h->tw.tok_emb);
  p.pos_emb = static_cast<const bf16 *>(h->tw.pos_emb);
  p.mask_emb = static_cast<const bf16 *>(h->dw.mask_emb);
  p.lnf_g = static_cast<const bf16 *>(h->tw.lnf_g);
  p.lnf_b = static_cast<const bf16 *>(h->tw.lnf_b);
  p.rope_tab = h->rope;
  p.eps = h->cfg.ln_eps;
  p.taps = h->taps;
  p.ld_tap = h->cfg.n_taps * d;
  p.xn = h->xn;
  p.err = h->err;
  p.spin = kMkSpinCycles;
  h->mk_on = false;
  return cudaSuccess;
}

// Every block of one pass in a single persistent launch; the final
// LayerNorm's output is left in h->xn for the head.
cudaError_t persist_pass(wf_handle *h, bool drafter, int n_seq, int rps, const int32_t *slots,
                         const int32_t *forced, bool taps, cudaStream_t s) {
  MkParams p = h->mkp;
  if (h->spin > 0) p.spin = h->spin;
  p.layers = drafter ? h->mkl + h->nl : h->mkl;
  p.nl = drafter ? h->nd : h->nl;
  p.drafter = drafter ? 1 : 0;
  p.write_taps = taps ? 1 : 0;
  p.n_seq = n_seq;
  p.rps = rps;
  p.M = n_seq * rps;
  p.seq_slot = slots;
  p.forced = forced;
  p.cand_out = (drafter || rps == 1) ? nullptr : h->cand;
  p.kc = drafter ? h->hist_k : h->self_k;
  p.vc = drafter ? h->hist_v : h->self_v;
  p.tm_kc = drafter ? h->tm_hist_k : h->tm_self_k;
  p.tm_vc = p.tm_kc + 1;
  h->launches++;
  prof_begin(h, s);
  cudaError_t e = launch_persist(p, s);
  // algorithmic bytes: every block's six projection matrices and each
  // sequence's acoustic keys and values (self/history K/V, a few percent at
  // these lengths, and the activations are not counted)
  const double d = h->d, F = h->F;
  const double block_bytes = 2.0 * (6.0 * d * d + 2.0 * d * F) + 2.0 * 2.0 * n_seq * h->cfg.enc_frames * d;
  prof_end(h, s, WF_FAM_PERSIST, p.nl * block_bytes);
  return e;
}

wf_status check_weights(const wf_layer_weights &w) {
  const void *ptrs[] = {w.ln1_g, w.ln1_b, w.qkv_w, w.qkv_b, w.out_w, w.out_b, w.ln2_g,
                        w.ln2_b, w.xq_w,  w.xq_b,  w.xkv_w, w.xkv_b, w.xout_w, w.xout_b,
                        w.ln3_g, w.ln3_b, w.fc1_w, w.fc1_b, w.fc2_w, w.fc2_b};
  for (const void *p : ptrs) {
    if (!p) return WF_ERR_INVALID;
    if (reinterpret_cast<uintptr_t>(p) & 15) return WF_ERR_INVALID;
  }
  return WF_OK;
}

}  // namespace

// ====================================================================== ABI
extern "C" {

const char *wf_status_str(wf_status s) {
  switch (s) {
    case WF_OK: return "ok";
    case WF_ERR_INVALID: return "invalid argument";
    case WF_ERR_CAPACITY: return "capacity exceeded";
    case WF_ERR_CUDA: return "CUDA error";
    case WF_ERR_UNSUPPORTED: return "unsupported shape";
    case WF_ERR_DEVICE: return "device error word set";
  }
  return "unknown status";
}

wf_status wf_workspace_bytes(const wf_config *cfg, int32_t max_batch, int32_t max_ctx,
                             size_t *out_bytes) {
  if (!out_bytes || !cfg) return WF_ERR_INVALID;
  if (!cfg_ok(cfg)) return WF_ERR_UNSUPPORTED;
  if (max_batch <= 0 || max_ctx <= cfg->block_k + 1 || max_ctx > cfg->max_pos) return WF_ERR_INVALID;
  *out_bytes = layout(nullptr, cfg, max_batch, max_ctx, nullptr);
  return WF_OK;
}

wf_status wf_create(const wf_config *cfg, const wf_target_weights *tw, const wf_drafter_weights *dw,
                    int32_t max_batch, int32_t max_ctx, void *d_workspace, size_t workspace_bytes,
                    void *stream, wf_handle **out) {
  if (!cfg || !tw || !dw || !out || !d_workspace) return WF_ERR_INVALID;
  *out = nullptr;
  size_t need = 0;
  wf_status st = wf_workspace_bytes(cfg, max_batch, max_ctx, &need);
  if (st != WF_OK) return st;
  if (workspace_bytes < need) return WF_ERR_CAPACITY;
  if (reinterpret_cast<uintptr_t>(d_workspace) % kAlign) return WF_ERR_INVALID;
  if (!tw->tok_emb || !tw->pos_emb || !tw->lnf_g || !tw->lnf_b || !tw->layers) return WF_ERR_INVALID;
  if (!dw->layers || !dw->proj_w || !dw->proj_b || !dw->hln_g || !dw->hln_b || !dw->mask_emb)
    return WF_ERR_INVALID;
  {
    const void *ptrs[] = {tw->tok_emb, tw->pos_emb, tw->lnf_g, tw->lnf_b, dw->proj_w,
                          dw->proj_b,  dw->hln_g,   dw->hln_b, dw->mask_emb};
    for (const void *p : ptrs)
      if (reinterpret_cast<uintptr_t>(p) & 15) return WF_ERR_INVALID;
  }
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return WF_ERR_CUDA;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return WF_ERR_CUDA;
  if (major != 10 || minor != 3) return WF_ERR_UNSUPPORTED;
  wf_handle *h = new (std::nothrow) wf_handle;
  if (!h) return WF_ERR_CAPACITY;
  h->cfg = *cfg;
  h->Bmax = max_batch;
  h->ctx = max_ctx;
  h->Mmax = rows_max(cfg, max_batch, max_ctx);
  h->d = cfg->d_model;
  h->H = cfg->n_heads;
  h->F = cfg->d_ff;
  h->V = cfg->vocab;
  h->K = cfg->block_k;
  h->nl = cfg->n_layers;
  h->nd = cfg->n_draft_layers;
  h->n_vtiles = (cfg->vocab + 127) / 128;
  h->tl.assign(tw->layers, tw->layers + cfg->n_layers);
  h->dl.assign(dw->layers, dw->layers + cfg->n_draft_layers);
  for (auto &w : h->tl)
    if (check_weights(w) != WF_OK) { delete h; return WF_ERR_INVALID; }
  for (auto &w : h->dl)
    if (check_weights(w) != WF_OK) { delete h; return WF_ERR_INVALID; }
  h->tw = *tw;
  h->tw.layers = h->tl.data();
  h->dw = *dw;
  h->dw.layers = h->dl.data();
  layout(h, cfg, max_batch, max_ctx, static_cast<char *>(d_workspace));
  cudaStream_t s = S(stream);
  const size_t sl = static_cast<size_t>(max_batch) * sizeof(int32_t);
  bool ok = cudaMemsetAsync(h->L, 0, sl, s) == cudaSuccess &&
            cudaMemsetAsync(h->anchor, 0, sl, s) == cudaSuccess &&
            cudaMemsetAsync(h->remaining, 0, sl, s) == cudaSuccess &&
            cudaMemsetAsync(h->done, 0x01, sl, s) == cudaSuccess &&  // no slot is active yet
            cudaMemsetAsync(h->step, 0, sl, s) == cudaSuccess &&
            cudaMemsetAsync(h->cand, 0, sl * h->K, s) == cudaSuccess &&
            cudaMemsetAsync(h->n_active_dev, 0, sizeof(int32_t), s) == cudaSuccess &&
            cudaMemsetAsync(h->err, 0, sizeof(uint32_t), s) == cudaSuccess &&
            cudaMemsetAsync(h->attn_counters, 0, h->attn_counter_cap * sizeof(int32_t), s) == cudaSuccess &&
            launch_rope_table(h->rope, cfg->max_pos, cfg->rope_base, s) == cudaSuccess;
  h->sk_rows = max_batch * (cfg->block_k + 1);
  h->skinny_ok = skinny_shapes_fit(h->d, h->F, h->sk_rows);
  // on by default where one operand tile holds a pass (single-sequence
  // handles); the batched form (2-16 sequences) is opt-in: it measured 3-12%
  // slower per step than the tcgen05 projections at 2-8 sequences, a tie at 16
  h->skinny = h->skinny_ok && h->sk_rows <= kSkMaxFoldRows;
  ok = ok && gemm_init() == cudaSuccess && skinny_init() == cudaSuccess && skinny_mt_init() == cudaSuccess &&
       attention_init() == cudaSuccess &&
       step_kernels_init() == cudaSuccess &&
       cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking) == cudaSuccess;
  if (ok && h->mk_ok) ok = persist_setup(h, s) == cudaSuccess;
  if (!ok) {
    if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
    delete h;
    return WF_ERR_CUDA;
  }
  *out = h;
  return WF_OK;
}

wf_status wf_destroy(wf_handle *h) {
  if (!h) return WF_ERR_INVALID;
  for (cudaEvent_t e : h->ev_pool) cudaEventDestroy(e);
  for (auto &kv : h->graphs) cudaGraphExecDestroy(kv.second.exec);
  if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
  delete h;
  return WF_OK;
}

int32_t wf_last_launch_count(const wf_handle *h) { return h ? h->launches : -1; }

wf_status wf_set_option(wf_handle *h, int32_t option, int32_t value) {
  if (!h) return WF_ERR_INVALID;
  if (option == WF_OPT_KEEP_LOGITS) {
    h->keep_logits = value != 0;
    return WF_OK;
  }
  if (option == WF_OPT_PDL) {
    g_pdl = value != 0;
    for (auto &kv : h->graphs) cudaGraphExecDestroy(kv.second.exec);
    h->graphs.clear();
    return WF_OK;
  }
  if (option == WF_OPT_GRAPHS) {
    h->use_graphs = value != 0;
    return WF_OK;
  }
  if (option == WF_OPT_PERSIST) {
    if (value && !h->mk_ok) return WF_ERR_UNSUPPORTED;
    h->mk_on = value != 0;
    for (auto &kv : h->graphs) cudaGraphExecDestroy(kv.second.exec);
    h->graphs.clear();
    return WF_OK;
  }
  if (option == WF_OPT_SKINNY) {
    if (value && !h->skinny_ok) return WF_ERR_UNSUPPORTED;
    h->skinny = value != 0;
    for (auto &kv : h->graphs) cudaGraphExecDestroy(kv.second.exec);
    h->graphs.clear();
    return WF_OK;
  }
  if (option == WF_OPT_SPIN_LIMIT) {
    if (value < 0) return WF_ERR_INVALID;
    h->spin = value;
    for (auto &kv : h->graphs) cudaGraphExecDestroy(kv.second.exec);
    h->graphs.clear();
    return WF_OK;
  }
  if (option == WF_OPT_PROFILE) {
    h->profile = value != 0;
    h->prof.clear();
    h->ev_next = 0;
    return WF_OK;
  }
  return WF_ERR_INVALID;
}

wf_status wf_profile_read(wf_handle *h, void *stream, double *h_ms, int32_t *h_launches,
                          double *h_bytes) {
  if (!h || !h_ms || !h_launches || !h_bytes) return WF_ERR_INVALID;
  WF_TRY(cudaStreamSynchronize(S(stream)));
  for (int f = 0; f < WF_PROF_FAMILIES; ++f) {
    h_ms[f] = 0.0;
    h_launches[f] = 0;
    h_bytes[f] = 0.0;
  }
  for (auto &r : h->prof) {
    float ms = 0.f;
    WF_TRY(cudaEventElapsedTime(&ms, r.a, r.b));
    h_ms[r.fam] += ms;
    h_launches[r.fam] += 1;
    h_bytes[r.fam] += r.bytes;
  }
  h->prof.clear();
  h->ev_next = 0;
  return WF_OK;
}

wf_status wf_debug_view(wf_handle *h, int32_t which, void **d_ptr, size_t *bytes) {
  if (!h || !d_ptr || !bytes) return WF_ERR_INVALID;
  const size_t M = static_cast<size_t>(h->Mmax);
  switch (which) {
    case WF_VIEW_TARGET_LOGITS:
      *d_ptr = h->logits_t;
      *bytes = M * h->V * sizeof(float);
      return WF_OK;
    case WF_VIEW_DRAFT_LOGITS:
      *d_ptr = h->logits_d;
      *bytes = M * h->V * sizeof(float);
      return WF_OK;
    case WF_VIEW_TAPS:
      *d_ptr = h->taps;
      *bytes = M * h->cfg.n_taps * h->d * sizeof(bf16);
      return WF_OK;
    case WF_VIEW_CANDIDATES:
      *d_ptr = h->cand;
      *bytes = static_cast<size_t>(h->Bmax) * h->K * sizeof(int32_t);
      return WF_OK;
  }
  return WF_ERR_INVALID;
}

wf_status wf_prefill_cross_kv(wf_handle *h, int32_t n, const int32_t *d_slots, const void *d_enc,
                              const int32_t *d_prompt, int32_t P, const int32_t *d_budget,
                              int32_t *d_first, const wf_sample_params *sp, void *stream) {
  if (!h || !d_slots || !d_enc || !d_prompt || !d_budget || n <= 0 || P <= 0) return WF_ERR_INVALID;
  if (h->n_active + n > h->Bmax) return WF_ERR_CAPACITY;
  if (P + h->K + 1 > h->ctx || P > h->Mmax) return WF_ERR_CAPACITY;
  if (reinterpret_cast<uintptr_t>(d_enc) & 15) return WF_ERR_INVALID;
  cudaStream_t s = S(stream);
  h->launches = 0;
  const int d = h->d, T = h->cfg.enc_frames;
  // acoustic keys/values of every target and drafter block (App. A.5)
  for (int l = 0; l < h->nl + h->nd; ++l) {
    const wf_layer_weights &lw = l < h->nl ? h->tl[l] : h->dl[l - h->nl];
    GemmParams p = gemm_base(h, n * T, 2 * d, d, EPI_KV);
    p.splits = 1;
    p.bias = static_cast<const bf16 *>(lw.xkv_b);
    p.q_cols = 0;
    p.kc = h->cross_k + layer_cache_off(h, l, T);
    p.vc = h->cross_v + layer_cache_off(h, l, T);
    p.ctx = T;
    p.rows_per_seq = T;
    p.seq_slot = d_slots;
    p.pos_base = nullptr;
    WF_TRY(gemm(h, d_enc, lw.xkv_w, p, s));
  }
  StateParams sp0 = {};
  sp0.op = 0;
  sp0.n = n;
  sp0.slots = d_slots;
  sp0.max_batch = h->Bmax;
  sp0.L = h->L;
  sp0.anchor = h->anchor;
  sp0.remaining = h->remaining;
  sp0.done = h->done;
  sp0.step = h->step;
  h->launches++;
  WF_TRY(launch_state(sp0, s, kPDL));
  const int g = std::max(1, std::min(n, h->Mmax / P));
  const bool sampling = sp && sp->temperature > 0.f;
  for (int i0 = 0; i0 < n; i0 += g) {
    const int gn = std::min(g, n - i0);
    const int32_t *slots = d_slots + i0;
    WF_TRY(target_pass(h, gn, P, slots, TOK_PROMPT, d_prompt + static_cast<size_t>(i0) * P, P,
                       nullptr, true, s));
    WF_TRY(ingest(h, gn, P, slots, s));
    WF_TRY(head(h, h->x, use_skinny(h, gn * P) ? nullptr : h->st_x, P, P - 1, gn, slots, 1, h->recs_t,
                h->hout_t, h->logits_t, sp, kTagBonus, nullptr, s));
    StateParams sp1 = sp0;
    sp1.op = 1;
    sp1.n = gn;
    sp1.slots = slots;
    sp1.budget = d_budget + i0;
    sp1.hout = h->hout_t;
    sp1.first = d_first ? d_first + i0 : nullptr;
    sp1.P = P;
    sp1.eos = h->cfg.eos_id;
    sp1.sampling = sampling ? 1 : 0;
    sp1.snap_L = h->snap_L;
    sp1.snap_anchor = h->snap_anchor;
    sp1.snap_remaining = h->snap_rem;
    sp1.active = h->active;
    sp1.n_active_dev = h->n_active_dev;
    sp1.active_offset = h->n_active + i0;
    h->launches++;
    WF_TRY(launch_state(sp1, s, kPDL));
  }
  h->n_active += n;
  return WF_OK;
}

static wf_status draft_body(wf_handle *h, const wf_sample_params *sp, cudaStream_t s) {
  if (h->n_active == 0) return WF_OK;
  const int n = h->n_active, rps = h->K + 1;
  if (h->mk_on) {
    WF_TRY(persist_pass(h, true, n, rps, h->active, nullptr, false, s));
    WF_TRY(head(h, nullptr, nullptr, 1, 0, n * rps, h->active, rps, h->recs_d, h->hout_d, h->logits_d, sp,
                kTagDraft, h->cand, s));
    return WF_OK;
  }
  EmbedParams ep = {};
  ep.tok_emb = static_cast<const bf16 *>(h->tw.tok_emb);
  ep.mask_emb = static_cast<const bf16 *>(h->dw.mask_emb);
  ep.seq_slot = h->active;
  ep.anchor = h->anchor;
  ep.x = h->xd;
  if (use_skinny(h, n * rps)) {  // the first block's folded LN1 operand
    ep.xg = h->xg;
    ep.g_next = static_cast<const bf16 *>(h->dl[0].ln1_g);
    ep.b_next = static_cast<const bf16 *>(h->dl[0].ln1_b);
    ep.part_out = h->fpart;
    ep.part_stride = kSkMaxParts;
    h->fold_np = 1;
  }
  ep.stats_out = h->st_xd;
  ep.n_seq = n;
  ep.rps = rps;
  ep.d = h->d;
  ep.K = h->K;
  ep.vocab = h->V;
  ep.src = TOK_ANCHOR;
  ep.drafter = 1;
  ep.err = h->err;
  h->launches++;
  prof_begin(h, s);
  WF_TRY(launch_embed(ep, s, kPDL));
  prof_end(h, s, WF_FAM_OTHER, 0.0);
  Pass ps{n, rps, h->active, true, h->xd, h->st_xd, false, use_skinny(h, n * rps)};
  for (int l = 0; l < h->nd; ++l) WF_TRY(run_block(h, ps, h->dl[l], l, l + 1 < h->nd ? &h->dl[l + 1] : nullptr, s));
  WF_TRY(head(h, h->xd, ps.sk ? nullptr : h->st_xd, 1, 0, n * rps, h->active, rps, h->recs_d, h->hout_d,
              h->logits_d, sp, kTagDraft, h->cand, s));
  return WF_OK;
}

static wf_status verify_body(wf_handle *h, const wf_sample_params *sp, const int32_t *d_forced,
                             const float *d_forced_q, int32_t *d_out_tokens, int32_t *d_out_count,
                             cudaStream_t s) {
  const int n = h->n_active, rps = h->K + 1;
  if (n > 0) {
    if (h->mk_on) {
      WF_TRY(persist_pass(h, false, n, rps, h->active, d_forced, true, s));
      WF_TRY(head(h, nullptr, nullptr, 1, 0, n * rps, h->active, rps, h->recs_t, h->hout_t, h->logits_t,
                  sp, kTagBonus, nullptr, s));
    } else {
      WF_TRY(target_pass(h, n, rps, h->active, TOK_VERIFY, nullptr, 0, d_forced, true, s));
      WF_TRY(head(h, h->x, use_skinny(h, n * rps) ? nullptr : h->st_x, 1, 0, n * rps, h->active, rps,
                  h->recs_t, h->hout_t, h->logits_t, sp, kTagBonus, nullptr, s));
    }
    WF_TRY(ingest(h, n, rps, h->active, s));
  }
  AcceptParams ap = {};
  ap.seq_slot = h->active;
  ap.n_seq = n;
  ap.rps = rps;
  ap.K = h->K;
  ap.max_batch = h->Bmax;
  ap.vocab = h->V;
  ap.eos = h->cfg.eos_id;
  ap.max_ctx = h->ctx;
  ap.greedy_step = 0;
  ap.tout = h->hout_t;
  ap.dout = h->hout_d;
  ap.cand = h->cand;
  ap.tlogits = h->logits_t;
  ap.dlogits = h->logits_d;
  ap.forced_q = d_forced_q;
  ap.suppress = sp ? sp->d_suppress : nullptr;
  ap.temperature = (sp && sp->temperature > 0.f) ? sp->temperature : 0.f;
  ap.seed = sp ? sp->seed : 0;
  ap.L = h->L;
  ap.anchor = h->anchor;
  ap.remaining = h->remaining;
  ap.done = h->done;
  ap.step = h->step;
  ap.out_tokens = d_out_tokens;
  ap.out_count = d_out_count;
  ap.err = h->err;
  h->launches++;
  prof_begin(h, s);
  WF_TRY(launch_accept(ap, s, kPDL));
  prof_end(h, s, WF_FAM_OTHER, 0.0);
  return WF_OK;
}

static wf_status greedy_body(wf_handle *h, const wf_sample_params *sp, int32_t *d_out_tokens,
                             int32_t *d_out_count, cudaStream_t s) {
  const int n = h->n_active;
  if (n > 0) {
    if (h->mk_on) {
      WF_TRY(persist_pass(h, false, n, 1, h->active, nullptr, false, s));
      WF_TRY(head(h, nullptr, nullptr, 1, 0, n, h->active, 1, h->recs_t, h->hout_t, h->logits_t, sp,
                  kTagBonus, nullptr, s));
    } else {
      WF_TRY(target_pass(h, n, 1, h->active, TOK_ANCHOR, nullptr, 0, nullptr, false, s));
      WF_TRY(head(h, h->x, use_skinny(h, n) ? nullptr : h->st_x, 1, 0, n, h->active, 1, h->recs_t, h->hout_t,
                  h->logits_t, sp, kTagBonus, nullptr, s));
    }
  }
  AcceptParams ap = {};
  ap.seq_slot = h->active;
  ap.n_seq = n;
  ap.rps = 1;
  ap.K = h->K;
  ap.max_batch = h->Bmax;
  ap.vocab = h->V;
  ap.eos = h->cfg.eos_id;
  ap.max_ctx = h->ctx;
  ap.greedy_step = 1;
  ap.tout = h->hout_t;
  ap.cand = h->cand;
  ap.temperature = (sp && sp->temperature > 0.f) ? sp->temperature : 0.f;
  ap.seed = sp ? sp->seed : 0;
  ap.L = h->L;
  ap.anchor = h->anchor;
  ap.remaining = h->remaining;
  ap.done = h->done;
  ap.step = h->step;
  ap.out_tokens = d_out_tokens;
  ap.out_count = d_out_count;
  ap.err = h->err;
  h->launches++;
  prof_begin(h, s);
  WF_TRY(launch_accept(ap, s, kPDL));
  prof_end(h, s, WF_FAM_OTHER, 0.0);
  return WF_OK;
}

}  // extern "C"

// Run `body` through a CUDA graph captured once per key on the handle's capture
// stream and replayed on the caller's stream; eager when graphs are off, when
// profiling, or when the caller's stream is itself being captured.
template <typename Body>
static wf_status run_graphed(wf_handle *h, wf_handle::GraphKey key, cudaStream_t s, Body body) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (s && cudaStreamIsCapturing(s, &cs) != cudaSuccess) return WF_ERR_CUDA;
  if (!h->use_graphs || h->profile || cs != cudaStreamCaptureStatusNone) {
    h->launches = 0;
    return body(s);
  }
  auto it = h->graphs.find(key);
  if (it == h->graphs.end()) {
    if (cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
      return WF_ERR_CUDA;
    h->launches = 0;
    wf_status st = body(h->cap_stream);
    cudaGraph_t g = nullptr;
    cudaError_t e = cudaStreamEndCapture(h->cap_stream, &g);
    if (st != WF_OK || e != cudaSuccess) {
      if (e != cudaSuccess) report_cuda("cudaStreamEndCapture", e, __LINE__);
      if (g) cudaGraphDestroy(g);
      return st != WF_OK ? st : WF_ERR_CUDA;
    }
    cudaGraphExec_t ex = nullptr;
    e = cudaGraphInstantiate(&ex, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess) {
      report_cuda("cudaGraphInstantiate", e, __LINE__);
      return WF_ERR_CUDA;
    }
    it = h->graphs.emplace(key, wf_handle::GraphEntry{ex, h->launches}).first;
  }
  h->launches = it->second.launches;
  WF_TRY(cudaGraphLaunch(it->second.exec, s));
  return WF_OK;
}

static wf_handle::GraphKey graph_key(wf_handle *h, int kind, const wf_sample_params *sp,
                                     bool forced, bool forced_q = false) {
  wf_handle::GraphKey k;
  k.kind = kind;
  k.n_active = h->n_active;
  k.forced = (forced ? 1 : 0) | (forced_q ? 2 : 0);
  const bool sampling = sp && sp->temperature > 0.f;
  k.temperature = sampling ? sp->temperature : 0.f;
  k.seed = sampling ? sp->seed : 0;
  k.suppress = sp ? sp->d_suppress : nullptr;
  return k;
}

extern "C" {

wf_status wf_draft(wf_handle *h, const wf_sample_params *sp, void *stream) {
  if (!h) return WF_ERR_INVALID;
  h->launches = 0;
  return draft_body(h, sp, S(stream));
}

wf_status wf_verify_accept(wf_handle *h, const wf_sample_params *sp, const int32_t *d_forced,
                           const float *d_forced_q, int32_t *d_out_tokens, int32_t *d_out_count,
                           void *stream) {
  if (!h || !d_out_tokens || !d_out_count || (d_forced_q && !d_forced)) return WF_ERR_INVALID;
  h->launches = 0;
  const bool sampling = sp && sp->temperature > 0.f;
  return verify_body(h, sp, d_forced, sampling ? d_forced_q : nullptr, d_out_tokens, d_out_count,
                     S(stream));
}

wf_status wf_step(wf_handle *h, const wf_sample_params *sp, const int32_t *d_forced,
                  const float *d_forced_q, int32_t *d_out_tokens, int32_t *d_out_count, void *stream) {
  if (!h || !d_out_tokens || !d_out_count || (d_forced_q && !d_forced)) return WF_ERR_INVALID;
  cudaStream_t s = S(stream);
  const size_t kb = static_cast<size_t>(h->Bmax) * h->K * sizeof(int32_t);
  if (d_forced) WF_TRY(cudaMemcpyAsync(h->forced_buf, d_forced, kb, cudaMemcpyDeviceToDevice, s));
  const int32_t *forced = d_forced ? h->forced_buf : nullptr;
  const bool use_q = d_forced_q && sp && sp->temperature > 0.f;
  if (use_q)
    WF_TRY(cudaMemcpyAsync(h->fq_buf, d_forced_q,
                           static_cast<size_t>(h->Bmax) * h->K * h->V * sizeof(float),
                           cudaMemcpyDeviceToDevice, s));
  const float *fq = use_q ? h->fq_buf : nullptr;
  wf_status st = run_graphed(h, graph_key(h, 1, sp, d_forced != nullptr, use_q), s,
                             [&](cudaStream_t cs) -> wf_status {
                               wf_status r = draft_body(h, sp, cs);
                               if (r != WF_OK) return r;
                               return verify_body(h, sp, forced, fq, h->tok_buf, h->cnt_buf, cs);
                             });
  if (st != WF_OK) return st;
  WF_TRY(cudaMemcpyAsync(d_out_tokens, h->tok_buf, kb / h->K * (h->K + 1), cudaMemcpyDeviceToDevice, s));
  WF_TRY(cudaMemcpyAsync(d_out_count, h->cnt_buf, static_cast<size_t>(h->Bmax) * sizeof(int32_t),
                         cudaMemcpyDeviceToDevice, s));
  return WF_OK;
}

wf_status wf_greedy_step(wf_handle *h, const wf_sample_params *sp, int32_t *d_out_tokens,
                         int32_t *d_out_count, void *stream) {
  if (!h || !d_out_tokens || !d_out_count) return WF_ERR_INVALID;
  cudaStream_t s = S(stream);
  wf_status st = run_graphed(h, graph_key(h, 2, sp, false), s, [&](cudaStream_t cs) -> wf_status {
    return greedy_body(h, sp, h->tok_buf, h->cnt_buf, cs);
  });
  if (st != WF_OK) return st;
  const size_t kb = static_cast<size_t>(h->Bmax) * (h->K + 1) * sizeof(int32_t);
  WF_TRY(cudaMemcpyAsync(d_out_tokens, h->tok_buf, kb, cudaMemcpyDeviceToDevice, s));
  WF_TRY(cudaMemcpyAsync(d_out_count, h->cnt_buf, static_cast<size_t>(h->Bmax) * sizeof(int32_t),
                         cudaMemcpyDeviceToDevice, s));
  return WF_OK;
}

wf_status wf_compact(wf_handle *h, void *stream, int32_t *h_n_active) {
  if (!h) return WF_ERR_INVALID;
  cudaStream_t s = S(stream);
  h->launches = 1;
  WF_TRY(launch_compact(h->done, h->Bmax, h->active, h->n_active_dev, s));
  int32_t n = 0;
  WF_TRY(cudaMemcpyAsync(&n, h->n_active_dev, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
  WF_TRY(cudaStreamSynchronize(s));
  h->n_active = n;
  if (h_n_active) *h_n_active = n;
  return WF_OK;
}

wf_status wf_reset_slots(wf_handle *h, int32_t n, const int32_t *d_slots, void *stream) {
  if (!h || !d_slots || n <= 0) return WF_ERR_INVALID;
  StateParams p = {};
  p.op = 2;
  p.n = n;
  p.slots = d_slots;
  p.max_batch = h->Bmax;
  p.L = h->L;
  p.anchor = h->anchor;
  p.remaining = h->remaining;
  p.done = h->done;
  p.step = h->step;
  p.snap_L = h->snap_L;
  p.snap_anchor = h->snap_anchor;
  p.snap_remaining = h->snap_rem;
  h->launches = 1;
  WF_TRY(launch_state(p, S(stream), kPDL));
  return WF_OK;
}

wf_status wf_get_state(wf_handle *h, int32_t *h_len, int32_t *h_anchor, int32_t *h_remaining,
                       int32_t *h_done, void *stream) {
  if (!h) return WF_ERR_INVALID;
  cudaStream_t s = S(stream);
  const size_t sz = static_cast<size_t>(h->Bmax) * sizeof(int32_t);
  if (h_len) WF_TRY(cudaMemcpyAsync(h_len, h->L, sz, cudaMemcpyDeviceToHost, s));
  if (h_anchor) WF_TRY(cudaMemcpyAsync(h_anchor, h->anchor, sz, cudaMemcpyDeviceToHost, s));
  if (h_remaining) WF_TRY(cudaMemcpyAsync(h_remaining, h->remaining, sz, cudaMemcpyDeviceToHost, s));
  if (h_done) WF_TRY(cudaMemcpyAsync(h_done, h->done, sz, cudaMemcpyDeviceToHost, s));
  WF_TRY(cudaStreamSynchronize(s));
  return WF_OK;
}

wf_status wf_get_error(wf_handle *h, uint32_t *h_err, int32_t clear, void *stream) {
  if (!h || !h_err) return WF_ERR_INVALID;
  cudaStream_t s = S(stream);
  WF_TRY(cudaMemcpyAsync(h_err, h->err, sizeof(uint32_t), cudaMemcpyDeviceToHost, s));
  WF_TRY(cudaStreamSynchronize(s));
  if (clear) {
    WF_TRY(cudaMemsetAsync(h->err, 0, sizeof(uint32_t), s));
    WF_TRY(cudaStreamSynchronize(s));
  }
  return WF_OK;
}

}  // extern "C"
