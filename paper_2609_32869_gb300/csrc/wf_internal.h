// Host-side declarations shared by the translation units of libwf: kernel
// parameter blocks and launchers.  Not part of the public ABI.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/wf.h"
#include "wf_skinny_mt_layout.h"

namespace wf {

using bf16 = __nv_bfloat16;

// Every kernel of the library runs with the same shared-memory carveout (the
// largest), so consecutive kernels of a pass, whose CTAs overlap under
// programmatic dependent launch, can share an SM without it first draining
// to change its L1 / shared-memory split.
inline cudaError_t prefer_max_shared(const void *fn) {
  return cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout,
                              cudaSharedmemCarveoutMaxShared);
}
// The row-wise kernels of wf_step_kernels.cu (once per process).
cudaError_t step_kernels_init();

// ------------------------------------------------------------------ GEMM --
// Y[t, n] = sum_k X[t, k] W[n, k] for token rows t < M and features n < N,
// computed as a 128 x BT tile of D = W_tile * X_tile^T on tcgen05 ("swap-AB":
// the weights fill the 128-row MMA side, the few tokens the N side).
enum EpiMode : int {
  EPI_F32 = 0,    // out_f32[t*ld_out + n] = y + b
  EPI_BF16 = 1,   // out_bf16[t*ld_out + n] = bf16(y + b)
  EPI_GELU = 2,   // out_bf16[t*ld_out + n] = bf16(gelu(y + b))
  EPI_RESID = 3,  // resid[t*ld_resid + n] += y + b; optional bf16 copies (taps)
  EPI_KV = 4,     // n < q_cols: out_bf16 (query); else keys/values into a cache
  EPI_HEAD = 5    // output-head records: per (token, 128-id tile) max/argmax,
                  // sum of exponentials and Gumbel-max (sampling)
};

struct HeadRec {  // one (token row, 128-id vocabulary tile) of the output head
  float m;        // max of x = z/T (z when greedy) over the tile
  float s;        // sum of exp(x - m) over the tile
  float gm;       // max of x + Gumbel noise (sampling only)
  int32_t arg;    // lowest id attaining m
  int32_t garg;   // lowest id attaining gm
  int32_t _pad[3];
};

struct GemmParams {
  int M, N, K;
  int BT, n_tt, splits, kps, stages, pipe_bytes;
  uint32_t tmem_cols;
  // fold != 0: one CTA computes every split of its tile in turn (the split
  // partials alternate between two TMEM accumulators of acc_cols columns and
  // are added in split order into a third), with the same arithmetic as the
  // cluster reduction
  int fold;
  uint32_t acc_cols;
  int epi;
  const bf16 *bias;
  float *out_f32;
  bf16 *out_bf16;
  int ld_out;
  float *resid;
  int ld_resid;
  bf16 *tap0, *tap1;
  int ld_tap;
  // EPI_KV: row t -> sequence i = t / rows_per_seq, j = t % rows_per_seq;
  // slot = seq_slot[i]; position = (pos_base ? pos_base[slot] : 0) + j;
  // cache layout [slot][head][ctx][64].
  int q_cols, d_model, n_heads, ctx, rows_per_seq;
  bf16 *kc, *vc;
  const int32_t *seq_slot, *pos_base;
  // EPI_HEAD
  HeadRec *recs;  // [M][n_tiles]
  float *logits;  // nullable [M][N] raw logits (sampling, or kept for inspection)
  int keep_logits;
  float temperature;  // 0: greedy
  uint64_t seed;
  const uint8_t *suppress;
  const int32_t *step;  // per slot
  uint32_t tag;
  uint32_t *err;
  long long spin;  // clock cycles a bounded wait spins before it gives up
  // LayerNorm-fused token operand: when ln_x is set the CTA builds its bf16
  // B tiles as LN(x) = (x - mean) * rstd * g + b from fp32 rows ln_x (row
  // stride ln_ld) and per-row statistics ln_stats[t][0..ln_tiles) (mean, M2
  // over each 128-feature tile, merged in tile order); X is then unused.
  const float *ln_x;
  int ln_ld, ln_tiles;
  const float2 *ln_stats;
  const bf16 *ln_g, *ln_b;
  float ln_eps;
  // Statistics of this GEMM's outputs for the next LayerNorm: per output row
  // and 128-feature tile, (mean, M2) of the final values (the updated
  // residual for EPI_RESID, the output for EPI_F32); [M][N/128].
  float2 *stats_out;
};

// Cache of TMA descriptors keyed by (address, rows, cols, box rows).
const CUtensorMap *tmap_bf16_2d(const void *ptr, uint64_t rows, uint64_t cols, uint32_t box_rows);
// A whole 8-row unit of a [rows][cols] matrix per copy: box {64, 8, kblocks}.
bool tmap_bf16_units(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint32_t kblocks);
// All `rows` rows of a [rows][cols] matrix (row stride ld elements) over
// kblocks 64-column blocks per copy: box {64, rows, kblocks}.
bool tmap_bf16_rows(CUtensorMap *m, const void *ptr, uint32_t rows, uint64_t cols, uint64_t ld, uint32_t kblocks);
// A key/value cache [outer][ctx][64] bf16 as (64 dims, position, outer) with a
// box of {64, box_rows, 1}, 128-byte swizzled; positions past ctx read as 0.
bool tmap_bf16_cache(CUtensorMap *m, const void *ptr, uint64_t ctx, uint64_t outer, uint32_t box_rows);

// Token tile for M rows: a multiple of 16, at most 128.
void gemm_token_tiling(int M, int *BT, int *n_tt);
// Split-K count for a projection of N outputs over K inputs (a function of
// the shape only, so a row's result never depends on how many rows run).
int gemm_splits(int N, int K);

// Opt every GEMM instantiation into large dynamic shared memory (once).
cudaError_t gemm_init();
// Launch one GEMM.  W is [N, K] bf16, X is [M, K] bf16 (row stride K), or
// X is null and the token operand is LN(p.ln_x) built inside the kernel.
cudaError_t launch_gemm(const void *X, const void *W, GemmParams p, cudaStream_t s, bool pdl);
// Whether to use the LayerNorm-fused form of a launch: one token tile, and
// all of the CTA's token tiles fit in shared memory; otherwise run
// launch_layernorm first (same bits either way).
bool gemm_ln_fits(int M, int N, int K, int epi);

// ------------------------------------------------------ skinny projections --
// Y = X W^T for M <= 16 token rows (wf_skinny.cu): each CTA prefetches its
// whole weight slab (U units of 8 rows over K / S) with TMA before the
// dependency wait and reduces K in a fixed order.  The operand is bf16 rows
// x, the folded LayerNorm of a residual (rows written by its producer), or
// LN(ln_x) computed in the kernel from fp32 rows.  Epilogues as EpiMode (no
// EPI_HEAD; EPI_RESID writes no tile statistics).
constexpr int kSkMaxRows = 16;
constexpr int kSkMaxFoldRows = kSkMaxRows - 2;  // token rows of a folded LayerNorm operand
constexpr int kSkMaxParts = 160;                // partial row sums of one residual update
struct SkinnyParams {
  int M, N, K;
  // token rows the plan (U, S) is chosen for, >= M (0: M): every pass of a
  // handle plans for its largest, so a row's arithmetic (K split, partial
  // sums) does not depend on how many rows run with it
  int plan_M;
  int U, S, C;  // set by launch_skinny (C: CTAs of a cluster sharing a LayerNorm operand)
  int ns;       // set by launch_skinny_mt: k-blocks of its operand ring
  int epi;
  const bf16 *x;
  int ld_x;
  const float *ln_x;
  int ln_ld;
  const bf16 *ln_g, *ln_b;
  float ln_eps;
  // Folded LayerNorm (fold != 0): LN(x) W^T = r (W (g . x)) - r mu (W g) + W b
  // per row, with the row's mean mu and r = 1 / sqrt(var + eps).  The
  // operand x holds M + 2 bf16 rows (row stride ld_x): g, b, then g . x of
  // every token row, all written by the residual's producer, so one MMA gives
  // W g and W b beside the token rows.  The row statistics are the sums of
  // n_part partials (sum x, sum x^2) per row, fold_part[t * part_stride + i].
  int fold;
  const float2 *fold_part;
  int n_part, part_stride;
  const bf16 *bias;
  float *out_f32;
  bf16 *out_bf16;
  int ld_out;
  float *resid;
  int ld_resid;
  // EPI_RESID, for a folded LayerNorm next (nullable): the next projection's
  // operand rows into xg_out (row stride ld_resid): g_next, b_next, then
  // bf16 (g_next . x) of every row; and per row the (sum x, sum x^2) of the
  // outputs this CTA finishes into part_out[t * part_stride + blockIdx.x * S
  // + rank]
  bf16 *xg_out;
  const bf16 *g_next, *b_next;
  float2 *part_out;  // (row stride part_stride, shared with fold_part)
  bf16 *tap0, *tap1;
  int ld_tap;
  int q_cols, d_model, n_heads, ctx, rows_per_seq;
  bf16 *kc, *vc;
  const int32_t *seq_slot, *pos_base;
  // skinny_xattn: frames per CTA of the fused cross-attention (kc, vc: the
  // acoustic keys and values, ctx frames; out_bf16: the attention output)
  int xa_kpc;
  int xa_outer;  // bound on slot * n_heads + head (the caches' tensor maps)
  // skinny_sattn: 0 causal (target), 1 block (drafter: all of [0, L + M), RoPE)
  int xa_mode;
  const float2 *rope_tab;  // [max_pos][32] (cos, sin), mode 1
  uint32_t *err;
  long long spin;
};
// Whether a projection of M operand rows, N outputs and K inputs has a
// skinny plan (units per CTA U, K split S).  ln: an fp32 LayerNorm operand
// (gain and bias staged, S == 1); whole_k: S == 1 (a folded LayerNorm).
bool skinny_plan(int M, int N, int K, bool ln, bool whole_k, int *U, int *S);
cudaError_t skinny_init();
cudaError_t launch_skinny(const void *W, SkinnyParams p, cudaStream_t s, bool pdl);
// The same projections for up to kMtMaxRows token rows (wf_skinny_mt.cu): the
// weights resident as above, the operand streamed by k-block, warps over
// units and 16-row tiles.  No fp32 LayerNorm operand (ln_x).  The plan of Mr
// operand rows (a folded LayerNorm's two included): units per CTA U, K split
// S, operand ring stages ns.
bool skinny_mt_plan(int Mr, int N, int K, bool fold, bool resid, int *U, int *S, int *ns);
cudaError_t skinny_mt_init();
cudaError_t launch_skinny_mt(const void *W, SkinnyParams p, cudaStream_t s, bool pdl);
// The cross-query projection (folded LN2, one sequence) fused with the
// cross-attention of its queries: one cluster of 8 CTAs per 64-dim head.
// False when the shapes do not allow it (then run the two separately).
bool skinny_xattn_fits(int M, int d, int n_heads, int frames);
cudaError_t launch_skinny_xattn(const void *W, SkinnyParams p, cudaStream_t s, bool pdl);
// The QKV projection (folded LN1, one sequence) fused with the self-attention
// of its rows: one cluster of 8 CTAs per head, each projecting 8 query, 8 key
// and 8 value columns; the new keys and values also go to the cache.
bool skinny_sattn_fits(int M, int d, int n_heads, int ctx);
cudaError_t launch_skinny_sattn(const void *W, SkinnyParams p, cudaStream_t s, bool pdl);

// ------------------------------------------------------------- attention --
struct AttnParams {
  const bf16 *q;
  const bf16 *kc, *vc;
  bf16 *out;
  const int32_t *seq_slot, *pos_base;
  const float2 *rope_tab;  // [max_pos][32] (cos, sin); nullable
  float *part;
  int32_t *counters;
  uint32_t *err;
  long long spin;  // bounded-wait limit (clock cycles; 0: the default)
  int n_seq, rps, n_heads, ctx, mode, n_chunks, qgroups;
  int outer;    // bound on slot * n_heads + head (the caches' tensor maps)
  int cluster;  // the n_chunks blocks of a (sequence, head, group) form a cluster
  int loop;     // one CTA per (sequence, head, group) walks its key blocks in order
};
constexpr int kAttnKeysPerCTA = 256;  // keys per CTA (32 per warp), aligned to absolute positions
constexpr int kAttnQGroup = 16;       // query rows per CTA
// slot * n_heads + head stays below this in calls that do not state the
// number of cache slots (the kernel-level entry points)
constexpr int kAttnOuterBound = 1 << 20;
cudaError_t attention_init();
size_t attn_partial_floats(int n_seq, int rps, int n_heads, int ctx);
int attn_counter_slots(int n_seq, int rps, int n_heads);
cudaError_t launch_attention(const AttnParams &p, cudaStream_t s, bool pdl);
cudaError_t launch_rope_table(float2 *tab, int max_pos, float base, cudaStream_t s);

// -------------------------------------------------------- small kernels --
enum TokSrc : int { TOK_VERIFY = 0, TOK_PROMPT = 1, TOK_ANCHOR = 2 };
struct EmbedParams {
  const bf16 *tok_emb, *pos_emb, *mask_emb;
  const int32_t *seq_slot, *L, *anchor, *cand_in, *forced, *prompt;
  int32_t *cand_out;   // effective proposals (after forcing) [slot][K]
  float *x;
  // nullable: the operand rows of a folded LayerNorm over x (g_next, b_next,
  // then bf16 g_next . x per row; row stride d) and each row's (sum x, sum
  // x^2) as its one partial (part_out[r * part_stride])
  bf16 *xg;
  const bf16 *g_next, *b_next;
  float2 *part_out;
  int part_stride;
  float2 *stats_out;  // nullable: per row and 128-feature tile (mean, M2) of x
  int n_seq, rps, d, K, P, vocab, src, drafter;
  uint32_t *err;
};
cudaError_t launch_embed(const EmbedParams &p, cudaStream_t s, bool pdl);

// y[r] = LN(x[i]) as bf16 with i = r*in_stride + in_off, using the row's
// per-tile statistics stats[i][0..d/128) (mean, M2) written by its producer,
// or (stats == nullptr) the row's mean and variance computed here.
cudaError_t launch_layernorm(const float *x, const float2 *stats, int in_stride, int in_off,
                             const bf16 *g, const bf16 *b, bf16 *y, int rows, int d, float eps,
                             cudaStream_t s, bool pdl);

// Reduce head records over the vocabulary tiles of each row.
struct HeadOut {
  int32_t arg;   // greedy argmax
  int32_t garg;  // Gumbel-max sample
  float lse;     // log sum exp(x) (x = z/T)
  float m;
};
struct HeadReduceParams {
  const HeadRec *recs;
  HeadOut *out;
  int rows, n_tiles;
  // drafter: write proposals cand[slot*K + j-1] for rows j >= 1
  int32_t *cand;
  const int32_t *seq_slot;
  int rps, K, sampling;
};
cudaError_t launch_head_reduce(const HeadReduceParams &p, cudaStream_t s, bool pdl);

struct AcceptParams {
  const int32_t *seq_slot;
  int n_seq, rps, K, max_batch, vocab, eos, max_ctx;
  int greedy_step;  // 1: plain autoregressive step (k = 0)
  const HeadOut *tout, *dout;
  const int32_t *cand;  // effective proposals [slot][K]
  const float *tlogits, *dlogits;  // sampling: raw logits [rows][V]
  const float *forced_q;  // nullable [max_batch][K][V]: logits of the forced proposals' distributions
  const uint8_t *suppress;
  float temperature;
  uint64_t seed;
  int32_t *L, *anchor, *remaining, *done, *step;
  int32_t *out_tokens, *out_count;
  uint32_t *err;
};
cudaError_t launch_accept(const AcceptParams &p, cudaStream_t s, bool pdl);

struct StateParams {
  int op;  // 0: begin prefill, 1: finish prefill, 2: reset to snapshot, 3: append active
  int n;
  const int32_t *slots;
  const int32_t *budget;
  const HeadOut *hout;
  int32_t *first;
  int P, eos, sampling, max_batch;
  int32_t *L, *anchor, *remaining, *done, *step;
  int32_t *snap_L, *snap_anchor, *snap_remaining;
  int32_t *active, *n_active_dev;
  int active_offset;
};
cudaError_t launch_state(const StateParams &p, cudaStream_t s, bool pdl);
cudaError_t launch_compact(const int32_t *done, int max_batch, int32_t *active,
                           int32_t *n_active_dev, cudaStream_t s);

// ------------------------------------------------- persistent decode pass --
// One cooperative launch runs every block of a small-batch pass (M <= 16
// token rows).  See wf_persist.cu.
constexpr int kMkRows = 16;       // token rows a persistent pass supports
constexpr int kMkMaxSeq = 16;     // sequences per persistent pass
constexpr int kMkPhases = 8;      // QKV, self-attn, out, cross-query, cross-attn, cross-out, fc1, fc2
constexpr int kMkMaxG = 256;      // CTAs a persistent pass may use
constexpr int kMkCounters = 8 * 64 + 2;  // phase counters: embedding + 8 phases x 64 blocks
constexpr long long kMkSpinCycles = 400000000LL;  // default bounded-wait limit (~0.2 s)
struct MkLayer {
  const bf16 *ln1_g, *ln1_b, *qkv_b, *out_b, *ln2_g, *ln2_b, *xq_b, *xout_b;
  const bf16 *ln3_g, *ln3_b, *fc1_b, *fc2_b;
  int32_t tm[6];        // tensor-map index of qkv_w, out_w, xq_w, xout_w, fc1_w, fc2_w
  int32_t self_layer;   // layer of the self (target) or history (drafter) cache
  int32_t cross_layer;  // layer of the acoustic cache
  int32_t tap[2];       // tap column blocks written after the block (-1: none)
};
struct MkParams {
  const CUtensorMap *tmaps;  // device table: weight maps, then the cache maps below
  const MkLayer *layers;     // device array [nl]
  int nl, drafter, src, write_taps;
  int G, n_seq, rps, M;
  int d, H, F, T, ctx, Bmax, K, vocab;
  int tm_kc, tm_vc, tm_xk, tm_xv;
  const int32_t *seq_slot, *L, *anchor, *cand_in, *forced;
  int32_t *cand_out;
  const bf16 *tok_emb, *pos_emb, *mask_emb, *lnf_g, *lnf_b;
  bf16 *kc, *vc;             // self or history cache, layer 0
  const float2 *rope_tab;
  float eps;
  // buffers between CTAs (rows: token rows of the pass)
  float *x;                    // [kMkRows][d]    residual stream
  bf16 *q_x, *att_x, *xq_x, *xatt_x;  // [kMkRows][d]
  bf16 *h_x;                   // [kMkRows][F]    fc1 output
  float *part2;                // [d/8][3][kMkRows][8] fc2 split-K partials
  float *xpart;                // [n_seq*H*nch][kMkRows][68] cross-attention partials
  uint32_t *cnt;               // [kMkCounters] CTAs that finished each phase
  uint32_t *cnt2;              // [d/8] fc2 partials published per output unit (cumulative)
  uint32_t *cntx;              // [max_batch*H] cross-attention partials published per head
  bf16 *taps;
  int ld_tap;
  bf16 *xn;                    // [M][d] final LayerNorm output (plain bf16)
  uint32_t *sync;              // [1] CTAs finished (reset by the last)
  uint32_t *err;
  long long spin;              // clock cycles a bounded wait spins before it gives up
};
size_t mk_xpart_words(int M, int H, int T);
cudaError_t persist_init(int *G);
bool persist_supported(int d, int H, int F, int T, int rows);
// Whether a grid of G CTAs leaves at most five projection units per CTA and
// phase (the persistent pass reduces one CTA's units in one batch).
bool persist_grid_fits(int d, int F, int G);
cudaError_t launch_persist(const MkParams &p, cudaStream_t s);

}  // namespace wf
