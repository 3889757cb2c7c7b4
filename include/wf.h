/*
 * wf.h -- C ABI of the GB300 (sm_103a) Whisper-Flash speculative decode step.
 *
 * One speculative decode step of a Whisper-shaped encoder-decoder (Whisper-Flash,
 * arXiv 2609.32869): a 2-layer parallel drafter proposes K=8 tokens in one
 * forward pass from the encoded audio and the target's accepted decoder states
 * (Sec. 3.2, Eq. 2, App. A.2); the frozen target decoder verifies the anchor
 * and the K proposals in one causal pass, keeps the longest agreeing prefix
 * plus its own correction or bonus token (greedy), or applies speculative
 * rejection sampling at temperature T (Sec. 3.1, App. A.4), and rolls back its
 * key/value cache to L+1+a positions (App. A.1).
 *
 * Conventions that hold for every entry point:
 *  - All pointers named d_* / device are DEVICE pointers; the library never
 *    copies them to the host unless an entry point says so.  Host pointers are
 *    named h_*.
 *  - Weights, the workspace and every output buffer are owned by the caller and
 *    borrowed by the handle; they must stay valid until wf_destroy.  Nothing is
 *    allocated by the library on the device: the caller passes one workspace
 *    of at least wf_workspace_bytes() bytes, 256-byte aligned.
 *  - Parameters are bfloat16, row-major; matrices are [out_features, in_features]
 *    (y = x W^T + b); every weight pointer is 16-byte aligned.  Token ids are
 *    int32.
 *  - Calls are asynchronous and ordered on the given stream unless stated.  The
 *    return value reports host-side validation and launch errors; conditions
 *    found on the device (capacity overflow, a bounded wait that gave up) are
 *    recorded in a device error word read by wf_get_state / wf_get_error.
 *  - A handle is not thread-safe.  No C++ exception crosses this boundary.
 *    There is no CPU fallback: without a usable sm_103a device every compute
 *    entry point returns WF_ERR_CUDA.
 */
#ifndef WF_H
#define WF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum wf_status {
  WF_OK = 0,
  WF_ERR_INVALID = 1,     /* a null pointer, a bad size, a misaligned buffer */
  WF_ERR_CAPACITY = 2,    /* max_batch / max_ctx / workspace too small for the call */
  WF_ERR_CUDA = 3,        /* a CUDA runtime or driver call failed */
  WF_ERR_UNSUPPORTED = 4, /* a shape the kernels do not support (see wf_config) */
  WF_ERR_DEVICE = 5       /* the device error word is set (see wf_get_error) */
} wf_status;

/* Device error word bits (wf_get_error). */
#define WF_DEV_ERR_TIMEOUT 0x1u  /* a bounded spin-wait gave up; results are invalid */
#define WF_DEV_ERR_CAPACITY 0x2u /* a sequence would pass max_ctx; it was frozen */
#define WF_DEV_ERR_TOKEN 0x4u    /* a token id outside [0, vocab) was clamped */
#define WF_DEV_ERR_LAUNCH 0x8u   /* a kernel found its launch inconsistent with its plan
                                    (grid, cluster or shared memory) and did nothing */

#define WF_MAX_TAPS 8
#define WF_MAX_LAYERS 64

/* Model shape.  Supported: head_dim = d_model / n_heads = 64; d_model a multiple
 * of 128 and at most 1536; d_ff a multiple of 64; block_k <= 8; max_pos <= 4096. */
typedef struct wf_config {
  int32_t d_model;        /* 1280 (Whisper large), 384 (tiny) */
  int32_t n_heads;        /* 20, 6 */
  int32_t d_ff;           /* 5120, 1536 */
  int32_t n_layers;       /* target decoder blocks: 32, 4 */
  int32_t vocab;          /* 51866, 51865 */
  int32_t max_pos;        /* learned text positions: 448 */
  int32_t enc_frames;     /* encoder frames per request: 1500 (30 s window) */
  int32_t n_draft_layers; /* drafter blocks: 2 (Sec. 3.2) */
  int32_t block_k;        /* proposals per round K: 8 (Eq. 2) */
  int32_t n_taps;         /* history taps: 5 (App. A.2) */
  int32_t taps[WF_MAX_TAPS]; /* zero-based target blocks tapped: 1,8,15,22,29 (App. A.2) */
  int32_t eos_id;         /* end-of-transcript id (App. A.1) */
  float rope_base;        /* drafter RoPE base: 10000 (App. A.2) */
  float ln_eps;           /* LayerNorm epsilon: 1e-5 */
} wf_config;

/* One Whisper decoder block (pre-LayerNorm).  qkv_w stacks the query, key and
 * value projections [3d, d] (bias [3d], key part zero); xkv_w stacks the
 * acoustic key and value projections [2d, d] (bias [2d], key part zero). */
typedef struct wf_layer_weights {
  const void *ln1_g, *ln1_b;    /* [d] */
  const void *qkv_w, *qkv_b;    /* [3d, d], [3d] */
  const void *out_w, *out_b;    /* [d, d], [d] */
  const void *ln2_g, *ln2_b;    /* [d] */
  const void *xq_w, *xq_b;      /* [d, d], [d] */
  const void *xkv_w, *xkv_b;    /* [2d, d], [2d] */
  const void *xout_w, *xout_b;  /* [d, d], [d] */
  const void *ln3_g, *ln3_b;    /* [d] */
  const void *fc1_w, *fc1_b;    /* [F, d], [F] */
  const void *fc2_w, *fc2_b;    /* [d, F], [d] */
} wf_layer_weights;

/* Frozen target decoder.  tok_emb is also the output head (tied). */
typedef struct wf_target_weights {
  const void *tok_emb;          /* [vocab, d] */
  const void *pos_emb;          /* [max_pos, d] */
  const void *lnf_g, *lnf_b;    /* [d] final LayerNorm, shared with the drafter */
  const wf_layer_weights *layers; /* HOST array of n_layers entries (copied at create) */
} wf_target_weights;

/* Drafter (Sec. 3.2, App. A.2).  Its blocks reuse wf_layer_weights: the key and
 * value rows of qkv_w also project the history memory.  It shares tok_emb, the
 * final LayerNorm and the head with the target. */
typedef struct wf_drafter_weights {
  const wf_layer_weights *layers; /* HOST array of n_draft_layers entries */
  const void *proj_w, *proj_b;  /* [d, n_taps*d], [d]: history projection */
  const void *hln_g, *hln_b;    /* [d]: LayerNorm after the projection */
  const void *mask_emb;         /* [d]: learned mask vector m (Eq. 2) */
} wf_drafter_weights;

/* Sampling parameters (App. A.4).  temperature == 0 selects greedy decoding.
 * d_suppress (nullable) is a device uint8 [vocab] mask; ids with a nonzero
 * entry get -inf logits in both the drafter and the target. */
typedef struct wf_sample_params {
  float temperature;
  uint32_t _pad;
  uint64_t seed;                /* Philox4x32-10 key */
  const uint8_t *d_suppress;
} wf_sample_params;

typedef struct wf_handle wf_handle;

/* Size of the workspace wf_create needs for these limits.  max_ctx <= max_pos. */
wf_status wf_workspace_bytes(const wf_config *cfg, int32_t max_batch, int32_t max_ctx,
                             size_t *out_bytes);

/* Build a handle over caller-owned weights and workspace.  Encodes the TMA
 * descriptors of every weight matrix and clears the per-sequence state on
 * `stream` (asynchronously).  d_workspace must be 256-byte aligned and every
 * weight pointer 16-byte aligned (else WF_ERR_INVALID). */
wf_status wf_create(const wf_config *cfg, const wf_target_weights *tw,
                    const wf_drafter_weights *dw, int32_t max_batch, int32_t max_ctx,
                    void *d_workspace, size_t workspace_bytes, void *stream,
                    wf_handle **out);

wf_status wf_destroy(wf_handle *h);

/* Admit n requests into batch slots (App. A.1, A.5): project the acoustic keys
 * and values of every target and drafter block from the encoder output (one
 * dense GEMM per block), run the prompt through the target in one causal pass
 * (filling its cache and the drafter's history memory), and emit the first
 * transcript token, which becomes the first anchor.
 *   d_slots   int32 [n]          distinct slots in [0, max_batch)
 *   d_enc     bf16  [n, enc_frames, d]   encoder output
 *   d_prompt  int32 [n, P]       prompt ids; P + 1 + block_k <= max_ctx
 *   d_budget  int32 [n]          output tokens allowed, >= 1
 *   d_first   int32 [n]          out: the first emitted token
 *   sp        nullable: greedy when null or temperature == 0
 * The admitted slots are appended to the active list. */
wf_status wf_prefill_cross_kv(wf_handle *h, int32_t n, const int32_t *d_slots,
                              const void *d_enc, const int32_t *d_prompt, int32_t P,
                              const int32_t *d_budget, int32_t *d_first,
                              const wf_sample_params *sp, void *stream);

/* Drafter forward for every active sequence (Sec. 3.2): one pass over
 * [Emb(anchor), m x K] per sequence, attending to its history memory and its
 * audio; writes K proposals per sequence into the handle (and, when sampling,
 * the draft logits). */
wf_status wf_draft(wf_handle *h, const wf_sample_params *sp, void *stream);

/* Verify [anchor, c_1..c_K] in one causal target pass, extend the drafter's
 * history with the block's states, and accept (Sec. 3.1, App. A.1):
 *   d_out_tokens int32 [max_batch, K+1] (per slot; entries past the count are -1)
 *   d_out_count  int32 [max_batch]      tokens emitted this step (0 if inactive)
 * d_forced (nullable) int32 [max_batch, K] replaces the drafter's proposals
 * (teacher forcing); the drafter's own pass is unaffected.
 * d_forced_q (nullable; needs d_forced) fp32 [max_batch, K, vocab]: the logits of
 * the distributions the forced proposals were drawn from, row j for proposal
 * c_{j+1}, in the units of the drafter's logits (they get the same temperature
 * and suppression).  When sampling, the rejection rule then uses
 * q = softmax(d_forced_q / T) in place of the drafter's distribution: the rule
 * preserves the target's distribution only if q is the distribution the
 * proposals actually came from (Sec. 3.1, App. A.4).  Ignored when greedy. */
wf_status wf_verify_accept(wf_handle *h, const wf_sample_params *sp,
                           const int32_t *d_forced, const float *d_forced_q,
                           int32_t *d_out_tokens, int32_t *d_out_count, void *stream);

/* wf_draft followed by wf_verify_accept. */
wf_status wf_step(wf_handle *h, const wf_sample_params *sp, const int32_t *d_forced,
                  const float *d_forced_q, int32_t *d_out_tokens, int32_t *d_out_count,
                  void *stream);

/* One plain autoregressive step of the target (Eq. 1; sampling when T > 0)
 * through the same kernels: the identity reference for the speculative path.
 * Outputs as wf_verify_accept (at most one token per slot). */
wf_status wf_greedy_step(wf_handle *h, const wf_sample_params *sp, int32_t *d_out_tokens,
                         int32_t *d_out_count, void *stream);

/* Rebuild the active list from the done flags (ascending slot order),
 * synchronise `stream`, and return the number of active sequences. */
wf_status wf_compact(wf_handle *h, void *stream, int32_t *h_n_active);

/* Rewind n slots to the state their prefill left (cache length, anchor,
 * budget, step counter) and re-activate them; the acoustic keys/values and
 * the prompt's cache rows are kept, so the same request decodes again. */
wf_status wf_reset_slots(wf_handle *h, int32_t n, const int32_t *d_slots, void *stream);

/* Copy per-slot state to HOST arrays (each [max_batch], any may be null) and
 * synchronise `stream`. */
wf_status wf_get_state(wf_handle *h, int32_t *h_len, int32_t *h_anchor, int32_t *h_remaining,
                       int32_t *h_done, void *stream);

/* Read (and optionally clear) the device error word; synchronises `stream`. */
wf_status wf_get_error(wf_handle *h, uint32_t *h_err, int32_t clear, void *stream);

/* Number of kernels the last call to a compute entry point launched. */
int32_t wf_last_launch_count(const wf_handle *h);

/* Inspection hooks for tests and profiling.  wf_set_option(WF_OPT_KEEP_LOGITS,
 * 1) makes every output-head pass also store raw fp32 logits (they are
 * stored anyway when sampling).  wf_debug_view returns the device address and
 * size of an internal buffer of the workspace (valid until wf_destroy; the
 * contents are those left by the last call that wrote them):
 *   WF_VIEW_TARGET_LOGITS  fp32 [rows][vocab]  rows of the last target head pass
 *   WF_VIEW_DRAFT_LOGITS   fp32 [rows][vocab]  rows of the last drafter pass
 *                          (row 9*i + j: sequence i of the active list, block row j)
 *   WF_VIEW_TAPS           bf16 [rows][n_taps*d] tapped residual streams (App. A.2)
 *   WF_VIEW_CANDIDATES     int32 [max_batch][K] proposals verified by the last step */
#define WF_OPT_KEEP_LOGITS 1
#define WF_OPT_PROFILE 2     /* 1: bracket every launch with CUDA events (serialises launches) */
#define WF_OPT_PDL 4         /* 1 (default): kernels use programmatic dependent launch */
#define WF_OPT_GRAPHS 3      /* 1 (default): wf_step / wf_greedy_step replay a CUDA graph
                                captured on first use per (active count, forcing, sampling
                                parameters); 0: launch kernel by kernel */
#define WF_OPT_PERSIST 5     /* 1: the blocks of every drafter, verify and greedy pass run
                                in one persistent cooperative launch (one CTA per SM, so
                                no other kernel may hold SMs meanwhile).  Off by default:
                                on GB300 it is slower than launch by launch.  Supported
                                when max_batch * (block_k + 1) <= 16, 64-wide heads,
                                d_model <= 1280, d_ff a multiple of 512 with
                                d_ff / 4 <= 1280, at most 2048 encoder frames and enough
                                SMs for at most five projection units per CTA; otherwise
                                setting it returns WF_ERR_UNSUPPORTED.  0: one launch per
                                projection and attention.  Both give results within the
                                tolerances of the method, not bit-identical ones. */
#define WF_OPT_SPIN_LIMIT 6  /* clock cycles a bounded wait in the projection kernels and the
                                persistent pass spins before it gives up (records
                                WF_DEV_ERR_TIMEOUT in the error word and returns; the kernel
                                still waits, with the default limit, for its own copies and
                                tensor-core work in flight before it exits).  0 (default)
                                restores about 1 s (projections) and 0.2 s (persistent pass).
                                Meant for tests of the failure path: a limit below a wait's
                                normal duration makes the results of that call invalid. */
#define WF_OPT_SKINNY 7      /* 1: passes of at most max_batch * (block_k + 1) <= 144 token
                                rows run their projections as low-latency kernels that hold
                                a CTA's whole weight slab in shared memory and reduce K in a
                                fixed order (up to 14 rows with the whole token operand
                                resident, more with it streamed by k-block); 0: the tcgen05
                                projections.  Default 1 when max_batch * (block_k + 1) <= 14
                                (single-sequence handles), else 0 (the streamed form is
                                slower than tcgen05 at 2-8 sequences and ties it at 16).
                                Setting 1 on a handle of more than 144 step rows returns
                                WF_ERR_UNSUPPORTED.
                                The two forms agree within the method's tolerances, not bit
                                for bit; a handle's speculative and plain greedy steps
                                always take the same form. */
#define WF_VIEW_TARGET_LOGITS 1
#define WF_VIEW_DRAFT_LOGITS 2
#define WF_VIEW_TAPS 3
#define WF_VIEW_CANDIDATES 4
wf_status wf_set_option(wf_handle *h, int32_t option, int32_t value);

/* Kernel families reported by wf_profile_read. */
#define WF_FAM_GEMM 0       /* tcgen05 projections (all but the output head) */
#define WF_FAM_HEAD 1       /* tcgen05 output head with its fused reduction records */
#define WF_FAM_ATTN_SELF 2  /* causal verify / prompt attention and the drafter's block attention */
#define WF_FAM_ATTN_CROSS 3 /* cross-attention over the encoder frames */
#define WF_FAM_LAYERNORM 4
#define WF_FAM_OTHER 5      /* embeddings, head reduction, accept, slot state */
#define WF_FAM_PERSIST 6    /* persistent small-batch pass: every block of a drafter,
                               verify or greedy pass in one launch (WF_OPT_PERSIST) */
#define WF_PROF_FAMILIES 7
/* With WF_OPT_PROFILE on: synchronise `stream`, then return per family the
 * summed kernel time (ms, CUDA events on the launching stream), the number of
 * launches and, for the GEMM and head families, the algorithmic bytes those
 * launches move (weights + token rows in + results out; split-K scratch is
 * not counted); for the persistent family the blocks' projection weights and
 * acoustic keys/values.  Each array has WF_PROF_FAMILIES entries; accumulators reset. */
wf_status wf_profile_read(wf_handle *h, void *stream, double *h_ms, int32_t *h_launches,
                          double *h_bytes);
wf_status wf_debug_view(wf_handle *h, int32_t which, void **d_ptr, size_t *bytes);

const char *wf_status_str(wf_status s);

/* ------------------------------------------------------------------------
 * Kernel-level entry points (device pointers, stream ordered).  They run one
 * kernel family of the step on caller buffers so each can be checked alone.
 * ---------------------------------------------------------------------- */

/* Y = X W^T (+ b): the skinny-M tcgen05 GEMM of every projection in the step.
 *   d_x bf16 [M, K], d_w bf16 [N, K], d_b bf16 [N] (nullable), d_y fp32 [M, N].
 *   K % 64 == 0, 1 <= M, 1 <= N.  Split-K partial sums are reduced on chip
 *   (thread-block cluster shared memory), so wf_gemm_scratch_bytes returns 0 and
 *   d_scratch may be null. */
wf_status wf_gemm_bf16(const void *d_x, const void *d_w, const void *d_b, float *d_y,
                       int32_t M, int32_t N, int32_t K, void *d_scratch,
                       size_t scratch_bytes, void *stream);
size_t wf_gemm_scratch_bytes(int32_t M, int32_t N, int32_t K);

/* Multi-head attention of RPS query rows per sequence against per-sequence
 * key/value caches laid out [slot][head][position][64] (bf16):
 *   d_q     bf16 [n_seq*RPS, n_heads*64]  queries, row r = seq*RPS + j
 *   d_kc/vc bf16 [n_slots, n_heads, ctx, 64]
 *   d_slot  int32 [n_seq]   cache slot of each sequence
 *   d_base  int32 [n_slots] position of query row 0 (the cache length L)
 *   mode 0: causal (query j sees keys [0, base+j]);  mode 1: all keys
 *   [0, base+RPS) (drafter block);  mode 2: all ctx keys (cross-attention)
 *   rope: nonzero applies RoPE (rope_base) to queries and keys by position
 *   d_out  bf16 [n_seq*RPS, n_heads*64] */
wf_status wf_attention(const void *d_q, const void *d_kc, const void *d_vc,
                       const int32_t *d_slot, const int32_t *d_base, int32_t n_seq,
                       int32_t RPS, int32_t n_heads, int32_t ctx, int32_t mode, int32_t rope,
                       float rope_base, void *d_out, void *d_scratch, size_t scratch_bytes,
                       void *stream);
size_t wf_attention_scratch_bytes(int32_t n_seq, int32_t RPS, int32_t n_heads, int32_t ctx);

/* wf_attention without a scratch argument, for callers that cannot allocate
 * device memory (a graph being captured in a mode that forbids cudaMalloc, a
 * plugin whose host framework owns every allocation, a latency-critical loop
 * that must not synchronise).  The paper has no counterpart: this is a
 * deployment convenience of this library.  Its scratch is one 8 MiB device
 * array inside the library, held by every GPU that loads it until exit;
 * calls needing more (wf_attention_scratch_bytes > 8 MiB) return
 * WF_ERR_CAPACITY.  The first call on a device looks the array up and may
 * load the library's module, so make it before any stream capture.  Every
 * call shares the array: calls that may overlap on the GPU race and must not
 * be issued.  Arguments and results are those of wf_attention. */
wf_status wf_attention_noalloc(const void *d_q, const void *d_kc, const void *d_vc,
                               const int32_t *d_slot, const int32_t *d_base, int32_t n_seq,
                               int32_t RPS, int32_t n_heads, int32_t ctx, int32_t mode,
                               int32_t rope, float rope_base, void *d_out, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* WF_H */
