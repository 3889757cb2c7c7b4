// Row-wise kernels of the decode step: block embeddings (Eq. 2 for the
// drafter; token + learned position for the target), LayerNorm, the
// cross-tile reduction of the output head, the per-sequence accept/rollback
// rule (Sec. 3.1, App. A.1, A.4) and per-slot state bookkeeping.
#include "wf_device.cuh"
#include "wf_internal.h"

namespace wf {

static cudaError_t launch_ex(const void *fn, dim3 grid, dim3 block, void **args, cudaStream_t s,
                             bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelExC(&cfg, fn, args);
}

// ------------------------------------------------------------ embedding --
// Target rows: x = Emb(tok) + PosEmb(L + j).  Drafter rows (Eq. 2): row 0 is
// Emb(anchor), rows 1..K are the mask vector m; no position embedding (the
// drafter marks positions with RoPE).
__global__ void embed_kernel(const EmbedParams p) {
  pdl_wait();
  pdl_launch_dependents();
  const int r = blockIdx.x;
  const int i = r / p.rps, j = r - i * p.rps;
  const int slot = p.seq_slot[i];
  int tok = -1;
  if (p.src == TOK_PROMPT) {
    tok = p.prompt[i * p.P + j];
  } else if (j == 0) {
    tok = p.anchor[slot];
  } else if (!p.drafter) {
    const int src = p.forced ? p.forced[slot * p.K + j - 1] : p.cand_in[slot * p.K + j - 1];
    tok = src;
    if (threadIdx.x == 0) p.cand_out[slot * p.K + j - 1] = src;
  }
  const bool use_mask = p.drafter && j > 0;
  if (!use_mask && (tok < 0 || tok >= p.vocab)) {
    if (threadIdx.x == 0) set_error(p.err, WF_DEV_ERR_TOKEN);
    tok = tok < 0 ? 0 : p.vocab - 1;
  }
  const int pos = (p.drafter || !p.L) ? 0 : ((p.src == TOK_PROMPT ? 0 : p.L[slot]) + j);
  float *x = p.x + static_cast<size_t>(r) * p.d;
  // thread tid holds feature 128k + tid of every 128-feature tile k
  const int tiles = p.d >> 7;
  float v[kMaxStatTiles];
#pragma unroll
  for (int k = 0; k < kMaxStatTiles; ++k) {
    if (k >= tiles) continue;
    const int e = k * 128 + threadIdx.x;
    float val;
    if (use_mask) {
      val = bf2f(p.mask_emb[e]);
    } else {
      val = bf2f(p.tok_emb[static_cast<size_t>(tok) * p.d + e]);
      if (!p.drafter) val += bf2f(p.pos_emb[static_cast<size_t>(pos) * p.d + e]);
    }
    v[k] = val;
    x[e] = val;
  }
  if (!p.stats_out) return;
  // per-tile (mean, M2) of the row for the next LayerNorm
  __shared__ float red[4][kMaxStatTiles];
  __shared__ float mean_s[kMaxStatTiles];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int k = 0; k < kMaxStatTiles; ++k) {
    if (k >= tiles) continue;
    const float sum = warp_sum(v[k]);
    if (lane == 0) red[warp][k] = sum;
  }
  __syncthreads();
  if (threadIdx.x < tiles) {
    const int k = threadIdx.x;
    mean_s[k] = ((red[0][k] + red[1][k]) + (red[2][k] + red[3][k])) * (1.0f / 128.f);
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kMaxStatTiles; ++k) {
    if (k >= tiles) continue;
    const float dv = v[k] - mean_s[k];
    const float sq = warp_sum(dv * dv);
    if (lane == 0) red[warp][k] = sq;
  }
  __syncthreads();
  if (threadIdx.x < tiles) {
    const int k = threadIdx.x;
    p.stats_out[static_cast<size_t>(r) * tiles + k] =
        make_float2(mean_s[k], (red[0][k] + red[1][k]) + (red[2][k] + red[3][k]));
  }
}

cudaError_t launch_embed(const EmbedParams &p0, cudaStream_t s, bool pdl) {
  EmbedParams p = p0;
  void *args[] = {&p};
  return launch_ex(reinterpret_cast<const void *>(embed_kernel), dim3(p.n_seq * p.rps), dim3(128),
                   args, s, pdl);
}

// ------------------------------------------------------------ LayerNorm --
// One warp per row; lane l owns the float4 chunks l, l+32, ... of the row.
// The row's statistics come from the kernel that wrote it (per 128-feature
// tile, merged in tile order), so this kernel and the GEMMs that normalise
// their own token operand produce identical bits.  Every load is issued
// before any arithmetic so the latencies overlap.
__global__ void __launch_bounds__(128) layernorm_kernel(const float *__restrict__ x,
                                                        const float2 *__restrict__ stats,
                                                        int in_stride, int in_off,
                                                        const bf16 *__restrict__ g,
                                                        const bf16 *__restrict__ b,
                                                        bf16 *__restrict__ y, int rows, int d,
                                                        float eps) {
  pdl_wait();
  pdl_launch_dependents();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= rows) return;
  const size_t row = static_cast<size_t>(warp) * in_stride + in_off;
  const float4 *xr = reinterpret_cast<const float4 *>(x + row * d);
  const uint2 *gr = reinterpret_cast<const uint2 *>(g);
  const uint2 *br = reinterpret_cast<const uint2 *>(b);
  const int chunks = d >> 7;
  float4 v[kMaxStatTiles];
  uint2 gv[kMaxStatTiles], bv[kMaxStatTiles];
#pragma unroll
  for (int k = 0; k < kMaxStatTiles; ++k) {
    if (k < chunks) {
      v[k] = xr[k * 32 + lane];
      gv[k] = gr[k * 32 + lane];
      bv[k] = br[k * 32 + lane];
    }
  }
  const float2 ms = merge_tile_stats(stats + row * chunks, chunks, eps);
  uint2 *yr = reinterpret_cast<uint2 *>(y + static_cast<size_t>(warp) * d);
#pragma unroll
  for (int k = 0; k < kMaxStatTiles; ++k) {
    if (k < chunks) {
      const __nv_bfloat162 g01 = *reinterpret_cast<const __nv_bfloat162 *>(&gv[k].x);
      const __nv_bfloat162 g23 = *reinterpret_cast<const __nv_bfloat162 *>(&gv[k].y);
      const __nv_bfloat162 b01 = *reinterpret_cast<const __nv_bfloat162 *>(&bv[k].x);
      const __nv_bfloat162 b23 = *reinterpret_cast<const __nv_bfloat162 *>(&bv[k].y);
      const __nv_bfloat162 o01 =
          __floats2bfloat162_rn(ln_apply(v[k].x, ms, __low2float(g01), __low2float(b01)),
                                ln_apply(v[k].y, ms, __high2float(g01), __high2float(b01)));
      const __nv_bfloat162 o23 =
          __floats2bfloat162_rn(ln_apply(v[k].z, ms, __low2float(g23), __low2float(b23)),
                                ln_apply(v[k].w, ms, __high2float(g23), __high2float(b23)));
      uint2 o;
      o.x = *reinterpret_cast<const uint32_t *>(&o01);
      o.y = *reinterpret_cast<const uint32_t *>(&o23);
      yr[k * 32 + lane] = o;
    }
  }
}

cudaError_t launch_layernorm(const float *x, const float2 *stats, int in_stride, int in_off,
                             const bf16 *g, const bf16 *b, bf16 *y, int rows, int d, float eps,
                             cudaStream_t s, bool pdl) {
  if (d % 128 || d / 128 > kMaxStatTiles || !stats) return cudaErrorInvalidValue;
  void *args[] = {&x, &stats, &in_stride, &in_off, &g, &b, &y, &rows, &d, &eps};
  const int threads = 128;
  const int blocks = (rows * 32 + threads - 1) / threads;
  return launch_ex(reinterpret_cast<const void *>(layernorm_kernel), dim3(blocks), dim3(threads),
                   args, s, pdl);
}

// ---------------------------------------------------------- head reduce --
// Combine the per-tile records of each row in tile order (deterministic):
// argmax with the lowest id on ties, log-sum-exp, and the Gumbel-max draw.
__device__ __forceinline__ void rec_combine(float &m, float &s, int &arg, float &gm, int &garg,
                                            const HeadRec &r) {
  const float M = fmaxf(m, r.m);
  float ns = 0.f;
  if (M != -INFINITY)
    ns = (m == -INFINITY ? 0.f : s * __expf(m - M)) + (r.m == -INFINITY ? 0.f : r.s * __expf(r.m - M));
  if (r.m > m || (r.m == m && r.arg < arg)) arg = r.arg;
  m = M;
  s = ns;
  if (r.gm > gm || (r.gm == gm && r.garg < garg)) {
    gm = r.gm;
    garg = r.garg;
  }
}

__global__ void head_reduce_kernel(const HeadReduceParams p) {
  pdl_wait();
  pdl_launch_dependents();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= p.rows) return;
  const HeadRec *rr = p.recs + static_cast<size_t>(warp) * p.n_tiles;
  // lane l reduces tiles l, l+32, ... in order; lanes then combine in order
  float m = -INFINITY, s = 0.f, gm = -INFINITY;
  int arg = 0x7fffffff, garg = 0x7fffffff;
  for (int t = lane; t < p.n_tiles; t += 32) rec_combine(m, s, arg, gm, garg, rr[t]);
  for (int off = 1; off < 32; off <<= 1) {
    HeadRec o;
    o.m = __shfl_down_sync(0xffffffffu, m, off);
    o.s = __shfl_down_sync(0xffffffffu, s, off);
    o.gm = __shfl_down_sync(0xffffffffu, gm, off);
    o.arg = __shfl_down_sync(0xffffffffu, arg, off);
    o.garg = __shfl_down_sync(0xffffffffu, garg, off);
    if ((lane & (2 * off - 1)) == 0 && lane + off < 32) rec_combine(m, s, arg, gm, garg, o);
  }
  if (lane == 0) {
    HeadOut out;
    out.arg = arg;
    out.garg = garg;
    out.m = m;
    out.lse = m + logf(s);
    p.out[warp] = out;
    if (p.cand) {
      const int i = warp / p.rps, j = warp - i * p.rps;
      if (j >= 1 && j <= p.K) p.cand[p.seq_slot[i] * p.K + j - 1] = p.sampling ? garg : arg;
    }
  }
}

cudaError_t launch_head_reduce(const HeadReduceParams &p0, cudaStream_t s, bool pdl) {
  HeadReduceParams p = p0;
  void *args[] = {&p};
  const int threads = 256;
  return launch_ex(reinterpret_cast<const void *>(head_reduce_kernel),
                   dim3((p.rows * 32 + threads - 1) / threads), dim3(threads), args, s, pdl);
}

// --------------------------------------------------------------- accept --
// One warp per active sequence.  Greedy (Sec. 3.1): keep proposals while they
// equal the target's argmax, then emit the target's token (correction, or
// bonus after K agreements).  Sampling (Sec. 3.1, App. A.4): accept c_i when
// u_i < p_i(c_i)/q_i(c_i) in FP32; at the first rejection draw from the
// normalised residual (p_i - q_i)_+ by Gumbel-max; after a full block emit
// the bonus drawn from the target.  An accepted EOS ends the transcript
// without a bonus; with R tokens left at most R-1 proposals are live; the
// cache keeps L+1+a positions (App. A.1).
__device__ int residual_draw(const AcceptParams &p, int slot, int step, int i, const float *xt,
                             float lse_t, const float *xd, float lse_d, int lane) {
  // i: 1-based candidate index; xt/xd: raw logit rows
  float best = -INFINITY;
  int barg = 0x7fffffff;
  bool any = false;
  for (int v = lane; v < p.vocab; v += 32) {
    if (p.suppress && p.suppress[v]) continue;
    const float pt = expf(__fdiv_rn(xt[v], p.temperature) - lse_t);
    const float qd = expf(__fdiv_rn(xd[v], p.temperature) - lse_d);
    const float r = fmaxf(pt - qd, 0.f);
    if (r > 0.f) {
      any = true;
      const float sc = logf(r) + gumbel(p.seed, slot, step, i, kTagResidual, v);
      if (sc > best) {
        best = sc;
        barg = v;
      }
    }
  }
  any = __any_sync(0xffffffffu, any);
  if (!any) {  // empty residual (rounding only): draw from the target itself
    for (int v = lane; v < p.vocab; v += 32) {
      if (p.suppress && p.suppress[v]) continue;
      const float sc = __fdiv_rn(xt[v], p.temperature) + gumbel(p.seed, slot, step, i, kTagResidual, v);
      if (sc > best) {
        best = sc;
        barg = v;
      }
    }
  }
  for (int off = 16; off > 0; off >>= 1) {
    const float b2 = __shfl_xor_sync(0xffffffffu, best, off);
    const int a2 = __shfl_xor_sync(0xffffffffu, barg, off);
    if (b2 > best || (b2 == best && a2 < barg)) {
      best = b2;
      barg = a2;
    }
  }
  return barg;
}

__global__ void __launch_bounds__(512) accept_kernel(const AcceptParams p) {
  pdl_wait();
  pdl_launch_dependents();
  const int Kp1 = p.K + 1;
  for (int sidx = threadIdx.x; sidx < p.max_batch; sidx += blockDim.x) {
    p.out_count[sidx] = 0;
    for (int j = 0; j < Kp1; ++j) p.out_tokens[sidx * Kp1 + j] = -1;
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = blockDim.x >> 5;
  const bool sampling = p.temperature > 0.f;
  for (int i = warp; i < p.n_seq; i += nwarps) {
    const int slot = p.seq_slot[i];
    if (p.done[slot]) continue;
    const int R = p.remaining[slot];
    const int step = p.step[slot];
    int k = p.greedy_step ? 0 : min(p.K, R - 1);
    if (k < 0) k = 0;
    const int r0 = i * p.rps;
    int emitted[16];
    int n_em = 0, a = 0;
    bool stop = false;
    for (int c = 1; c <= k; ++c) {
      const int cand = p.cand[slot * p.K + c - 1];
      bool acc;
      if (!sampling) {
        acc = cand == p.tout[r0 + c - 1].arg;
      } else {
        const int rt = r0 + c - 1, rd = r0 + c;  // drafter row c holds mask position c
        const float lse_t = p.tout[rt].lse, lse_d = p.dout[rd].lse;
        const float xt = __fdiv_rn(p.tlogits[static_cast<size_t>(rt) * p.vocab + cand], p.temperature);
        const float xd = __fdiv_rn(p.dlogits[static_cast<size_t>(rd) * p.vocab + cand], p.temperature);
        const bool sup = p.suppress && p.suppress[cand];
        const float pc = sup ? 0.f : expf(xt - lse_t);
        const float qc = sup ? 0.f : expf(xd - lse_d);
        Philox4 o = philox4x32_10(0, c, step, (kTagAccept << 24) | (slot & 0xFFFFFF),
                                  static_cast<uint32_t>(p.seed), static_cast<uint32_t>(p.seed >> 32));
        const float u = word_to_uniform(o.x[0]);
        acc = u < __fdiv_rn(pc, qc);
        if (!acc) {
          const int t = residual_draw(p, slot, step, c,
                                      p.tlogits + static_cast<size_t>(rt) * p.vocab, lse_t,
                                      p.dlogits + static_cast<size_t>(rd) * p.vocab, lse_d, lane);
          emitted[n_em++] = t;
          stop = (t == p.eos);
          a = c - 1;
          k = -1;  // mark: finished by a rejection
          break;
        }
      }
      if (!acc) break;
      emitted[n_em++] = cand;
      a = c;
      if (cand == p.eos) {
        stop = true;
        k = -1;
        break;
      }
    }
    if (k >= 0) {  // correction (greedy mismatch) or bonus
      const HeadOut &ho = p.tout[r0 + a];
      const int t = sampling ? ho.garg : ho.arg;
      emitted[n_em++] = t;
      stop = (t == p.eos);
    }
    if (lane == 0) {
      for (int e = 0; e < n_em; ++e) p.out_tokens[slot * Kp1 + e] = emitted[e];
      p.out_count[slot] = n_em;
      const int newL = p.L[slot] + 1 + a;
      p.L[slot] = newL;
      p.anchor[slot] = emitted[n_em - 1];
      const int left = R - n_em;
      p.remaining[slot] = left;
      p.step[slot] = step + 1;
      bool done = stop || left <= 0;
      if (!done && newL + Kp1 > p.max_ctx) {
        set_error(p.err, WF_DEV_ERR_CAPACITY);
        done = true;
      }
      p.done[slot] = done ? 1 : 0;
    }
    __syncwarp();
  }
}

cudaError_t launch_accept(const AcceptParams &p0, cudaStream_t s, bool pdl) {
  AcceptParams p = p0;
  void *args[] = {&p};
  return launch_ex(reinterpret_cast<const void *>(accept_kernel), dim3(1), dim3(512), args, s, pdl);
}

// ---------------------------------------------------------------- state --
__global__ void state_kernel(const StateParams p) {
  pdl_wait();
  pdl_launch_dependents();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= p.n) return;
  const int slot = p.slots[i];
  if (slot < 0 || slot >= p.max_batch) return;
  if (p.op == 0) {  // begin prefill: empty cache, step 0
    p.L[slot] = 0;
    p.step[slot] = 0;
    p.done[slot] = 0;
  } else if (p.op == 1) {  // finish prefill: the first token becomes the anchor
    const HeadOut &ho = p.hout[i];
    const int first = p.sampling ? ho.garg : ho.arg;
    const int left = p.budget[i] - 1;
    p.L[slot] = p.P;
    p.anchor[slot] = first;
    p.remaining[slot] = left;
    p.step[slot] = 1;
    p.done[slot] = (first == p.eos || left <= 0) ? 1 : 0;
    p.snap_L[slot] = p.P;
    p.snap_anchor[slot] = first;
    p.snap_remaining[slot] = left;
    if (p.first) p.first[i] = first;
    p.active[p.active_offset + i] = slot;
    if (i == 0) *p.n_active_dev = p.active_offset + p.n;
  } else if (p.op == 2) {  // rewind to the post-prefill snapshot
    p.L[slot] = p.snap_L[slot];
    p.anchor[slot] = p.snap_anchor[slot];
    p.remaining[slot] = p.snap_remaining[slot];
    p.step[slot] = 1;
    p.done[slot] = (p.snap_remaining[slot] <= 0) ? 1 : 0;
  }
}

cudaError_t launch_state(const StateParams &p0, cudaStream_t s, bool pdl) {
  StateParams p = p0;
  void *args[] = {&p};
  return launch_ex(reinterpret_cast<const void *>(state_kernel), dim3((p.n + 127) / 128), dim3(128),
                   args, s, pdl);
}

// Active list = slots whose done flag is clear, ascending.
__global__ void compact_kernel(const int32_t *done, int max_batch, int32_t *active,
                               int32_t *n_active) {
  if (threadIdx.x == 0) {
    int c = 0;
    for (int s = 0; s < max_batch; ++s)
      if (!done[s]) active[c++] = s;
    *n_active = c;
  }
}

cudaError_t launch_compact(const int32_t *done, int max_batch, int32_t *active,
                           int32_t *n_active_dev, cudaStream_t s) {
  compact_kernel<<<1, 32, 0, s>>>(done, max_batch, active, n_active_dev);
  return cudaGetLastError();
}

}  // namespace wf
