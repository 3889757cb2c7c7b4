// Row-wise kernels of the decode step: block embeddings (Eq. 2 for the
// drafter; token + learned position for the target), LayerNorm, the
// cross-tile reduction of the output head, the per-sequence accept/rollback
// rule (Sec. 3.1, App. A.1, A.4) and per-slot state bookkeeping.
#include <mutex>

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
    if (p.xg) {
      p.xg[static_cast<size_t>(r + 2) * p.d + e] = __float2bfloat16(val * bf2f(p.g_next[e]));
      if (r == 0) {
        p.xg[e] = p.g_next[e];
        p.xg[static_cast<size_t>(p.d) + e] = p.b_next[e];
      }
    }
  }
  if (p.part_out) {  // the whole row's (sum x, sum x^2), summed in a fixed order
    __shared__ float red2[4][2];
    float s1 = 0.f, s2 = 0.f;
#pragma unroll
    for (int k = 0; k < kMaxStatTiles; ++k)
      if (k < tiles) {
        s1 += v[k];
        s2 = __fmaf_rn(v[k], v[k], s2);
      }
    s1 = warp_sum(s1);
    s2 = warp_sum(s2);
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) {
      red2[w][0] = s1;
      red2[w][1] = s2;
    }
    __syncthreads();
    if (threadIdx.x == 0)
      p.part_out[static_cast<size_t>(r) * p.part_stride] =
          make_float2((red2[0][0] + red2[1][0]) + (red2[2][0] + red2[3][0]),
                      (red2[0][1] + red2[1][1]) + (red2[2][1] + red2[3][1]));
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
  float2 ms;
  if (stats) {
    ms = merge_tile_stats(stats + row * chunks, chunks, eps);
  } else {  // the row's own mean and variance (two passes over the registers)
    float sum = 0.f;
#pragma unroll
    for (int k = 0; k < kMaxStatTiles; ++k)
      if (k < chunks) sum += (v[k].x + v[k].y) + (v[k].z + v[k].w);
    const float mean = warp_sum(sum) / static_cast<float>(d);
    float q = 0.f;
#pragma unroll
    for (int k = 0; k < kMaxStatTiles; ++k) {
      if (k < chunks) {
        const float a = v[k].x - mean, b = v[k].y - mean, c = v[k].z - mean, e = v[k].w - mean;
        q += (a * a + b * b) + (c * c + e * e);
      }
    }
    ms = make_float2(mean, rsqrtf(warp_sum(q) / static_cast<float>(d) + eps));
  }
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
  if (d % 128 || d / 128 > kMaxStatTiles) return cudaErrorInvalidValue;
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
// One CTA per active sequence.  Greedy (Sec. 3.1): keep proposals while they
// equal the target's argmax, then emit the target's token (correction, or
// bonus after K agreements).  Sampling (Sec. 3.1, App. A.4): accept c_i when
// u_i < p_i(c_i)/q_i(c_i) in FP32; at the first rejection draw from the
// normalised residual (p_i - q_i)_+ by Gumbel-max; after a full block emit
// the bonus drawn from the target.  An accepted EOS ends the transcript
// without a bonus; with R tokens left at most R-1 proposals are live; the
// cache keeps L+1+a positions (App. A.1).  The decisions are sequential and
// taken by one thread; the residual draw and the normalisers of forced
// proposal distributions reduce over the vocabulary with the whole CTA.
constexpr int kAccThreads = 256;

// The CTA's maximum (value, lowest id on ties) of (v, arg) over its threads.
__device__ __forceinline__ void block_argmax(float &v, int &arg, float *sv, int *sa) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, v, off);
    const int a2 = __shfl_xor_sync(0xffffffffu, arg, off);
    if (v2 > v || (v2 == v && a2 < arg)) {
      v = v2;
      arg = a2;
    }
  }
  __syncthreads();
  if (lane == 0) {
    sv[warp] = v;
    sa[warp] = arg;
  }
  __syncthreads();
  v = sv[0];
  arg = sa[0];
  for (int w = 1; w < kAccThreads / 32; ++w)
    if (sv[w] > v || (sv[w] == v && sa[w] < arg)) {
      v = sv[w];
      arg = sa[w];
    }
}
// log sum exp over the CTA of per-thread (max, sum of exp(x - max)).
__device__ __forceinline__ float block_lse(float m, float sum, float *sm, float *ss) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
    const float s2 = __shfl_xor_sync(0xffffffffu, sum, off);
    const float M = fmaxf(m, m2);
    sum = (M == -INFINITY) ? 0.f : sum * expf(m - M) + s2 * expf(m2 - M);
    m = M;
  }
  __syncthreads();
  if (lane == 0) {
    sm[warp] = m;
    ss[warp] = sum;
  }
  __syncthreads();
  float M = -INFINITY, S = 0.f;
  for (int w = 0; w < kAccThreads / 32; ++w) {
    const float M2 = fmaxf(M, sm[w]);
    S = (M2 == -INFINITY) ? 0.f : S * expf(M - M2) + ss[w] * expf(sm[w] - M2);
    M = M2;
  }
  return M + logf(S);
}

__global__ void __launch_bounds__(kAccThreads) accept_kernel(const AcceptParams p) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float s_v[kAccThreads / 32], s_w[kAccThreads / 32];
  __shared__ int s_a[kAccThreads / 32];
  __shared__ float s_qlse[8];
  __shared__ int s_em[16];
  __shared__ int s_state[4];  // emitted count, accepted a, stopped, rejected row (0: none)
  const int Kp1 = p.K + 1;
  const int tid = threadIdx.x;
  // slots outside the active list emit nothing this step
  for (int sl = blockIdx.x; sl < p.max_batch; sl += gridDim.x) {
    bool active = false;
    for (int i = 0; i < p.n_seq; ++i) active = active || p.seq_slot[i] == sl;
    if (!active) {
      for (int j = tid; j < Kp1; j += kAccThreads) p.out_tokens[sl * Kp1 + j] = -1;
      if (tid == 0) p.out_count[sl] = 0;
    }
  }
  const int i = blockIdx.x;
  if (i >= p.n_seq) return;
  const int slot = p.seq_slot[i];
  if (p.done[slot]) {
    for (int j = tid; j < Kp1; j += kAccThreads) p.out_tokens[slot * Kp1 + j] = -1;
    if (tid == 0) p.out_count[slot] = 0;
    return;
  }
  const bool sampling = p.temperature > 0.f;
  const int R = p.remaining[slot];
  const int step = p.step[slot];
  int k = p.greedy_step ? 0 : min(p.K, R - 1);
  if (k < 0) k = 0;
  const int r0 = i * p.rps;
  const float *fq = p.forced_q ? p.forced_q + static_cast<size_t>(slot) * p.K * p.vocab : nullptr;
  // normalisers of the forced proposal distributions softmax(q / T)
  if (sampling && fq) {
    for (int c = 0; c < k; ++c) {
      const float *row = fq + static_cast<size_t>(c) * p.vocab;
      float m = -INFINITY, sum = 0.f;
      for (int v = tid; v < p.vocab; v += kAccThreads) {
        if (p.suppress && p.suppress[v]) continue;
        const float x = __fdiv_rn(row[v], p.temperature);
        if (x > m) {
          sum = sum * expf(m - x) + 1.f;
          m = x;
        } else {
          sum += expf(x - m);
        }
      }
      const float l = block_lse(m, sum, s_v, s_w);
      if (tid == 0) s_qlse[c] = l;
    }
  }
  if (tid == 0) {
    int n_em = 0, a = 0, stop = 0, rej = 0;
    bool finished = false;
    for (int c = 1; c <= k; ++c) {
      const int cand = p.cand[slot * p.K + c - 1];
      bool acc;
      if (!sampling) {
        acc = cand == p.tout[r0 + c - 1].arg;
      } else {
        const int rt = r0 + c - 1, rd = r0 + c;  // drafter row c holds mask position c
        const float lse_t = p.tout[rt].lse;
        const float lse_d = fq ? s_qlse[c - 1] : p.dout[rd].lse;
        const float zd = fq ? fq[static_cast<size_t>(c - 1) * p.vocab + cand]
                            : p.dlogits[static_cast<size_t>(rd) * p.vocab + cand];
        const float xt = __fdiv_rn(p.tlogits[static_cast<size_t>(rt) * p.vocab + cand], p.temperature);
        const float xd = __fdiv_rn(zd, p.temperature);
        const bool sup = p.suppress && p.suppress[cand];
        const float pc = sup ? 0.f : expf(xt - lse_t);
        const float qc = sup ? 0.f : expf(xd - lse_d);
        Philox4 o = philox4x32_10(0, c, step, (kTagAccept << 24) | (slot & 0xFFFFFF),
                                  static_cast<uint32_t>(p.seed), static_cast<uint32_t>(p.seed >> 32));
        const float u = word_to_uniform(o.x[0]);
        acc = u < __fdiv_rn(pc, qc);
        if (!acc) {
          rej = c;  // the residual draw below supplies the token
          a = c - 1;
          finished = true;
          break;
        }
      }
      if (!acc) break;
      s_em[n_em++] = cand;
      a = c;
      if (cand == p.eos) {
        stop = 1;
        finished = true;
        break;
      }
    }
    if (!finished) {  // correction (greedy mismatch) or bonus
      const HeadOut &ho = p.tout[r0 + a];
      const int t = sampling ? ho.garg : ho.arg;
      s_em[n_em++] = t;
      stop = t == p.eos;
    }
    s_state[0] = n_em;
    s_state[1] = a;
    s_state[2] = stop;
    s_state[3] = rej;
  }
  __syncthreads();
  const int rej = s_state[3];
  if (rej) {
    // residual (p - q)_+ of row rej by Gumbel-max over log r; if it is empty
    // (rounding only) the token is drawn from the target itself
    const int rt = r0 + rej - 1, rd = r0 + rej;
    const float *xt = p.tlogits + static_cast<size_t>(rt) * p.vocab;
    const float *xd = fq ? fq + static_cast<size_t>(rej - 1) * p.vocab
                         : p.dlogits + static_cast<size_t>(rd) * p.vocab;
    const float lse_t = p.tout[rt].lse;
    const float lse_d = fq ? s_qlse[rej - 1] : p.dout[rd].lse;
    float best = -INFINITY;
    int barg = 0x7fffffff;
    bool any = false;
    for (int v = tid; v < p.vocab; v += kAccThreads) {
      if (p.suppress && p.suppress[v]) continue;
      const float pt = expf(__fdiv_rn(xt[v], p.temperature) - lse_t);
      const float qd = expf(__fdiv_rn(xd[v], p.temperature) - lse_d);
      const float r = fmaxf(pt - qd, 0.f);
      if (r > 0.f) {
        any = true;
        const float sc = logf(r) + gumbel(p.seed, slot, step, rej, kTagResidual, v);
        if (sc > best || (sc == best && v < barg)) {
          best = sc;
          barg = v;
        }
      }
    }
    if (!__syncthreads_or(any)) {
      for (int v = tid; v < p.vocab; v += kAccThreads) {
        if (p.suppress && p.suppress[v]) continue;
        const float sc = __fdiv_rn(xt[v], p.temperature) + gumbel(p.seed, slot, step, rej, kTagResidual, v);
        if (sc > best || (sc == best && v < barg)) {
          best = sc;
          barg = v;
        }
      }
    }
    block_argmax(best, barg, s_v, s_a);
    if (tid == 0) {
      s_em[s_state[0]++] = barg;
      s_state[2] = barg == p.eos;
    }
  }
  __syncthreads();
  const int n_em = s_state[0], a = s_state[1];
  for (int j = tid; j < Kp1; j += kAccThreads) p.out_tokens[slot * Kp1 + j] = j < n_em ? s_em[j] : -1;
  if (tid == 0) {
    p.out_count[slot] = n_em;
    const int newL = p.L[slot] + 1 + a;
    p.L[slot] = newL;
    p.anchor[slot] = s_em[n_em - 1];
    const int left = R - n_em;
    p.remaining[slot] = left;
    p.step[slot] = step + 1;
    bool done = s_state[2] || left <= 0;
    if (!done && newL + Kp1 > p.max_ctx) {
      set_error(p.err, WF_DEV_ERR_CAPACITY);
      done = true;
    }
    p.done[slot] = done ? 1 : 0;
  }
}

cudaError_t launch_accept(const AcceptParams &p0, cudaStream_t s, bool pdl) {
  AcceptParams p = p0;
  if (p.K > 8) return cudaErrorInvalidValue;
  void *args[] = {&p};
  return launch_ex(reinterpret_cast<const void *>(accept_kernel), dim3(p.n_seq > 0 ? p.n_seq : 1),
                   dim3(kAccThreads), args, s, pdl);
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

cudaError_t step_kernels_init() {
  static cudaError_t status = cudaErrorNotReady;
  static std::once_flag once;
  std::call_once(once, [] {
    const void *fns[] = {reinterpret_cast<const void *>(embed_kernel), reinterpret_cast<const void *>(layernorm_kernel),
                         reinterpret_cast<const void *>(head_reduce_kernel), reinterpret_cast<const void *>(accept_kernel),
                         reinterpret_cast<const void *>(state_kernel), reinterpret_cast<const void *>(compact_kernel)};
    status = cudaSuccess;
    for (const void *f : fns)
      if (status == cudaSuccess) status = prefer_max_shared(f);
  });
  return status;
}

cudaError_t launch_compact(const int32_t *done, int max_batch, int32_t *active,
                           int32_t *n_active_dev, cudaStream_t s) {
  compact_kernel<<<1, 32, 0, s>>>(done, max_batch, active, n_active_dev);
  return cudaGetLastError();
}

}  // namespace wf
