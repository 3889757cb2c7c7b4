// Decode-time multi-head attention of a few query rows per sequence against a
// per-sequence key/value cache laid out [slot][head][position][64] (bf16).
//
// One kernel serves the three attentions of the step:
//  - mode 0, causal: the target's self-attention over its cache, query row j
//    of a block starting at position L sees positions [0, L+j] (verify block,
//    prompt, plain greedy step; Sec. 3.1 "one causal target pass");
//  - mode 1, block: the drafter's joint softmax over its history memory at
//    positions [0, L) and the 9 block positions [L, L+9), bidirectional inside
//    the block, with RoPE on queries and keys (Sec. 3.2, App. A.2);
//  - mode 2, cross: all encoder frames (cross-attention, Sec. 3.2).
// A CTA takes one (sequence, head, group of <= 16 queries, chunk of 64 keys);
// chunks are aligned to absolute positions and combined by the last CTA of a
// (sequence, head, group) in chunk order with the log-sum-exp rule, so a
// query's result does not depend on how many other rows run with it.
#include "wf_device.cuh"
#include "wf_internal.h"

namespace wf {

constexpr int kCK = kAttnChunk;
constexpr int kQG = kAttnQGroup;
constexpr int kPartStride = 2 + 64;  // m, l, o[64]

__global__ void __launch_bounds__(128) attention_kernel(const AttnParams p) {
  __shared__ float sq[kQG][64];
  __shared__ float sk[kCK][65];
  __shared__ float sv[kCK][64];
  __shared__ float sp[kQG][kCK];
  __shared__ int s_last;

  const int c = blockIdx.x;
  const int h = blockIdx.y % p.n_heads;
  const int qg = blockIdx.y / p.n_heads;
  const int i = blockIdx.z;
  const int tid = threadIdx.x;

  pdl_wait();
  pdl_launch_dependents();

  const int slot = p.seq_slot[i];
  const int base = (p.mode == 2 || !p.pos_base) ? 0 : p.pos_base[slot];
  const int q0 = qg * kQG;
  const int nq = min(kQG, p.rps - q0);
  int n_keys;
  if (p.mode == 2)
    n_keys = p.ctx;
  else if (p.mode == 1)
    n_keys = base + p.rps;
  else
    n_keys = base + q0 + nq;  // keys visible to the last query of the group
  if (n_keys > p.ctx || (p.mode != 2 && base + p.rps > p.ctx)) {
    // the block would pass the cache: record it and leave the output untouched
    if (c == 0 && tid == 0) set_error(p.err, WF_DEV_ERR_CAPACITY);
    return;
  }
  const int n_chunks = (n_keys + kCK - 1) / kCK;
  if (c >= n_chunks) return;

  const int d_model = p.n_heads * 64;
  const size_t cache_off = (static_cast<size_t>(slot) * p.n_heads + h) * p.ctx;

  // ---- queries (pre-scaled by 1/8 = 1/sqrt(64): exact in binary)
  for (int e = tid; e < kQG * 64; e += blockDim.x) {
    const int qi = e >> 6, dd = e & 63;
    float v = 0.f;
    if (qi < nq) {
      const bf16 *qrow = p.q + static_cast<size_t>(i * p.rps + q0 + qi) * d_model + h * 64;
      v = bf2f(qrow[dd]);
      if (p.rope_tab) {
        const int pos = base + q0 + qi;
        const int pr = dd & 31;
        const float2 cs = p.rope_tab[pos * 32 + pr];
        const float other = bf2f(qrow[dd ^ 32]);
        v = dd < 32 ? v * cs.x - other * cs.y : v * cs.x + other * cs.y;
      }
    }
    sq[qi][dd] = v * 0.125f;
  }
  // ---- keys and values of this chunk
  for (int e = tid; e < kCK * 64; e += blockDim.x) {
    const int kk = e >> 6, dd = e & 63;
    const int pos = c * kCK + kk;
    float kv = 0.f, vv = 0.f;
    if (pos < n_keys) {
      const bf16 *krow = p.kc + (cache_off + pos) * 64;
      kv = bf2f(krow[dd]);
      vv = bf2f(p.vc[(cache_off + pos) * 64 + dd]);
      if (p.rope_tab) {
        const int pr = dd & 31;
        const float2 cs = p.rope_tab[pos * 32 + pr];
        const float other = bf2f(krow[dd ^ 32]);
        kv = dd < 32 ? kv * cs.x - other * cs.y : kv * cs.x + other * cs.y;
      }
    }
    sk[kk][dd] = kv;
    sv[kk][dd] = vv;
  }
  __syncthreads();

  // ---- scores: thread -> (query qi = tid/8, keys kg + 8m)
  const int qi = tid >> 3, kg = tid & 7;
  float s[8];
  float mloc = -INFINITY;
#pragma unroll
  for (int m = 0; m < 8; ++m) {
    const int kk = kg + 8 * m;
    const int pos = c * kCK + kk;
    bool vis = qi < nq && pos < n_keys;
    if (p.mode == 0) vis = vis && pos <= base + q0 + qi;
    float acc = -INFINITY;
    if (vis) {
      acc = 0.f;
#pragma unroll 16
      for (int dd = 0; dd < 64; ++dd) acc = fmaf(sq[qi][dd], sk[kk][dd], acc);
    }
    s[m] = acc;
    mloc = fmaxf(mloc, acc);
  }
  mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, 4));
  mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, 2));
  mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, 1));
  float l = 0.f;
#pragma unroll
  for (int m = 0; m < 8; ++m) {
    const float pv = (s[m] == -INFINITY) ? 0.f : expf(s[m] - mloc);
    sp[qi][kg + 8 * m] = pv;
    l += pv;
  }
  l += __shfl_xor_sync(0xffffffffu, l, 4);
  l += __shfl_xor_sync(0xffffffffu, l, 2);
  l += __shfl_xor_sync(0xffffffffu, l, 1);
  __syncthreads();

  // ---- partial output: thread -> (query qi, dims d0..d0+7)
  const int d0 = kg * 8;
  float o[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) o[e] = 0.f;
  if (qi < nq) {
    for (int kk = 0; kk < kCK; ++kk) {
      const float pv = sp[qi][kk];
#pragma unroll
      for (int e = 0; e < 8; ++e) o[e] = fmaf(pv, sv[kk][d0 + e], o[e]);
    }
  }

  const int group_id = (i * p.n_heads + h) * p.qgroups + qg;
  float *part = p.part + (static_cast<size_t>(group_id) * p.n_chunks + c) * kQG * kPartStride;
  if (qi < nq) {
    float *pe = part + qi * kPartStride;
    if (kg == 0) {
      pe[0] = mloc;
      pe[1] = l;
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) pe[2 + d0 + e] = o[e];
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const int prev = atomicAdd(&p.counters[group_id], 1);
    s_last = (prev == n_chunks - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // ---- the last CTA combines the chunks in order
  if (qi < nq) {
    const float *pg = p.part + static_cast<size_t>(group_id) * p.n_chunks * kQG * kPartStride;
    float M = -INFINITY;
    for (int cc = 0; cc < n_chunks; ++cc) M = fmaxf(M, __ldcg(pg + (cc * kQG + qi) * kPartStride));
    float L = 0.f;
    float acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.f;
    for (int cc = 0; cc < n_chunks; ++cc) {
      const float *pe = pg + (cc * kQG + qi) * kPartStride;
      const float mc = __ldcg(pe);
      if (mc == -INFINITY) continue;
      const float w = expf(mc - M);
      L += __ldcg(pe + 1) * w;
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] += __ldcg(pe + 2 + d0 + e) * w;
    }
    const float inv = 1.0f / L;
    bf16 *orow = p.out + static_cast<size_t>(i * p.rps + q0 + qi) * d_model + h * 64 + d0;
#pragma unroll
    for (int e = 0; e < 8; ++e) orow[e] = __float2bfloat16(acc[e] * inv);
  }
  if (tid == 0) p.counters[group_id] = 0;
}

__global__ void rope_table_kernel(float2 *tab, int max_pos, float base) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= max_pos * 32) return;
  const int pos = idx / 32, i = idx % 32;
  // inverse frequency base^(-2i/64) and the phase pos * inv_freq in FP32 (App. A.2)
  const float inv = static_cast<float>(pow(static_cast<double>(base), -2.0 * i / 64.0));
  const float ang = __fmul_rn(static_cast<float>(pos), inv);
  tab[idx] = make_float2(static_cast<float>(cos(static_cast<double>(ang))),
                         static_cast<float>(sin(static_cast<double>(ang))));
}

size_t attn_partial_floats(int n_seq, int rps, int n_heads, int ctx) {
  const int qgroups = (rps + kQG - 1) / kQG;
  const int n_chunks = (ctx + kCK - 1) / kCK;
  return static_cast<size_t>(n_seq) * n_heads * qgroups * n_chunks * kQG * kPartStride;
}

int attn_counter_slots(int n_seq, int rps, int n_heads) {
  return n_seq * n_heads * ((rps + kQG - 1) / kQG);
}

cudaError_t launch_attention(const AttnParams &p0, cudaStream_t s, bool pdl) {
  AttnParams p = p0;
  p.qgroups = (p.rps + kQG - 1) / kQG;
  p.n_chunks = (p.ctx + kCK - 1) / kCK;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_chunks, p.n_heads * p.qgroups, p.n_seq);
  cfg.blockDim = dim3(128, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, attention_kernel, p);
}

cudaError_t launch_rope_table(float2 *tab, int max_pos, float base, cudaStream_t s) {
  const int n = max_pos * 32;
  rope_table_kernel<<<(n + 255) / 256, 256, 0, s>>>(tab, max_pos, base);
  return cudaGetLastError();
}

}  // namespace wf

extern "C" size_t wf_attention_scratch_bytes(int32_t n_seq, int32_t RPS, int32_t n_heads,
                                             int32_t ctx) {
  if (n_seq <= 0 || RPS <= 0 || n_heads <= 0 || ctx <= 0) return 0;
  const size_t counters = static_cast<size_t>(wf::attn_counter_slots(n_seq, RPS, n_heads)) * 4;
  return wf::attn_partial_floats(n_seq, RPS, n_heads, ctx) * sizeof(float) +
         ((counters + 255) / 256) * 256 + static_cast<size_t>(ctx) * 32 * sizeof(float2) + 256;
}

extern "C" wf_status wf_attention(const void *d_q, const void *d_kc, const void *d_vc,
                                  const int32_t *d_slot, const int32_t *d_base, int32_t n_seq,
                                  int32_t RPS, int32_t n_heads, int32_t ctx, int32_t mode,
                                  int32_t rope, float rope_base, void *d_out, void *d_scratch,
                                  size_t scratch_bytes, void *stream) {
  if (!d_q || !d_kc || !d_vc || !d_slot || !d_out || n_seq <= 0 || RPS <= 0 || n_heads <= 0 ||
      ctx <= 0 || mode < 0 || mode > 2)
    return WF_ERR_INVALID;
  if (mode != 2 && !d_base) return WF_ERR_INVALID;
  if (scratch_bytes < wf_attention_scratch_bytes(n_seq, RPS, n_heads, ctx) || !d_scratch)
    return WF_ERR_CAPACITY;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  wf::AttnParams p = {};
  p.q = static_cast<const wf::bf16 *>(d_q);
  p.kc = static_cast<const wf::bf16 *>(d_kc);
  p.vc = static_cast<const wf::bf16 *>(d_vc);
  p.out = static_cast<wf::bf16 *>(d_out);
  p.seq_slot = d_slot;
  p.pos_base = d_base;
  p.n_seq = n_seq;
  p.rps = RPS;
  p.n_heads = n_heads;
  p.ctx = ctx;
  p.mode = mode;
  const size_t pf = wf::attn_partial_floats(n_seq, RPS, n_heads, ctx);
  p.part = static_cast<float *>(d_scratch);
  p.counters = reinterpret_cast<int32_t *>(static_cast<char *>(d_scratch) + pf * sizeof(float));
  float2 *tab = nullptr;
  if (rope) {
    // the RoPE table lives in the scratch tail, after the counters
    const size_t counters = static_cast<size_t>(wf::attn_counter_slots(n_seq, RPS, n_heads)) * 4;
    tab = reinterpret_cast<float2 *>(static_cast<char *>(d_scratch) + pf * sizeof(float) +
                                     ((counters + 255) / 256) * 256);
    if (wf::launch_rope_table(tab, ctx, rope_base, s) != cudaSuccess) return WF_ERR_CUDA;
  }
  p.rope_tab = tab;
  if (cudaMemsetAsync(p.counters, 0, wf::attn_counter_slots(n_seq, RPS, n_heads) * sizeof(int32_t),
                      s) != cudaSuccess)
    return WF_ERR_CUDA;
  return wf::launch_attention(p, s, false) == cudaSuccess ? WF_OK : WF_ERR_CUDA;
}
