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
//
// A CTA takes one (sequence, head, group of <= 16 query rows, block of 256
// keys).  Keys and values arrive as two TMA copies of 32 KB (the caches are
// 3-D tensors (64, position, slot * heads), 128-byte swizzled in shared
// memory; rows past the cache are zero-filled by the copy, value rows past
// the visible keys are zeroed after it); each of the eight
// warps multiplies the 16 query rows against its 32 keys on the tensor cores
// (mma.sync m16n8k16, bf16 in, fp32 accumulate), keeps the row maxima and
// sums in fp32 and forms P V the same way.  Warps combine in order, and the
// blocks of a (sequence, head, group) are combined by the last CTA in block
// order.  Blocks and warps are aligned to absolute key positions and a key a
// query cannot see contributes an exact zero, so a query's result does not
// depend on how many other rows run with it.
#include <map>
#include <mutex>
#include <tuple>

#include "wf_device.cuh"
#include "wf_internal.h"

namespace wf {

constexpr int kKB = kAttnKeysPerCTA;  // 256 keys per CTA
constexpr int kQG = kAttnQGroup;      // 16 query rows per CTA
constexpr int kWarps = 8;             // each takes kKW consecutive keys of the block
constexpr int kThreadsA = 32 * kWarps;
constexpr int kKW = kKB / kWarps;     // 32 keys per warp
constexpr int kNT = kKW / 8;          // 8-key score tiles per warp
constexpr int kKS = kKW / 16;         // 16-key steps per warp
constexpr int kDPT = kQG * 64 / kThreadsA;  // output dims per thread in the combine
constexpr int kPartStride = 2 + 64;   // m, l, o[64]
// Scores are kept in base-2 units (times log2 e): every softmax weight, and
// every weight of the merges of partial results, is one exp2.
constexpr float kLog2e = 1.4426950408889634f;
constexpr int kSmemK = kKB * 128;     // bytes
constexpr int kSmemQ = kQG * 128;
// K, V, Q, then the warps' (m, l); the warps' O partials reuse the K tile.
// The K and V tiles start 1024-aligned (the copies swizzle by address).
constexpr int kSmemAttn = 1024 + 2 * kSmemK + kSmemQ + kWarps * kQG * 2 * 4 + 16;
static_assert(kWarps * kQG * 64 * 4 <= kSmemK, "O partials must fit in the key tile");
static_assert(kQG * 8 <= kThreadsA && kDPT * kThreadsA == kQG * 64, "thread mapping");
// A launch with fewer CTAs than SMs asks for enough shared memory that no two
// of its CTAs share an SM (it runs beside the neighbouring kernels' CTAs
// under programmatic dependent launch); a larger one packs three per SM.
constexpr int kSmemAttnSpread = 116 * 1024;

// kDPT consecutive output dims (scaled by inv) as bf16
__device__ __forceinline__ void store_row(bf16 *orow, const float (&v)[kDPT], float inv) {
  uint32_t w[kDPT / 2];
#pragma unroll
  for (int e = 0; e < kDPT / 2; ++e) w[e] = pack_bf16(v[2 * e] * inv, v[2 * e + 1] * inv);
  if constexpr (kDPT == 8) {
    *reinterpret_cast<uint4 *>(orow) = make_uint4(w[0], w[1], w[2], w[3]);
  } else {
    static_assert(kDPT == 4, "combine width");
    *reinterpret_cast<uint2 *>(orow) = make_uint2(w[0], w[1]);
  }
}
__global__ void __launch_bounds__(kThreadsA) attention_kernel(const __grid_constant__ CUtensorMap tmK,
                                                              const __grid_constant__ CUtensorMap tmV,
                                                              const AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_u32 = smem_u32(smem_raw);
  uint8_t *smem = smem_raw + (((raw_u32 + 1023u) & ~1023u) - raw_u32);
  uint8_t *sK = smem;
  uint8_t *sV = smem + kSmemK;
  uint8_t *sQ = smem + 2 * kSmemK;
  float *sm = reinterpret_cast<float *>(smem + 2 * kSmemK + kSmemQ);  // [kWarps][16]
  float *sl = sm + kWarps * kQG;                                     // [kWarps][16]
  // [kWarps][16][64]: the warps' O, in the key tile once every warp is done
  // with it (in the value tile for a looping CTA, whose next keys are by
  // then streaming into the key tile)
  float *so = reinterpret_cast<float *>(p.loop ? sV : sK);
  __shared__ int s_last;
  __shared__ uint64_t s_bar[2];  // [0] keys, [1] values

  const int blk = blockIdx.x;
  const int h = blockIdx.y % p.n_heads;
  const int qg = blockIdx.y / p.n_heads;
  const int i = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // Before griddepcontrol.wait only data the previous kernel cannot be
  // writing is touched: the active list and cache lengths change only between
  // steps (the kernels that precede an attention launch in a call all wait
  // for their predecessors before allowing it to start), the acoustic memory
  // only at prefill, and self-attention cache rows below L only in earlier
  // steps.  Those rows stream in while the producer of this layer's queries
  // (and of rows L..L+rps-1) finishes.

  const int slot = __ldcg(p.seq_slot + i);
  const int base = (p.mode == 2 || !p.pos_base) ? 0 : __ldcg(p.pos_base + slot);
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
    if (blk == 0 && tid == 0) set_error(p.err, WF_DEV_ERR_CAPACITY);
    return;
  }
  const int n_blocks = (n_keys + kKB - 1) / kKB;
  // In a cluster launch every CTA of a multi-block group takes part in the
  // merge; a block past the keys computes over masked keys only and yields
  // the exact empty partial (m = -inf, l = 0, o = 0).
  if (!p.loop && blk >= n_blocks && !(p.cluster && n_blocks > 1)) return;

  const int d_model = p.n_heads * 64;
  // the key blocks this CTA computes: its own, or (loop) all of its group's
  // in order, each leaving its partial as a CTA of its own would
  const int b_first = p.loop ? 0 : blk, b_end = p.loop ? n_blocks : blk + 1;
  const int group_id = (i * p.n_heads + h) * p.qgroups + qg;

  // ---- keys and values: one TMA copy each.  A block holding rows that this
  // step's projection writes (positions from `fresh` on) loads after the
  // wait; a block of settled rows streams in while the producer of the
  // queries finishes.  A looping CTA requests each later block once the
  // previous one is done with the tiles.
  const int fresh = p.mode == 2 ? n_keys : base;
  const int cache_row = slot * p.n_heads + h;
  const uint32_t tile_bytes = static_cast<uint32_t>(min(kKB, p.ctx)) * 128u;  // the maps' box
  auto issue_k = [&](int b) {
    mbar_arrive_expect_tx(&s_bar[0], tile_bytes);
    tma_load_3d(sK, &tmK, 0, b * kKB, cache_row, &s_bar[0]);
  };
  auto issue_v = [&](int b) {
    mbar_arrive_expect_tx(&s_bar[1], tile_bytes);
    tma_load_3d(sV, &tmV, 0, b * kKB, cache_row, &s_bar[1]);
  };
  auto issue = [&](int b) {
    issue_k(b);
    issue_v(b);
  };
  const bool first_keys = b_first * kKB < n_keys;
  const bool first_fresh = first_keys && fresh < n_keys && b_first * kKB + kKB > fresh;
  if (tid == 0) {
    mbar_init(&s_bar[0], 1);
    mbar_init(&s_bar[1], 1);
    fence_barrier_init();
    if (first_keys && !first_fresh) {
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      issue(b_first);
    }
  }
  pdl_wait();
  pdl_launch_dependents();
  if (tid == 0 && first_fresh) issue(b_first);
  const long long spin = p.spin > 0 ? p.spin : kSpinLimitCycles;
  // ---- queries, pre-scaled by 1/8 = 1/sqrt(64) (exact in binary), RoPE in fp32
  if (tid < kQG * 8) {
    const int r = tid >> 3, ch = tid & 7;
    uint4 raw = make_uint4(0, 0, 0, 0), par = make_uint4(0, 0, 0, 0);
    if (r < nq) {
      const bf16 *qrow = p.q + static_cast<size_t>(i * p.rps + q0 + r) * d_model + h * 64;
      raw = *reinterpret_cast<const uint4 *>(qrow + ch * 8);
      if (p.rope_tab) par = *reinterpret_cast<const uint4 *>(qrow + ((ch * 8) ^ 32));
    }
    const bf16 *qv = reinterpret_cast<const bf16 *>(&raw);
    const bf16 *qp = reinterpret_cast<const bf16 *>(&par);
    float f[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      float v = bf2f(qv[e]);
      if (p.rope_tab && r < nq) {
        const int dd = ch * 8 + e;
        const float2 cs = __ldg(p.rope_tab + (base + q0 + r) * 32 + (dd & 31));
        const float other = bf2f(qp[e]);
        v = dd < 32 ? v * cs.x - other * cs.y : v * cs.x + other * cs.y;
      }
      f[e] = v * 0.125f;
    }
    uint4 o;
    o.x = pack_bf16(f[0], f[1]);
    o.y = pack_bf16(f[2], f[3]);
    o.z = pack_bf16(f[4], f[5]);
    o.w = pack_bf16(f[6], f[7]);
    *reinterpret_cast<uint4 *>(sQ + swz(r, ch)) = o;
  }
  // thread -> (row qi, dims d0..d0+kDPT-1) in the combines
  const int qi = tid / (64 / kDPT), d0 = (tid % (64 / kDPT)) * kDPT;
  for (int bi = b_first; bi < b_end; ++bi) {
  const int key0 = bi * kKB;
  const bool any_keys = key0 < n_keys;
  const uint32_t ph = static_cast<uint32_t>((bi - b_first) & 1);  // the tiles' copy of this block
  if (bi > b_first && tid == 0) {  // this block's keys were requested under the previous block's P V
    fence_proxy_async();  // the previous block's generic writes to the value tile come before the copy
    issue_v(bi);
  }
  // keys first; the values keep streaming while the scores are formed.  After
  // a timeout thread 0 waits (bounded) for both copies before going on, so
  // no copy lands in a CTA that has exited.
  __syncthreads();
  if (any_keys && !mbar_wait(&s_bar[0], ph, p.err, spin) && tid == 0) {
    mbar_drain(&s_bar[0], ph);
    mbar_drain(&s_bar[1], ph);
  }

  // ---- RoPE on the keys (drafter): dims i and i+32 rotate by pos * base^(-2i/64)
  if (p.rope_tab) {
    for (int idx = tid; idx < kKB * 4; idx += kThreadsA) {
      const int kr = idx >> 2, c = idx & 3;  // chunk c (dims 8c..8c+7) pairs with chunk c+4
      const int pos = key0 + kr;
      if (pos >= n_keys) continue;
      uint4 *lo = reinterpret_cast<uint4 *>(sK + swz(kr, c));
      uint4 *hi = reinterpret_cast<uint4 *>(sK + swz(kr, c + 4));
      uint4 a = *lo, b = *hi;
      bf16 *av = reinterpret_cast<bf16 *>(&a);
      bf16 *bv = reinterpret_cast<bf16 *>(&b);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float2 cs = __ldg(p.rope_tab + pos * 32 + c * 8 + e);
        const float x1 = bf2f(av[e]), x2 = bf2f(bv[e]);
        av[e] = __float2bfloat16(x1 * cs.x - x2 * cs.y);
        bv[e] = __float2bfloat16(x2 * cs.x + x1 * cs.y);
      }
      *lo = a;
      *hi = b;
    }
    __syncthreads();
  }

  // ---- per warp: 16 query rows x kKW keys on the tensor cores
  const int g = lane >> 2, c4 = lane & 3;
  const int kw = warp * kKW;  // first key of this warp within the block
  const uint32_t q_u32 = smem_u32(sQ), k_u32 = smem_u32(sK), v_u32 = smem_u32(sV);
  float s[kNT][4];
#pragma unroll
  for (int nt = 0; nt < kNT; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
  for (int ks = 0; ks < 4; ++ks) {
    uint32_t a0, a1, a2, a3;
    {
      const int mi = lane >> 3;
      ldsm_x4(q_u32 + swz((mi & 1) * 8 + (lane & 7), 2 * ks + (mi >> 1)), a0, a1, a2, a3);
    }
#pragma unroll
    for (int np = 0; np < kKS; ++np) {
      uint32_t b0, b1, b2, b3;
      const int mi = lane >> 3;
      ldsm_x4(k_u32 + swz(kw + np * 16 + (mi >> 1) * 8 + (lane & 7), 2 * ks + (mi & 1)), b0, b1, b2,
              b3);
      mma_bf16(s[2 * np], a0, a1, a2, a3, b0, b1);
      mma_bf16(s[2 * np + 1], a0, a1, a2, a3, b2, b3);
    }
  }
  // masks, row maxima and exponentials (rows g and g+8 of the group)
  float mrow[2] = {-INFINITY, -INFINITY};
#pragma unroll
  for (int nt = 0; nt < kNT; ++nt) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int row = g + (e >> 1) * 8;
      const int pos = key0 + kw + nt * 8 + c4 * 2 + (e & 1);
      bool vis = row < nq && pos < n_keys;
      if (p.mode == 0) vis = vis && pos <= base + q0 + row;
      s[nt][e] = vis ? s[nt][e] * kLog2e : -INFINITY;  // base-2 logits
      mrow[e >> 1] = fmaxf(mrow[e >> 1], s[nt][e]);
    }
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    mrow[r] = fmaxf(mrow[r], __shfl_xor_sync(0xffffffffu, mrow[r], 1));
    mrow[r] = fmaxf(mrow[r], __shfl_xor_sync(0xffffffffu, mrow[r], 2));
  }
  float lrow[2] = {0.f, 0.f};
#pragma unroll
  for (int nt = 0; nt < kNT; ++nt) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float v = s[nt][e] == -INFINITY ? 0.f : exp2f(s[nt][e] - mrow[e >> 1]);
      s[nt][e] = v;
      lrow[e >> 1] += v;
    }
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
  // the values; rows past the visible keys (stale cache rows, rows past the
  // copy, or a block with no visible key at all) become zeros, so P V adds
  // exact zeros there
  if (any_keys && !mbar_wait(&s_bar[1], ph, p.err, spin) && tid == 0) mbar_drain(&s_bar[1], ph);
  {
    const int z0 = min(max(n_keys - key0, 0), kKB);
    for (int idx = tid; idx < (kKB - z0) * 8; idx += kThreadsA)
      *reinterpret_cast<uint4 *>(sV + swz(z0 + (idx >> 3), idx & 7)) = make_uint4(0u, 0u, 0u, 0u);
  }
  __syncthreads();
  // every warp is done with the keys: a looping CTA requests the next block's
  if (p.loop && bi + 1 < b_end && tid == 0) {
    fence_proxy_async();  // generic writes to the key tile (RoPE) come before the copy
    issue_k(bi + 1);
  }
  // O = P V (P rounded to bf16 as the A operand)
  float o[8][4];
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
#pragma unroll
  for (int kk = 0; kk < kKS; ++kk) {
    const uint32_t a0 = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
    const uint32_t a1 = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
    const uint32_t a2 = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
    const uint32_t a3 = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
    for (int dp = 0; dp < 4; ++dp) {
      uint32_t b0, b1, b2, b3;
      const int mi = lane >> 3;
      ldsm_x4_t(v_u32 + swz(kw + kk * 16 + (mi & 1) * 8 + (lane & 7), 2 * dp + (mi >> 1)), b0, b1,
                b2, b3);
      mma_bf16(o[2 * dp], a0, a1, a2, a3, b0, b1);
      mma_bf16(o[2 * dp + 1], a0, a1, a2, a3, b2, b3);
    }
  }
  __syncthreads();  // every warp is done with the tile that now holds O
  // stage this warp's (m, l, O) for the in-order combine
  if (c4 == 0) {
    sm[warp * kQG + g] = mrow[0];
    sm[warp * kQG + g + 8] = mrow[1];
    sl[warp * kQG + g] = lrow[0];
    sl[warp * kQG + g + 8] = lrow[1];
  }
  // O rows of 64 floats, 8-float column groups XOR-swizzled by the row's
  // low two bits: a half-warp's fragment stores fall in distinct banks
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) {
    const int col = (nd ^ (g & 3)) * 8 + c4 * 2;
    *reinterpret_cast<float2 *>(so + (warp * kQG + g) * 64 + col) = make_float2(o[nd][0], o[nd][1]);
    *reinterpret_cast<float2 *>(so + (warp * kQG + g + 8) * 64 + col) = make_float2(o[nd][2], o[nd][3]);
  }
  __syncthreads();

  // ---- combine the warps in order
  float M = -INFINITY;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sm[w * kQG + qi]);
  float L = 0.f, acc[kDPT];
#pragma unroll
  for (int e = 0; e < kDPT; ++e) acc[e] = 0.f;
  static_assert(kDPT == 4, "one float4 of O per warp and thread");
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    const float mw = sm[w * kQG + qi];
    const float wt = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
    L += sl[w * kQG + qi] * wt;
    // dims d0..d0+3 stay contiguous under the swizzle (it flips bits 3 and 4)
    const float4 o4 = *reinterpret_cast<const float4 *>(so + (w * kQG + qi) * 64 + (d0 ^ ((qi & 3) << 3)));
    acc[0] += o4.x * wt;
    acc[1] += o4.y * wt;
    acc[2] += o4.z * wt;
    acc[3] += o4.w * wt;
  }

  if (n_blocks == 1) {
    if (qi < nq) {
      const float inv = 1.0f / L;
      bf16 *orow = p.out + static_cast<size_t>(i * p.rps + q0 + qi) * d_model + h * 64 + d0;
      store_row(orow, acc, inv);
    }
    return;
  }

  if (p.cluster) {
    // ---- several key blocks in one cluster: each CTA leaves its partial in
    // its shared memory ([16][68]: m, l, -, -, o[64]); CTA 0 combines them in
    // block order over DSMEM with the same arithmetic as the global path.
    float *pb = reinterpret_cast<float *>(sV);
    if (d0 == 0) {
      pb[qi * 68] = M;
      pb[qi * 68 + 1] = L;
    }
#pragma unroll
    for (int e = 0; e < kDPT; ++e) pb[qi * 68 + 4 + d0 + e] = acc[e];
    cluster_sync();
    float MM = -INFINITY, LL = 0.f, oo[kDPT];
    if (blk == 0) {
      // every peer's (m, l, o) load in flight at once (at most 8 blocks), then
      // merged in block order; an absent block adds exact zeros
      const uint32_t pb_u32 = smem_u32(pb);
      float mc[8], lc[8];
      float4 o4[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        mc[u] = -INFINITY;
        lc[u] = 0.f;
        o4[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (u < p.n_chunks) {
          mc[u] = dsmem_ld_f32(dsmem_map(pb_u32 + 4u * (qi * 68), u));
          lc[u] = dsmem_ld_f32(dsmem_map(pb_u32 + 4u * (qi * 68 + 1), u));
          o4[u] = dsmem_ld_f32x4(dsmem_map(pb_u32 + 4u * (qi * 68 + 4 + d0), u));
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) MM = fmaxf(MM, mc[u]);
#pragma unroll
      for (int e = 0; e < kDPT; ++e) oo[e] = 0.f;
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float ov[4] = {o4[u].x, o4[u].y, o4[u].z, o4[u].w};
        const float wt = (mc[u] == -INFINITY) ? 0.f : exp2f(mc[u] - MM);
        LL = __fmaf_rn(lc[u], wt, LL);
#pragma unroll
        for (int e = 0; e < kDPT; ++e) oo[e] = __fmaf_rn(ov[e], wt, oo[e]);
      }
    }
    cluster_arrive();  // CTA 0 has read every partial; peers may exit
    cluster_wait();
    if (blk == 0 && qi < nq) {
      bf16 *orow = p.out + static_cast<size_t>(i * p.rps + q0 + qi) * d_model + h * 64 + d0;
      store_row(orow, oo, 1.0f / LL);
    }
    return;
  }

  // ---- several key blocks: partials to global, the last CTA combines in order
  float *part = p.part + (static_cast<size_t>(group_id) * p.n_chunks + bi) * kQG * kPartStride;
  if (qi < nq) {
    float *pe = part + qi * kPartStride;
    if (d0 == 0) {
      pe[0] = M;
      pe[1] = L;
    }
#pragma unroll
    for (int e = 0; e < kDPT; ++e) pe[2 + d0 + e] = acc[e];
  }
  // one fence per CTA: after the barrier thread 0 releases the whole CTA's
  // partial at GPU scope and counts it; the last CTA's thread 0 fences again
  // (acquire) before the barrier that releases its threads into the combine.
  // A looping CTA goes on to its next block once every thread is done with
  // this one (its partials are then visible to all its threads).
  __syncthreads();
  if (p.loop) continue;
  if (tid == 0) {
    __threadfence();
    const int last = atomicAdd(&p.counters[group_id], 1) == n_blocks - 1;
    if (last) __threadfence();
    s_last = last;
  }
  __syncthreads();
  if (!s_last) return;
  }  // key blocks
  // A block the query cannot see carries m = -inf, l = 0, o = 0 and gets
  // weight 0, so it adds exact zeros; the loads of all blocks are independent.
  if (qi < nq) {
    const float *pg = p.part + static_cast<size_t>(group_id) * p.n_chunks * kQG * kPartStride;
    // blocks in groups of 8 with every load of a group in flight, merged in
    // block order; a block past n_blocks adds exact zeros
    float MM = -INFINITY;
    for (int u0 = 0; u0 < n_blocks; u0 += 8) {
      float mc[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        mc[u] = u0 + u < n_blocks ? __ldcg(pg + ((u0 + u) * kQG + qi) * kPartStride) : -INFINITY;
#pragma unroll
      for (int u = 0; u < 8; ++u) MM = fmaxf(MM, mc[u]);
    }
    float LL = 0.f, oo[kDPT];
#pragma unroll
    for (int e = 0; e < kDPT; ++e) oo[e] = 0.f;
    for (int u0 = 0; u0 < n_blocks; u0 += 8) {
      float mc[8], lc[8], ov[8][kDPT];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        mc[u] = -INFINITY;
        lc[u] = 0.f;
#pragma unroll
        for (int e = 0; e < kDPT; ++e) ov[u][e] = 0.f;
        if (u0 + u < n_blocks) {
          const float *pe = pg + ((u0 + u) * kQG + qi) * kPartStride;
          mc[u] = __ldcg(pe);
          lc[u] = __ldcg(pe + 1);
#pragma unroll
          for (int e = 0; e < kDPT; ++e) ov[u][e] = __ldcg(pe + 2 + d0 + e);
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float wt = (mc[u] == -INFINITY) ? 0.f : exp2f(mc[u] - MM);
        LL = __fmaf_rn(lc[u], wt, LL);
#pragma unroll
        for (int e = 0; e < kDPT; ++e) oo[e] = __fmaf_rn(ov[u][e], wt, oo[e]);
      }
    }
    const float inv = 1.0f / LL;
    bf16 *orow = p.out + static_cast<size_t>(i * p.rps + q0 + qi) * d_model + h * 64 + d0;
    store_row(orow, oo, inv);
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
  const int n_blocks = (ctx + kKB - 1) / kKB;
  return static_cast<size_t>(n_seq) * n_heads * qgroups * n_blocks * kQG * kPartStride;
}

int attn_counter_slots(int n_seq, int rps, int n_heads) {
  return n_seq * n_heads * ((rps + kQG - 1) / kQG);
}

// Tensor maps of the caches, encoded once per (cache, ctx, outer): 3-D
// (64 dims, ctx positions, outer = slot * heads + head) with a box of one
// (slot, head)'s 256 positions, 128-byte swizzled; positions past ctx read
// as zeros.
static const CUtensorMap *attn_tmap(const void *cache, int ctx, int outer) {
  static std::mutex mu;
  static std::map<std::tuple<uintptr_t, int, int>, CUtensorMap *> maps;
  std::lock_guard<std::mutex> lock(mu);
  const auto key = std::make_tuple(reinterpret_cast<uintptr_t>(cache), ctx, outer);
  auto it = maps.find(key);
  if (it != maps.end()) return it->second;
  CUtensorMap *m = new CUtensorMap;
  if (!tmap_bf16_cache(m, cache, static_cast<uint64_t>(ctx), static_cast<uint64_t>(outer),
                       static_cast<uint32_t>(ctx < kKB ? ctx : kKB))) {
    delete m;
    return nullptr;
  }
  maps.emplace(key, m);
  return m;
}

cudaError_t attention_init() {
  static cudaError_t status = cudaErrorNotReady;
  static std::once_flag once;
  std::call_once(once, [] {
    status = cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  kSmemAttnSpread);
    if (status == cudaSuccess) status = prefer_max_shared(reinterpret_cast<const void *>(attention_kernel));
  });
  return status;
}

cudaError_t launch_attention(const AttnParams &p0, cudaStream_t s, bool pdl) {
  AttnParams p = p0;
  p.qgroups = (p.rps + kQG - 1) / kQG;
  p.n_chunks = (p.ctx + kKB - 1) / kKB;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.n_chunks, p.n_heads * p.qgroups, p.n_seq);
  cfg.blockDim = dim3(kThreadsA, 1, 1);
  static const int n_sm = [] {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return 0;
    return n;
  }();
  long long ctas = static_cast<long long>(cfg.gridDim.x) * cfg.gridDim.y * cfg.gridDim.z;
  // small launches merge their blocks over DSMEM (no global round trip);
  // large ones keep the global partials, where cluster placement costs more
  // than it saves.  With at least two (sequence, head, query group)s per SM
  // one CTA per group walks its key blocks in order, leaving the same
  // partials and merging them itself: a single wave of CTAs streams every
  // key, with no counter and no second wave.  All three paths do the same
  // arithmetic in the same order.
  p.cluster = (p.n_chunks > 1 && p.n_chunks <= 8 && ctas <= n_sm) ? 1 : 0;
  const long long groups = static_cast<long long>(cfg.gridDim.y) * cfg.gridDim.z;
  p.loop = (!p.cluster && p.n_chunks > 1 && n_sm > 0 && groups >= 2LL * n_sm) ? 1 : 0;
  if (p.loop) {
    cfg.gridDim.x = 1;
    ctas = groups;
  }
  cfg.dynamicSmemBytes = ctas <= n_sm ? kSmemAttnSpread : kSmemAttn;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (p.cluster) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = p.n_chunks;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  if (p.outer < 1) return cudaErrorInvalidValue;
  const CUtensorMap *tk = attn_tmap(p.kc, p.ctx, p.outer), *tv = attn_tmap(p.vc, p.ctx, p.outer);
  if (!tk || !tv) return cudaErrorInvalidValue;
  return cudaLaunchKernelEx(&cfg, attention_kernel, *tk, *tv, p);
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
  if (wf::attention_init() != cudaSuccess) return WF_ERR_CUDA;
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
  p.outer = wf::kAttnOuterBound;
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

// ---------------------------------------------------------------------------
// wf_attention_noalloc: the same attention for callers that cannot allocate
// device memory.
//
// Some callers have no way to obtain scratch: code that runs while a CUDA
// graph is being captured in a mode that forbids cudaMalloc, plugins hosted
// by a framework that owns every device allocation, and latency-critical
// loops where an allocation (which can synchronise the device) is not
// acceptable.  For them the partial sums and counters live in one file-scope
// device array of kNoAllocScratchBytes, which every GPU that loads this
// library holds until the process exits.  The first call on a device looks
// the array's device address up (cudaGetSymbolAddress), which can load the
// library's module; make that first call before any stream capture.  All
// calls share the array: calls that can overlap on the GPU (different
// streams, or without ordering between them) race on it and must not be
// issued.  The counters are cleared on every call; the partial sums need no
// clearing.
namespace {
constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;  // 8 MiB
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];
constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mu;
void *g_noalloc_ptr[kNoAllocMaxDevices] = {};
}  // namespace

extern "C" wf_status wf_attention_noalloc(const void *d_q, const void *d_kc, const void *d_vc,
                                          const int32_t *d_slot, const int32_t *d_base,
                                          int32_t n_seq, int32_t RPS, int32_t n_heads,
                                          int32_t ctx, int32_t mode, int32_t rope,
                                          float rope_base, void *d_out, void *stream) {
  if (!d_q || !d_kc || !d_vc || !d_slot || !d_out || n_seq <= 0 || RPS <= 0 || n_heads <= 0 ||
      ctx <= 0 || mode < 0 || mode > 2)
    return WF_ERR_INVALID;
  if (mode != 2 && !d_base) return WF_ERR_INVALID;
  const size_t need = wf_attention_scratch_bytes(n_seq, RPS, n_heads, ctx);
  if (need > kNoAllocScratchBytes) return WF_ERR_CAPACITY;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return WF_ERR_CUDA;
  if (dev < 0 || dev >= kNoAllocMaxDevices) return WF_ERR_UNSUPPORTED;
  void *scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
      void *ptr = nullptr;
      if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return WF_ERR_CUDA;
      g_noalloc_ptr[dev] = ptr;
    }
    scratch = g_noalloc_ptr[dev];
  }
  if (wf::attention_init() != cudaSuccess) return WF_ERR_CUDA;
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
  p.outer = wf::kAttnOuterBound;
  const size_t pf = wf::attn_partial_floats(n_seq, RPS, n_heads, ctx);
  const size_t counters = static_cast<size_t>(wf::attn_counter_slots(n_seq, RPS, n_heads)) * 4;
  p.part = static_cast<float *>(scratch);
  p.counters = reinterpret_cast<int32_t *>(static_cast<char *>(scratch) + pf * sizeof(float));
  float2 *tab = nullptr;
  if (rope) {
    tab = reinterpret_cast<float2 *>(static_cast<char *>(scratch) + pf * sizeof(float) +
                                     ((counters + 255) / 256) * 256);
    if (wf::launch_rope_table(tab, ctx, rope_base, s) != cudaSuccess) return WF_ERR_CUDA;
  }
  p.rope_tab = tab;
  if (cudaMemsetAsync(p.counters, 0, counters, s) != cudaSuccess) return WF_ERR_CUDA;
  return wf::launch_attention(p, s, false) == cudaSuccess ? WF_OK : WF_ERR_CUDA;
}
