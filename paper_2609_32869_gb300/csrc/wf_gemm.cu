// Skinny-M bf16 GEMM on the sm_103a tensor cores (tcgen05 + TMEM + TMA).
//
// Every projection of the decode step is Y = X W^T with few token rows
// (M = 9 per sequence: the anchor and K = 8 proposals, Sec. 3.1) against a
// large weight matrix, so the weights stream from HBM once and set the time.
// The kernel computes a 128 x BT tile of D = W_tile X_tile^T ("swap-AB"): the
// 128 weight rows fill the MMA's M side, the token tile (a multiple of 16,
// <= 128) its N side.  Weight and token tiles stream into shared memory by
// TMA (128-byte swizzle) through an mbarrier ring; one thread issues
// tcgen05.mma into a TMEM accumulator; eight warps read it back with
// tcgen05.ld for a fused epilogue (bias, GELU, residual add, taps, key/value
// cache scatter, or the output-head reduction).
//
// K is split into a fixed number of chunks per (N, K) shape so that ~150 CTAs
// stream weights even for a single sequence.  The S split CTAs of a tile form
// a thread-block cluster; after the MMAs each stages its fp32 partial tile in
// its own shared memory and, past a cluster barrier, reduces a slice of the
// tile by reading the S partials over distributed shared memory in split
// order, so results are deterministic and independent of M, and no partial
// ever travels through global memory.  When the token tiles alone give
// enough CTAs (many sequences), one CTA computes all S splits of its tile in
// turn ("fold"): the MMA thread alternates the splits between two TMEM
// accumulators while four warps add each finished partial, in split order,
// into a third -- the same sums in the same order as the cluster reduction,
// without its S-fold CTAs, barriers and partial tiles.
//
// With programmatic dependent launch the weight tiles of the first pipeline
// stages are requested before griddepcontrol.wait: they do not depend on the
// previous kernel, so their HBM latency overlaps its tail.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <mutex>
#include <map>
#include <tuple>
#include <algorithm>

#include "wf_device.cuh"
#include "wf_internal.h"

namespace wf {

constexpr int kBlockN = 128;   // weight rows per tile (MMA M)
constexpr int kThreads = 256;  // 8 warps: two per TMEM lane quarter
constexpr int kBlockK = 64;    // K per pipeline stage (one 128-byte swizzle atom)
constexpr int kStageA = kBlockN * kBlockK * 2;  // 16 KB
// Shared memory a CTA plans for: two CTAs fit on an SM, so one CTA's
// epilogue overlaps the other's weight stream.
constexpr int kSmemBudget = 110 * 1024;
constexpr int kSmemBudgetAlone = 200 * 1024;  // a CTA that holds all 512 TMEM columns
constexpr int kSmemBudgetLn = 110 * 1024;  // LN mode: resident token tiles + weight ring
constexpr int kMaxBT = 128;                // token rows per tile (MMA N)
constexpr size_t kSmemPerSM = 228 * 1024;  // shared memory of one SM
constexpr int kLnFuseMaxM = 256;              // token rows up to which LN is fused
constexpr int kFoldMinTiles = 64;             // output tiles from which split-K folds into one CTA

__device__ __forceinline__ void head_combine(float &m, float &s, int &arg, float &gm, int &garg,
                                             float m2, float s2, int arg2, float gm2, int garg2) {
  const float M = fmaxf(m, m2);
  float ns = 0.f;
  if (M != -INFINITY) {
    ns = (m == -INFINITY ? 0.f : s * __expf(m - M)) + (m2 == -INFINITY ? 0.f : s2 * __expf(m2 - M));
  }
  if (m2 > m || (m2 == m && arg2 < arg)) arg = arg2;
  m = M;
  s = ns;
  if (gm2 > gm || (gm2 == gm && garg2 < garg)) {
    gm = gm2;
    garg = garg2;
  }
}

// Epilogue of 16 consecutive token columns t0..t0+15 for output feature n.
// acc[] holds the 16 accumulated values; every global load of the chunk (the
// residual) is issued before its stores so the latencies overlap.
template <int EPI>
__device__ __forceinline__ void epi_chunk(const GemmParams &p, int t0, int n, float bn,
                                          const float (&acc)[16], const int2 *tok) {
  if (n >= p.N) return;
  if constexpr (EPI == EPI_F32) {
#pragma unroll
    for (int jj = 0; jj < 16; ++jj)
      if (t0 + jj < p.M) p.out_f32[static_cast<size_t>(t0 + jj) * p.ld_out + n] = acc[jj] + bn;
  } else if constexpr (EPI == EPI_BF16) {
#pragma unroll
    for (int jj = 0; jj < 16; ++jj)
      if (t0 + jj < p.M)
        p.out_bf16[static_cast<size_t>(t0 + jj) * p.ld_out + n] = __float2bfloat16(acc[jj] + bn);
  } else if constexpr (EPI == EPI_GELU) {
#pragma unroll
    for (int jj = 0; jj < 16; ++jj)
      if (t0 + jj < p.M)
        p.out_bf16[static_cast<size_t>(t0 + jj) * p.ld_out + n] =
            __float2bfloat16(gelu_erf(acc[jj] + bn));
  } else if constexpr (EPI == EPI_RESID) {
    float r[16];
#pragma unroll
    for (int jj = 0; jj < 16; ++jj)
      r[jj] = (t0 + jj < p.M) ? p.resid[static_cast<size_t>(t0 + jj) * p.ld_resid + n] : 0.f;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      if (t0 + jj >= p.M) continue;
      const float nr = r[jj] + (acc[jj] + bn);
      p.resid[static_cast<size_t>(t0 + jj) * p.ld_resid + n] = nr;
      if (p.tap0) p.tap0[static_cast<size_t>(t0 + jj) * p.ld_tap + n] = __float2bfloat16(nr);
      if (p.tap1) p.tap1[static_cast<size_t>(t0 + jj) * p.ld_tap + n] = __float2bfloat16(nr);
    }
  } else if constexpr (EPI == EPI_KV) {
    if (n < p.q_cols) {
#pragma unroll
      for (int jj = 0; jj < 16; ++jj)
        if (t0 + jj < p.M)
          p.out_bf16[static_cast<size_t>(t0 + jj) * p.ld_out + n] = __float2bfloat16(acc[jj] + bn);
      return;
    }
    const int c = n - p.q_cols;
    const int which = c / p.d_model;
    const int hd = c - which * p.d_model;
    const int h = hd >> 6, dd = hd & 63;
    bf16 *dst = which == 0 ? p.kc : p.vc;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      if (t0 + jj >= p.M) continue;
      const int2 sp = tok[jj];  // (slot, position) of this token row
      if (sp.y >= p.ctx) {
        set_error(p.err, WF_DEV_ERR_CAPACITY);
        continue;
      }
      dst[((static_cast<size_t>(sp.x) * p.n_heads + h) * p.ctx + sp.y) * 64 + dd] =
          __float2bfloat16(acc[jj] + bn);
    }
  }
}

// Four floats as four bf16 (round to nearest even) in one 8-byte word.
__device__ __forceinline__ uint2 pack4_bf16(const float (&v)[4]) {
  __nv_bfloat162 h[2] = {__floats2bfloat162_rn(v[0], v[1]), __floats2bfloat162_rn(v[2], v[3])};
  return *reinterpret_cast<const uint2 *>(h);
}
// Non-residual epilogues of four features: GELU, then fp32, bf16 or the
// query / key / value split with the cache scatter.
template <int EPI>
__device__ __forceinline__ void epi_quad_out(const GemmParams &p, int t, int n, float (&v)[4],
                                             const int2 *tok_local, float (&fin)[4]) {
  if constexpr (EPI == EPI_GELU) {
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = gelu_erf(v[i]);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) fin[i] = v[i];
  const bool whole = n + 3 < p.N && (p.ld_out & 3) == 0;
  if constexpr (EPI == EPI_F32) {
    float *o = p.out_f32 + static_cast<size_t>(t) * p.ld_out + n;
    if (whole) {
      *reinterpret_cast<float4 *>(o) = make_float4(v[0], v[1], v[2], v[3]);
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (n + i < p.N) o[i] = v[i];
    }
  } else if constexpr (EPI == EPI_BF16 || EPI == EPI_GELU) {
    bf16 *o = p.out_bf16 + static_cast<size_t>(t) * p.ld_out + n;
    if (whole) {
      *reinterpret_cast<uint2 *>(o) = pack4_bf16(v);
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (n + i < p.N) o[i] = __float2bfloat16(v[i]);
    }
  } else if constexpr (EPI == EPI_KV) {
    // N, q_cols and d_model are multiples of 4 (checked at launch)
    if (n >= p.N) return;
    if (n < p.q_cols) {
      *reinterpret_cast<uint2 *>(p.out_bf16 + static_cast<size_t>(t) * p.ld_out + n) = pack4_bf16(v);
      return;
    }
    const int c = n - p.q_cols;
    const int which = c / p.d_model;
    const int hd = c - which * p.d_model;
    const int2 sp = *tok_local;
    if (sp.y >= p.ctx) {
      set_error(p.err, WF_DEV_ERR_CAPACITY);
      return;
    }
    bf16 *dst = which == 0 ? p.kc : p.vc;
    *reinterpret_cast<uint2 *>(
        dst + ((static_cast<size_t>(sp.x) * p.n_heads + (hd >> 6)) * p.ctx + sp.y) * 64 + (hd & 63)) =
        pack4_bf16(v);
  }
}

// Epilogue of four consecutive output features n..n+3 of token row t (the
// staged path).  `old` is the residual row's current value (EPI_RESID).
// fin[] returns the final values (the updated residual for EPI_RESID) for the
// LayerNorm statistics.  Four consecutive features never straddle a head or
// the key/value boundary (multiples of 4), so each store is one vector.
template <int EPI>
__device__ __forceinline__ void epi_quad(const GemmParams &p, int t, int n, const float4 &a,
                                         const float (&b4)[4], const float4 &old,
                                         const int2 *tok_local, float (&fin)[4]) {
  float v[4] = {a.x + b4[0], a.y + b4[1], a.z + b4[2], a.w + b4[3]};
  if constexpr (EPI == EPI_RESID) {
    // N % 128 == 0 and ld_resid % 4 == 0 (checked at launch): one float4
    float4 *r = reinterpret_cast<float4 *>(p.resid + static_cast<size_t>(t) * p.ld_resid + n);
    const float4 nr = make_float4(old.x + v[0], old.y + v[1], old.z + v[2], old.w + v[3]);
    *r = nr;
    fin[0] = nr.x;
    fin[1] = nr.y;
    fin[2] = nr.z;
    fin[3] = nr.w;
    const uint2 h = pack4_bf16(fin);
    if (p.tap0) *reinterpret_cast<uint2 *>(p.tap0 + static_cast<size_t>(t) * p.ld_tap + n) = h;
    if (p.tap1) *reinterpret_cast<uint2 *>(p.tap1 + static_cast<size_t>(t) * p.ld_tap + n) = h;
  } else {
    epi_quad_out<EPI>(p, t, n, v, tok_local, fin);
  }
}

// Build the CTA's token operand for all kps k-steps from the fp32 residual:
// B[i][r][k] = LN(x[t0 + r])[(kit0 + i) * 64 + k] as bf16, stored in the
// 128-byte-swizzled K-major layout the TMA would have produced (16-byte
// chunk j of row r at chunk position j ^ (r % 8)); rows past M are zero.
__device__ __forceinline__ void ln_build_operand(const GemmParams &p, uint8_t *sB, uint32_t stageB,
                                                 float2 *lnst, int t0, int kit0) {
  const int BT = p.BT;
  const int per_stage = BT * 8;
  const int total = p.kps * per_stage;
  constexpr int U = 4;
  float4 xa[U], xb[U];
  uint4 gv[U], bv[U];
  // chunk c -> (k-step i, token row r, 16-byte chunk j of the 64-feature step)
  auto load = [&](int c0) {
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int c = c0 + u * kThreads + static_cast<int>(threadIdx.x);
      xa[u] = xb[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      gv[u] = bv[u] = make_uint4(0u, 0u, 0u, 0u);
      if (c < total) {
        const int i = c / per_stage, rem = c - i * per_stage, r = rem >> 3, j = rem & 7;
        const int t = t0 + r, f = (kit0 + i) * kBlockK + j * 8;
        gv[u] = *reinterpret_cast<const uint4 *>(p.ln_g + f);
        bv[u] = *reinterpret_cast<const uint4 *>(p.ln_b + f);
        if (t < p.M) {
          const float4 *src =
              reinterpret_cast<const float4 *>(p.ln_x + static_cast<size_t>(t) * p.ln_ld + f);
          xa[u] = src[0];
          xb[u] = src[1];
        }
      }
    }
  };
  load(0);  // the first rows are in flight while the statistics merge
  for (int j = threadIdx.x; j < BT; j += blockDim.x) {
    const int t = t0 + j;
    lnst[j] = t < p.M ? merge_tile_stats(p.ln_stats + static_cast<size_t>(t) * p.ln_tiles,
                                         p.ln_tiles, p.ln_eps)
                      : make_float2(0.f, 0.f);
  }
  __syncthreads();
  for (int c0 = 0; c0 < total; c0 += U * kThreads) {
    if (c0) load(c0);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int c = c0 + u * kThreads + static_cast<int>(threadIdx.x);
      if (c >= total) continue;
      const int i = c / per_stage, rem = c - i * per_stage, r = rem >> 3, j = rem & 7;
      uint4 o = make_uint4(0u, 0u, 0u, 0u);
      if (t0 + r < p.M) {
        const float2 ms = lnst[r];
        const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gv[u]);
        const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&bv[u]);
        const float xs[8] = {xa[u].x, xa[u].y, xa[u].z, xa[u].w, xb[u].x, xb[u].y, xb[u].z, xb[u].w};
        __nv_bfloat162 h[4];
#pragma unroll
        for (int q = 0; q < 4; ++q)
          h[q] = __floats2bfloat162_rn(
              ln_apply(xs[2 * q], ms, __low2float(g2[q]), __low2float(b2[q])),
              ln_apply(xs[2 * q + 1], ms, __high2float(g2[q]), __high2float(b2[q])));
        o = *reinterpret_cast<const uint4 *>(h);
      }
      *reinterpret_cast<uint4 *>(sB + static_cast<size_t>(i) * stageB + r * 128 + ((j ^ (r & 7)) << 4)) = o;
    }
  }
}

template <int EPI>
__global__ void __launch_bounds__(kThreads) gemm_tc_kernel(const __grid_constant__ CUtensorMap tmW,
                                                      const __grid_constant__ CUtensorMap tmX,
                                                      const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t *smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int BT = p.BT, stages = p.stages, kps = p.kps;
  const uint32_t stageB = static_cast<uint32_t>(BT) * kBlockK * 2;
  uint8_t *sA = smem;
  uint8_t *sB = smem + static_cast<size_t>(stages) * kStageA;
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + p.pipe_bytes);
  uint64_t *empty = full + stages;
  uint64_t *done = empty + stages;
  uint64_t *part_bar = done + 1;  // fold: split partial r finished in accumulator r % 2
  uint64_t *free_bar = done + 3;  // fold: accumulator r % 2 added into the sum, free again
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 5);
  // per-token (slot, position) for EPI_KV, (slot, step) for sampling heads
  int2 *tok = reinterpret_cast<int2 *>(smem + p.pipe_bytes + (2 * stages + 5) * 8 + 16 + 16);
  float2 *lnst = reinterpret_cast<float2 *>(tok + BT);  // per-token (mean, rstd), LN mode
  const bool ln = p.ln_x != nullptr;
  // a bounded wait of this CTA gave up (in the 32 bytes reserved after the
  // barriers, beside the TMEM address; the kernel has no static shared memory)
  volatile int &s_timed_out = *reinterpret_cast<int *>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tt = blockIdx.x, ntile = blockIdx.y, split = blockIdx.z;
  const bool fold = p.fold != 0;
  const int nk = fold ? kps * p.splits : kps;  // k-steps of this CTA
  const int n0 = ntile * kBlockN, t0 = tt * BT, kit0 = fold ? 0 : split * kps;

  if (threadIdx.x == 0) {
    s_timed_out = 0;
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    mbar_init(&part_bar[0], 1);
    mbar_init(&part_bar[1], 1);
    mbar_init(&free_bar[0], 4);
    mbar_init(&free_bar[1], 4);
    fence_barrier_init();
    fence_proxy_async();
  }
  if (warp == 2) tmem_alloc(tmem_slot, p.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_launch_dependents();

  // Weight tiles of the first stages do not depend on the previous kernel:
  // request them before the dependency wait.  In LN mode each stage carries
  // only its weight tile; the token operand is built once for all k-steps.
  const int npre = nk < stages ? nk : stages;
  const uint32_t tx = ln ? static_cast<uint32_t>(kStageA) : kStageA + stageB;
  if (threadIdx.x == 0) {
    for (int i = 0; i < npre; ++i) {
      mbar_arrive_expect_tx(&full[i], tx);
      tma_load_2d(sA + static_cast<size_t>(i) * kStageA, &tmW, (kit0 + i) * kBlockK, n0, &full[i]);
    }
  }
  if (ln) {
    pdl_wait();  // the residual rows and their statistics come from the previous kernels
    ln_build_operand(p, sB, stageB, lnst, t0, kit0);
    fence_proxy_async();  // generic-proxy writes -> visible to tcgen05.mma
    __syncthreads();
  }

  int issued = npre;  // k-steps whose tiles the producer (thread 0) has requested
  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer
    if (!ln) {
      pdl_wait();  // token rows come from the previous kernel
      for (int i = 0; i < npre; ++i)
        tma_load_2d(sB + static_cast<size_t>(i) * stageB, &tmX, (kit0 + i) * kBlockK, t0, &full[i]);
    }
    for (int it = npre; it < nk; ++it) {
      const int s = it % stages;
      const uint32_t ph = static_cast<uint32_t>((it / stages) - 1) & 1u;
      if (!mbar_wait(&empty[s], ph, p.err, p.spin)) {
        s_timed_out = 1;
        break;
      }
      issued = it + 1;
      mbar_arrive_expect_tx(&full[s], tx);
      tma_load_2d(sA + static_cast<size_t>(s) * kStageA, &tmW, (kit0 + it) * kBlockK, n0, &full[s]);
      if (!ln)
        tma_load_2d(sB + static_cast<size_t>(s) * stageB, &tmX, (kit0 + it) * kBlockK, t0, &full[s]);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    // Descriptors are built once and stepped: a 16-deep K step is 32 bytes,
    // +2 in the descriptor's start-address field (shared address >> 4, 14
    // bits; shared memory is below 256 KB, so the field never carries).  At
    // small N the single issuing thread, not the tensor pipe, sets the MMA
    // rate, so the loop keeps everything but the MMAs out of the way.
    const uint32_t idesc = umma_idesc_bf16(kBlockN, BT);
    const uint64_t a_base = umma_desc_sw128(smem_u32(sA)), b_base = umma_desc_sw128(smem_u32(sB));
    if (!fold && kps <= stages) {
      // every k-step has its own stage and none is refilled: wait for all
      // of them, then issue the MMAs back to back (no per-stage commit)
      bool landed = true;
      for (int it = 0; it < kps && landed; ++it) landed = mbar_wait(&full[it], 0u, p.err, p.spin);
      if (!landed) s_timed_out = 1;
      if (landed) {
        tc_fence_after();
        for (int it = 0; it < kps; ++it) {
          const uint64_t ad = a_base + static_cast<uint64_t>((it * kStageA) >> 4);
          const uint64_t bd = b_base + static_cast<uint64_t>((it * stageB) >> 4);
#pragma unroll
          for (int kk = 0; kk < kBlockK / 16; ++kk)
            umma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (it | kk) != 0 ? 1u : 0u);
        }
      }
    } else {
      for (int it = 0; it < nk; ++it) {
        const int s = it % stages;
        const uint32_t ph = static_cast<uint32_t>(it / stages) & 1u;
        if (!mbar_wait(&full[s], ph, p.err, p.spin)) {
          s_timed_out = 1;
          break;
        }
        // fold: split r = it / kps accumulates in columns (r % 2) acc_cols,
        // once the sum has taken split r - 2 out of them
        const int r = it / kps, kin = it - r * kps;
        if (fold && kin == 0 && r >= 2 &&
            !mbar_wait(&free_bar[r & 1], static_cast<uint32_t>((r >> 1) - 1) & 1u, p.err, p.spin)) {
          s_timed_out = 1;
          break;
        }
        tc_fence_after();
        const uint32_t dacc = tmem + (fold ? static_cast<uint32_t>(r & 1) * p.acc_cols : 0u);
        const uint64_t ad = a_base + static_cast<uint64_t>((s * kStageA) >> 4);
        const uint64_t bd = b_base + static_cast<uint64_t>(((ln ? it : s) * stageB) >> 4);
#pragma unroll
        for (int kk = 0; kk < kBlockK / 16; ++kk)
          umma_bf16(dacc, ad + 2 * kk, bd + 2 * kk, idesc, (kin | kk) != 0 ? 1u : 0u);
        umma_commit(&empty[s]);
        if (fold && kin == kps - 1) umma_commit(&part_bar[r & 1]);
      }
    }
    umma_commit(done);
  }
  __syncwarp();

  // ---------------- fold: warps 4..7 (TMEM lane quarters 0..3) add each split
  // partial into the sum columns 2 acc_cols.., in split order from zero
  if (fold && warp >= 4) {
    const uint32_t lbase = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    const uint32_t sum_col = lbase + 2 * p.acc_cols;
    const int n_ch = BT / 16;
    for (int r = 0; r < p.splits; ++r) {
      if (!mbar_wait(&part_bar[r & 1], static_cast<uint32_t>(r >> 1) & 1u, p.err, p.spin)) {
        s_timed_out = 1;
        break;
      }
      tc_fence_after();
      const uint32_t part_col = lbase + static_cast<uint32_t>(r & 1) * p.acc_cols;
      for (int c = 0; c < n_ch; ++c) {
        float v[16], a[16];
        tmem_ld16(part_col + c * 16, v);
        if (r == 0) {
#pragma unroll
          for (int e = 0; e < 16; ++e) a[e] = 0.f + v[e];
        } else {
          tmem_ld16(sum_col + c * 16, a);
#pragma unroll
          for (int e = 0; e < 16; ++e) a[e] += v[e];
        }
        tmem_st16(sum_col + c * 16, a);
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cta(&free_bar[r & 1]);
    }
  }

  // ---------------- epilogue: warp w owns TMEM lanes [32w, 32w+32) = weight rows
  // (fold: the sum columns; S_eff = 1, the CTA finishes every row of its tile)
  const int S_eff = fold ? 1 : p.splits;
  pdl_wait();
  if constexpr (EPI == EPI_HEAD) {
    if (p.temperature > 0.f) {
      for (int j = threadIdx.x; j < BT; j += blockDim.x) {
        const int t = t0 + j;
        int2 ss = make_int2(0, 0);
        if (t < p.M) {
          const int i = t / p.rows_per_seq;
          ss.x = p.seq_slot[i];
          ss.y = p.step[ss.x];
        }
        tok[j] = ss;
      }
    }
  }
  if constexpr (EPI == EPI_KV) {
    for (int j = threadIdx.x; j < BT; j += blockDim.x) {
      const int t = t0 + j;
      int2 sp = make_int2(0, 0x7fffffff);
      if (t < p.M) {
        const int i = t / p.rows_per_seq, jr = t - i * p.rows_per_seq;
        sp.x = p.seq_slot[i];
        sp.y = (p.pos_base ? p.pos_base[sp.x] : 0) + jr;
      }
      tok[j] = sp;
    }
  }
  // Inputs of the four-feature epilogue that do not depend on this GEMM's
  // result load while the MMAs run: the bias of the lane's four features and,
  // for a residual update, the first row this warp will own.
  const int cols = max(0, min(BT, p.M - t0));
  float b4[4] = {0.f, 0.f, 0.f, 0.f};
  float4 pre = make_float4(0.f, 0.f, 0.f, 0.f);
  bool has_pre = false;
  if (EPI != EPI_HEAD && (S_eff > 1 || p.stats_out)) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int nn = n0 + 4 * lane + i;
      b4[i] = (p.bias && nn < p.N) ? bf2f(p.bias[nn]) : 0.f;
    }
    if constexpr (EPI == EPI_RESID) {
      const int S = S_eff, tl = cols * split / S + warp;
      if (tl < cols * (split + 1) / S) {
        pre = *reinterpret_cast<const float4 *>(p.resid + static_cast<size_t>(t0 + tl) * p.ld_resid +
                                                n0 + 4 * lane);
        has_pre = true;
      }
    }
  }
  __syncthreads();
  const bool ok = mbar_wait(done, 0, p.err, p.spin);
  if (!ok) s_timed_out = 1;
  tc_fence_after();
  __syncwarp();
  // warp w reads TMEM lane quarter w % 4 (weight rows 32 (w % 4) ..) and the
  // token-column chunks [c_lo, c_hi) of its half of the tile
  const int quarter = warp & 3, half = warp >> 2;
  const int n = n0 + quarter * 32 + lane;
  const uint32_t trow =
      tmem + (static_cast<uint32_t>(quarter * 32) << 16) + (fold ? 2 * p.acc_cols : 0u);
  const int n_chunks = BT / 16, c_per = (n_chunks + 1) / 2;
  const int c_lo = half * c_per, c_hi = min(n_chunks, c_lo + c_per);

  if constexpr (EPI == EPI_HEAD) {
    // Stage the [BT][128] logit tile in shared memory (the pipeline buffers
    // are free once the MMAs completed); then a warp owns a token row, lane l
    // folds features 4l..4l+3 in order and the warp combines its lanes:
    // running max with the lowest id on ties, sum of exp(x - max), and the
    // Gumbel-max draw.  One record per (row, vocabulary tile).
    const bool sampling = p.temperature > 0.f;
    const int n_tiles = gridDim.y;
    float *tile = reinterpret_cast<float *>(smem);
    const int r = quarter * 32 + lane;
    for (int c = c_lo; c < c_hi; ++c) {
      float v[16];
      tmem_ld16(trow + c * 16, v);
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) tile[(c * 16 + jj) * kBlockN + r] = v[jj];
    }
    __syncthreads();
    constexpr int W = kThreads / 32;
    for (int tl = warp; tl < cols; tl += W) {
      const int t = t0 + tl;
      const float4 z4 = *reinterpret_cast<const float4 *>(tile + tl * kBlockN + 4 * lane);
      const float z[4] = {z4.x, z4.y, z4.z, z4.w};
      const int2 ss = sampling ? tok[tl] : make_int2(0, 0);
      const int j = t % p.rows_per_seq;
      float m = -INFINITY, sum = 0.f, gm = -INFINITY;
      int arg = 0x7fffffff, garg = 0x7fffffff;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int nn = n0 + 4 * lane + i;
        const bool masked = nn >= p.N || (p.suppress && p.suppress[nn]);
        if (ok && p.logits && nn < p.N) p.logits[static_cast<size_t>(t) * p.N + nn] = z[i];
        const float x = masked ? -INFINITY : (sampling ? __fdiv_rn(z[i], p.temperature) : z[i]);
        float g = -INFINITY;
        if (sampling && !masked)
          g = x + gumbel(p.seed, static_cast<uint32_t>(ss.x), static_cast<uint32_t>(ss.y),
                         static_cast<uint32_t>(j), p.tag, static_cast<uint32_t>(nn));
        head_combine(m, sum, arg, gm, garg, x, masked ? 0.f : 1.f, nn, g, nn);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float m2 = __shfl_down_sync(0xffffffffu, m, off);
        const float s2 = __shfl_down_sync(0xffffffffu, sum, off);
        const float gm2 = __shfl_down_sync(0xffffffffu, gm, off);
        const int a2 = __shfl_down_sync(0xffffffffu, arg, off);
        const int ga2 = __shfl_down_sync(0xffffffffu, garg, off);
        head_combine(m, sum, arg, gm, garg, m2, s2, a2, gm2, ga2);
      }
      if (lane == 0 && ok) {
        HeadRec rec;
        rec.m = m;
        rec.s = sum;
        rec.gm = gm;
        rec.arg = arg;
        rec.garg = garg;
        rec._pad[0] = rec._pad[1] = rec._pad[2] = 0;
        p.recs[static_cast<size_t>(t) * n_tiles + ntile] = rec;
      }
    }
  } else if (S_eff == 1 && !p.stats_out) {
    const float bn = (p.bias && n < p.N) ? bf2f(p.bias[n]) : 0.f;
    for (int c = c_lo; c < c_hi; ++c) {
      float v[16];
      tmem_ld16(trow + c * 16, v);
      if (ok) epi_chunk<EPI>(p, t0 + c * 16, n, bn, v, tok + c * 16);
    }
  } else {
    // Four-feature epilogue: a warp owns a token row (lane l: features
    // 4l..4l+3), so the row's LayerNorm statistics over this 128-feature tile
    // are two warp reductions.  Split-K partials are summed in split order.
    const int S = S_eff;
    const int rank = fold ? 0 : split;  // cluster (1, 1, S) over gridDim.z == S: rank == blockIdx.z
    const int rlo = cols * rank / S, rhi = cols * (rank + 1) / S;
    const int stat_tiles = p.N / kBlockN;
    // the residual row a warp updates next (EPI_RESID; the first one was
    // loaded under the MMAs)
    auto load_old = [&](int tl) {
      float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
      if constexpr (EPI == EPI_RESID) {
        o = (has_pre && tl == rlo + warp)
                ? pre
                : *reinterpret_cast<const float4 *>(p.resid + static_cast<size_t>(t0 + tl) * p.ld_resid +
                                                    n0 + 4 * lane);
      }
      return o;
    };
    auto finish_row = [&](int tl, const float4 &acc, bool valid, const float4 &old) {
      float fin[4] = {0.f, 0.f, 0.f, 0.f};
      if (valid) epi_quad<EPI>(p, t0 + tl, n0 + 4 * lane, acc, b4, old, tok + tl, fin);
      if (p.stats_out) {
        const float mean = warp_sum((fin[0] + fin[1]) + (fin[2] + fin[3])) * (1.0f / 128.f);
        const float d0 = fin[0] - mean, d1 = fin[1] - mean, d2 = fin[2] - mean, d3 = fin[3] - mean;
        const float m2 = warp_sum((d0 * d0 + d1 * d1) + (d2 * d2 + d3 * d3));
        if (lane == 0 && valid)
          p.stats_out[static_cast<size_t>(t0 + tl) * stat_tiles + ntile] = make_float2(mean, m2);
      }
    };
    const int r = quarter * 32 + lane;
    // Every CTA stages its fp32 tile [BT][128] in its own shared memory (the
    // pipeline buffers are free once the MMAs completed); with split-K the S
    // CTAs of the tile form a cluster and each reduces its share of the token
    // rows by reading the S partials over DSMEM.
    float *tile = reinterpret_cast<float *>(smem);
    for (int c = c_lo; c < c_hi; ++c) {
      float v[16];
      tmem_ld16(trow + c * 16, v);
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) tile[(c * 16 + jj) * kBlockN + r] = v[jj];
    }
    if (S > 1) cluster_sync();
    else __syncthreads();
    const uint32_t tile_u32 = smem_u32(tile);
    auto reduce_row = [&](int tl) {
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      const int e = tl * kBlockN + 4 * lane;
      if (S == 1) {
        acc = *reinterpret_cast<const float4 *>(tile + e);
      } else {
#pragma unroll
        for (int sp = 0; sp < 16; ++sp) {
          if (sp < S) {
            const float4 v = dsmem_ld_f32x4(dsmem_map(tile_u32 + 4u * e, sp));
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
          }
        }
      }
      return acc;
    };
    constexpr int W = kThreads / 32;
    if (S > 1 && rhi - rlo <= 2 * W) {
      // at most two rows per warp: read every partial first, tell the peers
      // their tiles are free, then run the epilogue while they finish
      float4 acc[2], old[2];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        if (rlo + warp + W * k < rhi) {
          old[k] = load_old(rlo + warp + W * k);
          acc[k] = reduce_row(rlo + warp + W * k);
        }
      }
      cluster_arrive();
#pragma unroll
      for (int k = 0; k < 2; ++k)
        if (rlo + warp + W * k < rhi) finish_row(rlo + warp + W * k, acc[k], ok, old[k]);
      cluster_wait();
    } else {
      // two rows per warp at a time, so their loads overlap
      for (int tl = rlo + warp; tl < rhi; tl += 2 * W) {
        const int tl2 = tl + W;
        const bool two = tl2 < rhi;
        const float4 old1 = load_old(tl);
        const float4 old2 = two ? load_old(tl2) : make_float4(0.f, 0.f, 0.f, 0.f);
        const float4 acc1 = reduce_row(tl);
        const float4 acc2 = two ? reduce_row(tl2) : make_float4(0.f, 0.f, 0.f, 0.f);
        finish_row(tl, acc1, ok, old1);
        if (two) finish_row(tl2, acc2, ok, old2);
      }
      if (S > 1) cluster_sync();
    }
  }

  // After a timeout, copies this CTA requested may still be landing and
  // MMAs it issued may still be running: wait for both (bounded) before the
  // CTA frees its TMEM and leaves.  Otherwise every copy was consumed by the
  // MMA thread and the MMAs completed before the epilogue read TMEM.
  __syncthreads();
  if (threadIdx.x == 0 && s_timed_out) {
    for (int q = max(0, issued - stages); q < issued; ++q)
      mbar_drain(&full[q % stages], static_cast<uint32_t>(q / stages) & 1u);
    mbar_drain(done, 0u);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) tmem_dealloc(tmem, p.tmem_cols);
}

// --------------------------------------------------------------- host ----
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

const CUtensorMap *tmap_bf16_2d(const void *ptr, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  static std::mutex mu;
  static std::map<std::tuple<uintptr_t, uint64_t, uint64_t, uint32_t>, CUtensorMap *> cache;
  std::lock_guard<std::mutex> lock(mu);
  auto key = std::make_tuple(reinterpret_cast<uintptr_t>(ptr), rows, cols, box_rows);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  auto fn = encode_fn();
  if (!fn) return nullptr;
  if ((reinterpret_cast<uintptr_t>(ptr) & 15) || (cols * 2) % 16 || box_rows == 0 || box_rows > 256)
    return nullptr;
  CUtensorMap *m = new CUtensorMap;
  cuuint64_t gdim[2] = {cols, rows};
  cuuint64_t gstride[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBlockK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), gdim, gstride,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    delete m;
    return nullptr;
  }
  cache.emplace(key, m);
  return m;
}

// 3-D view of a row-major [rows][cols] bf16 matrix as (64 columns, row,
// 64-column block) with strides (cols * 2 bytes, 128 bytes): a box of
// {64, 8, kblocks} is 8 consecutive rows by kblocks * 64 columns, landing in
// shared memory as [kblock][8 rows][128 B] with 128-byte swizzling (one
// swizzle atom per k-block), in a single copy.
bool tmap_bf16_units(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint32_t kblocks) {
  auto fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(ptr) & 15) || cols % 64 || kblocks == 0 || kblocks > 256 ||
      kblocks > cols / 64)
    return false;
  cuuint64_t gdim[3] = {64, rows, cols / 64};
  cuuint64_t gstride[2] = {cols * 2, 128};
  cuuint32_t box[3] = {64, 8, kblocks};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), gdim, gstride, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool tmap_bf16_rows(CUtensorMap *m, const void *ptr, uint32_t rows, uint64_t cols, uint64_t ld, uint32_t kblocks) {
  auto fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(ptr) & 15) || cols % 64 || (ld * 2) % 16 || ld < cols || rows == 0 ||
      rows > 256 || kblocks == 0 || kblocks > 256 || kblocks > cols / 64)
    return false;
  cuuint64_t gdim[3] = {64, rows, cols / 64};
  cuuint64_t gstride[2] = {ld * 2, 128};
  cuuint32_t box[3] = {64, rows, kblocks};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), gdim, gstride, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool tmap_bf16_cache(CUtensorMap *m, const void *ptr, uint64_t ctx, uint64_t outer, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(ptr) & 15) || ctx == 0 || outer == 0 || box_rows == 0 || box_rows > 256 ||
      box_rows > ctx)
    return false;
  cuuint64_t gdim[3] = {64, ctx, outer};
  cuuint64_t gstride[2] = {128, ctx * 128};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), gdim, gstride, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

void gemm_token_tiling(int M, int *BT, int *n_tt) {
  const int nt = (M + kMaxBT - 1) / kMaxBT;
  const int per = (M + nt - 1) / nt;
  *n_tt = nt;
  *BT = ((per + 15) / 16) * 16;
}

int gemm_splits(int N, int K) {
  const int n_tiles = (N + kBlockN - 1) / kBlockN;
  const int k_iters = K / kBlockK;
  int best = 1;
  for (int s = 1; s <= k_iters && s <= 16; ++s) {
    if (k_iters % s) continue;
    if (n_tiles * s > 160) break;
    if (k_iters / s < 2) break;
    best = s;
  }
  return best;
}

template <int EPI>
static cudaError_t cluster_fits(int splits, size_t smem, dim3 grid) {
  static std::mutex mu;
  static std::map<std::pair<int, size_t>, int> seen;
  std::lock_guard<std::mutex> lock(mu);
  auto key = std::make_pair(splits, smem);
  auto it = seen.find(key);
  if (it == seen.end()) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 1;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = splits;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    cudaError_t e = cudaOccupancyMaxActiveClusters(&n, gemm_tc_kernel<EPI>, &cfg);
    if (e != cudaSuccess) return e;
    it = seen.emplace(key, n).first;
  }
  return it->second > 0 ? cudaSuccess : cudaErrorInvalidConfiguration;
}

template <int EPI>
static cudaError_t launch_typed(const CUtensorMap *tw, const CUtensorMap *tx, const GemmParams &p,
                                size_t smem, cudaStream_t s, bool pdl) {
  const bool clustered = p.splits > 1 && !p.fold;
  const dim3 grid(p.n_tt, (p.N + kBlockN - 1) / kBlockN, clustered ? p.splits : 1);
  if (clustered) {
    cudaError_t e = cluster_fits<EPI>(p.splits, smem, grid);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (clustered) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 1;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = p.splits;
    ++na;
  }
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<EPI>, *tw, *tx, p);
}

cudaError_t gemm_init() {
  static cudaError_t status = cudaErrorNotReady;
  static std::once_flag once;
  std::call_once(once, [] {
    const int lim = 227 * 1024;
    status = cudaFuncSetAttribute(gemm_tc_kernel<EPI_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
    if (status == cudaSuccess)
      status = cudaFuncSetAttribute(gemm_tc_kernel<EPI_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
    if (status == cudaSuccess)
      status = cudaFuncSetAttribute(gemm_tc_kernel<EPI_GELU>, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
    if (status == cudaSuccess)
      status = cudaFuncSetAttribute(gemm_tc_kernel<EPI_RESID>, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
    if (status == cudaSuccess)
      status = cudaFuncSetAttribute(gemm_tc_kernel<EPI_KV>, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
    if (status == cudaSuccess)
      status = cudaFuncSetAttribute(gemm_tc_kernel<EPI_HEAD>, cudaFuncAttributeMaxDynamicSharedMemorySize, lim);
    // split-K clusters of up to 16 CTAs
    const void *fns[] = {reinterpret_cast<const void *>(gemm_tc_kernel<EPI_F32>),
                         reinterpret_cast<const void *>(gemm_tc_kernel<EPI_BF16>),
                         reinterpret_cast<const void *>(gemm_tc_kernel<EPI_GELU>),
                         reinterpret_cast<const void *>(gemm_tc_kernel<EPI_RESID>),
                         reinterpret_cast<const void *>(gemm_tc_kernel<EPI_KV>)};
    for (const void *f : fns)
      if (status == cudaSuccess)
        status = cudaFuncSetAttribute(f, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    for (const void *f : fns)
      if (status == cudaSuccess) status = prefer_max_shared(f);
    if (status == cudaSuccess) status = prefer_max_shared(reinterpret_cast<const void *>(gemm_tc_kernel<EPI_HEAD>));
  });
  return status;
}

// Tiling, split and shared-memory plan of one launch; false if it does not fit.
static bool plan_gemm(GemmParams &p, size_t *smem_out) {
  if (p.M <= 0 || p.N <= 0 || p.K <= 0 || p.K % kBlockK) return false;
  gemm_token_tiling(p.M, &p.BT, &p.n_tt);
  if (p.epi == EPI_HEAD) p.splits = 1;
  if (p.splits < 1) p.splits = 1;
  const int k_iters = p.K / kBlockK;
  if (k_iters % p.splits) return false;
  p.kps = k_iters / p.splits;
  const bool ln = p.ln_x != nullptr;
  // fold the splits into one CTA when the token tiles alone fill the GPU
  const int n_tiles = (p.N + kBlockN - 1) / kBlockN;
  p.fold = (!ln && p.epi != EPI_HEAD && p.splits > 1 && p.n_tt * n_tiles >= kFoldMinTiles) ? 1 : 0;
  const size_t stageA = kStageA, stageB = static_cast<size_t>(p.BT) * kBlockK * 2;
  const size_t red = static_cast<size_t>(p.BT) * sizeof(int2) * (ln ? 2 : 1);
  const size_t fixed = red;
  uint32_t cols = 32;
  while (cols < static_cast<uint32_t>(p.BT)) cols <<= 1;
  p.acc_cols = cols;
  if (p.fold) {  // two split accumulators and their sum
    uint32_t all = 32;
    while (all < 3 * cols) all <<= 1;
    if (all > 512) return false;
    cols = all;
  }
  p.tmem_cols = cols;
  // a CTA that holds all of TMEM is alone on its SM: it may take a deeper ring
  const size_t budget = cols == 512 ? kSmemBudgetAlone : kSmemBudget;
  int stages;
  size_t pipe;
  if (ln) {
    // every k-step's token tile stays resident; the weight tiles cycle through a ring
    const size_t btiles = static_cast<size_t>(p.kps) * stageB;
    if (btiles + 2 * stageA + fixed > kSmemBudgetLn) return false;
    stages = static_cast<int>((kSmemBudgetLn - fixed - btiles) / stageA);
    if (stages > p.kps) stages = p.kps;
    if (stages > 16) stages = 16;
    pipe = stages * stageA + btiles;
  } else {
    if (fixed + stageA + stageB > budget) return false;
    stages = static_cast<int>((budget - fixed) / (stageA + stageB));
    const int nk = p.fold ? p.kps * p.splits : p.kps;
    if (stages > nk) stages = nk;
    if (stages > 16) stages = 16;
    pipe = stages * (stageA + stageB);
  }
  p.stages = stages;
  // the staged epilogues reuse the pipeline buffers for a [BT][128] fp32 tile
  if ((p.splits > 1 && !p.fold) || p.stats_out || p.epi == EPI_HEAD)
    pipe = std::max<size_t>(pipe, 512 * static_cast<size_t>(p.BT));
  size_t smem = 1024 + pipe + (2 * stages + 5) * 8 + 32 + 16 + red;
  // A CTA blocks in tcgen05.alloc while co-resident CTAs hold the SM's 512
  // TMEM columns; CTAs of one cluster wait for each other, so no more CTAs
  // may fit on an SM (by shared memory) than can hold TMEM at once.
  const int tmem_ctas = 512 / static_cast<int>(cols);
  if (tmem_ctas < 4)
    smem = std::max<size_t>(smem, kSmemPerSM / (tmem_ctas + 1) + 1);
  if (smem > 227 * 1024) return false;
  p.pipe_bytes = static_cast<int>(pipe);
  *smem_out = smem;
  return true;
}

bool gemm_ln_fits(int M, int N, int K, int epi) {
  // Every weight tile of the projection normalises the same token rows again;
  // past one token tile that repeated work outweighs the launch it saves.
  if (M > kLnFuseMaxM) return false;
  GemmParams p = {};
  p.M = M;
  p.N = N;
  p.K = K;
  p.epi = epi;
  p.splits = gemm_splits(N, K);
  p.ln_x = reinterpret_cast<const float *>(16);  // only tested for non-null
  size_t smem = 0;
  return plan_gemm(p, &smem);
}

cudaError_t launch_gemm(const void *X, const void *W, GemmParams p, cudaStream_t s, bool pdl) {
  const bool ln = p.ln_x != nullptr;
  if (p.spin <= 0) p.spin = kSpinLimitCycles;
  const bool quad = p.splits > 1 || p.stats_out;  // the staged (four-feature) epilogue
  if (p.epi == EPI_HEAD && (ln || p.stats_out)) return cudaErrorInvalidValue;
  if ((p.stats_out || p.epi == EPI_RESID) && p.N % kBlockN) return cudaErrorInvalidValue;
  if (p.epi == EPI_RESID && (p.ld_resid % 4 || (reinterpret_cast<uintptr_t>(p.resid) & 15)))
    return cudaErrorInvalidValue;
  if (quad && p.epi == EPI_KV && (p.N % 4 || p.q_cols % 4 || p.d_model % 4 || p.ld_out % 4))
    return cudaErrorInvalidValue;
  if (quad && p.epi == EPI_RESID && (p.tap0 || p.tap1) && p.ld_tap % 4) return cudaErrorInvalidValue;
  if (ln) {
    const uintptr_t al = reinterpret_cast<uintptr_t>(p.ln_x) | reinterpret_cast<uintptr_t>(p.ln_g) |
                         reinterpret_cast<uintptr_t>(p.ln_b);
    if (!p.ln_stats || !p.ln_g || !p.ln_b || (al & 15) || p.ln_ld % 4 || p.ln_tiles < 1 || p.ln_tiles > kMaxStatTiles ||
        p.K > p.ln_tiles * 128 || p.ln_ld < p.K)
      return cudaErrorInvalidValue;
  } else if (!X) {
    return cudaErrorInvalidValue;
  }
  size_t smem = 0;
  if (!plan_gemm(p, &smem)) return cudaErrorInvalidValue;
  const CUtensorMap *tw = tmap_bf16_2d(W, p.N, p.K, kBlockN);
  const CUtensorMap *tx = ln ? tw : tmap_bf16_2d(X, p.M, p.K, p.BT);
  if (!tw || !tx) return cudaErrorInvalidValue;
  switch (p.epi) {
    case EPI_F32: return launch_typed<EPI_F32>(tw, tx, p, smem, s, pdl);
    case EPI_BF16: return launch_typed<EPI_BF16>(tw, tx, p, smem, s, pdl);
    case EPI_GELU: return launch_typed<EPI_GELU>(tw, tx, p, smem, s, pdl);
    case EPI_RESID: return launch_typed<EPI_RESID>(tw, tx, p, smem, s, pdl);
    case EPI_KV: return launch_typed<EPI_KV>(tw, tx, p, smem, s, pdl);
    case EPI_HEAD: return launch_typed<EPI_HEAD>(tw, tx, p, smem, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace wf

// ------------------------------------------------------- C entry points --
extern "C" size_t wf_gemm_scratch_bytes(int32_t M, int32_t N, int32_t K) {
  // split-K partials are reduced on chip (cluster shared memory): no scratch
  (void)M;
  (void)N;
  (void)K;
  return 0;
}

extern "C" wf_status wf_gemm_bf16(const void *d_x, const void *d_w, const void *d_b, float *d_y,
                                  int32_t M, int32_t N, int32_t K, void *d_scratch,
                                  size_t scratch_bytes, void *stream) {
  (void)d_scratch;
  (void)scratch_bytes;
  if (!d_x || !d_w || !d_y || M <= 0 || N <= 0 || K <= 0) return WF_ERR_INVALID;
  if (K % 64) return WF_ERR_UNSUPPORTED;
  wf::GemmParams p = {};
  p.M = M;
  p.N = N;
  p.K = K;
  p.epi = wf::EPI_F32;
  p.bias = static_cast<const wf::bf16 *>(d_b);
  p.out_f32 = d_y;
  p.ld_out = N;
  p.splits = wf::gemm_splits(N, K);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (wf::gemm_init() != cudaSuccess) return WF_ERR_CUDA;
  return wf::launch_gemm(d_x, d_w, p, s, false) == cudaSuccess ? WF_OK : WF_ERR_CUDA;
}
