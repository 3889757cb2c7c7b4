// Projections of a batch of up to 16 sequences (Sec. 3.1: one verify block of
// 9 rows per sequence, up to 146 operand rows with a folded LayerNorm's two
// extra rows) on the skinny kernels' scheme, for M too large to hold the
// whole token operand of a CTA's K range beside its weights.  Opt-in per
// handle (WF_OPT_SKINNY): the tcgen05 GEMM is the default for such batches.
//
// Each CTA owns U units of 8 weight rows over a K range (all of K, or 1/S of
// it in a cluster of S CTAs) and requests its whole weight slab with TMA
// before griddepcontrol.wait, as the single-sequence kernel does.  The token
// operand streams through a ring of ns k-blocks ([M rows][64] bf16, one TMA
// copy each, 128-byte swizzled).  The 8 warps form a grid of WU unit groups
// by WT tile groups: warp (wu, wt) multiplies the 16-row token tiles wt,
// wt + WT, ... by the units of group wu over the CTA's K range, so no sums
// cross warps (mma.sync m16n8k16, tokens as the 16-row A operand, a unit's 8
// weight rows as B).  Results go to shared memory; with S > 1 the rank that
// finishes a row adds the S ranks' sums in rank order over distributed shared
// memory.  The partial row sums of a folded LayerNorm and the residual rows
// an EPI_RESID update reads are copied in (cp.async) while the MMAs run.  A
// row's arithmetic is a fixed function of the plan, which the caller fixes
// per handle, so it does not depend on how many rows run with it.  Operands,
// folded LayerNorm and epilogues are those of the single-sequence kernel
// (wf_skinny.cu).
#include <cstdio>
#include <cstdlib>
#include <map>
#include <mutex>
#include <tuple>

#include "wf_device.cuh"
#include "wf_internal.h"
#include "wf_skinny_mt_layout.h"

namespace wf {

namespace {

constexpr int kMtQuadsPerPass = 2;  // epilogue column quads a thread finishes per pass

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void st_bf16x4(bf16 *dst, float a, float b, float c, float d) {
  uint2 v;
  v.x = pack_bf16(a, b);
  v.y = pack_bf16(c, d);
  *reinterpret_cast<uint2 *>(dst) = v;
}

}  // namespace

template <int U>
__global__ void __launch_bounds__(kMtThreads, 2) skinny_mt_kernel(const __grid_constant__ CUtensorMap tmW,
                                                                  const __grid_constant__ CUtensorMap tmX,
                                                                  const SkinnyParams p) {
  using G = MtGrid<U>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t *smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int M = p.M, S = p.S, ns = p.ns;
  const bool fold = p.fold != 0, resid = p.epi == EPI_RESID;
  const int t0 = fold ? 2 : 0;  // first token row of the operand
  const int Mr = M + t0;
  const int Ks = p.K / S, kb = Ks / 64;
  const int split = blockIdx.z;
  // rank `split` finishes token rows [r_lo, r_hi)
  const int r_lo = M * split / S, r_hi = M * (split + 1) / S, rows_o = r_hi - r_lo;
  const MtLayout L(Mr, Ks, U, ns, (M + S - 1) / S, fold, resid);
  uint8_t *sW = smem + L.w_off;
  uint8_t *ring = smem + L.ring_off;
  float *sRes = reinterpret_cast<float *>(ring);  // [Mr][res_ld], after the last k-block
  float2 *sPart = reinterpret_cast<float2 *>(smem + L.part_off);
  float *sOld = reinterpret_cast<float *>(smem + L.old_off);
  float *sBias = reinterpret_cast<float *>(smem + L.bias_off);
  float *sWg = reinterpret_cast<float *>(smem + L.wgb_off);  // W g, then W b, summed over ranks
  float *sGn = reinterpret_cast<float *>(smem + L.gn_off);   // the next LayerNorm's gain, these columns
  float2 *sStat = reinterpret_cast<float2 *>(smem + L.stat_off);
  int2 *sRow = reinterpret_cast<int2 *>(smem + L.row_off);   // (cache slot, position) of each row finished
  uint64_t *wbar = reinterpret_cast<uint64_t *>(smem + L.bar_off);
  uint64_t *full = wbar + 1;
  uint4 *sZero = reinterpret_cast<uint4 *>(smem + L.zero_off);
  int *s_flag = reinterpret_cast<int *>(smem + L.flag_off);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cta = blockIdx.x;
  constexpr int kUC = U * 8;
  const int n_base = cta * kUC;
  const int res_ld = L.res_ld;
  const int unit_bytes = kb * 1024;
  const long long spin = p.spin > 0 ? p.spin : kSpinLimitCycles;

  // the launch the plan implies (uniform over the grid: a mismatch ends every
  // CTA before any barrier or copy)
  {
    uint32_t dyn, ncta = 1, crank = 0;
    asm volatile("mov.u32 %0, %%dynamic_smem_size;" : "=r"(dyn));
    if (S > 1) {
      asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(ncta));
      crank = cluster_ctarank();
    }
    const uint32_t need = static_cast<uint32_t>(L.total) + static_cast<uint32_t>(smem - smem_raw);
    if (dyn < need || ncta != static_cast<uint32_t>(S) || crank != static_cast<uint32_t>(split) || ns < 1 ||
        ns > kMtMaxStages || ns > kb || Mr > kMtMaxTiles * 16 || static_cast<int>(gridDim.x) * kUC != p.N ||
        static_cast<int>(gridDim.z) != S || kb * 64 * S != p.K) {
      if (tid == 0) set_error(p.err, WF_DEV_ERR_LAUNCH);
      return;
    }
  }

  if (tid == 0) {
    *s_flag = 0;
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
    mbar_init(wbar, 1);
    for (int s = 0; s < kMtMaxStages; ++s) mbar_init(&full[s], 1);
    fence_barrier_init();
    *sZero = make_uint4(0u, 0u, 0u, 0u);
    mbar_arrive_expect_tx(wbar, static_cast<uint32_t>(U * unit_bytes));
    for (int u = 0; u < U; ++u)
      tma_load_3d(sW + u * unit_bytes, &tmW, 0, (cta * U + u) * 8, split * kb, wbar);
  }
  for (int i = tid; i < kUC; i += kMtThreads) {
    sBias[i] = p.bias ? bf2f(p.bias[n_base + i]) : 0.f;
    if (p.xg_out) sGn[i] = bf2f(p.g_next[n_base + i]);
  }
  // a key/value row's cache slot and position are fixed for the step (the
  // kernels before this one in the pass do not write them)
  if (p.epi == EPI_KV)
    for (int r = tid; r < rows_o; r += kMtThreads) {
      const int t = r_lo + r, ii = t / p.rows_per_seq, jr = t - ii * p.rows_per_seq;
      const int slot = p.seq_slot[ii];
      sRow[r] = make_int2(slot, (p.pos_base ? p.pos_base[slot] : 0) + jr);
    }
  __syncthreads();  // the barriers and the zero line are initialised before any thread uses them
  pdl_wait();

  // ---------------- the first k-blocks of the operand; the partial row sums
  // and the residual rows this rank finishes copy in meanwhile
  const uint32_t stage_tx = static_cast<uint32_t>(Mr * 128);
  if (tid == 0) {
    for (int q = 0; q < ns; ++q) {
      mbar_arrive_expect_tx(&full[q], stage_tx);
      tma_load_3d(ring + q * L.stage_bytes, &tmX, 0, 0, split * kb + q, &full[q]);
    }
  }
  const bool staged = fold && p.n_part <= kMtStageParts;
  if (staged) {  // 16-byte pairs of partials (a row's last pair may carry one unused)
    const uint32_t dst = smem_u32(sPart);
    const int pairs = (p.n_part + 1) / 2;
    for (int i = tid; i < rows_o * pairs; i += kMtThreads) {
      const int r = i / pairs, j = 2 * (i - r * pairs);
      cp_async16(dst + 8u * (r * kMtStageParts + j), p.fold_part + static_cast<size_t>(r_lo + r) * p.part_stride + j);
    }
  }
  constexpr int kQ = kUC / 4;  // column quads of a row
  if (resid) {
    const uint32_t dst = smem_u32(sOld);
    for (int i = tid; i < rows_o * kQ; i += kMtThreads) {
      const int r = i / kQ, c = (i - r * kQ) * 4;
      cp_async16(dst + 16u * i, p.resid + static_cast<size_t>(r_lo + r) * p.ld_resid + n_base + c);
    }
  }
  bool ok = mbar_wait(wbar, 0, p.err, spin);
  if (!ok) *s_flag = 1;

  // ---------------- MMAs: warp (wu, wt) owns the units of group wu and the
  // 16-row tiles wt, wt + WT, ...
  const int n_tiles = (Mr + 15) / 16;
  const int wu = warp % G::kWU, wt = warp / G::kWU;
  float acc[G::kTW][G::kUW][4];
#pragma unroll
  for (int h = 0; h < G::kTW; ++h)
#pragma unroll
    for (int u = 0; u < G::kUW; ++u) acc[h][u][0] = acc[h][u][1] = acc[h][u][2] = acc[h][u][3] = 0.f;
  const int ar = (lane & 7) + ((lane >> 3) & 1) * 8, c0 = lane >> 4;
  const int br = lane & 7, bg = lane >> 3;
  const uint32_t offB0 = br * 128 + (((bg) ^ br) << 4), offB1 = br * 128 + (((bg + 4) ^ br) << 4);
  const uint32_t w_base = smem_u32(sW) + wu * G::kUW * unit_bytes, ring_base = smem_u32(ring),
                 z_addr = smem_u32(sZero);
  for (int q = 0; q < kb; ++q) {
    const int s = q % ns;
    const bool landed = mbar_wait(&full[s], static_cast<uint32_t>(q / ns) & 1u, p.err, spin);
    if (!landed) *s_flag = 1;
    if (ok && landed) {
      const uint32_t st = ring_base + s * L.stage_bytes;
      uint32_t b[G::kUW][8];
#pragma unroll
      for (int u = 0; u < G::kUW; ++u) {
        const uint32_t wq = w_base + u * unit_bytes + q * 1024;
        ldsm_x4(wq + offB0, b[u][0], b[u][1], b[u][2], b[u][3]);
        ldsm_x4(wq + offB1, b[u][4], b[u][5], b[u][6], b[u][7]);
      }
      // consecutive MMAs go to different accumulators (units, and tiles when
      // the registers allow): a k-step's result is not waited on before the
      // next independent MMA issues; each accumulator still adds its k-steps
      // in order
      if constexpr (G::kAllTiles) {
        uint32_t a[G::kTW][4][4];
#pragma unroll
        for (int h = 0; h < G::kTW; ++h) {
          const int row = (wt + G::kWT * h) * 16 + ar;
          const bool real = row < Mr;
          const uint32_t aq = st + row * 128, sw = row & 7;
#pragma unroll
          for (int j = 0; j < 4; ++j)
            ldsm_x4(real ? aq + (((2 * j + c0) ^ sw) << 4) : z_addr, a[h][j][0], a[h][j][1], a[h][j][2], a[h][j][3]);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j)
#pragma unroll
          for (int h = 0; h < G::kTW; ++h)
#pragma unroll
            for (int u = 0; u < G::kUW; ++u)
              mma_bf16(acc[h][u], a[h][j][0], a[h][j][1], a[h][j][2], a[h][j][3], b[u][2 * j], b[u][2 * j + 1]);
      } else {
#pragma unroll
        for (int h = 0; h < G::kTW; ++h) {
          const int tile = wt + G::kWT * h;
          if (tile >= n_tiles) break;
          const int row = tile * 16 + ar;
          const bool real = row < Mr;
          const uint32_t aq = st + row * 128, sw = row & 7;
          uint32_t a[4][4];
#pragma unroll
          for (int j = 0; j < 4; ++j)
            ldsm_x4(real ? aq + (((2 * j + c0) ^ sw) << 4) : z_addr, a[j][0], a[j][1], a[j][2], a[j][3]);
#pragma unroll
          for (int j = 0; j < 4; ++j)
#pragma unroll
            for (int u = 0; u < G::kUW; ++u)
              mma_bf16(acc[h][u], a[j][0], a[j][1], a[j][2], a[j][3], b[u][2 * j], b[u][2 * j + 1]);
        }
      }
    }
    __syncthreads();  // every warp is done with stage s: refill it
    if (tid == 0 && q + ns < kb) {
      mbar_arrive_expect_tx(&full[s], stage_tx);
      tma_load_3d(ring + s * L.stage_bytes, &tmX, 0, 0, split * kb + q + ns, &full[s]);
    }
  }
  // the next kernel may start once every CTA is past its MMAs (earlier, its
  // prefetches slow this kernel's gather of the split-K sums: measured)
  pdl_launch_dependents();
  // results -> shared memory over the ring (fp32 [Mr][res_ld]); lane holds
  // rows g, g + 8 and columns 2 c4, 2 c4 + 1 of each unit
  {
    const int g = lane >> 2, c4 = lane & 3;
#pragma unroll
    for (int h = 0; h < G::kTW; ++h) {
      const int tile = wt + G::kWT * h;
      if (tile >= n_tiles) break;
#pragma unroll
      for (int u = 0; u < G::kUW; ++u) {
        const int r0 = tile * 16 + g, r1 = r0 + 8, col = (wu * G::kUW + u) * 8 + 2 * c4;
        if (r0 < Mr) *reinterpret_cast<float2 *>(sRes + r0 * res_ld + col) = make_float2(acc[h][u][0], acc[h][u][1]);
        if (r1 < Mr) *reinterpret_cast<float2 *>(sRes + r1 * res_ld + col) = make_float2(acc[h][u][2], acc[h][u][3]);
      }
    }
  }
  cp_async_wait_all();
  if (S > 1) cluster_sync();  // every rank's results are in its shared memory
  else __syncthreads();

  // ---------------- W g and W b summed over the ranks in rank order (warps
  // 0-3); the statistics of the rows this rank finishes (warps 4-7, four rows
  // in flight per warp): lane l sums partials l + 32 i in order of i, then
  // the warp adds across lanes
  const uint32_t res_u32 = smem_u32(sRes);
  if (fold) {
    constexpr int kHalf = kMtWarps / 2;
    if (warp < kHalf) {
      for (int i = tid; i < 2 * kUC; i += kHalf * 32) {
        const int e = (i / kUC) * res_ld + (i % kUC);
        float v = 0.f;
        if (S > 1) {
          // every load issued unconditionally (a rank past S reads this
          // CTA's own value, unused) so none waits on another
          float part[8];
#pragma unroll
          for (int r = 0; r < 8; ++r) part[r] = dsmem_ld_f32(dsmem_map(res_u32 + 4u * e, r < S ? r : split));
#pragma unroll
          for (int r = 0; r < 8; ++r)
            if (r < S) v += part[r];
        } else {
          v = sRes[e];
        }
        sWg[i] = v;
      }
    } else {
      constexpr int kR = 4;
      for (int r0 = warp - kHalf; r0 < rows_o; r0 += kHalf * kR) {
        float s1[kR], s2[kR];
#pragma unroll
        for (int k = 0; k < kR; ++k) {
          const int r = r0 + kHalf * k;
          s1[k] = s2[k] = 0.f;
          if (r < rows_o) {
            const float2 *src = staged ? sPart + r * kMtStageParts
                                       : p.fold_part + static_cast<size_t>(r_lo + r) * p.part_stride;
            for (int i = lane; i < p.n_part; i += 32) {
              const float2 v = staged ? src[i] : __ldcg(src + i);
              s1[k] += v.x;
              s2[k] += v.y;
            }
          }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1)
#pragma unroll
          for (int k = 0; k < kR; ++k) {
            s1[k] += __shfl_xor_sync(0xffffffffu, s1[k], off);
            s2[k] += __shfl_xor_sync(0xffffffffu, s2[k], off);
          }
        if (lane == 0)
#pragma unroll
          for (int k = 0; k < kR; ++k) {
            const int r = r0 + kHalf * k;
            if (r >= rows_o) continue;
            const float mu = s1[k] / static_cast<float>(p.K);
            const float var = fmaxf(s2[k] / static_cast<float>(p.K) - mu * mu, 0.f);
            sStat[r] = make_float2(mu, rsqrtf(var + p.ln_eps));
          }
      }
    }
    __syncthreads();
  }

  // ---------------- epilogue: thread f finishes the 4 columns 4 (f % kQ) of
  // row r_lo + f / kQ (a row's quads in consecutive lanes of one warp)
  const int n_q = rows_o * kQ;
  const bool good = ok && !*s_flag;
  // a rank arrives at the closing cluster barrier once it has read its
  // peers' sums for the last time (its own stores then overlap the barrier)
  bool arrived = false;
  for (int f0 = 0; f0 < n_q; f0 += kMtThreads * kMtQuadsPerPass) {
    float4 val[kMtQuadsPerPass];
    if (S > 1) {
      // every load issued unconditionally, all in flight before the sums: a
      // quad past the rows reads row r_lo's first quad and a rank past S this
      // CTA's own value, neither used
      float4 part[kMtQuadsPerPass][8];
#pragma unroll
      for (int e = 0; e < kMtQuadsPerPass; ++e) {
        const int f = f0 + e * kMtThreads + tid;
        const int r = f < n_q ? f / kQ : 0, c = f < n_q ? (f - r * kQ) * 4 : 0;
        const uint32_t a = res_u32 + 4u * ((r_lo + r + t0) * res_ld + c);
#pragma unroll
        for (int k = 0; k < 8; ++k) part[e][k] = dsmem_ld_f32x4(dsmem_map(a, k < S ? k : split));
      }
#pragma unroll
      for (int e = 0; e < kMtQuadsPerPass; ++e) {
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (k < S) {
            v.x += part[e][k].x;
            v.y += part[e][k].y;
            v.z += part[e][k].z;
            v.w += part[e][k].w;
          }
        }
        val[e] = v;
      }
      if (f0 + kMtThreads * kMtQuadsPerPass >= n_q) {
        cluster_arrive();
        arrived = true;
      }
    } else {
#pragma unroll
      for (int e = 0; e < kMtQuadsPerPass; ++e) {
        const int f = f0 + e * kMtThreads + tid;
        const int r = f / kQ, c = (f - r * kQ) * 4;
        val[e] = f < n_q ? *reinterpret_cast<const float4 *>(sRes + (r_lo + r + t0) * res_ld + c)
                         : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
#pragma unroll
    for (int e = 0; e < kMtQuadsPerPass; ++e) {
      const int f = f0 + e * kMtThreads + tid;
      const int r = f / kQ, c = (f - r * kQ) * 4;
      const int t = r_lo + r, n = n_base + c;
      const bool live = f < n_q && good;
      float v[4] = {val[e].x, val[e].y, val[e].z, val[e].w};
      float s1 = 0.f, s2 = 0.f;
      if (live) {
        if (fold) {  // r (W (g . x) - mu W g) + W b
          const float2 ms = sStat[r];
#pragma unroll
          for (int j = 0; j < 4; ++j) v[j] = __fmaf_rn(ms.y, __fmaf_rn(-ms.x, sWg[c + j], v[j]), sWg[kUC + c + j]);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) v[j] += sBias[c + j];
        if (p.epi == EPI_F32) {
          *reinterpret_cast<float4 *>(p.out_f32 + static_cast<size_t>(t) * p.ld_out + n) =
              make_float4(v[0], v[1], v[2], v[3]);
        } else if (p.epi == EPI_BF16) {
          st_bf16x4(p.out_bf16 + static_cast<size_t>(t) * p.ld_out + n, v[0], v[1], v[2], v[3]);
        } else if (p.epi == EPI_GELU) {
          st_bf16x4(p.out_bf16 + static_cast<size_t>(t) * p.ld_out + n, gelu_erf(v[0]), gelu_erf(v[1]),
                    gelu_erf(v[2]), gelu_erf(v[3]));
        } else if (p.epi == EPI_RESID) {
          const float4 old = *reinterpret_cast<const float4 *>(sOld + r * kUC + c);
          const float nr[4] = {old.x + v[0], old.y + v[1], old.z + v[2], old.w + v[3]};
          *reinterpret_cast<float4 *>(p.resid + static_cast<size_t>(t) * p.ld_resid + n) =
              make_float4(nr[0], nr[1], nr[2], nr[3]);
          if (p.xg_out) {
            st_bf16x4(p.xg_out + static_cast<size_t>(t + 2) * p.ld_resid + n, nr[0] * sGn[c], nr[1] * sGn[c + 1],
                      nr[2] * sGn[c + 2], nr[3] * sGn[c + 3]);
            if (t == 0) {
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                p.xg_out[n + j] = p.g_next[n + j];
                p.xg_out[static_cast<size_t>(p.ld_resid) + n + j] = p.b_next[n + j];
              }
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              s1 += nr[j];
              s2 += nr[j] * nr[j];
            }
          }
          if (p.tap0) st_bf16x4(p.tap0 + static_cast<size_t>(t) * p.ld_tap + n, nr[0], nr[1], nr[2], nr[3]);
          if (p.tap1) st_bf16x4(p.tap1 + static_cast<size_t>(t) * p.ld_tap + n, nr[0], nr[1], nr[2], nr[3]);
        } else if (p.epi == EPI_KV) {
          if (n < p.q_cols) {
            st_bf16x4(p.out_bf16 + static_cast<size_t>(t) * p.ld_out + n, v[0], v[1], v[2], v[3]);
          } else {
            const int cc = n - p.q_cols, which = cc / p.d_model, hd = cc - which * p.d_model;
            const int slot = sRow[r].x, pos = sRow[r].y;
            if (pos >= p.ctx) {
              set_error(p.err, WF_DEV_ERR_CAPACITY);
            } else {
              bf16 *dst = which == 0 ? p.kc : p.vc;
              st_bf16x4(dst + ((static_cast<size_t>(slot) * p.n_heads + (hd >> 6)) * p.ctx + pos) * 64 + (hd & 63),
                        v[0], v[1], v[2], v[3]);
            }
          }
        }
      }
      // this CTA's partial (sum x, sum x^2) of the row, for the next
      // LayerNorm: the row's kQ quads sit in consecutive lanes
      if (p.xg_out) {  // uniform over the block
#pragma unroll
        for (int off = kQ / 2; off > 0; off >>= 1) {
          s1 += __shfl_xor_sync(0xffffffffu, s1, off);
          s2 += __shfl_xor_sync(0xffffffffu, s2, off);
        }
        if (live && (f % kQ) == 0) p.part_out[static_cast<size_t>(t) * p.part_stride + cta] = make_float2(s1, s2);
      }
    }
  }
  if (S > 1) {  // peers may read this CTA's results until they have all arrived
    if (!arrived) cluster_arrive();
    cluster_wait();
  }
  // after a timeout a copy may still be landing
  __syncthreads();
  if (tid == 0 && *s_flag) {
    mbar_drain(wbar, 0);
    const int last = kb - 1;  // every stage's latest copy
    for (int q = last; q >= 0 && q > last - ns; --q)
      mbar_drain(&full[q % ns], static_cast<uint32_t>(q / ns) & 1u);
  }
}

// ------------------------------------------------------------------ host ----
namespace {
size_t mt_smem(int Mr, int M, int K, int U, int S, int ns, bool fold, bool resid) {
  return static_cast<size_t>(mt_smem_bytes(Mr, M, K, U, S, ns, fold, resid));
}

const CUtensorMap *mt_wmap(const void *W, int N, int K, int kblocks) {
  static std::mutex mu;
  static std::map<std::tuple<uintptr_t, int, int, int>, CUtensorMap *> cache;
  std::lock_guard<std::mutex> lock(mu);
  const auto key = std::make_tuple(reinterpret_cast<uintptr_t>(W), N, K, kblocks);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  CUtensorMap *m = new CUtensorMap;
  if (!tmap_bf16_units(m, W, N, K, kblocks)) {
    delete m;
    return nullptr;
  }
  cache.emplace(key, m);
  return m;
}

// the operand as (64 columns, row, 64-column block) with a box of one k-block
// of all Mr rows
const CUtensorMap *mt_xmap(const void *X, int Mr, int K, int ld) {
  static std::mutex mu;
  static std::map<std::tuple<uintptr_t, int, int, int>, CUtensorMap *> cache;
  std::lock_guard<std::mutex> lock(mu);
  const auto key = std::make_tuple(reinterpret_cast<uintptr_t>(X), Mr, K, ld);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  CUtensorMap *m = new CUtensorMap;
  if (!tmap_bf16_rows(m, X, Mr, K, ld, 1)) {
    delete m;
    return nullptr;
  }
  cache.emplace(key, m);
  return m;
}

template <int U>
cudaError_t mt_attrs() {
  const void *f = reinterpret_cast<const void *>(skinny_mt_kernel<U>);
  cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
  if (e == cudaSuccess) e = prefer_max_shared(f);
  return e;
}

const void *mt_kernel(int U) {
  switch (U) {
    case 1: return reinterpret_cast<const void *>(skinny_mt_kernel<1>);
    case 2: return reinterpret_cast<const void *>(skinny_mt_kernel<2>);
    case 4: return reinterpret_cast<const void *>(skinny_mt_kernel<4>);
    case 8: return reinterpret_cast<const void *>(skinny_mt_kernel<8>);
    default: return nullptr;
  }
}

int mt_sms() {
  static int n = [] {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return 0;
    return v;
  }();
  return n > 0 ? n : 152;
}

// CTAs (S == 1) or clusters of S CTAs of this shared-memory size that the
// GPU holds at once (a cluster's CTAs share one GPC, so clusters of 3, 5, 6
// or 7 CTAs leave SMs idle)
int mt_resident(int U, int S, size_t smem) {
  static std::mutex mu;
  static std::map<std::tuple<int, int, size_t>, int> cache;
  std::lock_guard<std::mutex> lock(mu);
  const auto key = std::make_tuple(U, S, smem);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  int n = 0;
  const void *f = mt_kernel(U);
  if (S == 1) {
    int per_sm = 0;
    if (f && cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, f, kMtThreads, smem) == cudaSuccess)
      n = per_sm * mt_sms();
  } else if (f) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1, 1, S);
    cfg.blockDim = dim3(kMtThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 1;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = S;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, f, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();  // a failed query leaves no error behind
  cache.emplace(key, n);
  return n;
}

// Estimated SM clock cycles of one launch: the waves of CTAs (clusters) the
// GPU holds at once, each paying a fixed latency (launch, weights, first
// operand block, about 4000 cycles; 1500 more for a cluster reduction) and
// its k-blocks.  A k-block costs the longer of the busiest warp's MMAs (about
// 10 cycles each with four or more independent accumulators) and the SM's
// MMA throughput over the CTAs sharing it (about 2.2 cycles per MMA), plus
// about 300 cycles of waiting and block synchronisation.
double mt_cost(int Mr, int N, int K, int u, int s, size_t smem) {
  const int T = (Mr + 15) / 16, wu = u >= 8 ? 2 : 1, wt = 8 / wu, uw = u / wu;
  const int tw_max = (kMtMaxTiles + wt - 1) / wt;
  const int tw = tw_max * uw <= 8 ? tw_max : (T + wt - 1) / wt;  // every tile slot, or the real ones
  const int kb = K / 64 / s;
  const int ctas = N / 8 / u * s;
  const int resident = mt_resident(u, s, smem);
  if (resident <= 0) return 1e30;
  const int units = s > 1 ? ctas / s : ctas;  // clusters or CTAs
  const int waves = (units + resident - 1) / resident;
  const int per_sm = (ctas / waves + mt_sms() - 1) / mt_sms();  // CTAs sharing an SM in a wave
  const double warp_mma = tw * uw * 4 * 10.0, sm_mma = per_sm * T * u * 4 * 2.2;
  const double t_kb = (warp_mma > sm_mma ? warp_mma : sm_mma) + 300.0;
  return waves * (4000.0 + (s > 1 ? 1500.0 : 0.0) + kb * t_kb);
}
}  // namespace

bool skinny_mt_plan(int Mr, int N, int K, bool fold, bool resid, int *U, int *S, int *ns) {
  if (Mr < 1 || Mr > kMtMaxTiles * 16 || N % 8 || K % 64) return false;
  if (skinny_mt_init() != cudaSuccess) return false;
  const int units = N / 8, kbt = K / 64;
  double best = 0.0;
  bool found = false;
  for (int u : {8, 4, 2, 1}) {
    if (units % u) continue;
    if (resid && units / u > kSkMaxParts) continue;  // one partial row sum per CTA column block
    for (int s = 1; s <= 8; ++s) {
      if (kbt % s) continue;
      const int kb = kbt / s;
      const int qmax = kb < kMtMaxStages ? kb : kMtMaxStages, qmin = kb < 2 ? kb : 2;
      // the deepest ring that lets two CTAs share an SM, else the deepest for one
      int pick = 0;
      for (int q = qmax; q >= qmin && !pick; --q)
        if (mt_smem(Mr, Mr, K, u, s, q, fold, resid) <= static_cast<size_t>(kMtSmemPair)) pick = q;
      for (int q = qmax; q >= qmin && !pick; --q)
        if (mt_smem(Mr, Mr, K, u, s, q, fold, resid) <= static_cast<size_t>(kMtSmemAlone)) pick = q;
      if (!pick) continue;
      const double c = mt_cost(Mr, N, K, u, s, mt_smem(Mr, Mr, K, u, s, pick, fold, resid));
      if (!found || c < best) {
        best = c;
        found = true;
        *U = u;
        *S = s;
        *ns = pick;
      }
    }
  }
  return found;
}

cudaError_t skinny_mt_init() {
  static cudaError_t status = cudaErrorNotReady;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaError_t e = mt_attrs<1>();
    if (e == cudaSuccess) e = mt_attrs<2>();
    if (e == cudaSuccess) e = mt_attrs<4>();
    if (e == cudaSuccess) e = mt_attrs<8>();
    status = e;
  });
  return status;
}

namespace {
bool aligned(const void *ptr, uintptr_t a) { return (reinterpret_cast<uintptr_t>(ptr) & (a - 1)) == 0; }
// a rejected launch; WF_DEBUG in the environment names the reason on stderr
cudaError_t mt_reject(const char *why, const SkinnyParams &p) {
  static const bool on = getenv("WF_DEBUG") != nullptr;
  if (on) fprintf(stderr, "libwf: skinny_mt rejects M=%d N=%d K=%d epi=%d: %s\n", p.M, p.N, p.K, p.epi, why);
  return cudaErrorInvalidValue;
}
}  // namespace

cudaError_t launch_skinny_mt(const void *W, SkinnyParams p, cudaStream_t s, bool pdl) {
  if (p.spin <= 0) p.spin = kSpinLimitCycles;
  const bool fold = p.fold != 0, resid = p.epi == EPI_RESID;
  if (p.ln_x || p.M < 1) return mt_reject("an fp32 LayerNorm operand or no rows", p);
  if (fold && (!p.fold_part || p.n_part < 1 || p.n_part > p.part_stride || p.part_stride % 2 ||
               !aligned(p.fold_part, 16)))
    return mt_reject("partial row sums", p);
  if (!p.x || p.ld_x % 8 || !aligned(p.x, 16)) return mt_reject("operand", p);
  // the epilogue moves 4 columns at a time: 16-byte fp32 and 8-byte bf16 stores
  if (p.epi == EPI_F32 && (p.ld_out % 4 || !aligned(p.out_f32, 16))) return mt_reject("fp32 output", p);
  if ((p.epi == EPI_BF16 || p.epi == EPI_GELU || (p.epi == EPI_KV && p.q_cols > 0)) &&
      (p.ld_out % 4 || !aligned(p.out_bf16, 8)))
    return mt_reject("bf16 output", p);
  if (p.epi == EPI_KV && (p.q_cols % 4 || p.d_model % 64 || !aligned(p.kc, 8) || !aligned(p.vc, 8)))
    return mt_reject("key/value caches", p);
  if (resid && (p.ld_resid % 4 || !aligned(p.resid, 16) || (p.xg_out && !aligned(p.xg_out, 8))))
    return mt_reject("residual rows", p);
  if ((p.tap0 || p.tap1) && (p.ld_tap % 4 || !aligned(p.tap0, 8) || !aligned(p.tap1, 8)))
    return mt_reject("taps", p);
  const int Mr = p.M + (fold ? 2 : 0);
  if (p.plan_M && p.plan_M < p.M) return mt_reject("more rows than planned", p);
  const int Mp = (p.plan_M ? p.plan_M : p.M) + (fold ? 2 : 0);
  if (!skinny_mt_plan(Mp, p.N, p.K, fold, resid, &p.U, &p.S, &p.ns)) return mt_reject("no plan", p);
  if (p.xg_out && (p.epi != EPI_RESID || !p.g_next || !p.b_next || !p.part_out || p.N / 8 / p.U > p.part_stride))
    return mt_reject("next LayerNorm operand", p);
  const CUtensorMap *tm = mt_wmap(W, p.N, p.K, p.K / p.S / 64);
  const CUtensorMap *tx = mt_xmap(p.x, Mr, p.K, p.ld_x);
  if (!tm || !tx) return mt_reject("tensor maps", p);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.N / 8 / p.U, 1, p.S);
  cfg.blockDim = dim3(kMtThreads, 1, 1);
  cfg.dynamicSmemBytes = mt_smem(Mr, p.M, p.K, p.U, p.S, p.ns, fold, resid);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (p.S > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 1;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = p.S;
    ++na;
  }
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  switch (p.U) {
    case 1: return cudaLaunchKernelEx(&cfg, skinny_mt_kernel<1>, *tm, *tx, p);
    case 2: return cudaLaunchKernelEx(&cfg, skinny_mt_kernel<2>, *tm, *tx, p);
    case 4: return cudaLaunchKernelEx(&cfg, skinny_mt_kernel<4>, *tm, *tx, p);
    case 8: return cudaLaunchKernelEx(&cfg, skinny_mt_kernel<8>, *tm, *tx, p);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace wf
