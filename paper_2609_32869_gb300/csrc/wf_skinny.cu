// Low-latency projections for a handful of token rows (M <= 16: one
// speculative block of K + 1 = 9 rows, a plain greedy step, a short prompt).
//
// At batch 1 a decoder block is a chain of dependent steps over 46 MB of
// weights (Sec. 3.1: one verify pass; Sec. 3.2: one drafter pass), so each
// projection's time after its dependency wait, not its weight stream, sets
// the step time.  The kernels here are shaped for that (the QKV and the
// cross-query projections of one sequence also carry their attention, in
// skinny_sattn_kernel and skinny_xattn_kernel below):
//  - every CTA owns U units of 8 weight rows over a K range (the whole K, or
//    1/S of it inside a cluster of S CTAs) and requests its entire weight slab
//    with TMA before griddepcontrol.wait, one 3-D tensor copy per unit that
//    lands 128-byte swizzled ([k-block][8 rows][64 features]); the slab
//    streams while the previous kernels run;
//  - after the wait the token operand lands in shared memory by one TMA
//    copy.  A LayerNorm operand is folded into the projection: with the
//    row's mean mu and r = 1 / sqrt(var + eps),
//      LN(x) W^T = r (W (g . x) - mu W g) + W b,
//    so the producer of the residual writes the bf16 rows g, b and g . x
//    (and per row its partial sums of x and x^2), one MMA over those rows
//    gives W g and W b beside the token rows, and the row statistics are
//    applied in the epilogue: no normalisation sits between the operand's
//    arrival and the MMAs.  (The history memory's LN_h, over fp32 rows, is
//    computed in the kernel instead: the CTAs of a cluster split the rows and
//    write the normalised bf16 rows into every CTA over distributed shared
//    memory.)
//  - all eight warps issue mma.sync m16n8k16 at once (tokens on the 16-row
//    side, weight rows on the 8-column side), each over its own slice of K;
//    the slices are summed in warp order, then (S > 1) the S CTAs' sums in
//    rank order over distributed shared memory, so a row's result never
//    depends on how many rows run with it;
//  - the epilogue adds the bias and applies GELU, the residual update with
//    the history taps, or the key/value cache scatter.
// At these shapes tcgen05.mma would be issued by one thread per CTA, 64 or
// more rows wide, for 9 useful rows; the warp-level MMA issues from every
// warp at once, and the tensor pipe is idle either way: the weights bound it.
#include <map>
#include <mutex>
#include <tuple>

#include "wf_device.cuh"
#include "wf_internal.h"

namespace wf {

namespace {

constexpr int kSkThreads = 256;
constexpr int kSkWarps = kSkThreads / 32;
// Shared memory a CTA may plan for: two CTAs (of this kernel and the next)
// fit on one SM's 228 KB with the per-CTA reserve.
constexpr int kSkSmemBudget = 113 * 1024;


// Shared-memory layout of one CTA (offsets from the 1024-aligned base).  The
// warps' partial sums reuse the weight slab once every MMA has read it.
struct SkLayout {
  int unit_bytes, w_bytes, a_off, a_bytes, sum_off, bias_off, gb_off, stat_off, bar_off, zero_off, flag_off,
      total;
  // M: operand rows; K_ln: features of an fp32 LayerNorm operand (its gain
  // and bias are staged), else 0
  __host__ __device__ SkLayout(int M, int Ks, int U, int K_ln) {
    const int kb = Ks / 64;
    unit_bytes = kb * 1024;
    w_bytes = U * unit_bytes;
    a_off = w_bytes;  // 1024-aligned: the operand's TMA copy swizzles by address
    a_bytes = kb * M * 128;
    sum_off = (a_off + a_bytes + 15) & ~15;
    bias_off = sum_off + U * 128 * 4;
    gb_off = (bias_off + U * 8 * 4 + 15) & ~15;
    stat_off = (gb_off + K_ln * 4 + 15) & ~15;
    bar_off = stat_off + kSkMaxRows * 8;
    zero_off = bar_off + 16;
    flag_off = zero_off + 16;
    total = flag_off + 16;
  }
};

// Byte offset of element k of token row r in the operand tile [k-block][M
// rows][128 B]: 128-byte line l = kb * M + r holds 16-byte chunk j at
// position j ^ (l & 7), the pattern a 128-byte-swizzled TMA copy writes into
// a 1024-aligned destination.
__device__ __forceinline__ uint32_t a_off(int M, int r, int k) {
  const int line = (k >> 6) * M + r;
  return static_cast<uint32_t>(line * 128 + ((((k >> 3) & 7) ^ (line & 7)) << 4) + (k & 7) * 2);
}

__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void dsmem_st_f32(uint32_t cluster_addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(cluster_addr), "f"(v) : "memory");
}
__device__ __forceinline__ void dsmem_st_u32x4(uint32_t cluster_addr, uint4 v) {
  asm volatile("st.shared::cluster.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(cluster_addr), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}

}  // namespace

template <int U>
__global__ void __launch_bounds__(kSkThreads, 2) skinny_kernel(const __grid_constant__ CUtensorMap tmW,
                                                               const __grid_constant__ CUtensorMap tmX,
                                                               const SkinnyParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t *smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int M = p.M, S = p.S, C = p.C;
  const bool ln = p.ln_x != nullptr;  // LayerNorm of fp32 rows computed here (gain and bias staged)
  const bool fold = p.fold != 0;      // folded LayerNorm: rows g, b, then the M token rows
  const bool tma_op = !ln;            // the operand's rows arrive by one TMA copy
  const int t0 = fold ? 2 : 0;        // first token row of the operand
  const int Mr = M + t0;              // operand rows
  const int Ks = p.K / S;  // K range of this CTA
  const int kb = Ks / 64;  // 64-wide k-blocks
  const SkLayout L(Mr, Ks, U, ln ? p.K : 0);
  const int unit_bytes = L.unit_bytes;             // one unit: [kb][8 rows][128 B]
  uint8_t *sW = smem;
  uint8_t *sA = smem + L.a_off;                    // [kb][Mr][128 B]
  float *sPart = reinterpret_cast<float *>(smem);  // [warps][U][16][8], over the slab after the MMAs
  float *sSum = reinterpret_cast<float *>(smem + L.sum_off);    // [U][16][8]
  float *sBias = reinterpret_cast<float *>(smem + L.bias_off);  // [U * 8]
  bf16 *sG = reinterpret_cast<bf16 *>(smem + L.gb_off);         // [K] LayerNorm gain, then [K] bias
  bf16 *sB = sG + p.K;
  float2 *sStat = reinterpret_cast<float2 *>(smem + L.stat_off);  // [M] (mu, r) of a folded LayerNorm
  uint64_t *bar = reinterpret_cast<uint64_t *>(smem + L.bar_off);  // [0] weights, [1] operand
  uint4 *sZero = reinterpret_cast<uint4 *>(smem + L.zero_off);
  int *s_flag = reinterpret_cast<int *>(smem + L.flag_off);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cta = blockIdx.x, split = blockIdx.z;
  const int unit0 = cta * U;  // first 8-row unit of this CTA
  const int n_base = unit0 * 8;
  const uint32_t crank = C > 1 ? cluster_ctarank() : 0u;  // cluster (C, 1, 1) when C > 1

  if (C > 1) cluster_arrive_relaxed();  // this CTA has started (peers write into it later)
  if (tid == 0) {
    *s_flag = 0;
    tma_prefetch_desc(&tmW);
    if (tma_op) tma_prefetch_desc(&tmX);
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    fence_barrier_init();
    *sZero = make_uint4(0u, 0u, 0u, 0u);
    // the whole weight slab: one copy per unit, before the dependency wait
    mbar_arrive_expect_tx(&bar[0], static_cast<uint32_t>(U * unit_bytes));
    for (int u = 0; u < U; ++u)
      tma_load_3d(sW + static_cast<size_t>(u) * unit_bytes, &tmW, 0, (unit0 + u) * 8, split * kb, &bar[0]);
  }
  for (int i = tid; i < U * 8; i += kSkThreads) {
    const int n = n_base + i;
    sBias[i] = (p.bias && n < p.N) ? bf2f(p.bias[n]) : 0.f;
  }
  if (ln) {  // parameters, not activations: staged before the wait
    for (int i = tid; i < p.K / 8; i += kSkThreads) {
      reinterpret_cast<uint4 *>(sG)[i] = reinterpret_cast<const uint4 *>(p.ln_g)[i];
      reinterpret_cast<uint4 *>(sB)[i] = reinterpret_cast<const uint4 *>(p.ln_b)[i];
    }
  }
  // epilogue outputs: rank `split` finishes the token rows [r_lo, r_hi) (all
  // of them when S == 1), every column u * 8 + j of each; its element
  // f = (t - r_lo) * U * 8 + u * 8 + j goes to thread f % threads, so a
  // warp holds whole rows when U * 8 divides 32.  The cache slot and
  // position of a key/value row are fixed for the step, so they are read
  // before the wait.
  constexpr int kEpi = (U * kSkMaxRows * 8 + kSkThreads - 1) / kSkThreads;
  constexpr int kUC = U * 8;  // columns of this CTA
  const int r_lo = M * split / S, r_hi = M * (split + 1) / S;
  const int n_out = (r_hi - r_lo) * kUC;
  auto elem = [&](int f, int &u, int &t, int &j) {
    t = r_lo + f / kUC;
    const int c = f - (t - r_lo) * kUC;
    u = c >> 3;
    j = c & 7;
  };
  int kv_dst[kEpi];  // EPI_KV: cache row index (slot * heads + head) * ctx + position, or -1
  // EPI_RESID with a folded LayerNorm next: its gain (and, on token row 0,
  // its bias) at this thread's outputs
  float g_nx[kEpi], b_nx[kEpi];
#pragma unroll
  for (int i = 0; i < kEpi; ++i) {
    kv_dst[i] = -1;
    const int f = tid + i * kSkThreads;
    g_nx[i] = b_nx[i] = 0.f;
    if (p.xg_out && f < n_out) {
      int u, t, j;
      elem(f, u, t, j);
      const int n = n_base + u * 8 + j;
      if (n < p.N) {
        g_nx[i] = bf2f(p.g_next[n]);
        if (t == 0) b_nx[i] = bf2f(p.b_next[n]);
      }
    }
    if (p.epi == EPI_KV && f < n_out) {
      int u, t, j;
      elem(f, u, t, j);
      const int n = n_base + u * 8 + j;
      if (n >= p.q_cols && n < p.N) {
        const int c = n - p.q_cols, hd = c % p.d_model;
        const int ii = t / p.rows_per_seq, jr = t - ii * p.rows_per_seq;
        const int slot = p.seq_slot[ii];
        const int pos = (p.pos_base ? p.pos_base[slot] : 0) + jr;
        kv_dst[i] = pos < p.ctx ? (slot * p.n_heads + (hd >> 6)) * p.ctx + pos : -2;
      }
    }
  }
  pdl_launch_dependents();
  __syncthreads();  // the barriers are initialised before any thread waits on them
  pdl_wait();

  // ---------------- operand: bf16 rows by one TMA copy (issued first), the
  // residual values this thread will update, or LN(x) shared by the cluster
  if (tma_op && tid == 0) {
    mbar_arrive_expect_tx(&bar[1], static_cast<uint32_t>(L.a_bytes));
    tma_load_3d(sA, &tmX, 0, 0, split * kb, &bar[1]);
  }
  float old[kEpi];
#pragma unroll
  for (int i = 0; i < kEpi; ++i) {
    old[i] = 0.f;
    const int f = tid + i * kSkThreads;
    if (p.epi == EPI_RESID && f < n_out) {
      int u, t, j;
      elem(f, u, t, j);
      const int n = n_base + u * 8 + j;
      if (n < p.N) old[i] = __ldcg(p.resid + static_cast<size_t>(t) * p.ld_resid + n);
    }
  }
  if (fold) {
    // row statistics of a folded LayerNorm: warp w sums the partials of rows
    // w and w + 8, lane l the partials l + 32 i (every load in flight at
    // once), added in order of i, then across lanes
    constexpr int kPL = (kSkMaxParts + 31) / 32;
    float2 v[2][kPL];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int t = warp + kSkWarps * h;
      const float2 *pr = p.fold_part + static_cast<size_t>(t) * p.part_stride;
#pragma unroll
      for (int q = 0; q < kPL; ++q) {
        const int i = lane + 32 * q;
        v[h][q] = (t < M && i < p.n_part) ? __ldcg(pr + i) : make_float2(0.f, 0.f);
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int t = warp + kSkWarps * h;
      float s1 = 0.f, s2 = 0.f;
#pragma unroll
      for (int q = 0; q < kPL; ++q) {
        s1 += v[h][q].x;
        s2 += v[h][q].y;
      }
      s1 = warp_sum(s1);
      s2 = warp_sum(s2);
      const float mu = s1 / static_cast<float>(p.K);
      const float var = fmaxf(s2 / static_cast<float>(p.K) - mu * mu, 0.f);
      if (lane == 0 && t < M) sStat[t] = make_float2(mu, rsqrtf(var + p.ln_eps));
    }
  }
  bool op_ok = true;
  if (ln) {
    // rows r = crank + C q of the cluster's operand belong to this CTA; warp w
    // normalises its rows q = w, w + 8 (lane l holds features 4l + 128 i)
    // into its own operand tile, then the CTA copies them to its peers
    constexpr int kMaxI = 12;  // K <= 1536
    const int nI = p.K / 128;
    if (C > 1) cluster_wait();  // every CTA of the cluster has started
    const uint32_t a_loc = smem_u32(sA);
    for (int h = 0; h < 2; ++h) {
      const int r = static_cast<int>(crank) + C * (warp + kSkWarps * h);
      if (r >= M) break;
      const float *xr = p.ln_x + static_cast<size_t>(r) * p.ln_ld;
      float4 v[kMaxI];
#pragma unroll
      for (int i = 0; i < kMaxI; ++i)
        if (i < nI) v[i] = __ldcg(reinterpret_cast<const float4 *>(xr + 4 * lane + 128 * i));
      float sum = 0.f;
#pragma unroll
      for (int i = 0; i < kMaxI; ++i)
        if (i < nI) sum += (v[i].x + v[i].y) + (v[i].z + v[i].w);
      const float mean = warp_sum(sum) / static_cast<float>(p.K);
      float q = 0.f;
#pragma unroll
      for (int i = 0; i < kMaxI; ++i) {
        if (i < nI) {
          const float a = v[i].x - mean, b = v[i].y - mean, c = v[i].z - mean, d = v[i].w - mean;
          q += (a * a + b * b) + (c * c + d * d);
        }
      }
      const float2 ms = make_float2(mean, rsqrtf(warp_sum(q) / static_cast<float>(p.K) + p.ln_eps));
#pragma unroll
      for (int i = 0; i < kMaxI; ++i) {
        if (i < nI) {
          const int k = 4 * lane + 128 * i;
          const uint2 gg = *reinterpret_cast<const uint2 *>(sG + k);
          const uint2 bb = *reinterpret_cast<const uint2 *>(sB + k);
          const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gg);
          const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&bb);
          const __nv_bfloat162 o0 = __floats2bfloat162_rn(ln_apply(v[i].x, ms, __low2float(g2[0]), __low2float(b2[0])),
                                                          ln_apply(v[i].y, ms, __high2float(g2[0]), __high2float(b2[0])));
          const __nv_bfloat162 o1 = __floats2bfloat162_rn(ln_apply(v[i].z, ms, __low2float(g2[1]), __low2float(b2[1])),
                                                          ln_apply(v[i].w, ms, __high2float(g2[1]), __high2float(b2[1])));
          *reinterpret_cast<uint2 *>(sA + a_off(M, r, k)) =
              make_uint2(*reinterpret_cast<const uint32_t *>(&o0), *reinterpret_cast<const uint32_t *>(&o1));
        }
      }
    }
    if (C > 1) {
      // fan this CTA's rows out to the other CTAs of the cluster: warp w
      // copies them to rank (crank + 1 + w) % C, 16 bytes per lane and store
      __syncthreads();
      const int my_rows = (M - static_cast<int>(crank) + C - 1) / C;  // rows crank, crank + C, ...
      const int lines = my_rows * kb;                                  // 128-byte lines to copy
      for (int w = warp; w < C - 1; w += kSkWarps) {
        const uint32_t dst = (crank + 1 + w) % C;
        for (int c = lane; c < lines * 8; c += 32) {
          const int li = c >> 3, ch = c & 7;
          const int rr = static_cast<int>(crank) + C * (li / kb), q = li % kb;
          const uint32_t off = static_cast<uint32_t>((q * M + rr) * 128 + ch * 16);
          const uint4 v4 = *reinterpret_cast<const uint4 *>(sA + off);
          dsmem_st_u32x4(dsmem_map(a_loc + off, dst), v4);
        }
      }
    }
    if (C > 1) cluster_sync();  // every row has landed in every CTA
    else __syncthreads();
  } else {
    op_ok = mbar_wait(&bar[1], 0, p.err, p.spin);
    if (!op_ok) *s_flag = 1;
  }
  // ---------------- MMAs: warp w takes the k-blocks [w kb / 8, (w + 1) kb / 8) of
  // every unit; within a k-block the k-steps alternate between two accumulators
  // (shorter dependency chains), added in a fixed order at the end
  const bool landed = mbar_wait(&bar[0], 0, p.err, p.spin) && op_ok;
  if (!landed) *s_flag = 1;
  float acc[U][2][4];
#pragma unroll
  for (int u = 0; u < U; ++u)
#pragma unroll
    for (int h = 0; h < 2; ++h) acc[u][h][0] = acc[u][h][1] = acc[u][h][2] = acc[u][h][3] = 0.f;
  if (landed) {
    const uint32_t w_base = smem_u32(sW);
    // A (ldmatrix.x4 per k-step): lanes 0-7 rows 0-7 and 16-23 rows 0-7 (second
    // 8 features), 8-15 and 24-31 rows 8-15; rows >= Mr read 16 zero bytes
    const int ar = (lane & 7) + ((lane >> 3) & 1) * 8, c0 = lane >> 4;
    const bool real = ar < Mr;
    const uint32_t a_base = smem_u32(sA), z_addr = smem_u32(sZero);
    // B (ldmatrix.x4 per pair of k-steps): lane group g reads 16-byte chunk g
    // (first pair) or g + 4 (second pair) of weight row lane & 7
    const int br = lane & 7, bg = lane >> 3;
    const uint32_t offB0 = br * 128 + (((bg) ^ br) << 4), offB1 = br * 128 + (((bg + 4) ^ br) << 4);
    const int kb_lo = warp * kb / kSkWarps, kb_hi = (warp + 1) * kb / kSkWarps;
    for (int q = kb_lo; q < kb_hi; ++q) {
      uint32_t a[4][4];
      const int line = q * Mr + ar;
      const uint32_t aq = a_base + line * 128, sw = line & 7;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        ldsm_x4(real ? aq + (((2 * j + c0) ^ sw) << 4) : z_addr, a[j][0], a[j][1], a[j][2], a[j][3]);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t wq = w_base + u * unit_bytes + q * 1024;
        uint32_t b0, b1, b2, b3, b4, b5, b6, b7;
        ldsm_x4(wq + offB0, b0, b1, b2, b3);
        ldsm_x4(wq + offB1, b4, b5, b6, b7);
        mma_bf16(acc[u][0], a[0][0], a[0][1], a[0][2], a[0][3], b0, b1);
        mma_bf16(acc[u][1], a[1][0], a[1][1], a[1][2], a[1][3], b2, b3);
        mma_bf16(acc[u][0], a[2][0], a[2][1], a[2][2], a[2][3], b4, b5);
        mma_bf16(acc[u][1], a[3][0], a[3][1], a[3][2], a[3][3], b6, b7);
      }
    }
  }
  __syncthreads();  // every warp is done with the slab, which now takes the partials
  // warp partials -> shared memory: lane holds rows g, g+8 and columns 2 c4, 2 c4 + 1
  {
    const int g = lane >> 2, c4 = lane & 3;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      float *pw = sPart + (warp * U + u) * 128;
      pw[g * 8 + 2 * c4] = acc[u][0][0] + acc[u][1][0];
      pw[g * 8 + 2 * c4 + 1] = acc[u][0][1] + acc[u][1][1];
      pw[(g + 8) * 8 + 2 * c4] = acc[u][0][2] + acc[u][1][2];
      pw[(g + 8) * 8 + 2 * c4 + 1] = acc[u][0][3] + acc[u][1][3];
    }
  }
  __syncthreads();
  // the CTA's sums, warps added in order
  for (int e = tid; e < U * 128; e += kSkThreads) {
    const int u = e >> 7, rc = e & 127;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kSkWarps; ++w) v += sPart[(w * U + u) * 128 + rc];
    sSum[e] = v;
  }
  // ---------------- S > 1: the cluster's CTAs add their sums in rank order;
  // rank r finishes the outputs e with e % S == r
  const bool ok = landed;
  if (S > 1) cluster_sync();
  else __syncthreads();
  // this CTA's partial (sum x, sum x^2) of each row it finishes, for the next
  // LayerNorm: reduced over the row's lanes when a warp holds whole rows
  constexpr bool kRowWarps = 32 % kUC == 0;
#pragma unroll
  for (int i = 0; i < kEpi; ++i) {
    const int f = tid + i * kSkThreads;
    float px = 0.f;  // the updated residual value this lane adds to its row's partial
    bool pv = false;
    if (f < n_out) {
      int u, t, j;
      elem(f, u, t, j);
      const int idx = u * 128 + (t + t0) * 8 + j;
      float v;
      if (S > 1) {
        float part[8];
        const uint32_t loc = smem_u32(sSum + idx);
#pragma unroll
        for (int r = 0; r < 8; ++r)  // every load in flight before the sum
          part[r] = r < S ? dsmem_ld_f32(dsmem_map(loc, r)) : 0.f;
        v = 0.f;
#pragma unroll
        for (int r = 0; r < 8; ++r)
          if (r < S) v += part[r];
      } else {
        v = sSum[idx];
      }
      const int n = n_base + u * 8 + j;
      if (n < p.N && ok) {
        if (fold) {  // r (W (g . x) - mu W g) + W b; rows 0 and 1 of the sums hold W g and W b
          const float2 ms = sStat[t];
          v = __fmaf_rn(ms.y, __fmaf_rn(-ms.x, sSum[u * 128 + j], v), sSum[u * 128 + 8 + j]);
        }
        v += sBias[u * 8 + j];
        if (p.epi == EPI_F32) {
          p.out_f32[static_cast<size_t>(t) * p.ld_out + n] = v;
        } else if (p.epi == EPI_BF16) {
          p.out_bf16[static_cast<size_t>(t) * p.ld_out + n] = __float2bfloat16(v);
        } else if (p.epi == EPI_GELU) {
          p.out_bf16[static_cast<size_t>(t) * p.ld_out + n] = __float2bfloat16(gelu_erf(v));
        } else if (p.epi == EPI_RESID) {
          const float nr = old[i] + v;
          p.resid[static_cast<size_t>(t) * p.ld_resid + n] = nr;
          if (p.xg_out) {
            p.xg_out[static_cast<size_t>(t + 2) * p.ld_resid + n] = __float2bfloat16(nr * g_nx[i]);
            if (t == 0) {  // bf16 values, converted back exactly
              p.xg_out[n] = __float2bfloat16(g_nx[i]);
              p.xg_out[static_cast<size_t>(p.ld_resid) + n] = __float2bfloat16(b_nx[i]);
            }
            px = nr;
            pv = true;
            if (!kRowWarps) sPart[u * 128 + t * 8 + j] = nr;  // the slab is free: the sums are in sSum
          }
          if (p.tap0) p.tap0[static_cast<size_t>(t) * p.ld_tap + n] = __float2bfloat16(nr);
          if (p.tap1) p.tap1[static_cast<size_t>(t) * p.ld_tap + n] = __float2bfloat16(nr);
        } else if (p.epi == EPI_KV) {
          if (n < p.q_cols) {
            p.out_bf16[static_cast<size_t>(t) * p.ld_out + n] = __float2bfloat16(v);
          } else if (kv_dst[i] == -2) {
            set_error(p.err, WF_DEV_ERR_CAPACITY);
          } else {
            const int c = n - p.q_cols, which = c / p.d_model;
            bf16 *dst = which == 0 ? p.kc : p.vc;
            dst[static_cast<size_t>(kv_dst[i]) * 64 + ((c - which * p.d_model) & 63)] = __float2bfloat16(v);
          }
        }
      }  // n < N && ok
    }  // f < n_out
    if (kRowWarps && p.xg_out && i * kSkThreads + warp * 32 < n_out) {  // warp-uniform
      float s1 = pv ? px : 0.f, s2 = pv ? px * px : 0.f;
#pragma unroll
      for (int off = kUC / 2; off > 0; off >>= 1) {
        s1 += __shfl_xor_sync(0xffffffffu, s1, off);
        s2 += __shfl_xor_sync(0xffffffffu, s2, off);
      }
      if (f < n_out && (f % kUC) == 0 && ok)
        p.part_out[static_cast<size_t>(r_lo + f / kUC) * p.part_stride + cta] = make_float2(s1, s2);
    }
  }
  if (!kRowWarps && p.xg_out) {
    // rows wider than a warp: warp w takes this rank's rows r_lo + w, + 8, ..,
    // lane l the outputs (u, j) with u = l / 8 + 4 i and j = l % 8, added in
    // order of i, then across lanes
    __syncthreads();
    for (int t = r_lo + warp; t < r_hi; t += kSkWarps) {
      float s1 = 0.f, s2 = 0.f;
      for (int u = lane >> 3; u < U; u += 4) {
        const int j = lane & 7;
        if (n_base + u * 8 + j >= p.N || !ok) continue;
        const float x = sPart[u * 128 + t * 8 + j];
        s1 += x;
        s2 += x * x;
      }
      s1 = warp_sum(s1);
      s2 = warp_sum(s2);
      if (lane == 0) p.part_out[static_cast<size_t>(t) * p.part_stride + cta] = make_float2(s1, s2);
    }
  }
  if (S > 1) cluster_sync();  // peers may read this CTA's sums until here
  // after a timeout a copy may still be landing: wait for it (bounded)
  __syncthreads();
  if (tid == 0 && *s_flag) {
    mbar_drain(&bar[0], 0);
    if (tma_op) mbar_drain(&bar[1], 0);
  }
}

// ------------------------------------------- cross-query + cross-attention --
// The cross-attention of a single sequence fused into the projection that
// forms its queries (Sec. 3.2: the drafter and the target attend to the
// acoustic memory; the query projection is LN2(x) W_q^T + b_q, folded as in
// the skinny projection).  A head's 64 query columns are 8 units of 8 weight
// rows, i.e. 8 CTAs with U = 1: the kernel runs them as one cluster per head.
// Each CTA projects its 8 columns for the M rows (MMA as above), scales them
// by 1/8 and writes them as one 16-byte chunk per row into the query tile of
// every CTA of the cluster.  Each CTA then attends to its own kpc frames
// (kpc = ceil(frames / 8) rounded up to 32; keys and values requested by TMA
// before the dependency wait: the acoustic memory is written once, at
// prefill), with the attention kernel's per-warp arithmetic (32 frames per
// warp, base-2 softmax, P rounded to bf16 for P V) and its in-order warp
// merge; the 8 CTAs' (m, l, o) then merge in rank order over distributed
// shared memory: each CTA pushes its partial of dims 8c .. 8c + 7 into CTA c,
// which merges the 8 it receives.  No query
// row and no partial leaves the cluster, and a row's result depends only on
// its own query (frames are split by position, not by rows).
namespace {
struct XaLayout {
  int w_off, a_off, k_off, v_off, q_off, pb_off, sum_off, bias_off, stat_off, ml_off, bar_off, zero_off, flag_off,
      total;
  __host__ __device__ XaLayout(int Mr, int K, int kpc) {
    const int kb = K / 64;
    w_off = 0;
    a_off = kb * 1024;
    k_off = (a_off + kb * Mr * 128 + 1023) & ~1023;
    v_off = k_off + kpc * 128;  // kpc a multiple of 32: 1024-aligned
    q_off = v_off + kpc * 128;
    // the partial inbox reuses the operand tile (dead in every CTA of the
    // cluster before the first partial is pushed) when it is large enough
    const bool inbox_in_a = kb * Mr * 128 >= 8 * 16 * 12 * 4;
    pb_off = inbox_in_a ? a_off : q_off + 16 * 128;
    sum_off = q_off + 16 * 128 + (inbox_in_a ? 0 : 8 * 16 * 12 * 4);
    bias_off = sum_off + 128 * 4;
    stat_off = bias_off + 8 * 4;
    ml_off = stat_off + kSkMaxRows * 8;
    bar_off = ml_off + 2 * 8 * 16 * 4;
    zero_off = bar_off + 4 * 8;
    flag_off = zero_off + 16;
    total = flag_off + 16;
  }
};
constexpr float kXaLog2e = 1.4426950408889634f;
}  // namespace

__global__ void __launch_bounds__(kSkThreads, 2) skinny_xattn_kernel(const __grid_constant__ CUtensorMap tmW,
                                                                     const __grid_constant__ CUtensorMap tmX,
                                                                     const __grid_constant__ CUtensorMap tmK,
                                                                     const __grid_constant__ CUtensorMap tmV,
                                                                     const SkinnyParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t *smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int M = p.M, Mr = M + 2, K = p.K, kb = K / 64, kpc = p.xa_kpc, ctx = p.ctx;
  const XaLayout L(Mr, K, kpc);
  uint8_t *sW = smem + L.w_off;
  uint8_t *sA = smem + L.a_off;
  uint8_t *sK = smem + L.k_off;
  uint8_t *sV = smem + L.v_off;
  uint8_t *sQ = smem + L.q_off;
  // [8 source CTAs][16 rows][12]: m, l, -, -, o[8] of this CTA's 8 dims, pushed by each CTA
  float *pin = reinterpret_cast<float *>(smem + L.pb_off);
  float *sPart = reinterpret_cast<float *>(smem + L.w_off);  // [8 warps][16][8], over the slab after the MMAs
  float *sSum = reinterpret_cast<float *>(smem + L.sum_off);  // [16][8]
  float *sBias = reinterpret_cast<float *>(smem + L.bias_off);
  float2 *sStat = reinterpret_cast<float2 *>(smem + L.stat_off);
  float *sm = reinterpret_cast<float *>(smem + L.ml_off);  // [8][16]
  float *sl = sm + 8 * 16;                                 // [8][16]
  float *so = reinterpret_cast<float *>(sK);               // [warps][16][64], once every warp is done with K
  uint64_t *bar = reinterpret_cast<uint64_t *>(smem + L.bar_off);  // weights, operand, keys, values
  uint4 *sZero = reinterpret_cast<uint4 *>(smem + L.zero_off);
  int *s_flag = reinterpret_cast<int *>(smem + L.flag_off);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cta = blockIdx.x, head = cta >> 3;
  const uint32_t crank = cluster_ctarank();  // == cta % 8: this CTA's 8 dims of the head
  const int n_base = cta * 8;
  const int nw = kpc / 32;                   // warps with frames
  const int key0 = static_cast<int>(crank) * kpc;
  const bool any_keys = key0 < ctx;
  const long long spin = p.spin > 0 ? p.spin : kSpinLimitCycles;

  cluster_arrive_relaxed();  // this CTA has started (peers write into it later)
  if (tid == 0) {
    *s_flag = 0;
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
    for (int i = 0; i < 4; ++i) mbar_init(&bar[i], 1);
    fence_barrier_init();
    *sZero = make_uint4(0u, 0u, 0u, 0u);
    mbar_arrive_expect_tx(&bar[0], static_cast<uint32_t>(kb * 1024));
    tma_load_3d(sW, &tmW, 0, n_base, 0, &bar[0]);
    if (any_keys) {  // the acoustic memory of this CTA's frames
      const int slot = p.seq_slot[0];
      const int outer = slot * p.n_heads + head;
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      mbar_arrive_expect_tx(&bar[2], static_cast<uint32_t>(kpc * 128));
      tma_load_3d(sK, &tmK, 0, key0, outer, &bar[2]);
      mbar_arrive_expect_tx(&bar[3], static_cast<uint32_t>(kpc * 128));
      tma_load_3d(sV, &tmV, 0, key0, outer, &bar[3]);
    }
  }
  if (tid < 8) sBias[tid] = p.bias ? bf2f(p.bias[n_base + tid]) : 0.f;
  pdl_launch_dependents();
  __syncthreads();  // the barriers are initialised before any thread waits on them
  pdl_wait();

  // ---------------- operand (rows g, b, then g . x) and the row statistics
  if (tid == 0) {
    mbar_arrive_expect_tx(&bar[1], static_cast<uint32_t>(kb * Mr * 128));
    tma_load_3d(sA, &tmX, 0, 0, 0, &bar[1]);
  }
  {
    constexpr int kPL = (kSkMaxParts + 31) / 32;
    float2 v[2][kPL];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int t = warp + kSkWarps * h;
      const float2 *pr = p.fold_part + static_cast<size_t>(t) * p.part_stride;
#pragma unroll
      for (int q = 0; q < kPL; ++q) {
        const int i = lane + 32 * q;
        v[h][q] = (t < M && i < p.n_part) ? __ldcg(pr + i) : make_float2(0.f, 0.f);
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int t = warp + kSkWarps * h;
      float s1 = 0.f, s2 = 0.f;
#pragma unroll
      for (int q = 0; q < kPL; ++q) {
        s1 += v[h][q].x;
        s2 += v[h][q].y;
      }
      s1 = warp_sum(s1);
      s2 = warp_sum(s2);
      const float mu = s1 / static_cast<float>(K);
      const float var = fmaxf(s2 / static_cast<float>(K) - mu * mu, 0.f);
      if (lane == 0 && t < M) sStat[t] = make_float2(mu, rsqrtf(var + p.ln_eps));
    }
  }
  bool ok = mbar_wait(&bar[1], 0, p.err, spin);
  ok = mbar_wait(&bar[0], 0, p.err, spin) && ok;
  if (!ok) *s_flag = 1;

  // ---------------- the 8 query columns: warp w over k-blocks [w kb / 8, (w + 1) kb / 8)
  float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
  if (ok) {
    const int ar = (lane & 7) + ((lane >> 3) & 1) * 8, c0 = lane >> 4;
    const bool real = ar < Mr;
    const uint32_t a_base = smem_u32(sA), z_addr = smem_u32(sZero), w_base = smem_u32(sW);
    const int br = lane & 7, bg = lane >> 3;
    const uint32_t offB0 = br * 128 + (((bg) ^ br) << 4), offB1 = br * 128 + (((bg + 4) ^ br) << 4);
    const int kb_lo = warp * kb / kSkWarps, kb_hi = (warp + 1) * kb / kSkWarps;
    for (int q = kb_lo; q < kb_hi; ++q) {
      uint32_t a[4][4];
      const int line = q * Mr + ar;
      const uint32_t aq = a_base + line * 128, sw = line & 7;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        ldsm_x4(real ? aq + (((2 * j + c0) ^ sw) << 4) : z_addr, a[j][0], a[j][1], a[j][2], a[j][3]);
      const uint32_t wq = w_base + q * 1024;
      uint32_t b0, b1, b2, b3, b4, b5, b6, b7;
      ldsm_x4(wq + offB0, b0, b1, b2, b3);
      ldsm_x4(wq + offB1, b4, b5, b6, b7);
      mma_bf16(acc[0], a[0][0], a[0][1], a[0][2], a[0][3], b0, b1);
      mma_bf16(acc[1], a[1][0], a[1][1], a[1][2], a[1][3], b2, b3);
      mma_bf16(acc[0], a[2][0], a[2][1], a[2][2], a[2][3], b4, b5);
      mma_bf16(acc[1], a[3][0], a[3][1], a[3][2], a[3][3], b6, b7);
    }
  }
  __syncthreads();  // the slab now takes the warps' partials
  {
    const int g = lane >> 2, c4 = lane & 3;
    float *pw = sPart + warp * 128;
    pw[g * 8 + 2 * c4] = acc[0][0] + acc[1][0];
    pw[g * 8 + 2 * c4 + 1] = acc[0][1] + acc[1][1];
    pw[(g + 8) * 8 + 2 * c4] = acc[0][2] + acc[1][2];
    pw[(g + 8) * 8 + 2 * c4 + 1] = acc[0][3] + acc[1][3];
  }
  __syncthreads();
  if (tid < 128) {
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kSkWarps; ++w) v += sPart[w * 128 + tid];
    sSum[tid] = v;
  }
  __syncthreads();

  // ---------------- queries into every CTA of the cluster: a lane group of 8
  // holds one row's 8 values; lane j of the group stores the row's chunk into
  // CTA j
  cluster_wait();  // every CTA of the cluster has started
  if (warp < (M * 8 + 31) / 32) {
    const int e = tid, t = e >> 3, j = e & 7;
    float qv = 0.f;
    if (t < M) {
      const float2 ms = sStat[t];
      float v = __fmaf_rn(ms.y, __fmaf_rn(-ms.x, sSum[j], sSum[(t + 2) * 8 + j]), sSum[8 + j]);
      v += sBias[j];
      qv = __bfloat162float(__float2bfloat16(v)) * 0.125f;  // the query in bf16, scaled by 1/sqrt(64)
    }
    const float nx = __shfl_down_sync(0xffffffffu, qv, 1);
    const uint32_t pr = pack_bf16(qv, nx);
    const int base = lane & ~7;
    uint4 chunk;
    chunk.x = __shfl_sync(0xffffffffu, pr, base + 0);
    chunk.y = __shfl_sync(0xffffffffu, pr, base + 2);
    chunk.z = __shfl_sync(0xffffffffu, pr, base + 4);
    chunk.w = __shfl_sync(0xffffffffu, pr, base + 6);
    if (t < M) dsmem_st_u32x4(dsmem_map(smem_u32(sQ) + swz(t, static_cast<int>(crank)), j), chunk);
  }
  cluster_sync();  // every row's 8 chunks have landed in every CTA

  // ---------------- attention over this CTA's frames (warps < nw, 32 each)
  const bool k_ok = !any_keys || mbar_wait(&bar[2], 0, p.err, spin);
  if (!k_ok) *s_flag = 1;
  const int g = lane >> 2, c4 = lane & 3;
  const int kw = warp * 32;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  float o[8][4];
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
  // warp-uniform: the MMAs below need the whole warp
  const bool mine = __all_sync(0xffffffffu, any_keys && warp < nw && k_ok && ok);
  float sc[4][4];
  if (mine) {
    const uint32_t q_u32 = smem_u32(sQ), k_u32 = smem_u32(sK);
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
      uint32_t a0, a1, a2, a3;
      const int mi = lane >> 3;
      ldsm_x4(q_u32 + swz((mi & 1) * 8 + (lane & 7), 2 * ks + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
      for (int np = 0; np < 2; ++np) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(k_u32 + swz(kw + np * 16 + (mi >> 1) * 8 + (lane & 7), 2 * ks + (mi & 1)), b0, b1, b2, b3);
        mma_bf16(sc[2 * np], a0, a1, a2, a3, b0, b1);
        mma_bf16(sc[2 * np + 1], a0, a1, a2, a3, b2, b3);
      }
    }
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int row = g + (e >> 1) * 8;
        const int pos = key0 + kw + nt * 8 + c4 * 2 + (e & 1);
        const bool vis = row < M && pos < ctx;
        sc[nt][e] = vis ? sc[nt][e] * kXaLog2e : -INFINITY;
        mrow[e >> 1] = fmaxf(mrow[e >> 1], sc[nt][e]);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mrow[r] = fmaxf(mrow[r], __shfl_xor_sync(0xffffffffu, mrow[r], 1));
      mrow[r] = fmaxf(mrow[r], __shfl_xor_sync(0xffffffffu, mrow[r], 2));
    }
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float v = sc[nt][e] == -INFINITY ? 0.f : exp2f(sc[nt][e] - mrow[e >> 1]);
        sc[nt][e] = v;
        lrow[e >> 1] += v;
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
      lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
    }
    if (!mbar_wait(&bar[3], 0, p.err, spin)) *s_flag = 1;
    const uint32_t v_u32 = smem_u32(sV);
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      const uint32_t a0 = pack_bf16(sc[2 * kk][0], sc[2 * kk][1]);
      const uint32_t a1 = pack_bf16(sc[2 * kk][2], sc[2 * kk][3]);
      const uint32_t a2 = pack_bf16(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
      const uint32_t a3 = pack_bf16(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
      for (int dp = 0; dp < 4; ++dp) {
        uint32_t b0, b1, b2, b3;
        const int mi = lane >> 3;
        ldsm_x4_t(v_u32 + swz(kw + kk * 16 + (mi & 1) * 8 + (lane & 7), 2 * dp + (mi >> 1)), b0, b1, b2, b3);
        mma_bf16(o[2 * dp], a0, a1, a2, a3, b0, b1);
        mma_bf16(o[2 * dp + 1], a0, a1, a2, a3, b2, b3);
      }
    }
  } else if (any_keys && warp < nw) {
    // a wait gave up: this warp still waits (bounded) for the values it would read
    mbar_wait(&bar[3], 0, p.err, spin);
  }
  __syncthreads();  // every warp is done with the key tile, which now holds O
  if (warp < nw) {
    if (c4 == 0) {
      sm[warp * 16 + g] = mrow[0];
      sm[warp * 16 + g + 8] = mrow[1];
      sl[warp * 16 + g] = lrow[0];
      sl[warp * 16 + g + 8] = lrow[1];
    }
#pragma unroll
    for (int nd = 0; nd < 8; ++nd) {
      const int col = (nd ^ (g & 3)) * 8 + c4 * 2;
      *reinterpret_cast<float2 *>(so + (warp * 16 + g) * 64 + col) = make_float2(o[nd][0], o[nd][1]);
      *reinterpret_cast<float2 *>(so + (warp * 16 + g + 8) * 64 + col) = make_float2(o[nd][2], o[nd][3]);
    }
  }
  __syncthreads();
  // the CTA's (m, l, o) per row: thread -> (row qi, dims d0 .. d0 + 3), warps in order
  {
    const int qi = tid >> 4, d0 = (tid & 15) * 4;
    float Mx = -INFINITY;
    for (int w = 0; w < nw; ++w) Mx = fmaxf(Mx, sm[w * 16 + qi]);
    float Ls = 0.f, a4[4] = {0.f, 0.f, 0.f, 0.f};
    for (int w = 0; w < nw; ++w) {
      const float mw = sm[w * 16 + qi];
      const float wt = (mw == -INFINITY) ? 0.f : exp2f(mw - Mx);
      Ls += sl[w * 16 + qi] * wt;
      const float4 o4 = *reinterpret_cast<const float4 *>(so + (w * 16 + qi) * 64 + (d0 ^ ((qi & 3) << 3)));
      a4[0] += o4.x * wt;
      a4[1] += o4.y * wt;
      a4[2] += o4.z * wt;
      a4[3] += o4.w * wt;
    }
    if (!any_keys) {  // no frame here: the empty partial
      Mx = -INFINITY;
      Ls = 0.f;
      a4[0] = a4[1] = a4[2] = a4[3] = 0.f;
    }
    // push to the CTA that owns dims d0 .. d0 + 3 (rank d0 / 8)
    const uint32_t dst = static_cast<uint32_t>(d0 >> 3);
    const uint32_t base = smem_u32(pin) + 4u * ((crank * 16 + qi) * 12);
    if ((d0 & 7) == 0) {
      dsmem_st_f32(dsmem_map(base, dst), Mx);
      dsmem_st_f32(dsmem_map(base + 4u, dst), Ls);
    }
    dsmem_st_u32x4(dsmem_map(base + 4u * (4 + (d0 & 7)), dst),
                   make_uint4(__float_as_uint(a4[0]), __float_as_uint(a4[1]), __float_as_uint(a4[2]),
                              __float_as_uint(a4[3])));
  }
  cluster_sync();  // every CTA's partial of this CTA's dims has arrived
  // ---------------- merge the 8 partials in rank order: thread -> (row, 4 of the 8 dims)
  if (tid < 2 * M) {
    const int qi = tid >> 1, half = tid & 1;
    float MM = -INFINITY;
#pragma unroll
    for (int r = 0; r < 8; ++r) MM = fmaxf(MM, pin[(r * 16 + qi) * 12]);
    float LL = 0.f, oo[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const float *pr = pin + (r * 16 + qi) * 12;
      const float mc = pr[0];
      const float wt = (mc == -INFINITY) ? 0.f : exp2f(mc - MM);
      const float4 o4 = *reinterpret_cast<const float4 *>(pr + 4 + 4 * half);
      LL = __fmaf_rn(pr[1], wt, LL);
      oo[0] = __fmaf_rn(o4.x, wt, oo[0]);
      oo[1] = __fmaf_rn(o4.y, wt, oo[1]);
      oo[2] = __fmaf_rn(o4.z, wt, oo[2]);
      oo[3] = __fmaf_rn(o4.w, wt, oo[3]);
    }
    if (!*s_flag) {
      const float inv = 1.0f / LL;
      const int d0 = static_cast<int>(crank) * 8 + 4 * half;
      *reinterpret_cast<uint2 *>(p.out_bf16 + static_cast<size_t>(qi) * p.ld_out + head * 64 + d0) =
          make_uint2(pack_bf16(oo[0] * inv, oo[1] * inv), pack_bf16(oo[2] * inv, oo[3] * inv));
    }
  }
  __syncthreads();
  if (tid == 0 && *s_flag) {  // after a timeout a copy may still be landing
    for (int i = 0; i < 4; ++i)
      if (i < 2 || any_keys) mbar_drain(&bar[i], 0);
  }
}

// ------------------------------------------------ QKV + self-attention --
// The self-attention of a single sequence fused into its QKV projection
// (Sec. 3.1: the verify block's causal pass, query j seeing positions
// 0 .. L + j; Sec. 3.2, App. A.2: the drafter's joint softmax over its
// history memory and the bidirectional block, RoPE on queries and keys).  A
// cluster of 8 CTAs owns a head: CTA c projects query, key and value columns
// 8c .. 8c + 7 of the head (three units of 8 weight rows) for the M rows.
// The new keys and values go to the cache at positions L + j, as in the
// unfused projection, and, as 16-byte chunks over distributed shared memory,
// straight into the key/value tile of the CTA that attends to position
// L + j (CTA c attends to positions c kpc .. (c + 1) kpc - 1, its settled
// rows requested by TMA before the dependency wait; the chunks are written
// only after every CTA's copy has landed).  The query chunks go to every
// CTA.  Attention, warp merge and the rank-order merge of the 8 CTAs are
// those of the cross-attention kernel above.
namespace {
struct SaLayout {
  int w_off, a_off, k_off, v_off, q_off, new_off, pb_off, sum_off, bias_off, stat_off, ml_off, bar_off, zero_off,
      flag_off, total;
  __host__ __device__ SaLayout(int Mr, int K, int kpc) {
    const int kb = K / 64;
    w_off = 0;
    a_off = 3 * kb * 1024;
    k_off = (a_off + kb * Mr * 128 + 1023) & ~1023;
    v_off = k_off + kpc * 128;
    q_off = v_off + kpc * 128;
    new_off = q_off + 16 * 128;  // the new key rows, then the new value rows: [2][16][128 B]
    // the partial inbox reuses the operand tile, as in the cross-attention
    // kernel, and the CTA sums sit in the slab behind the warps' partials
    const bool inbox_in_a = kb * Mr * 128 >= 8 * 16 * 12 * 4;
    pb_off = inbox_in_a ? a_off : new_off + 2 * 16 * 128;
    sum_off = w_off + 8 * 3 * 128 * 4;
    bias_off = new_off + 2 * 16 * 128 + (inbox_in_a ? 0 : 8 * 16 * 12 * 4);
    stat_off = bias_off + 24 * 4;
    ml_off = stat_off + kSkMaxRows * 8;
    bar_off = ml_off + 2 * 8 * 16 * 4;
    zero_off = bar_off + 4 * 8;
    flag_off = zero_off + 16;
    total = flag_off + 16;
  }
};
}  // namespace

__global__ void __launch_bounds__(kSkThreads, 2) skinny_sattn_kernel(const __grid_constant__ CUtensorMap tmW,
                                                                     const __grid_constant__ CUtensorMap tmX,
                                                                     const __grid_constant__ CUtensorMap tmK,
                                                                     const __grid_constant__ CUtensorMap tmV,
                                                                     const SkinnyParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t *smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int M = p.M, Mr = M + 2, K = p.K, kb = K / 64, kpc = p.xa_kpc, ctx = p.ctx, H = p.n_heads;
  const SaLayout L(Mr, K, kpc);
  uint8_t *sW = smem + L.w_off;
  uint8_t *sA = smem + L.a_off;
  uint8_t *sK = smem + L.k_off;
  uint8_t *sV = smem + L.v_off;
  uint8_t *sQ = smem + L.q_off;
  uint8_t *sKn = smem + L.new_off, *sVn = sKn + 16 * 128;  // new key / value rows, by block row
  float *pin = reinterpret_cast<float *>(smem + L.pb_off);   // [8 source CTAs][16][12]
  float *sPart = reinterpret_cast<float *>(smem + L.w_off);  // [8 warps][3 units][16][8]
  float *sSum = reinterpret_cast<float *>(smem + L.sum_off);  // [3][16][8]
  float *sBias = reinterpret_cast<float *>(smem + L.bias_off);  // [3][8]
  float2 *sStat = reinterpret_cast<float2 *>(smem + L.stat_off);
  float *sm = reinterpret_cast<float *>(smem + L.ml_off);
  float *sl = sm + 8 * 16;
  float *so = reinterpret_cast<float *>(sK);
  uint64_t *bar = reinterpret_cast<uint64_t *>(smem + L.bar_off);
  uint4 *sZero = reinterpret_cast<uint4 *>(smem + L.zero_off);
  int *s_flag = reinterpret_cast<int *>(smem + L.flag_off);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cta = blockIdx.x, head = cta >> 3;
  const uint32_t crank = cluster_ctarank();
  const int nw = kpc / 32;
  const int key0 = static_cast<int>(crank) * kpc;
  const long long spin = p.spin > 0 ? p.spin : kSpinLimitCycles;
  // query, key and value units of this CTA (rows of the [3 d][d] weight)
  auto unit_row = [&](int u) { return (u * H * 8 + head * 8 + static_cast<int>(crank)) * 8; };
  // the cache length and slot are fixed for the step (read before the wait)
  const int slot = p.seq_slot[0];
  const int Lc = p.pos_base[slot];
  const int n_keys = Lc + M;
  const bool fits = n_keys <= ctx;
  const bool any_keys = fits && key0 < n_keys;
  const int outer = slot * H + head;

  cluster_arrive_relaxed();  // this CTA has started (peers write into it later)
  if (tid == 0) {
    *s_flag = fits ? 0 : 1;
    if (!fits) set_error(p.err, WF_DEV_ERR_CAPACITY);
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
    for (int i = 0; i < 4; ++i) mbar_init(&bar[i], 1);
    fence_barrier_init();
    *sZero = make_uint4(0u, 0u, 0u, 0u);
    mbar_arrive_expect_tx(&bar[0], static_cast<uint32_t>(3 * kb * 1024));
    for (int u = 0; u < 3; ++u) tma_load_3d(sW + u * kb * 1024, &tmW, 0, unit_row(u), 0, &bar[0]);
    if (any_keys) {  // this CTA's positions; rows from L on are replaced below
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      mbar_arrive_expect_tx(&bar[2], static_cast<uint32_t>(kpc * 128));
      tma_load_3d(sK, &tmK, 0, key0, outer, &bar[2]);
      mbar_arrive_expect_tx(&bar[3], static_cast<uint32_t>(kpc * 128));
      tma_load_3d(sV, &tmV, 0, key0, outer, &bar[3]);
    }
  }
  if (tid < 24) sBias[tid] = p.bias ? bf2f(p.bias[unit_row(tid >> 3) + (tid & 7)]) : 0.f;
  pdl_launch_dependents();
  __syncthreads();  // the barriers are initialised before any thread waits on them
  pdl_wait();

  // ---------------- operand (rows g, b, then g . x) and the row statistics
  if (tid == 0) {
    mbar_arrive_expect_tx(&bar[1], static_cast<uint32_t>(kb * Mr * 128));
    tma_load_3d(sA, &tmX, 0, 0, 0, &bar[1]);
  }
  {
    constexpr int kPL = (kSkMaxParts + 31) / 32;
    float2 v[2][kPL];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int t = warp + kSkWarps * h;
      const float2 *pr = p.fold_part + static_cast<size_t>(t) * p.part_stride;
#pragma unroll
      for (int q = 0; q < kPL; ++q) {
        const int i = lane + 32 * q;
        v[h][q] = (t < M && i < p.n_part) ? __ldcg(pr + i) : make_float2(0.f, 0.f);
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int t = warp + kSkWarps * h;
      float s1 = 0.f, s2 = 0.f;
#pragma unroll
      for (int q = 0; q < kPL; ++q) {
        s1 += v[h][q].x;
        s2 += v[h][q].y;
      }
      s1 = warp_sum(s1);
      s2 = warp_sum(s2);
      const float mu = s1 / static_cast<float>(K);
      const float var = fmaxf(s2 / static_cast<float>(K) - mu * mu, 0.f);
      if (lane == 0 && t < M) sStat[t] = make_float2(mu, rsqrtf(var + p.ln_eps));
    }
  }
  bool ok = mbar_wait(&bar[1], 0, p.err, spin);
  ok = mbar_wait(&bar[0], 0, p.err, spin) && ok;
  if (!ok) *s_flag = 1;

  // ---------------- query, key and value columns: warp w over k-blocks [w kb / 8, (w + 1) kb / 8)
  float acc[3][2][4];
#pragma unroll
  for (int u = 0; u < 3; ++u)
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) acc[u][hh][0] = acc[u][hh][1] = acc[u][hh][2] = acc[u][hh][3] = 0.f;
  if (ok) {
    const int ar = (lane & 7) + ((lane >> 3) & 1) * 8, c0 = lane >> 4;
    const bool real = ar < Mr;
    const uint32_t a_base = smem_u32(sA), z_addr = smem_u32(sZero), w_base = smem_u32(sW);
    const int br = lane & 7, bg = lane >> 3;
    const uint32_t offB0 = br * 128 + (((bg) ^ br) << 4), offB1 = br * 128 + (((bg + 4) ^ br) << 4);
    const int kb_lo = warp * kb / kSkWarps, kb_hi = (warp + 1) * kb / kSkWarps;
    for (int q = kb_lo; q < kb_hi; ++q) {
      uint32_t a[4][4];
      const int line = q * Mr + ar;
      const uint32_t aq = a_base + line * 128, sw = line & 7;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        ldsm_x4(real ? aq + (((2 * j + c0) ^ sw) << 4) : z_addr, a[j][0], a[j][1], a[j][2], a[j][3]);
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        const uint32_t wq = w_base + u * kb * 1024 + q * 1024;
        uint32_t b0, b1, b2, b3, b4, b5, b6, b7;
        ldsm_x4(wq + offB0, b0, b1, b2, b3);
        ldsm_x4(wq + offB1, b4, b5, b6, b7);
        mma_bf16(acc[u][0], a[0][0], a[0][1], a[0][2], a[0][3], b0, b1);
        mma_bf16(acc[u][1], a[1][0], a[1][1], a[1][2], a[1][3], b2, b3);
        mma_bf16(acc[u][0], a[2][0], a[2][1], a[2][2], a[2][3], b4, b5);
        mma_bf16(acc[u][1], a[3][0], a[3][1], a[3][2], a[3][3], b6, b7);
      }
    }
  }
  __syncthreads();  // the slab now takes the warps' partials
  {
    const int g = lane >> 2, c4 = lane & 3;
#pragma unroll
    for (int u = 0; u < 3; ++u) {
      float *pw = sPart + (warp * 3 + u) * 128;
      pw[g * 8 + 2 * c4] = acc[u][0][0] + acc[u][1][0];
      pw[g * 8 + 2 * c4 + 1] = acc[u][0][1] + acc[u][1][1];
      pw[(g + 8) * 8 + 2 * c4] = acc[u][0][2] + acc[u][1][2];
      pw[(g + 8) * 8 + 2 * c4 + 1] = acc[u][0][3] + acc[u][1][3];
    }
  }
  __syncthreads();
  for (int e = tid; e < 3 * 128; e += kSkThreads) {
    const int u = e >> 7, rc = e & 127;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kSkWarps; ++w) v += sPart[(w * 3 + u) * 128 + rc];
    sSum[e] = v;
  }
  __syncthreads();
  cluster_wait();  // every CTA of the cluster has started

  // ---------------- the new rows: a lane group of 8 holds one (unit, row)'s
  // 8 values; lane j stores the row's chunk into CTA j (queries into the
  // query tile, keys and values into the new-row buffers), and every lane
  // writes its key or value to the cache
  const int n_el = 3 * M * 8;
  for (int e0 = 0; e0 < n_el; e0 += kSkThreads) {
    if (e0 + warp * 32 >= n_el) break;  // warp-uniform
    const int e = e0 + tid, u = e / (M * 8), rem = e - u * M * 8, t = rem >> 3, j = rem & 7;
    const bool live = e < n_el;
    float val = 0.f;
    if (live) {
      const float *su = sSum + (u < 3 ? u : 0) * 128;
      const float2 ms = sStat[t];
      float v = __fmaf_rn(ms.y, __fmaf_rn(-ms.x, su[j], su[(t + 2) * 8 + j]), su[8 + j]);
      v += sBias[u * 8 + j];
      val = __bfloat162float(__float2bfloat16(v));
      if (u > 0 && fits && !*s_flag) {
        bf16 *dst = u == 1 ? p.kc : p.vc;
        dst[(static_cast<size_t>(outer) * ctx + Lc + t) * 64 + static_cast<int>(crank) * 8 + j] = __float2bfloat16(v);
      }
    }
    const float nx = __shfl_down_sync(0xffffffffu, val, 1);
    const uint32_t pr = pack_bf16(val, nx);
    const int base = lane & ~7;
    uint4 chunk;
    chunk.x = __shfl_sync(0xffffffffu, pr, base + 0);
    chunk.y = __shfl_sync(0xffffffffu, pr, base + 2);
    chunk.z = __shfl_sync(0xffffffffu, pr, base + 4);
    chunk.w = __shfl_sync(0xffffffffu, pr, base + 6);
    if (live && fits) {
      uint8_t *dst = u == 0 ? sQ : (u == 1 ? sKn : sVn);
      dsmem_st_u32x4(dsmem_map(smem_u32(dst) + swz(t, static_cast<int>(crank)), j), chunk);
    }
  }
  cluster_sync();  // every chunk has landed
  // this CTA's settled keys and values have landed: the new rows it attends
  // to (positions L + t in its range) replace the stale cache rows there
  bool kv_ok = true;
  if (any_keys) {
    kv_ok = mbar_wait(&bar[2], 0, p.err, spin);
    kv_ok = mbar_wait(&bar[3], 0, p.err, spin) && kv_ok;
  }
  if (!kv_ok) *s_flag = 1;
  {
    const int t = tid >> 4, c = (tid >> 1) & 7, kv = tid & 1;  // 16 rows x 8 chunks x {K, V}
    const int pos = Lc + t;
    if (t < M && any_keys && pos >= key0 && pos < key0 + kpc) {
      const uint8_t *src = kv ? sVn : sKn;
      uint8_t *dst = kv ? sV : sK;
      *reinterpret_cast<uint4 *>(dst + swz(pos - key0, c)) = *reinterpret_cast<const uint4 *>(src + swz(t, c));
    }
  }
  __syncthreads();

  // ---------------- queries: RoPE (drafter) at L + r, then the 1/8 scale;
  // keys: RoPE at their positions; values past the visible keys: zeros
  const bool rope = p.xa_mode == 1 && p.rope_tab;
  if (tid < 16 * 4) {
    const int r = tid >> 2, c = tid & 3;  // chunk c pairs with chunk c + 4 (dims i and i + 32)
    uint4 *lo = reinterpret_cast<uint4 *>(sQ + swz(r, c));
    uint4 *hi = reinterpret_cast<uint4 *>(sQ + swz(r, c + 4));
    uint4 a = *lo, b = *hi;
    bf16 *av = reinterpret_cast<bf16 *>(&a);
    bf16 *bv = reinterpret_cast<bf16 *>(&b);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      float x1 = bf2f(av[e]), x2 = bf2f(bv[e]);
      if (rope && r < M) {
        const float2 cs = __ldg(p.rope_tab + (Lc + r) * 32 + c * 8 + e);
        const float y1 = x1 * cs.x - x2 * cs.y, y2 = x2 * cs.x + x1 * cs.y;
        x1 = y1;
        x2 = y2;
      }
      av[e] = __float2bfloat16(x1 * 0.125f);
      bv[e] = __float2bfloat16(x2 * 0.125f);
    }
    *lo = a;
    *hi = b;
  }
  if (rope && any_keys) {
    for (int idx = tid; idx < kpc * 4; idx += kSkThreads) {
      const int kr = idx >> 2, c = idx & 3;
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
  }
  {
    const int z0 = min(max(n_keys - key0, 0), kpc);
    for (int idx = tid; idx < (kpc - z0) * 8; idx += kSkThreads)
      *reinterpret_cast<uint4 *>(sV + swz(z0 + (idx >> 3), idx & 7)) = make_uint4(0u, 0u, 0u, 0u);
  }
  __syncthreads();

  // ---------------- attention over this CTA's positions (warps < nw, 32 each)
  const int g = lane >> 2, c4 = lane & 3;
  const int kw = warp * 32;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
  float o[8][4];
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
  const bool mine = __all_sync(0xffffffffu, any_keys && warp < nw && key0 + kw < n_keys && ok && kv_ok);
  if (mine) {
    float sc[4][4];
    const uint32_t q_u32 = smem_u32(sQ), k_u32 = smem_u32(sK);
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
      uint32_t a0, a1, a2, a3;
      const int mi = lane >> 3;
      ldsm_x4(q_u32 + swz((mi & 1) * 8 + (lane & 7), 2 * ks + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
      for (int np = 0; np < 2; ++np) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(k_u32 + swz(kw + np * 16 + (mi >> 1) * 8 + (lane & 7), 2 * ks + (mi & 1)), b0, b1, b2, b3);
        mma_bf16(sc[2 * np], a0, a1, a2, a3, b0, b1);
        mma_bf16(sc[2 * np + 1], a0, a1, a2, a3, b2, b3);
      }
    }
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int row = g + (e >> 1) * 8;
        const int pos = key0 + kw + nt * 8 + c4 * 2 + (e & 1);
        bool vis = row < M && pos < n_keys;
        if (p.xa_mode == 0) vis = vis && pos <= Lc + row;
        sc[nt][e] = vis ? sc[nt][e] * kXaLog2e : -INFINITY;
        mrow[e >> 1] = fmaxf(mrow[e >> 1], sc[nt][e]);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mrow[r] = fmaxf(mrow[r], __shfl_xor_sync(0xffffffffu, mrow[r], 1));
      mrow[r] = fmaxf(mrow[r], __shfl_xor_sync(0xffffffffu, mrow[r], 2));
    }
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float v = sc[nt][e] == -INFINITY ? 0.f : exp2f(sc[nt][e] - mrow[e >> 1]);
        sc[nt][e] = v;
        lrow[e >> 1] += v;
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
      lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
    }
    const uint32_t v_u32 = smem_u32(sV);
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      const uint32_t a0 = pack_bf16(sc[2 * kk][0], sc[2 * kk][1]);
      const uint32_t a1 = pack_bf16(sc[2 * kk][2], sc[2 * kk][3]);
      const uint32_t a2 = pack_bf16(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
      const uint32_t a3 = pack_bf16(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
      for (int dp = 0; dp < 4; ++dp) {
        uint32_t b0, b1, b2, b3;
        const int mi = lane >> 3;
        ldsm_x4_t(v_u32 + swz(kw + kk * 16 + (mi & 1) * 8 + (lane & 7), 2 * dp + (mi >> 1)), b0, b1, b2, b3);
        mma_bf16(o[2 * dp], a0, a1, a2, a3, b0, b1);
        mma_bf16(o[2 * dp + 1], a0, a1, a2, a3, b2, b3);
      }
    }
  }
  __syncthreads();  // every warp is done with the key tile, which now holds O
  if (warp < nw) {
    if (c4 == 0) {
      sm[warp * 16 + g] = mrow[0];
      sm[warp * 16 + g + 8] = mrow[1];
      sl[warp * 16 + g] = lrow[0];
      sl[warp * 16 + g + 8] = lrow[1];
    }
#pragma unroll
    for (int nd = 0; nd < 8; ++nd) {
      const int col = (nd ^ (g & 3)) * 8 + c4 * 2;
      *reinterpret_cast<float2 *>(so + (warp * 16 + g) * 64 + col) = make_float2(o[nd][0], o[nd][1]);
      *reinterpret_cast<float2 *>(so + (warp * 16 + g + 8) * 64 + col) = make_float2(o[nd][2], o[nd][3]);
    }
  }
  __syncthreads();
  {
    const int qi = tid >> 4, d0 = (tid & 15) * 4;
    float Mx = -INFINITY;
    for (int w = 0; w < nw; ++w) Mx = fmaxf(Mx, sm[w * 16 + qi]);
    float Ls = 0.f, a4[4] = {0.f, 0.f, 0.f, 0.f};
    for (int w = 0; w < nw; ++w) {
      const float mw = sm[w * 16 + qi];
      const float wt = (mw == -INFINITY) ? 0.f : exp2f(mw - Mx);
      Ls += sl[w * 16 + qi] * wt;
      const float4 o4 = *reinterpret_cast<const float4 *>(so + (w * 16 + qi) * 64 + (d0 ^ ((qi & 3) << 3)));
      a4[0] += o4.x * wt;
      a4[1] += o4.y * wt;
      a4[2] += o4.z * wt;
      a4[3] += o4.w * wt;
    }
    if (!any_keys) {
      Mx = -INFINITY;
      Ls = 0.f;
      a4[0] = a4[1] = a4[2] = a4[3] = 0.f;
    }
    const uint32_t dst = static_cast<uint32_t>(d0 >> 3);
    const uint32_t base = smem_u32(pin) + 4u * ((crank * 16 + qi) * 12);
    if ((d0 & 7) == 0) {
      dsmem_st_f32(dsmem_map(base, dst), Mx);
      dsmem_st_f32(dsmem_map(base + 4u, dst), Ls);
    }
    dsmem_st_u32x4(dsmem_map(base + 4u * (4 + (d0 & 7)), dst),
                   make_uint4(__float_as_uint(a4[0]), __float_as_uint(a4[1]), __float_as_uint(a4[2]),
                              __float_as_uint(a4[3])));
  }
  cluster_sync();  // every CTA's partial of this CTA's dims has arrived
  if (tid < 2 * M) {
    const int qi = tid >> 1, half = tid & 1;
    float MM = -INFINITY;
#pragma unroll
    for (int r = 0; r < 8; ++r) MM = fmaxf(MM, pin[(r * 16 + qi) * 12]);
    float LL = 0.f, oo[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const float *pr = pin + (r * 16 + qi) * 12;
      const float mc = pr[0];
      const float wt = (mc == -INFINITY) ? 0.f : exp2f(mc - MM);
      const float4 o4 = *reinterpret_cast<const float4 *>(pr + 4 + 4 * half);
      LL = __fmaf_rn(pr[1], wt, LL);
      oo[0] = __fmaf_rn(o4.x, wt, oo[0]);
      oo[1] = __fmaf_rn(o4.y, wt, oo[1]);
      oo[2] = __fmaf_rn(o4.z, wt, oo[2]);
      oo[3] = __fmaf_rn(o4.w, wt, oo[3]);
    }
    if (!*s_flag) {
      const float inv = 1.0f / LL;
      const int d0 = static_cast<int>(crank) * 8 + 4 * half;
      *reinterpret_cast<uint2 *>(p.out_bf16 + static_cast<size_t>(qi) * p.ld_out + head * 64 + d0) =
          make_uint2(pack_bf16(oo[0] * inv, oo[1] * inv), pack_bf16(oo[2] * inv, oo[3] * inv));
    }
  }
  __syncthreads();
  if (tid == 0 && *s_flag) {  // after a timeout a copy may still be landing
    for (int i = 0; i < 4; ++i)
      if (i < 2 || any_keys) mbar_drain(&bar[i], 0);
  }
}

// ------------------------------------------------------------------ host ----
namespace {
size_t skinny_smem(int M, int K, int U, int S, bool ln) {
  return 1024 + static_cast<size_t>(SkLayout(M, K / S, U, ln ? K : 0).total);
}
}  // namespace

bool skinny_plan(int M, int N, int K, bool ln, bool whole_k, int *U, int *S) {
  if (M < 1 || M > kSkMaxRows || N % 8 || K % 128) return false;
  const int units = N / 8;
  // the fewest CTAs' worth of units that keeps the grid within about one CTA
  // per SM (160 for 1280 rows of 8) and a CTA within 113 KB of shared memory
  // (two kernels' CTAs share an SM, so the next one's slab streams in while
  // this one runs); whole K per CTA unless that does not fit, then K split
  // over a cluster of S CTAs
  int best_u = 0, best_s = 0;
  for (int s = 1; s <= 8; s *= 2) {
    if (K % (s * 128) || K / s < 256 || ((ln || whole_k) && s > 1)) continue;
    for (int u = 1; u <= 8; ++u) {
      if (units % u) continue;
      const int ctas = units / u * s;
      if (ctas > kSkMaxParts) continue;
      if (skinny_smem(M, K, u, s, ln) > kSkSmemBudget) continue;
      if (!best_u) {
        best_u = u;
        best_s = s;
      }
      break;
    }
    if (best_u) break;
  }
  if (!best_u) return false;
  if (ln && K > 1536) return false;
  *U = best_u;
  *S = best_s;
  return true;
}

// Unit tensor maps, encoded once per (matrix, k-blocks per copy).
static const CUtensorMap *skinny_tmap(const void *W, int N, int K, int kblocks) {
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

template <int U>
static cudaError_t skinny_attrs() {
  const void *f = reinterpret_cast<const void *>(skinny_kernel<U>);
  cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, kSkSmemBudget);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(f, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess) e = prefer_max_shared(f);
  return e;
}

cudaError_t skinny_init() {
  static cudaError_t status = cudaErrorNotReady;
  static std::once_flag once;
  std::call_once(once, [] {
    const void *xa = reinterpret_cast<const void *>(skinny_xattn_kernel);
    const void *sa = reinterpret_cast<const void *>(skinny_sattn_kernel);
    cudaError_t e = cudaFuncSetAttribute(xa, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e == cudaSuccess) e = prefer_max_shared(xa);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(sa, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (e == cudaSuccess) e = prefer_max_shared(sa);
    if (e == cudaSuccess) e = skinny_attrs<1>();
    if (e == cudaSuccess) e = skinny_attrs<2>();
    if (e == cudaSuccess) e = skinny_attrs<3>();
    if (e == cudaSuccess) e = skinny_attrs<4>();
    if (e == cudaSuccess) e = skinny_attrs<5>();
    if (e == cudaSuccess) e = skinny_attrs<6>();
    if (e == cudaSuccess) e = skinny_attrs<7>();
    if (e == cudaSuccess) e = skinny_attrs<8>();
    status = e;
  });
  return status;
}

// Operand tensor maps: the M bf16 rows of X [M][K] (row stride ld) as
// (64 columns, row, 64-column block), one copy of {64, M, kblocks} per CTA
// landing as [k-block][M][128 B], 128-byte swizzled.
static const CUtensorMap *skinny_xmap(const void *X, int M, int K, int ld, int kblocks) {
  static std::mutex mu;
  static std::map<std::tuple<uintptr_t, int, int, int, int>, CUtensorMap *> cache;
  std::lock_guard<std::mutex> lock(mu);
  const auto key = std::make_tuple(reinterpret_cast<uintptr_t>(X), M, K, ld, kblocks);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  CUtensorMap *m = new CUtensorMap;
  if (!tmap_bf16_rows(m, X, M, K, ld, kblocks)) {
    delete m;
    return nullptr;
  }
  cache.emplace(key, m);
  return m;
}

cudaError_t launch_skinny(const void *W, SkinnyParams p, cudaStream_t s, bool pdl) {
  if (p.spin <= 0) p.spin = kSpinLimitCycles;
  const bool ln = p.ln_x != nullptr;
  const bool fold = p.fold != 0;
  if (fold && (ln || p.M > kSkMaxFoldRows || !p.fold_part || p.n_part < 1 || p.n_part > p.part_stride))
    return cudaErrorInvalidValue;
  const int Mr = p.M + (fold ? 2 : 0);  // operand rows
  if (p.plan_M && p.plan_M < p.M) return cudaErrorInvalidValue;
  const int Mp = (p.plan_M ? p.plan_M : p.M) + (fold ? 2 : 0);  // operand rows of the plan
  if (!skinny_plan(Mp, p.N, p.K, ln, fold, &p.U, &p.S)) return cudaErrorInvalidValue;
  if (ln && (!p.ln_g || !p.ln_b || p.ln_ld % 4 || (reinterpret_cast<uintptr_t>(p.ln_x) & 15)))
    return cudaErrorInvalidValue;
  if (!ln && (!p.x || p.ld_x % 8 || (reinterpret_cast<uintptr_t>(p.x) & 15))) return cudaErrorInvalidValue;
  if (p.xg_out && (p.epi != EPI_RESID || !p.g_next || !p.b_next || !p.part_out ||
                   p.N / 8 / p.U > p.part_stride))
    return cudaErrorInvalidValue;
  const CUtensorMap *tm = skinny_tmap(W, p.N, p.K, p.K / p.S / 64);
  if (!tm) return cudaErrorInvalidValue;
  const CUtensorMap *tx = ln ? tm : skinny_xmap(p.x, Mr, p.K, p.ld_x, p.K / p.S / 64);
  if (!tx) return cudaErrorInvalidValue;
  // fp32 LayerNorm operands: the CTAs of a cluster share the rows (at most 8)
  const int gx = p.N / 8 / p.U;
  p.C = 1;
  if (ln && p.S == 1)
    for (int c = 8; c >= 2; c >>= 1)
      if (gx % c == 0) {
        p.C = c;
        break;
      }
  const size_t smem = skinny_smem(Mr, p.K, p.U, p.S, ln);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.N / 8 / p.U, 1, p.S);
  cfg.blockDim = dim3(kSkThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (p.S > 1 || p.C > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = p.C;
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
    case 1: return cudaLaunchKernelEx(&cfg, skinny_kernel<1>, *tm, *tx, p);
    case 2: return cudaLaunchKernelEx(&cfg, skinny_kernel<2>, *tm, *tx, p);
    case 3: return cudaLaunchKernelEx(&cfg, skinny_kernel<3>, *tm, *tx, p);
    case 4: return cudaLaunchKernelEx(&cfg, skinny_kernel<4>, *tm, *tx, p);
    case 5: return cudaLaunchKernelEx(&cfg, skinny_kernel<5>, *tm, *tx, p);
    case 6: return cudaLaunchKernelEx(&cfg, skinny_kernel<6>, *tm, *tx, p);
    case 7: return cudaLaunchKernelEx(&cfg, skinny_kernel<7>, *tm, *tx, p);
    case 8: return cudaLaunchKernelEx(&cfg, skinny_kernel<8>, *tm, *tx, p);
    default: return cudaErrorInvalidValue;
  }
}

// ------------------------------------------- fused cross-attention, host ----
namespace {
// frames per CTA: an eighth of the memory, rounded up to whole warps of 32
int xattn_kpc(int frames) { return ((frames + 7) / 8 + 31) / 32 * 32; }
size_t xattn_smem(int Mr, int K, int kpc) { return 1024 + static_cast<size_t>(XaLayout(Mr, K, kpc).total); }
// Tensor maps of the acoustic caches with a box of kpc frames.
const CUtensorMap *xattn_tmap(const void *cache, int ctx, int outer, int kpc) {
  static std::mutex mu;
  static std::map<std::tuple<uintptr_t, int, int, int>, CUtensorMap *> maps;
  std::lock_guard<std::mutex> lock(mu);
  const auto key = std::make_tuple(reinterpret_cast<uintptr_t>(cache), ctx, outer, kpc);
  auto it = maps.find(key);
  if (it != maps.end()) return it->second;
  CUtensorMap *m = new CUtensorMap;
  if (!tmap_bf16_cache(m, cache, static_cast<uint64_t>(ctx), static_cast<uint64_t>(outer),
                       static_cast<uint32_t>(kpc))) {
    delete m;
    return nullptr;
  }
  maps.emplace(key, m);
  return m;
}
}  // namespace

bool skinny_xattn_fits(int M, int d, int n_heads, int frames) {
  if (M < 1 || M > kSkMaxFoldRows || n_heads < 1 || d != n_heads * 64 || d % 128 || frames < 1) return false;
  const int kpc = xattn_kpc(frames);
  if (kpc > 256 || kpc > frames) return false;
  int U = 0, S = 0;
  if (!skinny_plan(M + 2, d, d, false, true, &U, &S)) return false;
  return xattn_smem(M + 2, d, kpc) <= 227 * 1024;
}

cudaError_t launch_skinny_xattn(const void *W, SkinnyParams p, cudaStream_t s, bool pdl) {
  if (p.spin <= 0) p.spin = kSpinLimitCycles;
  if (!p.fold || !p.x || !p.fold_part || p.n_part < 1 || p.n_part > p.part_stride || !p.kc || !p.vc ||
      !p.seq_slot || !p.out_bf16 || p.K != p.N || p.ld_out % 4 || p.ld_x % 8 || p.xa_outer < 1 ||
      (reinterpret_cast<uintptr_t>(p.x) & 15) || (reinterpret_cast<uintptr_t>(p.out_bf16) & 7) ||
      !skinny_xattn_fits(p.M, p.N, p.n_heads, p.ctx))
    return cudaErrorInvalidValue;
  p.U = 1;
  p.S = 1;
  p.C = 8;
  p.xa_kpc = xattn_kpc(p.ctx);
  const int Mr = p.M + 2;
  const CUtensorMap *tm = skinny_tmap(W, p.N, p.K, p.K / 64);
  const CUtensorMap *tx = skinny_xmap(p.x, Mr, p.K, p.ld_x, p.K / 64);
  const CUtensorMap *tk = xattn_tmap(p.kc, p.ctx, p.xa_outer, p.xa_kpc);
  const CUtensorMap *tv = xattn_tmap(p.vc, p.ctx, p.xa_outer, p.xa_kpc);
  if (!tm || !tx || !tk || !tv) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.N / 8, 1, 1);
  cfg.blockDim = dim3(kSkThreads, 1, 1);
  cfg.dynamicSmemBytes = xattn_smem(Mr, p.K, p.xa_kpc);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  attr[na].id = cudaLaunchAttributeClusterDimension;
  attr[na].val.clusterDim.x = 8;
  attr[na].val.clusterDim.y = 1;
  attr[na].val.clusterDim.z = 1;
  ++na;
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, skinny_xattn_kernel, *tm, *tx, *tk, *tv, p);
}

bool skinny_sattn_fits(int M, int d, int n_heads, int ctx) {
  if (M < 1 || M > kSkMaxFoldRows || n_heads < 1 || d != n_heads * 64 || d % 128 || ctx < 1) return false;
  const int kpc = xattn_kpc(ctx);
  if (kpc > 256 || kpc > ctx) return false;
  return 1024 + static_cast<size_t>(SaLayout(M + 2, d, kpc).total) <= 227 * 1024;
}

cudaError_t launch_skinny_sattn(const void *W, SkinnyParams p, cudaStream_t s, bool pdl) {
  if (p.spin <= 0) p.spin = kSpinLimitCycles;
  if (!p.fold || !p.x || !p.fold_part || p.n_part < 1 || p.n_part > p.part_stride || !p.kc || !p.vc ||
      !p.seq_slot || !p.pos_base || !p.out_bf16 || p.N != 3 * p.K || p.ld_out % 4 || p.ld_x % 8 ||
      p.xa_outer < 1 || (p.xa_mode != 0 && p.xa_mode != 1) || (p.xa_mode == 1 && !p.rope_tab) ||
      (reinterpret_cast<uintptr_t>(p.x) & 15) || (reinterpret_cast<uintptr_t>(p.out_bf16) & 7) ||
      !skinny_sattn_fits(p.M, p.K, p.n_heads, p.ctx))
    return cudaErrorInvalidValue;
  p.U = 3;
  p.S = 1;
  p.C = 8;
  p.xa_kpc = xattn_kpc(p.ctx);
  const int Mr = p.M + 2;
  const CUtensorMap *tm = skinny_tmap(W, p.N, p.K, p.K / 64);
  const CUtensorMap *tx = skinny_xmap(p.x, Mr, p.K, p.ld_x, p.K / 64);
  const CUtensorMap *tk = xattn_tmap(p.kc, p.ctx, p.xa_outer, p.xa_kpc);
  const CUtensorMap *tv = xattn_tmap(p.vc, p.ctx, p.xa_outer, p.xa_kpc);
  if (!tm || !tx || !tk || !tv) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.K / 8, 1, 1);  // 8 CTAs per head
  cfg.blockDim = dim3(kSkThreads, 1, 1);
  cfg.dynamicSmemBytes = 1024 + static_cast<size_t>(SaLayout(Mr, p.K, p.xa_kpc).total);
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int na = 0;
  attr[na].id = cudaLaunchAttributeClusterDimension;
  attr[na].val.clusterDim.x = 8;
  attr[na].val.clusterDim.y = 1;
  attr[na].val.clusterDim.z = 1;
  ++na;
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, skinny_sattn_kernel, *tm, *tx, *tk, *tv, p);
}

}  // namespace wf
