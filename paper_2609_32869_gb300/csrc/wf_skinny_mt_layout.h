// Shared-memory plan of the batched skinny projections (wf_skinny_mt.cu):
// the CTA's thread and warp grid and the byte layout of its dynamic shared
// memory.  Plain C++ (no CUDA headers) so that a host-only checker can walk
// every plan against the same layout the kernel and its launcher use.
#pragma once

#if defined(__CUDACC__)
#define WF_MT_HD __host__ __device__
#else
#define WF_MT_HD
#endif

namespace wf {

constexpr int kMtMaxRows = 144;  // 16 sequences x (1 + 8)

constexpr int kMtThreads = 256;
constexpr int kMtWarps = kMtThreads / 32;
constexpr int kMtMaxStages = 4;
constexpr int kMtMaxTiles = (kMtMaxRows + 2 + 15) / 16;  // 16-row tiles of the largest operand
constexpr int kMtStageParts = 32;  // partial row sums staged per row (more are read in place)
// shared memory a CTA may plan for: alone on its SM, or two per SM
constexpr int kMtSmemAlone = 220 * 1024;
constexpr int kMtSmemPair = 112 * 1024;

// warp grid: unit groups x tile groups (fewest ldmatrix bytes per k-block at
// 10 tiles: 2 x 4 for 8 units, 1 x 8 below)
template <int U>
struct MtGrid {
  static constexpr int kWU = U >= 8 ? 2 : 1;
  static constexpr int kUW = U / kWU;                        // units per warp
  static constexpr int kWT = kMtWarps / kWU;                 // tile groups
  static constexpr int kTW = (kMtMaxTiles + kWT - 1) / kWT;  // tiles per warp at most
  // all of a warp's tiles' A fragments held at once (when few accumulators);
  // a tile past the operand reads the zero line and its results are dropped
  static constexpr bool kAllTiles = kTW * kUW <= 8;
};

// Shared-memory layout: Mr operand rows, Ks inputs, ns ring stages, at most
// rows_o rows finished per rank.
struct MtLayout {
  int w_off, ring_off, stage_bytes, res_ld, part_off, old_off, bias_off, wgb_off, gn_off, stat_off, row_off,
      bar_off, zero_off, flag_off, total;
  WF_MT_HD MtLayout(int Mr, int Ks, int U, int ns, int rows_o, bool fold, bool resid) {
    const int kb = Ks / 64;
    w_off = 0;
    ring_off = U * kb * 1024;
    stage_bytes = (Mr * 128 + 1023) & ~1023;  // stages start 1024-aligned (the copies swizzle by address)
    res_ld = U * 8 + 8;                       // fp32 results [Mr][U 8 + 8], over the ring once it is done
    int region = ns * stage_bytes;
    if (Mr * res_ld * 4 > region) region = Mr * res_ld * 4;
    part_off = ring_off + region;
    old_off = part_off + (fold ? rows_o * kMtStageParts * 8 : 0);
    bias_off = old_off + (resid ? rows_o * U * 8 * 4 : 0);
    wgb_off = bias_off + U * 8 * 4;
    gn_off = wgb_off + 2 * U * 8 * 4;
    stat_off = gn_off + U * 8 * 4;
    row_off = stat_off + rows_o * 8;
    bar_off = (row_off + rows_o * 8 + 15) & ~15;
    zero_off = (bar_off + (1 + kMtMaxStages) * 8 + 15) & ~15;
    flag_off = zero_off + 16;
    total = flag_off + 16;
  }
};

// Dynamic shared memory of a launch: the layout of Mr operand rows, M token
// rows split over S ranks, plus 1024 bytes to align its start.
inline unsigned long mt_smem_bytes(int Mr, int M, int K, int U, int S, int ns, bool fold, bool resid) {
  return 1024ul + static_cast<unsigned long>(MtLayout(Mr, K / S, U, ns, (M + S - 1) / S, fold, resid).total);
}

}  // namespace wf
