// Host-only check of the batched skinny projections' shared-memory plan
// (paper_2609_32869_gb300/csrc/wf_skinny_mt_layout.h, the header the kernel
// and its launcher use): for every plan the launcher may choose (units per
// CTA U, K split S, ring depth ns) and every pass size up to the handle's
// largest, each region the kernel addresses lies inside the launch's dynamic
// shared memory, the regions do not overlap, and the alignments the copies
// need hold.  Prints the number of violations and exits 1 if there is any.
#include <cstdio>
#include <initializer_list>

#include "wf_skinny_mt_layout.h"

using namespace wf;

static int errors = 0;
static void check(bool ok, const char *what, int N, int K, int U, int S, int ns, int M) {
  if (ok) return;
  if (++errors <= 20) std::printf("violation: %s (N %d K %d U %d S %d ns %d M %d)\n", what, N, K, U, S, ns, M);
}

// one projection shape: N outputs, K inputs, a folded LayerNorm operand
// (two more rows), a residual update; every plan at every pass of up to Mmax rows
static long shape(int N, int K, bool fold, bool resid, int Mmax) {
  long plans = 0;
  const int t0 = fold ? 2 : 0;
  for (int U : {1, 2, 4, 8}) {
    if ((N / 8) % U) continue;
    const int kUC = U * 8, WU = U >= 8 ? 2 : 1, WT = kMtWarps / WU, TW = (kMtMaxTiles + WT - 1) / WT;
    for (int S = 1; S <= 8; ++S) {
      if ((K / 64) % S) continue;
      const int kb = K / 64 / S;
      for (int ns = 1; ns <= (kb < kMtMaxStages ? kb : kMtMaxStages); ++ns) {
        if (mt_smem_bytes(Mmax + t0, Mmax + t0, K, U, S, ns, fold, resid) > static_cast<unsigned long>(kMtSmemAlone))
          continue;
        for (int M = 1; M <= Mmax; ++M) {
          ++plans;
          const int Mr = M + t0, cap = (M + S - 1) / S;
          const MtLayout L(Mr, K / S, U, ns, cap, fold, resid);
          const unsigned long dyn = mt_smem_bytes(Mr, M, K, U, S, ns, fold, resid);
          check(dyn <= 227ul * 1024, "launch asks for more than 227 KB", N, K, U, S, ns, M);
          check(static_cast<unsigned long>(L.total) + 1008 <= dyn, "no room to align the base", N, K, U, S, ns, M);
          // weights: one [kb][8 rows][128 B] slab per unit, 1024-aligned
          check(L.ring_off == U * kb * 1024 && L.ring_off % 1024 == 0, "weight slab", N, K, U, S, ns, M);
          // operand ring: ns stages of Mr rows x 128 B, each 1024-aligned
          check(L.stage_bytes % 1024 == 0 && Mr * 128 <= L.stage_bytes, "ring stage", N, K, U, S, ns, M);
          check(L.ring_off + ns * L.stage_bytes <= L.part_off, "ring past its region", N, K, U, S, ns, M);
          // results [Mr][res_ld] fp32 over the ring; the epilogue's float4 reads
          check(L.ring_off + Mr * L.res_ld * 4 <= L.part_off, "results past their region", N, K, U, S, ns, M);
          check((L.res_ld * 4) % 16 == 0 && L.res_ld >= kUC, "result row stride", N, K, U, S, ns, M);
          // staged partial sums (pairs of float2 by 16-byte copies) and residual rows
          check(L.part_off % 16 == 0 && L.old_off % 16 == 0, "copy alignment", N, K, U, S, ns, M);
          check(L.part_off + (fold ? cap * kMtStageParts * 8 : 0) <= L.old_off, "partials", N, K, U, S, ns, M);
          check(L.old_off + (resid ? cap * kUC * 4 : 0) <= L.bias_off, "residual rows", N, K, U, S, ns, M);
          // bias, W g / W b, next gain, row statistics, row slots: in order
          check(L.bias_off + kUC * 4 <= L.wgb_off && L.wgb_off + 2 * kUC * 4 <= L.gn_off &&
                    L.gn_off + kUC * 4 <= L.stat_off && L.stat_off % 8 == 0 && L.stat_off + cap * 8 <= L.row_off &&
                    L.row_off % 8 == 0 && L.row_off + cap * 8 <= L.bar_off,
                "small regions", N, K, U, S, ns, M);
          // mbarriers (weights + the stages), the zero line, the flag
          check(L.bar_off % 8 == 0 && L.bar_off + (1 + kMtMaxStages) * 8 <= L.zero_off && L.zero_off % 16 == 0 &&
                    L.zero_off + 16 <= L.flag_off && L.flag_off + 4 <= L.total,
                "barriers", N, K, U, S, ns, M);
          // every 16-row tile of the operand has a warp
          check((Mr + 15) / 16 <= WT * TW, "tiles without a warp", N, K, U, S, ns, M);
          // the rows a rank finishes stay inside the token rows
          for (int sp = 0; sp < S; ++sp) {
            const int lo = M * sp / S, hi = M * (sp + 1) / S;
            check(hi - lo <= cap && hi <= M, "rank rows", N, K, U, S, ns, M);
          }
        }
      }
    }
  }
  return plans;
}

int main() {
  long plans = 0;
  // (d, F): Whisper-large, Whisper-tiny, the toy decoder of the tests
  const int dims[3][2] = {{1280, 5120}, {384, 1536}, {128, 512}};
  for (const auto &df : dims) {
    const int d = df[0], F = df[1];
    plans += shape(3 * d, d, true, false, kMtMaxRows);  // QKV
    plans += shape(d, d, false, true, kMtMaxRows);      // out, cross-out
    plans += shape(d, d, true, false, kMtMaxRows);      // cross-query
    plans += shape(F, d, true, false, kMtMaxRows);      // fc1
    plans += shape(d, F, false, true, kMtMaxRows);      // fc2
  }
  std::printf("%d violations in %ld (plan, pass size) pairs\n", errors, plans);
  return errors ? 1 : 0;
}
