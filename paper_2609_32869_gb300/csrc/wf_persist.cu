// Persistent decode pass for small batches (M <= 16 token rows: one
// speculative sequence of K + 1 = 9 rows, or plain greedy steps).
//
// The verification pass of Sec. 3.1 (and the drafter pass of Sec. 3.2, and
// plain greedy steps) at small batch.  At batch 1 a decoder block is a chain
// of dependent, tiny computations over 46 MB of weights: LN1 -> QKV ->
// self-attention -> out + residual -> LN2 -> cross-query -> cross-attention
// -> cross-out + residual -> LN3 -> fc1 -> fc2 + residual (the Whisper
// decoder block, pre-LayerNorm).  Launched kernel by kernel, each link pays a
// launch edge and a cold start, so the step is bound by latency, not by HBM.
// Here one cooperative launch runs every block of the pass with one CTA per
// SM:
//
//  - A producer thread streams everything that does not depend on the
//    activations through a ring of eight 20 KB shared-memory slots with TMA,
//    running ahead of the dependency chain across phases and blocks: each
//    projection unit (8 weight rows by the unit's whole K range) is one
//    copy, each 128 cached keys (or values) of one head another.  Large
//    copies matter: a TMA instruction costs about the same for 1 KB as for
//    20 KB.
//  - Eight compute warps follow the chain.  Work is cut into units: 8 weight
//    rows of a projection (the n = 8 side of mma.sync m16n8k16; the <= 16
//    token rows fill the m side), a (sequence, head) of self-attention, a
//    (sequence, head, 256-frame chunk) of cross-attention.  Units are dealt
//    round robin over the CTAs, continuing from phase to phase, so every CTA
//    streams about the same bytes per block.
//  - CTAs hand activations to each other through plain global buffers.  A
//    CTA publishes a phase by adding one to the phase's counter with release
//    semantics; a consumer waits with one thread (acquire, with backoff) for
//    the counter to reach the number of CTAs and then reads through L2.  The
//    fc2 split-K partials and the cross-attention block partials have
//    counters of their own, so only their owners wait on them.
//  - Every result is a function of its own token row only: LayerNorm
//    statistics reduce each row in a fixed order, a token row is one row of
//    the MMA's A operand, attention key blocks are aligned to absolute
//    positions and merge in order, and the fc2 split-K partials add in
//    quarter order.  Speculative (9 rows) and plain greedy (1 row) steps
//    therefore produce identical bits for the same position.
//
// Precision follows the rest of the library: bf16 weights and activations
// into the tensor cores, fp32 accumulation, fp32 residual, fp32 softmax.
#include <cuda/atomic>
#include <mutex>

#include "wf_device.cuh"
#include "wf_internal.h"

namespace wf {

namespace {

constexpr int kW = 8;                     // compute warps
constexpr int kThr = (kW + 1) * 32;       // + one producer warp
constexpr int kCThr = kW * 32;            // compute threads
constexpr int kNS = 8;                    // ring slots
constexpr int kSlot = 20 * 1024;          // bytes per slot: one projection unit (8 rows x K,
                                          // K <= 1280) or 128 keys (or values) of one head
constexpr int kKeysPerSlot = 128;
constexpr int kScratch = 42 * 1024;       // operand tile, reductions, attention staging
constexpr int kUB = 5;                    // projection units per CTA and phase (at most)
constexpr int kKS = 10;                   // k16-steps per warp: operand width <= 1280
constexpr int kQ2 = 4;                    // fc2 split-K factor (partials add in order)
constexpr int kPS = 68;                   // attention partial: m, l, -, -, o[64] (o 16-byte aligned)
constexpr int kLnGB = 2 * 1280 * 2;        // LayerNorm gain and bias (bf16, d <= 1280)
constexpr int kSmemMk = 1024 + kNS * kSlot + kScratch + kLnGB + 2 * kNS * 8 + 2048;

enum : int { PH_QKV = 0, PH_SATT, PH_OUT, PH_XQ, PH_XATT, PH_XOUT, PH_FC1, PH_FC2 };

// ------------------------------------------------------ synchronisation --
// Phases hand data to each other through plain global buffers.  A CTA that
// has written its outputs of phase s adds one to counter s with release
// semantics (after a barrier of its compute warps, so every thread's stores
// are ordered before it); a CTA that needs them waits, with one thread and
// an acquire load, until the counter reaches the number of CTAs, then reads
// with L2 loads (ld.global.cg: L1 is not coherent across SMs).  One polling
// thread per CTA keeps the counters' cache lines cool; a measured hop (last
// arrival to every CTA holding a 46 KB operand) costs about 1.8 us.
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t *ptr) {
  cuda::atomic_ref<uint32_t, cuda::thread_scope_device> r(*const_cast<uint32_t *>(ptr));
  return r.load(cuda::memory_order_acquire);
}
__device__ __forceinline__ uint32_t ld_relaxed(const uint32_t *ptr) {
  cuda::atomic_ref<uint32_t, cuda::thread_scope_device> r(*const_cast<uint32_t *>(ptr));
  return r.load(cuda::memory_order_relaxed);
}
__device__ __forceinline__ void add_release(uint32_t *ptr, uint32_t v) {
  cuda::atomic_ref<uint32_t, cuda::thread_scope_device> r(*ptr);
  r.fetch_add(v, cuda::memory_order_release);
}
__device__ __forceinline__ uint4 ldcg_u128(const void *ptr) { return __ldcg(static_cast<const uint4 *>(ptr)); }
// Five 16-byte loads (L2, not L1) in one statement, so that they issue back
// to back: under the kernel's register budget the compiler otherwise places
// uses (or stores) of the first loads between them and serialises the round
// trips.
__device__ __forceinline__ void ldcg_f32x4x5(float4 *v, const float4 *p0, const float4 *p1, const float4 *p2,
                                             const float4 *p3, const float4 *p4) {
  asm volatile(
      "ld.global.cg.v4.f32 {%0, %1, %2, %3}, [%20];\n\t"
      "ld.global.cg.v4.f32 {%4, %5, %6, %7}, [%21];\n\t"
      "ld.global.cg.v4.f32 {%8, %9, %10, %11}, [%22];\n\t"
      "ld.global.cg.v4.f32 {%12, %13, %14, %15}, [%23];\n\t"
      "ld.global.cg.v4.f32 {%16, %17, %18, %19}, [%24];"
      : "=f"(v[0].x), "=f"(v[0].y), "=f"(v[0].z), "=f"(v[0].w), "=f"(v[1].x), "=f"(v[1].y), "=f"(v[1].z),
        "=f"(v[1].w), "=f"(v[2].x), "=f"(v[2].y), "=f"(v[2].z), "=f"(v[2].w), "=f"(v[3].x), "=f"(v[3].y),
        "=f"(v[3].z), "=f"(v[3].w), "=f"(v[4].x), "=f"(v[4].y), "=f"(v[4].z), "=f"(v[4].w)
      : "l"(p0), "l"(p1), "l"(p2), "l"(p3), "l"(p4)
      : "memory");
}
__device__ __forceinline__ void ldcg_u128x5(uint4 (&v)[5], const void *p0, const void *p1, const void *p2,
                                            const void *p3, const void *p4) {
  asm volatile(
      "ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%20];\n\t"
      "ld.global.cg.v4.u32 {%4, %5, %6, %7}, [%21];\n\t"
      "ld.global.cg.v4.u32 {%8, %9, %10, %11}, [%22];\n\t"
      "ld.global.cg.v4.u32 {%12, %13, %14, %15}, [%23];\n\t"
      "ld.global.cg.v4.u32 {%16, %17, %18, %19}, [%24];"
      : "=r"(v[0].x), "=r"(v[0].y), "=r"(v[0].z), "=r"(v[0].w), "=r"(v[1].x), "=r"(v[1].y), "=r"(v[1].z),
        "=r"(v[1].w), "=r"(v[2].x), "=r"(v[2].y), "=r"(v[2].z), "=r"(v[2].w), "=r"(v[3].x), "=r"(v[3].y),
        "=r"(v[3].z), "=r"(v[3].w), "=r"(v[4].x), "=r"(v[4].y), "=r"(v[4].z), "=r"(v[4].w)
      : "l"(p0), "l"(p1), "l"(p2), "l"(p3), "l"(p4)
      : "memory");
}
__device__ __forceinline__ int seq_of(int b, int ph) { return 1 + b * kMkPhases + ph; }

// Bounded spin: gives up (recording WF_DEV_ERR_TIMEOUT) after `limit` cycles
// (MkParams::spin), or at once when another thread of the grid has already
// given up.
struct Spin {
  long long limit;
  long long t0 = 0;
  int it = 0;
  __device__ __forceinline__ explicit Spin(long long lim) : limit(lim) {}
  __device__ __forceinline__ bool again(uint32_t *err) {
    if (it == 0) t0 = clock64();
    ++it;
    if ((it & 31) == 0) {
      if (ld_relaxed(err) & WF_DEV_ERR_TIMEOUT) return false;
      if (clock64() - t0 > limit) {
        set_error(err, WF_DEV_ERR_TIMEOUT);
        return false;
      }
    }
    return true;
  }
};
// One thread waits (acquire) until *ctr >= target.
__device__ __forceinline__ void wait_ge(const uint32_t *ctr, uint32_t target, uint32_t *err,
                                        long long limit) {
  Spin sp(limit);
  while (ld_acquire(ctr) < target && sp.again(err)) __nanosleep(100);
}
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t parity, uint32_t *err, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  Spin sp(limit);
  while (!mbar_try_wait(bar, parity))
    if (!sp.again(err)) return false;
  return true;
}
// The producer's wait for a free slot backs off between tries, leaving the
// issue slots of its scheduler to the two compute warps that share it.
__device__ __forceinline__ bool wait_bar_idle(uint64_t *bar, uint32_t parity, uint32_t *err,
                                              long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  Spin sp(limit);
  while (!mbar_try_wait(bar, parity)) {
    if (!sp.again(err)) return false;
    __nanosleep(64);
  }
  return true;
}
__device__ __forceinline__ void mbar_arrive1(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void cbar() {  // the compute warps only
  asm volatile("bar.sync 1, %0;" ::"n"(kCThr) : "memory");
}

// ------------------------------------------------------------ geometry ----
// Units per phase, recomputed from the parameters where needed (cheap integer
// arithmetic on kernel parameters keeps no registers live across phases).
__device__ __forceinline__ int n_chunks(const MkParams &p) { return (p.T + 255) / 256; }
__device__ __forceinline__ int fc2_k(const MkParams &p) { return p.F / kQ2; }
__device__ __forceinline__ int units_of(const MkParams &p, int ph) {
  switch (ph) {
    case PH_QKV: return 3 * p.d / 8;
    case PH_SATT: return p.n_seq * p.H;
    case PH_XATT: return p.n_seq * p.H * n_chunks(p);
    case PH_FC1: return p.F / 8;
    case PH_FC2: return p.d / 8 * kQ2;
    default: return p.d / 8;  // out, cross-query, cross-out
  }
}
// First unit of phase `ph` of block b dealt to CTA c (units go round robin,
// continuing across phases and blocks).
__device__ __forceinline__ int first_unit(const MkParams &p, int b, int ph, int c) {
  int pre = 0, per_block = 0;
#pragma unroll
  for (int i = 0; i < kMkPhases; ++i) {
    const int u = units_of(p, i);
    if (i < ph) pre += u;
    per_block += u;
  }
  const long long off = (static_cast<long long>(b) * per_block + pre) % p.G;
  return static_cast<int>((c - off + p.G) % p.G);
}
__device__ __forceinline__ bool is_gemm(int ph) { return ph != PH_SATT && ph != PH_XATT; }

// Shared memory: the ring, the scratch area, the ring's mbarriers and a few
// per-CTA values, at fixed offsets from one 1024-aligned base.
constexpr int kOffScratch = kNS * kSlot;
constexpr int kOffLnGB = kOffScratch + kScratch;
constexpr int kOffFull = kOffLnGB + kLnGB;
constexpr int kOffEmpty = kOffFull + kNS * 8;
constexpr int kOffNk = kOffEmpty + kNS * 8;                 // int[kMkMaxSeq]
constexpr int kOffSlot = kOffNk + kMkMaxSeq * 4;            // int[kMkMaxSeq]
constexpr int kOffZero = (kOffSlot + kMkMaxSeq * 4 + 15) / 16 * 16;  // 16 zero bytes (operand rows >= M)
constexpr int kOffIssued = kOffZero + 16;                  // uint32: ring copies the producer requested
constexpr int kOffParams = kOffIssued + 16;                // MkParams (a copy of the launch's)
constexpr int kSmemUsed = kOffParams + (static_cast<int>(sizeof(MkParams)) + 15) / 16 * 16;
static_assert(kSmemUsed + 1024 <= kSmemMk, "shared-memory plan");
struct Smem {
  uint8_t *base;
  __device__ __forceinline__ uint8_t *ring() const { return base; }
  __device__ __forceinline__ uint8_t *scratch() const { return base + kOffScratch; }
  __device__ __forceinline__ uint64_t *full(int s) const { return reinterpret_cast<uint64_t *>(base + kOffFull) + s; }
  __device__ __forceinline__ uint64_t *empty(int s) const { return reinterpret_cast<uint64_t *>(base + kOffEmpty) + s; }
  __device__ __forceinline__ int *nk() const { return reinterpret_cast<int *>(base + kOffNk); }
  __device__ __forceinline__ int *slot() const { return reinterpret_cast<int *>(base + kOffSlot); }
  __device__ __forceinline__ uint8_t *zero16() const { return base + kOffZero; }
  __device__ __forceinline__ bf16 *lngb() const { return reinterpret_cast<bf16 *>(base + kOffLnGB); }
  __device__ __forceinline__ MkParams *params() const { return reinterpret_cast<MkParams *>(base + kOffParams); }
  __device__ __forceinline__ uint32_t *issued() const { return reinterpret_cast<uint32_t *>(base + kOffIssued); }
};

// ------------------------------------------------------------ producer ----
__device__ void producer(const MkParams &p, const Smem sm, int c) {
  uint32_t sc = 0;
  bool ok = true;
  auto acquire = [&](uint32_t bytes, uint8_t *&dst, uint64_t *&bar) {
    const uint32_t s = sc % kNS, n = sc / kNS;
    if (n > 0 && !wait_bar_idle(sm.empty(s), (n - 1) & 1u, p.err, p.spin)) {
      ok = false;
      return;
    }
    bar = sm.full(s);
    dst = sm.ring() + static_cast<size_t>(s) * kSlot;
    mbar_arrive_expect_tx(bar, bytes);
    ++sc;
  };
  tma_prefetch_desc(p.tmaps + p.tm_kc);
  tma_prefetch_desc(p.tmaps + p.tm_vc);
  tma_prefetch_desc(p.tmaps + p.tm_xk);
  tma_prefetch_desc(p.tmaps + p.tm_xv);
  for (int b = 0; b < p.nl && ok; ++b) {
    const MkLayer &ly = p.layers[b];
    if (b + 1 < p.nl)  // the next block's weight descriptors
      for (int k = 0; k < 6; ++k) tma_prefetch_desc(p.tmaps + p.layers[b + 1].tm[k]);
    for (int ph = 0; ph < kMkPhases && ok; ++ph) {
      const int U = units_of(p, ph);
      for (int u = first_unit(p, b, ph, c); u < U && ok; u += p.G) {
        if (is_gemm(ph)) {
          const int wi = ph == PH_QKV ? 0 : ph == PH_OUT ? 1 : ph == PH_XQ ? 2 : ph == PH_XOUT ? 3
                                                                 : ph == PH_FC1 ? 4 : 5;
          const CUtensorMap *tm = p.tmaps + ly.tm[wi];
          int ru = u, k0 = 0, Kp = p.d;
          if (ph == PH_FC2) {
            ru = u / kQ2;
            k0 = (u % kQ2) * fc2_k(p);
            Kp = fc2_k(p);
          }
          // the whole unit (8 rows x Kp) in one copy
          uint8_t *dst;
          uint64_t *bar;
          acquire(static_cast<uint32_t>(8 * Kp * 2), dst, bar);
          if (ok) tma_load_3d(dst, tm, 0, 8 * ru, k0 / 64, bar);
        } else if (ph == PH_SATT) {
          const int i = u / p.H, h = u % p.H;
          const int nk = sm.nk()[i];
          const int row0 = ((ly.self_layer * p.Bmax + sm.slot()[i]) * p.H + h) * p.ctx;
          for (int ch = 0; ch * 256 < nk && ok; ++ch) {
            // keys, then values, of one 256-key block: 128 keys per copy, only
            // the halves that hold visible keys
            const int nh = (min(256, nk - ch * 256) + kKeysPerSlot - 1) / kKeysPerSlot;
            for (int kv = 0; kv < 2 && ok; ++kv)
              for (int hf = 0; hf < nh && ok; ++hf) {
                uint8_t *dst;
                uint64_t *bar;
                acquire(kKeysPerSlot * 128, dst, bar);
                if (ok)
                  tma_load_2d(dst, p.tmaps + (kv ? p.tm_vc : p.tm_kc), 0, row0 + ch * 256 + hf * kKeysPerSlot, bar);
              }
          }
        } else {  // PH_XATT: handled below, in two sweeps
          break;
        }
      }
      if (ph == PH_XATT) {
        // blocks 1.. first, then the merging block-0 units (as the consumer does)
        for (int sweep = 0; sweep < 2 && ok; ++sweep)
          for (int u = first_unit(p, b, ph, c); u < U && ok; u += p.G) {
          const int hu = u / n_chunks(p), cc = u % n_chunks(p);
          if ((cc == 0) != (sweep == 1)) continue;
          const int i = hu / p.H, h = hu % p.H;
          const int row0 = ((ly.cross_layer * p.Bmax + sm.slot()[i]) * p.H + h) * p.T;
          const int nh = (min(256, p.T - cc * 256) + kKeysPerSlot - 1) / kKeysPerSlot;
          for (int kv = 0; kv < 2 && ok; ++kv)
            for (int hf = 0; hf < nh && ok; ++hf) {
              uint8_t *dst;
              uint64_t *bar;
              acquire(kKeysPerSlot * 128, dst, bar);
              if (ok) tma_load_2d(dst, p.tmaps + (kv ? p.tm_xv : p.tm_xk), 0, row0 + cc * 256 + hf * kKeysPerSlot, bar);
            }
        }
      }
    }
  }
  *sm.issued() = sc;  // copies requested, for the drain at the end of the kernel
}


// ------------------------------------------------------------ consumer ----
struct Cons {
  const MkParams &p;
  const Smem sm;
  int c, warp, lane, tid;
  uint32_t rs, rp;  // ring cursor, advanced identically by every compute warp

  __device__ Cons(const MkParams &pp, const Smem s) : p(pp), sm(s) {
    refresh();
    rs = 0;
    rp = 0;
  }
  // Re-read the thread and CTA indices through volatile asm at the start of
  // every phase: values derived from them (addresses, unit lists) are then
  // recomputed per phase instead of being hoisted out of the block loop,
  // where they would stay live across all eight phases and spill.
  __device__ __forceinline__ void refresh() {
    asm volatile("mov.u32 %0, %%tid.x;" : "=r"(tid));
    asm volatile("mov.u32 %0, %%ctaid.x;" : "=r"(c));
    warp = tid >> 5;
    lane = tid & 31;
  }

  // Ring cursor: slot rs of lap parity rp is the next one to consume.  Slot
  // m ahead of the cursor (m < kNS) is rs + m, wrapped once at most.
  __device__ __forceinline__ int ahead(int m) const {
    const int s = static_cast<int>(rs) + m;
    return s >= kNS ? s - kNS : s;
  }
  __device__ __forceinline__ uint32_t ahead_par(int m) const {
    return (static_cast<int>(rs) + m >= kNS) ? (rp ^ 1u) : rp;
  }
  __device__ __forceinline__ uint8_t *slot_ptr(int m) const {
    return sm.ring() + static_cast<size_t>(ahead(m)) * kSlot;
  }
  __device__ __forceinline__ void wait_slot(int m) const { wait_bar(sm.full(ahead(m)), ahead_par(m), p.err, p.spin); }
  // The 32-key group gi (0..7) of a 256-key block whose keys fill the first
  // nh slots at the cursor and whose values the next nh.
  __device__ __forceinline__ uint8_t *kgroup(int gi) const { return slot_ptr(gi >> 2) + (gi & 3) * 4096; }
  __device__ __forceinline__ uint8_t *vgroup(int gi, int nh) const {
    return slot_ptr(nh + (gi >> 2)) + (gi & 3) * 4096;
  }
  // Hand the n slots at the cursor back to the producer and advance past them.
  __device__ __forceinline__ void release(int n) {
    __syncwarp();
    if (lane == 0)
      for (int i = 0; i < n; ++i) mbar_arrive1(sm.empty(ahead(i)));
    const int s = static_cast<int>(rs) + n;
    if (s >= kNS) {
      rs = static_cast<uint32_t>(s - kNS);
      rp ^= 1u;
    } else {
      rs = static_cast<uint32_t>(s);
    }
  }

  // -------------------------------------------------- phase completion --
  __device__ __forceinline__ void arrive(int s) {
    cbar();  // every compute thread's stores of the phase are issued
    if (tid == 0) add_release(p.cnt + s, 1u);
  }
  // Wait until every CTA has finished phase s.
  __device__ __forceinline__ void wait_phase(int s) {
    if (tid == 0) wait_ge(p.cnt + s, static_cast<uint32_t>(p.G), p.err, p.spin);
    cbar();
  }

  // ---------------------------------------------------------- embedding --
  // Target rows: Emb(tok) + PosEmb(L + j); drafter rows (Eq. 2): Emb(anchor),
  // then the mask vector m.  Row t is built by CTA t.
  __device__ __noinline__ void embed() {
    const int t = c;
    if (t >= p.M) return;
    const int i = t / p.rps, j = t - i * p.rps;
    const int slot = sm.slot()[i];
    int tok = 0;
    if (j == 0) {
      tok = p.anchor[slot];
    } else if (!p.drafter) {
      tok = p.forced ? p.forced[slot * p.K + j - 1] : p.cand_in[slot * p.K + j - 1];
      if (tid == 0 && p.cand_out) p.cand_out[slot * p.K + j - 1] = tok;
    }
    const bool use_mask = p.drafter && j > 0;
    if (!use_mask && (tok < 0 || tok >= p.vocab)) {
      if (tid == 0) set_error(p.err, WF_DEV_ERR_TOKEN);
      tok = tok < 0 ? 0 : p.vocab - 1;
    }
    const int pos = p.drafter ? 0 : min(p.L[slot] + j, p.ctx - 1);  // past ctx: error already recorded
    for (int e2 = tid; e2 < p.d / 2; e2 += kCThr) {
      const int e = 2 * e2;
      float v0, v1;
      if (use_mask) {
        v0 = bf2f(p.mask_emb[e]);
        v1 = bf2f(p.mask_emb[e + 1]);
      } else {
        v0 = bf2f(p.tok_emb[static_cast<size_t>(tok) * p.d + e]);
        v1 = bf2f(p.tok_emb[static_cast<size_t>(tok) * p.d + e + 1]);
        if (!p.drafter) {
          v0 += bf2f(p.pos_emb[static_cast<size_t>(pos) * p.d + e]);
          v1 += bf2f(p.pos_emb[static_cast<size_t>(pos) * p.d + e + 1]);
        }
      }
      *reinterpret_cast<float2 *>(p.x + static_cast<size_t>(t) * p.d + e) = make_float2(v0, v1);
    }
  }

  // ------------------------------------------------- token operand (A) ----
  // Warp w owns k16-steps s = w, w + 8, ... of the operand; lane (g, c4)
  // holds rows g and g + 8, columns 16s + 2c4 (+1, +8, +9) as in the
  // m16n8k16 A fragment.
  // LayerNorm operand: LN(x) as a bf16 tile [M][d] in shared memory (rows
  // >= M read zeros), from which every warp reads its A fragments with
  // ldmatrix.  Warp w normalises rows w and w + 8; lane l holds float4s
  // l + 32 j of a row, so a row's sums run in one fixed order (the lane's
  // elements, then the shuffle tree, whose result is the same in every lane)
  // whatever M is: a row's result never depends on the other rows.
  static constexpr int kLnJ = 10;  // float4s per lane and row (d <= 1280)
  // The LayerNorm's gain and bias go to shared memory before the phase
  // waits: they do not depend on the previous phase.
  __device__ __forceinline__ void stage_ln(const bf16 *lg, const bf16 *lb) {
    uint4 *dst = reinterpret_cast<uint4 *>(sm.lngb());
    const int n = p.d / 8;
    for (int i = tid; i < 2 * n; i += kCThr)
      dst[i] = i < n ? __ldg(reinterpret_cast<const uint4 *>(lg) + i)
                     : __ldg(reinterpret_cast<const uint4 *>(lb) + (i - n));
  }
  // Four independent running sums (one per float4 component), added in a
  // fixed order: short dependency chains, same result for any M.
  __device__ __forceinline__ float2 row_stats(const float4 (&v)[kLnJ], int nj, float inv_d, float eps) const {
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
    for (int j = 0; j < kLnJ; ++j) {
      if (j < nj) {
        s0 += v[j].x;
        s1 += v[j].y;
        s2 += v[j].z;
        s3 += v[j].w;
      }
    }
    const float mean = warp_sum((s0 + s1) + (s2 + s3)) * inv_d;
    float q0 = 0.f, q1 = 0.f, q2 = 0.f, q3 = 0.f;
#pragma unroll
    for (int j = 0; j < kLnJ; ++j) {
      if (j < nj) {
        const float a = v[j].x - mean, b = v[j].y - mean, c2 = v[j].z - mean, d2 = v[j].w - mean;
        q0 = __fmaf_rn(a, a, q0);
        q1 = __fmaf_rn(b, b, q1);
        q2 = __fmaf_rn(c2, c2, q2);
        q3 = __fmaf_rn(d2, d2, q3);
      }
    }
    return make_float2(mean, rsqrtf(__fadd_rn(warp_sum((q0 + q1) + (q2 + q3)) * inv_d, eps)));
  }
  __device__ __forceinline__ void row_out(bf16 *trow, const float4 (&v)[kLnJ], int nj, float2 ms) const {
    const bf16 *g = sm.lngb(), *bb = sm.lngb() + p.d;
#pragma unroll
    for (int j = 0; j < kLnJ; ++j) {
      if (j < nj) {
        const int col = 4 * (lane + 32 * j);
        const uint2 gr = *reinterpret_cast<const uint2 *>(g + col);
        const uint2 br = *reinterpret_cast<const uint2 *>(bb + col);
        const bf16 *ge = reinterpret_cast<const bf16 *>(&gr);
        const bf16 *be = reinterpret_cast<const bf16 *>(&br);
        uint2 o;
        o.x = pack_bf16(ln_apply(v[j].x, ms, bf2f(ge[0]), bf2f(be[0])), ln_apply(v[j].y, ms, bf2f(ge[1]), bf2f(be[1])));
        o.y = pack_bf16(ln_apply(v[j].z, ms, bf2f(ge[2]), bf2f(be[2])), ln_apply(v[j].w, ms, bf2f(ge[3]), bf2f(be[3])));
        *reinterpret_cast<uint2 *>(trow + col) = o;
      }
    }
  }
  // Row t of the residual: lane l's float4s l + 32 j, j < nj (those past the
  // row repeat its last and are never used), all ten loads in flight at once.
  __device__ __forceinline__ void load_row(float4 (&v)[kLnJ], int t, int nj) const {
    static_assert(kLnJ == 10, "two groups of five loads");
    const float4 *xr = reinterpret_cast<const float4 *>(p.x + static_cast<size_t>(t) * p.d) + lane;
    auto at = [&](int j) { return xr + 32 * min(j, nj - 1); };
    ldcg_f32x4x5(v, at(0), at(1), at(2), at(3), at(4));
    ldcg_f32x4x5(v + 5, at(5), at(6), at(7), at(8), at(9));
  }
  __device__ __forceinline__ void ln_tile() {
    static_assert(kMkRows <= 2 * kW, "two rows per warp at most");
    if (warp >= p.M) return;
    bf16 *tile = reinterpret_cast<bf16 *>(sm.scratch());
    const int nj = p.d / 128, ld = p.d + 8, t1 = warp + kW;
    const float inv_d = 1.0f / static_cast<float>(p.d), eps = p.eps;
    float4 v0[kLnJ], v1[kLnJ];
    load_row(v0, warp, nj);
    // both rows in flight together (a lone row loads itself twice), and
    // both statistics computed side by side
    load_row(v1, t1 < p.M ? t1 : warp, nj);
    const float2 ms0 = row_stats(v0, nj, inv_d, eps), ms1 = row_stats(v1, nj, inv_d, eps);
    row_out(tile + warp * ld, v0, nj, ms0);
    if (t1 < p.M) row_out(tile + t1 * ld, v1, nj, ms1);
  }
  // bf16 operand: rows [0, M), columns [k0, k0 + Kp) of buf (row stride
  // cols) copied into the tile with 16-byte loads, warp w taking rows w and
  // w + 8, every load in flight before the first store.
  static constexpr int kPlainJ = 5;  // uint4 per lane and row (Kp <= 1280)
  __device__ __forceinline__ void plain_tile(const bf16 *buf, int cols, int k0, int Kp) {
    if (warp >= p.M) return;
    bf16 *tile = reinterpret_cast<bf16 *>(sm.scratch());
    const int ld = Kp + 8, per = Kp / 8;
    const int r1 = warp + 8 < p.M ? warp + 8 : warp;
    const bf16 *s0 = buf + static_cast<size_t>(warp) * cols + k0;
    const bf16 *s1 = buf + static_cast<size_t>(r1) * cols + k0;
    static_assert(kPlainJ == 5, "five loads per row");
    // columns past the row read its last chunk (valid) and are not stored
    auto col = [&](int j) { return 8 * min(lane + 32 * j, per - 1); };
    uint4 v0[kPlainJ], v1[kPlainJ];
    ldcg_u128x5(v0, s0 + col(0), s0 + col(1), s0 + col(2), s0 + col(3), s0 + col(4));
    ldcg_u128x5(v1, s1 + col(0), s1 + col(1), s1 + col(2), s1 + col(3), s1 + col(4));
#pragma unroll
    for (int j = 0; j < kPlainJ; ++j) {
      const int q = lane + 32 * j;
      if (q < per) {
        *reinterpret_cast<uint4 *>(tile + warp * ld + 8 * q) = v0[j];
        if (r1 != warp) *reinterpret_cast<uint4 *>(tile + r1 * ld + 8 * q) = v1[j];
      }
    }
  }
  // A fragments of k-steps s = w + 8 j from the shared tile of row stride ld
  // (rows >= M read zeros).
  __device__ __forceinline__ void tile_frags(uint32_t (&a)[kKS][4], int nks, int ld) {
    const bf16 *tile = reinterpret_cast<const bf16 *>(sm.scratch());
    const int row = lane & 15, koff = (lane >> 4) * 8;
    const uint32_t rbase = row < p.M ? smem_u32(tile + row * ld + 16 * warp + koff) : smem_u32(sm.zero16());
    const uint32_t rstep = row < p.M ? 256u : 0u;  // 128 bf16 per j
#pragma unroll
    for (int j = 0; j < kKS; ++j) {
      if (j >= nks) continue;
      ldsm_x4(rbase + rstep * j, a[j][0], a[j][1], a[j][2], a[j][3]);
    }
  }

  // ------------------------------------------------------- projections ----
  // Phases are separate (non-inlined) functions: inlined into the block loop
  // their live ranges add up past the register budget of a 288-thread CTA.
  __device__ __noinline__ void gemm_phase(int b, const int PH) {
    refresh();
    const int U = units_of(p, PH);
    const int u0 = first_unit(p, b, PH, c);
    const int s = seq_of(b, PH);
    if (u0 >= U) {
      arrive(s);
      return;
    }
    const MkLayer &ly = p.layers[b];
    const bool ln = PH == PH_QKV || PH == PH_XQ || PH == PH_FC1;
    if (ln)
      stage_ln(PH == PH_QKV ? ly.ln1_g : PH == PH_XQ ? ly.ln2_g : ly.ln3_g,
               PH == PH_QKV ? ly.ln1_b : PH == PH_XQ ? ly.ln2_b : ly.ln3_b);
    // Thread tid finishes unit u0 + (tid / 32) G (if any): its bias pair is
    // loaded before the wait, the residual it updates right after it, both
    // in the shadow of the operand loads.
    const int eu = u0 + (tid >> 5) * p.G;
    const bool epi = (tid >> 5) < kUB && eu < U;
    const int en0 = 8 * (PH == PH_FC2 ? eu / kQ2 : eu) + 2 * (lane & 3);
    const bool resid = PH == PH_OUT || PH == PH_XOUT || (PH == PH_FC2 && u0 % kQ2 == 0);
    uint32_t bias2 = 0u;
    if (epi && (PH != PH_FC2 || resid)) {
      const bf16 *bias = PH == PH_QKV ? ly.qkv_b : PH == PH_OUT ? ly.out_b : PH == PH_XQ ? ly.xq_b
                       : PH == PH_XOUT ? ly.xout_b : PH == PH_FC1 ? ly.fc1_b : ly.fc2_b;
      bias2 = __ldg(reinterpret_cast<const unsigned int *>(bias + en0));
    }
    wait_phase(s - 1);  // its barrier also publishes the staged gain and bias
    float2 old[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
    if (epi && resid) {
#pragma unroll
      for (int hr = 0; hr < 2; ++hr) {
        const int t = (lane >> 2) + 8 * hr;
        if (t < p.M) old[hr] = __ldcg(reinterpret_cast<const float2 *>(p.x + static_cast<size_t>(t) * p.d + en0));
      }
    }
    const int Kp = PH == PH_FC2 ? fc2_k(p) : p.d;
    const int nks = Kp / 128;  // k16-steps per warp
    const int nslot = (Kp + 255) / 256;
    uint32_t a[kKS][4];
    if (ln)
      ln_tile();
    else  // G is a multiple of the fc2 split (checked at launch), so every fc2
          // unit of this CTA reads the same quarter of the fc1 output
      plain_tile(PH == PH_OUT ? p.att_x : PH == PH_XOUT ? p.xatt_x : p.h_x, PH == PH_FC2 ? p.F : p.d,
                 PH == PH_FC2 ? (u0 % kQ2) * Kp : 0, Kp);
    cbar();
    tile_frags(a, nks, Kp + 8);
    cbar();  // the reduction buffer of the projection overlaps the tile
    // ldmatrix addressing inside a unit: k-block atoms of [8 rows][64] bf16,
    // 128-byte swizzled; warp w's k-steps 16m + w and 16m + w + 8 sit in the
    // 4 KB (four k-blocks) at 4096 m
    const int lr = lane & 7, mi = lane >> 3;
    const int kb = (warp >> 2) + ((mi >> 1) << 1);
    const int ch = 2 * (warp & 3) + (mi & 1);
    const uint32_t ld_off = static_cast<uint32_t>(kb * 1024 + lr * 128 + ((ch ^ lr) << 4));
    float4 *red = reinterpret_cast<float4 *>(sm.scratch());
    {  // every unit of the CTA in one batch (at most kUB, checked at launch)
      const int ub = u0;
      float acc[kUB][4];
      int nb = 0;
#pragma unroll
      for (int k = 0; k < kUB; ++k) {
        acc[k][0] = acc[k][1] = acc[k][2] = acc[k][3] = 0.f;
        const int u = ub + k * p.G;
        if (u >= U) continue;
        nb = k + 1;
        wait_slot(0);
        const uint32_t ubase = smem_u32(slot_ptr(0)) + ld_off;
#pragma unroll
        for (int m = 0; m < kKS / 2; ++m) {
          if (m >= nslot) break;
          uint32_t b0, b1, b2, b3;
          ldsm_x4(ubase + 4096u * m, b0, b1, b2, b3);
          if (2 * m < nks) mma_bf16(acc[k], a[2 * m][0], a[2 * m][1], a[2 * m][2], a[2 * m][3], b0, b1);
          if (2 * m + 1 < nks)
            mma_bf16(acc[k], a[2 * m + 1][0], a[2 * m + 1][1], a[2 * m + 1][2], a[2 * m + 1][3], b2, b3);
        }
        release(1);
      }
#pragma unroll
      for (int k = 0; k < kUB; ++k)
        if (k < nb) red[(k * kW + warp) * 32 + lane] = make_float4(acc[k][0], acc[k][1], acc[k][2], acc[k][3]);
      cbar();
      if (PH == PH_FC2) {
        // a quarter-0 unit owns the output: wait for the other quarters'
        // partials (every fc2 unit of this CTA has the same quarter)
        if (u0 % kQ2 == 0) {
          if (tid == 0)
            for (int k = 0; k < nb; ++k)
              wait_ge(p.cnt2 + (ub + k * p.G) / kQ2, static_cast<uint32_t>((kQ2 - 1) * (b + 1)), p.err, p.spin);
          cbar();
        }
      }
      if (tid < nb * 32) {
        const int k = tid >> 5, ln = tid & 31;
        float4 v = red[(k * kW) * 32 + ln];
#pragma unroll
        for (int ww = 1; ww < kW; ++ww) {
          const float4 o = red[(k * kW + ww) * 32 + ln];
          v.x += o.x;
          v.y += o.y;
          v.z += o.z;
          v.w += o.w;
        }
        epilogue(PH, b, ly, ub + k * p.G, ln, v, bias2, old);
      }
      cbar();
      if (PH == PH_FC2) {  // partials of quarters 1..3 are published
        if (u0 % kQ2 != 0 && tid == 0)
          for (int k = 0; k < nb; ++k) add_release(p.cnt2 + (ub + k * p.G) / kQ2, 1u);
      }
    }
    arrive(s);
  }

  // D fragment of one unit: rows g, g+8; columns n0, n0+1 (n0 = 8 ru + 2 c4).
  __device__ __forceinline__ void epilogue(const int PH, int b, const MkLayer &ly, int u, int ln, float4 v,
                                          uint32_t bias2, const float2 (&old)[2]) {
    const float bias0 = __uint_as_float(bias2 << 16), bias1 = __uint_as_float(bias2 & 0xffff0000u);
    const int gr = ln >> 2, c4 = ln & 3;
    const int ru = PH == PH_FC2 ? u / kQ2 : u;
    const int n0 = 8 * ru + 2 * c4;
    const float vals[2][2] = {{v.x, v.y}, {v.z, v.w}};
#pragma unroll
    for (int hr = 0; hr < 2; ++hr) {
      const int t = gr + 8 * hr;
      if (t >= p.M) continue;
      float y0 = vals[hr][0], y1 = vals[hr][1];
      if (PH == PH_QKV) {
        y0 += bias0;
        y1 += bias1;
        const uint32_t pr = pack_bf16(y0, y1);
        if (n0 < p.d) {
          *reinterpret_cast<uint32_t *>(p.q_x + t * p.d + n0) = pr;
        } else {
          // keys and values go straight into the cache at position L + j
          const int cc = n0 - p.d;
          const int which = cc / p.d, hd = cc - which * p.d;
          const int i = t / p.rps, j = t - i * p.rps;
          const int slot = sm.slot()[i];
          const int pos = p.L[slot] + j;
          if (pos < p.ctx) {
            bf16 *dst = (which == 0 ? p.kc : p.vc) +
                        ((static_cast<size_t>(ly.self_layer * p.Bmax + slot) * p.H + (hd >> 6)) * p.ctx + pos) * 64 +
                        (hd & 63);
            *reinterpret_cast<uint32_t *>(dst) = pr;
          } else {
            set_error(p.err, WF_DEV_ERR_CAPACITY);
          }
        }
      } else if (PH == PH_XQ) {
        y0 += bias0;
        y1 += bias1;
        *reinterpret_cast<uint32_t *>(p.xq_x + t * p.d + n0) = pack_bf16(y0, y1);
      } else if (PH == PH_FC1) {
        y0 = gelu_erf(y0 + bias0);
        y1 = gelu_erf(y1 + bias1);
        *reinterpret_cast<uint32_t *>(p.h_x + t * p.F + n0) = pack_bf16(y0, y1);
      } else {
        // residual updates: OUT, XOUT, FC2
        if (PH == PH_FC2) {
          const int q = u % kQ2;
          float *pp = p.part2 + (static_cast<size_t>(ru) * (kQ2 - 1) * kMkRows) * 8;
          if (q != 0) {
            *reinterpret_cast<float2 *>(pp + ((q - 1) * kMkRows + t) * 8 + 2 * c4) = make_float2(y0, y1);
            continue;
          }
          // owner: the other quarters' partials, added in order
#pragma unroll
          for (int qq = 1; qq < kQ2; ++qq) {
            const float2 pq = __ldcg(reinterpret_cast<const float2 *>(pp + ((qq - 1) * kMkRows + t) * 8 + 2 * c4));
            y0 += pq.x;
            y1 += pq.y;
          }
        }
        float *xo = p.x + static_cast<size_t>(t) * p.d + n0;
        const float x0 = old[hr].x + (y0 + bias0);
        const float x1 = old[hr].y + (y1 + bias1);
        *reinterpret_cast<float2 *>(xo) = make_float2(x0, x1);
        if (PH == PH_FC2) {
          if (p.write_taps) {
            const uint32_t pr = pack_bf16(x0, x1);
#pragma unroll
            for (int k = 0; k < 2; ++k)
              if (ly.tap[k] >= 0)
                *reinterpret_cast<uint32_t *>(p.taps + static_cast<size_t>(t) * p.ld_tap +
                                              ly.tap[k] * p.d + n0) = pr;
          }
        }
      }
    }
  }

  // --------------------------------------------------------- attention ----
  // Scratch: query tile [16][64] bf16 (swizzled), per-warp (m, l) and O.
  __device__ __forceinline__ uint8_t *sQ() const { return sm.scratch(); }
  __device__ __forceinline__ float *sMax() const { return reinterpret_cast<float *>(sm.scratch() + 2048); }
  __device__ __forceinline__ float *sSum() const { return reinterpret_cast<float *>(sm.scratch() + 2560); }
  // per-warp O partials, rows padded to 72 floats: the fragment stores of
  // one half-warp fall in distinct banks
  static constexpr int kOLd = 72;
  static_assert(3072 + kW * 16 * kOLd * 4 <= kScratch, "attention scratch");
  // Scores are kept in base-2 units (times log2 e), so every weight of the
  // softmax, and of the merges of partial results, is one exp2.
  static constexpr float kLog2e = 1.4426950408889634f;
  __device__ __forceinline__ float *sO() const { return reinterpret_cast<float *>(sm.scratch() + 3072); }

  // Query rows of unit (sequence i, head h) of buf [rows][d], scaled by
  // 1/8 = 1/sqrt(64) after RoPE (drafter) in fp32.
  __device__ __noinline__ void load_q(const bf16 *buf, int i, int h, int base, bool rope) {
    if (tid < 16 * 8) {
      const int r = tid >> 3, chq = tid & 7;
      uint4 raw = make_uint4(0u, 0u, 0u, 0u), par = make_uint4(0u, 0u, 0u, 0u);
      if (r < p.rps) {
        const bf16 *row = buf + (i * p.rps + r) * p.d + h * 64;
        raw = ldcg_u128(row + chq * 8);
        if (rope) par = ldcg_u128(row + (chq ^ 4) * 8);  // the RoPE partner dims (d ^ 32)
      }
      const bf16 *qv = reinterpret_cast<const bf16 *>(&raw);
      const bf16 *qp = reinterpret_cast<const bf16 *>(&par);
      float f[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        float v = bf2f(qv[e]);
        if (rope && r < p.rps) {
          const int dd = chq * 8 + e;
          const float2 cs = __ldg(p.rope_tab + (base + r) * 32 + (dd & 31));
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
      *reinterpret_cast<uint4 *>(sQ() + swz(r, chq)) = o;
    }
  }

  // One warp: 16 query rows x the 32 keys of slot pair (k_u32, v_u32), keys
  // at absolute positions key0 .. key0 + 31; a key is visible when
  // pos < nk and, for causal rows, pos <= cbase + row.  Leaves the warp's
  // (m, l, O) in scratch.
  __device__ __noinline__ void attn_warp(bool active, uint32_t k_u32, uint32_t v_u32, int key0, int nk, int nq,
                            int cbase) {
    float *smx = sMax(), *ssm = sSum(), *so = sO();
    const int gq = lane >> 2, c4 = lane & 3;
    if (!active) {
      if (c4 == 0) {
        smx[warp * 16 + gq] = -INFINITY;
        smx[warp * 16 + gq + 8] = -INFINITY;
        ssm[warp * 16 + gq] = 0.f;
        ssm[warp * 16 + gq + 8] = 0.f;
      }
#pragma unroll
      for (int nd = 0; nd < 8; ++nd) {
        float *o0 = so + (warp * 16 + gq) * kOLd + nd * 8 + c4 * 2;
        float *o1 = so + (warp * 16 + gq + 8) * kOLd + nd * 8 + c4 * 2;
        *reinterpret_cast<float2 *>(o0) = make_float2(0.f, 0.f);
        *reinterpret_cast<float2 *>(o1) = make_float2(0.f, 0.f);
      }
      return;
    }
    const uint32_t q_u32 = smem_u32(sQ());
    float s[4][4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
      uint32_t a0, a1, a2, a3;
      const int mi = lane >> 3;
      ldsm_x4(q_u32 + swz((mi & 1) * 8 + (lane & 7), 2 * ks + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
      for (int np = 0; np < 2; ++np) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4(k_u32 + swz(np * 16 + (mi >> 1) * 8 + (lane & 7), 2 * ks + (mi & 1)), b0, b1, b2, b3);
        mma_bf16(s[2 * np], a0, a1, a2, a3, b0, b1);
        mma_bf16(s[2 * np + 1], a0, a1, a2, a3, b2, b3);
      }
    }
    float mrow[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int row = gq + (e >> 1) * 8;
        const int pos = key0 + nt * 8 + c4 * 2 + (e & 1);
        bool vis = row < nq && pos < nk;
        if (cbase >= 0) vis = vis && pos <= cbase + row;
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
    for (int nt = 0; nt < 4; ++nt) {
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
    float o[8][4];
#pragma unroll
    for (int nd = 0; nd < 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      const uint32_t a0 = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      const uint32_t a1 = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      const uint32_t a2 = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      const uint32_t a3 = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int dp = 0; dp < 4; ++dp) {
        uint32_t b0, b1, b2, b3;
        const int mi = lane >> 3;
        ldsm_x4_t(v_u32 + swz(kk * 16 + (mi & 1) * 8 + (lane & 7), 2 * dp + (mi >> 1)), b0, b1, b2, b3);
        mma_bf16(o[2 * dp], a0, a1, a2, a3, b0, b1);
        mma_bf16(o[2 * dp + 1], a0, a1, a2, a3, b2, b3);
      }
    }
    if (c4 == 0) {
      smx[warp * 16 + gq] = mrow[0];
      smx[warp * 16 + gq + 8] = mrow[1];
      ssm[warp * 16 + gq] = lrow[0];
      ssm[warp * 16 + gq + 8] = lrow[1];
    }
#pragma unroll
    for (int nd = 0; nd < 8; ++nd) {
      float *o0 = so + (warp * 16 + gq) * kOLd + nd * 8 + c4 * 2;
      float *o1 = so + (warp * 16 + gq + 8) * kOLd + nd * 8 + c4 * 2;
      *reinterpret_cast<float2 *>(o0) = make_float2(o[nd][0], o[nd][1]);
      *reinterpret_cast<float2 *>(o1) = make_float2(o[nd][2], o[nd][3]);
    }
  }

  // Combine the eight warps in order: thread -> (row qi, dims d0..d0+3).
  __device__ __forceinline__ void combine(float &M, float &L, float (&acc)[4]) const {
    const int qi = tid >> 4, d0 = (tid & 15) * 4;
    const float *smx = sMax(), *ssm = sSum(), *so = sO();
    M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kW; ++w) M = fmaxf(M, smx[w * 16 + qi]);
    L = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[e] = 0.f;
#pragma unroll
    for (int w = 0; w < kW; ++w) {
      const float mw = smx[w * 16 + qi];
      const float wt = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
      L += ssm[w * 16 + qi] * wt;
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[e] += so[(w * 16 + qi) * kOLd + d0 + e] * wt;
    }
  }
  // (Mr, Lr, ar) <- merge with (M, L, a), earlier block first.
  __device__ __forceinline__ static void merge(float &Mr, float &Lr, float (&ar)[4], float M, float L,
                                               const float (&a)[4]) {
    const float MM = fmaxf(Mr, M);
    const float wr = (Mr == -INFINITY) ? 0.f : exp2f(Mr - MM);
    const float wc = (M == -INFINITY) ? 0.f : exp2f(M - MM);
    Lr = __fmaf_rn(L, wc, Lr * wr);
#pragma unroll
    for (int e = 0; e < 4; ++e) ar[e] = __fmaf_rn(a[e], wc, ar[e] * wr);
    Mr = MM;
  }
  __device__ void store_out(bf16 *buf, int i, int h, float L, const float (&acc)[4]) const {
    const int qi = tid >> 4, d0 = (tid & 15) * 4;
    if (qi >= p.rps) return;
    const float inv = 1.0f / L;
    *reinterpret_cast<uint2 *>(buf + (i * p.rps + qi) * p.d + h * 64 + d0) =
        make_uint2(pack_bf16(acc[0] * inv, acc[1] * inv), pack_bf16(acc[2] * inv, acc[3] * inv));
  }
  // Zero value rows [from, 32) of a slot (keys past the end).
  __device__ void zero_rows(uint8_t *slot, int from) const {
    for (int idx = tid; idx < (32 - from) * 8; idx += kCThr) {
      const int r = from + (idx >> 3), chv = idx & 7;
      *reinterpret_cast<uint4 *>(slot + swz(r, chv)) = make_uint4(0u, 0u, 0u, 0u);
    }
  }

  // Self-attention: target rows see positions [0, L + j] (causal verify
  // block), drafter rows see the history [0, L) and the whole block (Eq. 2),
  // with RoPE on queries and keys.  A unit is one (sequence, head); its keys
  // come in 256-key blocks aligned to absolute positions.
  __device__ __noinline__ void satt_phase(int b) {
    refresh();
    const int U = units_of(p, PH_SATT);
    const int u0 = first_unit(p, b, PH_SATT, c);
    const bool rope = p.drafter != 0;
    if (u0 < U) wait_phase(seq_of(b, PH_SATT) - 1);
    for (int u = u0; u < U; u += p.G) {
      const int i = u / p.H, h = u % p.H;
      const int nk = sm.nk()[i];
      const int base = nk - p.rps;
      float Mr = -INFINITY, Lr = 0.f, ar[4] = {0.f, 0.f, 0.f, 0.f};
      const bf16 *kcache = p.kc + (static_cast<size_t>(p.layers[b].self_layer * p.Bmax + sm.slot()[i]) * p.H + h) * p.ctx * 64;
      const bf16 *vcache = p.vc + (kcache - p.kc);
      // This step's rows (positions base .. nk-1) were written by the
      // projection in this pass (the prefetched slots hold stale copies):
      // item tid + 256 r is (row jr, keys or values, 16-byte chunk chv),
      // fetched together with the queries.
      static_assert(kMkRows * 16 <= 2 * kCThr, "two fresh-row items per thread");
      uint4 fresh[2];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int idx = tid + r * kCThr;
        if (nk > 0 && idx < p.rps * 16) {
          const int jr = idx >> 4, kv = (idx >> 3) & 1, chv = idx & 7;
          fresh[r] = ldcg_u128((kv ? vcache : kcache) + static_cast<size_t>(base + jr) * 64 + chv * 8);
        }
      }
      if (nk > 0) load_q(p.q_x, i, h, base, rope);
      for (int ch = 0; ch * 256 < nk; ++ch) {
        const int ng = min(8, (nk - ch * 256 + 31) / 32);
        const int nh = (ng + 3) / 4;  // 128-key halves holding visible keys
        for (int m = 0; m < 2 * nh; ++m) wait_slot(m);
#pragma unroll
        for (int r2 = 0; r2 < 2; ++r2) {
          const int idx = tid + r2 * kCThr;
          if (idx >= p.rps * 16) continue;
          const int jr = idx >> 4, kv = (idx >> 3) & 1, chv = idx & 7;
          const int pos = base + jr;
          if (pos < ch * 256 || pos >= ch * 256 + 256) continue;
          const int gi = (pos - ch * 256) >> 5, r = pos & 31;
          *reinterpret_cast<uint4 *>((kv ? vgroup(gi, nh) : kgroup(gi)) + swz(r, chv)) = fresh[r2];
        }
        if ((nk & 31) && nk <= ch * 256 + 256) zero_rows(vgroup(ng - 1, nh), nk & 31);
        cbar();
        if (rope) {
          for (int idx = tid; idx < ng * 32 * 4; idx += kCThr) {
            const int kr = idx >> 2, cq = idx & 3;
            const int pos = ch * 256 + kr;
            if (pos >= nk) continue;
            uint8_t *ks = kgroup(kr >> 5);
            uint4 *lo = reinterpret_cast<uint4 *>(ks + swz(kr & 31, cq));
            uint4 *hi = reinterpret_cast<uint4 *>(ks + swz(kr & 31, cq + 4));
            uint4 av = *lo, bv = *hi;
            bf16 *ae = reinterpret_cast<bf16 *>(&av);
            bf16 *be = reinterpret_cast<bf16 *>(&bv);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float2 cs = __ldg(p.rope_tab + pos * 32 + cq * 8 + e);
              const float x1 = bf2f(ae[e]), x2 = bf2f(be[e]);
              ae[e] = __float2bfloat16(x1 * cs.x - x2 * cs.y);
              be[e] = __float2bfloat16(x2 * cs.x + x1 * cs.y);
            }
            *lo = av;
            *hi = bv;
          }
          cbar();
        }
        attn_warp(warp < ng, smem_u32(kgroup(warp)), smem_u32(vgroup(warp, nh)), ch * 256 + warp * 32, nk,
                  p.rps, p.drafter ? -1 : base);
        cbar();
        float M, L, a4[4];
        combine(M, L, a4);
        merge(Mr, Lr, ar, M, L, a4);
        fence_proxy_async();
        release(2 * nh);
        cbar();
      }
      if (nk > 0) {
        store_out(p.att_x, i, h, Lr, ar);
      } else {  // past the cache (error recorded): publish zeros so the pass completes
        const float one[4] = {0.f, 0.f, 0.f, 0.f};
        store_out(p.att_x, i, h, 1.f, one);
      }
    }
    arrive(seq_of(b, PH_SATT));
  }

  // Cross-attention over the encoder frames: a unit is one (sequence, head,
  // 256-frame block); the unit of block 0 merges the others' partials in
  // block order.
  __device__ __noinline__ void xatt_phase(int b) {
    refresh();
    const int U = units_of(p, PH_XATT);
    const int u0 = first_unit(p, b, PH_XATT, c);
    if (u0 < U) wait_phase(seq_of(b, PH_XATT) - 1);
    // Blocks 1.. first, then the block-0 units that merge them: a CTA never
    // waits on a merge while it still owes another head a partial.
    for (int sweep = 0; sweep < 2; ++sweep)
    for (int u = u0; u < U; u += p.G) {
      const int hu = u / n_chunks(p), cc = u % n_chunks(p);
      if ((cc == 0) != (sweep == 1)) continue;
      const int i = hu / p.H, h = hu % p.H;
      const int ng = min(8, (p.T - cc * 256 + 31) / 32);
      load_q(p.xq_x, i, h, 0, false);
      const int nh = (ng + 3) / 4;
      for (int m = 0; m < 2 * nh; ++m) wait_slot(m);
      const int valid = p.T - cc * 256;
      if (valid < 256 && (valid & 31)) zero_rows(vgroup(ng - 1, nh), valid & 31);
      cbar();
      attn_warp(warp < ng, smem_u32(kgroup(warp)), smem_u32(vgroup(warp, nh)), cc * 256 + warp * 32, p.T,
                p.rps, -1);
      cbar();
      float M, L, a4[4];
      combine(M, L, a4);
      fence_proxy_async();
      release(2 * nh);
      const int qi = tid >> 4, d0 = (tid & 15) * 4;
      if (n_chunks(p) == 1) {
        store_out(p.xatt_x, i, h, L, a4);
      } else if (cc != 0) {
        // partial (m, l, o) of this frame block, published on the head's counter
        if (qi < p.rps) {
          float *pt = p.xpart + (static_cast<size_t>(u) * kMkRows + qi) * kPS;
          if (d0 == 0) {
            pt[0] = M;
            pt[1] = L;
          }
          *reinterpret_cast<float4 *>(pt + 4 + d0) = make_float4(a4[0], a4[1], a4[2], a4[3]);
        }
        cbar();
        if (tid == 0) add_release(p.cntx + hu, 1u);
      } else {
        // merge the other blocks' partials in block order
        if (tid == 0) wait_ge(p.cntx + hu, static_cast<uint32_t>((n_chunks(p) - 1) * (b + 1)), p.err, p.spin);
        cbar();
        if (qi < p.rps) {
          constexpr int kMaxCh = 8;  // T <= 2048 frames
          const int nch = n_chunks(p);
          float4 o4[kMaxCh - 1];
          float2 ml[kMaxCh - 1];
#pragma unroll
          for (int c2 = 1; c2 < kMaxCh; ++c2) {  // every load first
            const float *pt = p.xpart + (static_cast<size_t>(u + (c2 < nch ? c2 : 1)) * kMkRows + qi) * kPS;
            o4[c2 - 1] = __ldcg(reinterpret_cast<const float4 *>(pt + 4 + d0));
            ml[c2 - 1] = __ldcg(reinterpret_cast<const float2 *>(pt));
          }
#pragma unroll
          for (int c2 = 1; c2 < kMaxCh; ++c2) {
            if (c2 >= nch) break;
            const float a2[4] = {o4[c2 - 1].x, o4[c2 - 1].y, o4[c2 - 1].z, o4[c2 - 1].w};
            merge(M, L, a4, ml[c2 - 1].x, ml[c2 - 1].y, a2);
          }
        }
        store_out(p.xatt_x, i, h, L, a4);
      }
      cbar();
    }
    arrive(seq_of(b, PH_XATT));
  }

  // ------------------------------------------------- final LayerNorm ----
  // Row t (CTA t): the target's final LayerNorm (shared with the drafter)
  // from the exact fp32 residual, written as plain bf16 for the head.
  __device__ __noinline__ void final_ln() {
    const int t = c;
    if (t >= p.M) return;
    stage_ln(p.lnf_g, p.lnf_b);
    wait_phase(seq_of(p.nl - 1, PH_FC2));  // its barrier also publishes the staged gain and bias
    if (warp != 0) return;
    const int nj = p.d / 128;
    float4 v[kLnJ];
    load_row(v, t, nj);
    row_out(p.xn + static_cast<size_t>(t) * p.d, v, nj, row_stats(v, nj, 1.0f / static_cast<float>(p.d), p.eps));
  }

  __device__ void run() {
    embed();
    arrive(0);
#pragma unroll 1
    for (int b = 0; b < p.nl; ++b) {
      gemm_phase(b, PH_QKV);
      satt_phase(b);
      gemm_phase(b, PH_OUT);
      gemm_phase(b, PH_XQ);
      xatt_phase(b);
      gemm_phase(b, PH_XOUT);
      gemm_phase(b, PH_FC1);
      gemm_phase(b, PH_FC2);
    }
    final_ln();
  }
};

}  // namespace

__global__ void __launch_bounds__(kThr, 1) persist_kernel(const __grid_constant__ MkParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  Smem sm;
  sm.base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int c = blockIdx.x;
  const int tid = threadIdx.x;
  // The phases read the parameters through a reference; pointing it at a
  // shared-memory copy keeps those reads out of local memory.
  static_assert(sizeof(MkParams) % 4 == 0, "parameter copy in words");
  for (int w = tid; w < static_cast<int>(sizeof(MkParams) / 4); w += kThr)
    reinterpret_cast<uint32_t *>(sm.params())[w] = reinterpret_cast<const uint32_t *>(&p)[w];
  if (tid == 0) {
    for (int s = 0; s < kNS; ++s) {
      mbar_init(sm.full(s), 1);
      mbar_init(sm.empty(s), kW);
    }
    fence_barrier_init();
    *reinterpret_cast<uint4 *>(sm.zero16()) = make_uint4(0u, 0u, 0u, 0u);
    *sm.issued() = 0u;
  }
  if (tid < p.n_seq) {
    const int slot = p.seq_slot[tid];
    const int L = p.L[slot];
    sm.slot()[tid] = slot;
    const int nk = L + p.rps;
    sm.nk()[tid] = nk <= p.ctx ? nk : 0;
    if (nk > p.ctx) set_error(p.err, WF_DEV_ERR_CAPACITY);
  }
  __syncthreads();
  if (tid >= kCThr) {
    if (tid == kCThr) producer(*sm.params(), sm, c);
  } else {
    Cons cons(*sm.params(), sm);
    cons.run();
  }
  __syncthreads();
  if (tid == 0 && (ld_relaxed(p.err) & WF_DEV_ERR_TIMEOUT)) {
    // After a timeout the compute warps may have left ring slots unconsumed:
    // wait (bounded) for the copies still landing before the CTA leaves.
    // Otherwise every copy was consumed before the barrier above.
    const uint32_t sc = *sm.issued();
    for (uint32_t q = sc > static_cast<uint32_t>(kNS) ? sc - kNS : 0u; q < sc; ++q)
      mbar_drain(sm.full(q % kNS), (q / kNS) & 1u);
  }
  if (tid == 0) {
    // The last CTA to finish resets the counters for the next pass: no CTA
    // reads them any more once all have finished.
    __threadfence();
    const uint32_t done = atomicAdd(p.sync + 1, 1u);
    if (done == static_cast<uint32_t>(p.G - 1)) {
      for (int s = 0; s <= seq_of(p.nl - 1, PH_FC2); ++s) p.cnt[s] = 0u;
      for (int r = 0; r < p.d / 8; ++r) p.cnt2[r] = 0u;
      for (int hh = 0; hh < p.n_seq * p.H; ++hh) p.cntx[hh] = 0u;
      __threadfence();
      p.sync[1] = 0u;
    }
  }
}

size_t mk_xpart_words(int M, int H, int T) {
  const int nch = (T + 255) / 256;
  return static_cast<size_t>(M) * H * nch * kMkRows * kPS;
}

bool persist_supported(int d, int H, int F, int T, int rows) {
  return rows <= kMkRows && d % 128 == 0 && d <= 1280 && H * 64 == d && F % (128 * kQ2) == 0 &&
         F / kQ2 <= 1280 && T <= 8 * 256;
}

bool persist_grid_fits(int d, int F, int G) {
  auto per_cta = [G](int units) { return (units + G - 1) / G; };
  return G > 0 && per_cta(3 * d / 8) <= kUB && per_cta(F / 8) <= kUB && per_cta(d / 8 * kQ2) <= kUB &&
         per_cta(d / 8) <= kUB;
}

// Per device: the shared-memory opt-in and the grid (one CTA per SM, rounded
// down to a multiple of the fc2 split), set up the first time a handle on
// that device asks.  A cooperative launch needs every CTA resident at once,
// so the grid must come from the device the pass runs on.
cudaError_t persist_init(int *G) {
  constexpr int kMaxDev = 64;
  static std::mutex mu;
  static cudaError_t status[kMaxDev];
  static int grid[kMaxDev];
  static bool ready[kMaxDev] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDev) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (!ready[dev]) {
    int n_sm = 0, per_sm = 0;
    e = cudaFuncSetAttribute(persist_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMk);
    if (e == cudaSuccess) e = prefer_max_shared(reinterpret_cast<const void *>(persist_kernel));
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, persist_kernel, kThr, kSmemMk);
    if (e == cudaSuccess && per_sm < 1) e = cudaErrorInvalidConfiguration;
    status[dev] = e;
    grid[dev] = (n_sm / kQ2) * kQ2;
    ready[dev] = true;
  }
  if (G) *G = grid[dev];
  return status[dev];
}

cudaError_t launch_persist(const MkParams &p, cudaStream_t s) {
  if (p.M > kMkRows || p.n_seq > kMkMaxSeq || p.rps > 16 || p.G < p.M || p.G % kQ2 ||
      !persist_grid_fits(p.d, p.F, p.G))
    return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.G, 1, 1);
  cfg.blockDim = dim3(kThr, 1, 1);
  cfg.dynamicSmemBytes = kSmemMk;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, persist_kernel, p);
}

}  // namespace wf
