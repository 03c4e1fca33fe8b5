// LM head fused with the verifier's row reduction (Pro-Router, Section 3.1:
// the features are a side product of the small model's own decoding): the
// logits x = W h of a batch of hidden states are produced on the tensor cores
// and reduced to the Eq. 3 row state in the epilogue, so they never reach
// device memory.
//
//   lm_fused   grid (vocabulary splits, 256-row tiles), 320 threads:
//              warp 0   TMA producer: 64-wide K blocks of H (256 x 64) and W
//                       (256 x 64), 128-byte swizzle, a 3-stage ring;
//              warp 1   TMEM owner and MMA issuer: tcgen05.mma kind::f16 (bf16
//                       in, fp32 accumulate), M = 128, N = 256, K = 16 per
//                       instruction; the two 128-row halves of the tile share
//                       each W block and accumulate into two 128 x 256 fp32
//                       TMEM accumulators (all 512 columns);
//              warps 2-9 epilogue: tcgen05.ld of the finished accumulators,
//                       one row per thread, folded into the row's online (max,
//                       sum of 2^t, sum of t 2^t) state, an exact running
//                       top-KC list and the chosen token's logit; the state of
//                       each (row, split) goes to a small buffer.  Each W
//                       block is read once per 256 rows: half the L2 traffic
//                       of 128-row tiles for the same MMA work.
//   lm_merge   one warp per row: merges the splits' states in split order
//              and writes the feature record with the verifier's own row
//              finalisation (row_finish).
// With a thread-block cluster of cm x cs CTAs, the cm CTAs of one split (same
// W tiles, different rows) and the cs CTAs of one row tile (same H tiles,
// different splits) each load a slice of the shared tile and multicast it;
// each stage is released to every CTA that writes into it by a multicast
// tcgen05.commit.  This divides the L2 traffic per MMA by up to four.
// Every mbarrier wait is bounded (2 s of %globaltimer); a wait that runs out
// sets an error flag and stops the CTA's loops; the producer then waits
// (bounded) for its copies in flight, the MMA issuer for its own MMAs, and the
// CTA frees its TMEM before it exits.
#pragma once

#include <cuda.h>

#include "pr_device.cuh"
#include "pr_kernels.cuh"

namespace prk {

constexpr int LM_BM = 256, LM_BN = 256, LM_BK = 64, LM_STAGES = 3;
constexpr int LM_MH = 128;                             // rows per MMA (M)
constexpr int LM_A_BYTES = LM_BM * LM_BK * 2;          // 32 KB
constexpr int LM_B_BYTES = LM_BN * LM_BK * 2;          // 32 KB
constexpr int LM_STAGE_BYTES = LM_A_BYTES + LM_B_BYTES;
constexpr int LM_NT = 320;
constexpr int LM_EPI_WARPS = 8;
constexpr int LM_TMEM_COLS = 512;                      // two 256-column fp32 accumulators
constexpr size_t LM_SMEM = (size_t)LM_STAGES * LM_STAGE_BYTES + 1024 + 256;
constexpr uint64_t LM_WAIT_NS = 2000000000ull;         // a wait gives up after 2 s
constexpr uint32_t LM_ERR_TIMEOUT = 32u;                 // PR_FLAG_TIMEOUT in the context flag word

// instruction descriptor of tcgen05.mma kind::f16: fp32 accumulator (bits
// 4-5 = 1), bf16 A and B (bits 7-9, 10-12 = 1), both K-major (bits 15, 16 =
// 0), N / 8 in bits 17-22, M / 16 in bits 24-28
constexpr uint32_t LM_IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                              ((uint32_t)(LM_BN >> 3) << 17) | ((uint32_t)(LM_MH >> 4) << 24);

struct LmPart {            // one row's state over one vocabulary split
  float m, S, U, xy;       // base-2 (m, S, U); the chosen token's logit if in range
  uint32_t bad, has_y, pad0, pad1;
  uint64_t top[32];        // descending keys (value, lower index first); 0 = empty
};

struct LmArgs {
  int64_t n_rows, vocab;
  int32_t d, kblocks, ntiles;
  int32_t tiles_per_split;  // equal for every split (the last may run past V: masked)
  int32_t cm, cs;           // cluster shape: CTAs sharing W slices (M), sharing H slices (split)
  const int32_t* chosen;
  LmPart* parts;           // [nsplit][n_rows]
  uint32_t* err;           // error word
};

__device__ __forceinline__ uint32_t lm_smem(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void lm_mbar_init(uint64_t* b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(lm_smem(b)), "r"(count) : "memory");
}
__device__ __forceinline__ void lm_mbar_expect(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(lm_smem(b)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void lm_mbar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(lm_smem(b)) : "memory");
}
__device__ __forceinline__ bool lm_mbar_test(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(lm_smem(b)), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded wait for the phase with the given parity: false (and the error
// flag) when it has not completed after LM_WAIT_NS nanoseconds or another role
// of the CTA gave up first
__device__ __forceinline__ uint64_t lm_clock() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ bool lm_wait(uint64_t* b, uint32_t parity, volatile uint32_t* abort_,
                                        uint32_t* err) {
  if (lm_mbar_test(b, parity)) return true;
  const uint64_t t0 = lm_clock();
  for (uint32_t i = 1;; ++i) {
    if (lm_mbar_test(b, parity)) return true;
    if ((i & 255u) == 0u) {
      if (*abort_) return false;
      if (lm_clock() - t0 > LM_WAIT_NS) break;
    }
  }
  *abort_ = 1u;
  atomicOr(err, LM_ERR_TIMEOUT);
  return false;
}

// 2-D TMA load of a box at (x = K element, y = row) into shared memory,
// completing bytes on the mbarrier
__device__ __forceinline__ void lm_tma_load(const CUtensorMap* map, void* dst, uint64_t* bar,
                                            int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(lm_smem(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(lm_smem(bar))
      : "memory");
}

// the same load delivered to the CTAs of `mask` in the cluster: each receives
// the box at the same shared-memory offset and the bytes on its own mbarrier
// at the same offset
__device__ __forceinline__ void lm_tma_load_mc(const CUtensorMap* map, void* dst, uint64_t* bar,
                                               int x, int y, uint16_t mask) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      ".multicast::cluster [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(lm_smem(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(lm_smem(bar)), "h"(mask)
      : "memory");
}

// shared-memory matrix descriptor of a K-major operand written by TMA with the
// 128-byte swizzle: rows of 128 bytes (64 bf16), 8-row atoms of 1,024 bytes
// (stride byte offset), start address >> 4 in bits 0-13, leading byte offset
// 16 (unused for this layout) in bits 16-29, stride 1,024 >> 4 in bits 32-45,
// version 1 in bits 46-47, layout "128-byte swizzle" (2) in bits 61-63
__device__ __forceinline__ uint64_t lm_sdesc(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr >> 4) & 0x3fffu);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

__device__ __forceinline__ void lm_mma(uint32_t dtmem, uint64_t adesc, uint64_t bdesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(dtmem),
      "l"(adesc), "l"(bdesc), "r"(LM_IDESC), "r"(accumulate)
      : "memory");
}
// arrive on the mbarrier (same offset) of every CTA in `mask` once every
// tcgen05.mma this thread issued has completed
__device__ __forceinline__ void lm_commit_mc(uint64_t* bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(lm_smem(bar)),
      "h"(mask)
      : "memory");
}
__device__ __forceinline__ void lm_cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ uint32_t lm_cluster_id(int dim) {
  uint32_t v;
  if (dim == 0)
    asm volatile("mov.u32 %0, %%cluster_ctaid.x;" : "=r"(v));
  else
    asm volatile("mov.u32 %0, %%cluster_ctaid.y;" : "=r"(v));
  return v;
}

// arrive on the mbarrier once every tcgen05.mma this thread issued has completed
__device__ __forceinline__ void lm_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          lm_smem(bar))
      : "memory");
}
__device__ __forceinline__ void lm_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void lm_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes (lane = row)
__device__ __forceinline__ void lm_tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}

// v[j] for a run-time j without indexing the register array (a select tree)
__device__ __forceinline__ float lm_pick(const float (&v)[32], uint32_t j) {
  float a[16], b[8], c[4], d[2];
#pragma unroll
  for (int i = 0; i < 16; ++i) a[i] = (j & 1u) ? v[2 * i + 1] : v[2 * i];
#pragma unroll
  for (int i = 0; i < 8; ++i) b[i] = (j & 2u) ? a[2 * i + 1] : a[2 * i];
#pragma unroll
  for (int i = 0; i < 4; ++i) c[i] = (j & 4u) ? b[2 * i + 1] : b[2 * i];
#pragma unroll
  for (int i = 0; i < 2; ++i) d[i] = (j & 8u) ? c[2 * i + 1] : c[2 * i];
  return (j & 16u) ? d[1] : d[0];
}

// insert key k into the descending list L (L[KC-1] the smallest kept)
template <int KC>
__device__ __forceinline__ void lm_insert(uint64_t (&L)[KC], uint64_t k) {
  L[KC - 1] = k;
#pragma unroll
  for (int j = KC - 1; j > 0; --j) {
    const uint64_t a = L[j - 1], b = L[j];
    const bool sw = b > a;
    L[j - 1] = sw ? b : a;
    L[j] = sw ? a : b;
  }
}

template <int KC>
__global__ void __launch_bounds__(LM_NT, 1)
    lm_fused(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
             const LmArgs a) {
  extern __shared__ __align__(16) uint8_t lm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(lm_raw) + 1023) &
                                           ~(uintptr_t)1023);
  uint64_t* full = reinterpret_cast<uint64_t*>(sm + LM_STAGES * LM_STAGE_BYTES);
  uint64_t* empty = full + LM_STAGES;
  uint64_t* tfull = empty + LM_STAGES;   // both accumulators hold a finished tile
  uint64_t* tempty = tfull + 1;          // the epilogue has read them
  uint64_t* mdone = tempty + 1;          // the MMA issuer's own completion
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mdone + 1);
  volatile uint32_t* abort_ = tmem_slot + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // grid x = vocabulary split (fastest), y = 256-row tile: a wave of CTAs covers a
  // few row tiles across all splits, so the H tiles it re-reads and the W tiles
  // it streams together fit in L2
  const int split = blockIdx.x, mt = blockIdx.y;
  const int t0 = split * a.tiles_per_split, t1 = t0 + a.tiles_per_split;
  // cluster position (cluster dims cs x cm): pm along the rows (CTAs with the
  // same ps share W slices, cm of them), ps along the splits (CTAs with the same
  // pm share H slices, cs of them); rank = ps + pm cs
  const int ps = a.cs > 1 ? (int)lm_cluster_id(0) : 0;
  const int pm = a.cm > 1 ? (int)lm_cluster_id(1) : 0;
  uint16_t mask_h = 0, mask_w = 0;  // CTAs receiving my H slice / my W slice
  for (int s2 = 0; s2 < a.cs; ++s2) mask_h |= (uint16_t)(1u << (s2 + pm * a.cs));
  for (int m2 = 0; m2 < a.cm; ++m2) mask_w |= (uint16_t)(1u << (ps + m2 * a.cs));
  const uint16_t mask_rel = mask_h | mask_w;  // writers into my stages = readers of mine
  const bool clustered = a.cm * a.cs > 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < LM_STAGES; ++s) {
      lm_mbar_init(full + s, 1);
      lm_mbar_init(empty + s, (uint32_t)(a.cm + a.cs - 1));  // one release per writer's reader
    }
    lm_mbar_init(tfull, 1);
    lm_mbar_init(tempty, LM_EPI_WARPS);  // one arrival per epilogue warp
    lm_mbar_init(mdone, 1);
    *abort_ = 0u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     lm_smem(tmem_slot)),
                 "r"(LM_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  __syncthreads();
  if (clustered) lm_cluster_sync();  // every CTA's barriers exist before any remote use
  lm_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {  // ---- TMA producer
      int it = 0;
      for (int t = t0; t < t1 && !*abort_; ++t)
        for (int kb = 0; kb < a.kblocks; ++kb, ++it) {
          const int s = it % LM_STAGES;
          const uint32_t ph = (uint32_t)(it / LM_STAGES) & 1u;
          if (!lm_wait(empty + s, ph ^ 1u, abort_, a.err)) {
            t = t1;  // leave both loops
            break;
          }
          uint8_t* st = sm + s * LM_STAGE_BYTES;
          lm_mbar_expect(full + s, LM_STAGE_BYTES);  // all slices, from every writer
          if (!clustered) {
            lm_tma_load(&tmA, st, full + s, kb * LM_BK, mt * LM_BM);
            lm_tma_load(&tmB, st + LM_A_BYTES, full + s, kb * LM_BK, t * LM_BN);
          } else {
            const int ha = LM_BM / a.cs, wb = LM_BN / a.cm;  // slice rows
            lm_tma_load_mc(&tmA, st + ps * ha * 128, full + s, kb * LM_BK, mt * LM_BM + ps * ha,
                           mask_h);
            lm_tma_load_mc(&tmB, st + LM_A_BYTES + pm * wb * 128, full + s, kb * LM_BK,
                           t * LM_BN + pm * wb, mask_w);
          }
        }
      // the copies still in flight land before the CTA exits (already true
      // unless a wait gave up): wait, bounded, for the last stages' loads
      for (int j = it - 1; j >= 0 && j >= it - LM_STAGES; --j) {
        volatile uint32_t no_abort = 0u;
        lm_wait(full + j % LM_STAGES, (uint32_t)(j / LM_STAGES) & 1u, &no_abort, a.err);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---- MMA issuer
      int it = 0;
      for (int i = 0, t = t0; t < t1 && !*abort_; ++t, ++i) {
        // the epilogue has read the previous tile out of both accumulators
        if (!lm_wait(tempty, ((uint32_t)i & 1u) ^ 1u, abort_, a.err)) break;
        lm_fence_after();
        bool ok = true;
        for (int kb = 0; kb < a.kblocks; ++kb, ++it) {
          const int s = it % LM_STAGES;
          const uint32_t ph = (uint32_t)(it / LM_STAGES) & 1u;
          if (!lm_wait(full + s, ph, abort_, a.err)) {
            ok = false;
            break;
          }
          lm_fence_after();
          const uint32_t sa = lm_smem(sm + s * LM_STAGE_BYTES), sb = sa + LM_A_BYTES;
#pragma unroll
          for (int k = 0; k < LM_BK / 16; ++k) {  // K = 16 per MMA: 32 bytes along the row
            const uint64_t bd = lm_sdesc(sb + 32 * k);
            const uint32_t acc = (kb | k) != 0 ? 1u : 0u;
            lm_mma(tmem, lm_sdesc(sa + 32 * k), bd, acc);                       // rows 0-127
            lm_mma(tmem + LM_BN, lm_sdesc(sa + LM_MH * 128 + 32 * k), bd, acc);  // rows 128-255
          }
          // the stage is free, in every CTA that writes into it, once these MMAs
          // have read it
          if (clustered)
            lm_commit_mc(empty + s, mask_rel);
          else
            lm_commit(empty + s);
        }
        if (!ok) break;
        lm_commit(tfull);
      }
      // every MMA this thread issued has completed before TMEM is freed
      lm_commit(mdone);
      volatile uint32_t no_abort = 0u;
      lm_wait(mdone, 0u, &no_abort, a.err);
    }
  } else {  // ---- epilogue: warps 2..9, TMEM lanes 32 (warp % 4) .., accumulator h
    const int q = warp & 3, h = (warp - 2) >> 2;
    const int64_t row = (int64_t)mt * LM_BM + LM_MH * h + 32 * q + lane;
    const bool live = row < a.n_rows;
    const int32_t y = live ? a.chosen[row] : -1;
    const int32_t V = (int32_t)a.vocab;
    float m = M2_INIT, xy = NAN;
    float2 S2 = make_float2(0.f, 0.f), U2 = make_float2(0.f, 0.f);  // even / odd columns
    bool bad = false, has_y = false;
    uint64_t L[KC];
#pragma unroll
    for (int j = 0; j < KC; ++j) L[j] = 0ull;
    float thr = -INFINITY;  // value of the KC-th key kept (-inf while the list is not full)
    for (int i = 0, t = t0; t < t1; ++t, ++i) {
      int ok = 1;
      if (lane == 0) ok = lm_wait(tfull, (uint32_t)i & 1u, abort_, a.err) ? 1 : 0;
      ok = __shfl_sync(FULL, ok, 0);  // the warp stays converged for tcgen05.ld
      if (!ok) break;
      lm_fence_after();
      const uint32_t tbase = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(h * LM_BN);
      for (int c = 0; c < LM_BN / 32; ++c) {
        float v[32];
        lm_tmem_ld32(tbase + 32 * c, v);
        const int32_t col0 = t * LM_BN + 32 * c;
        const bool whole = col0 + 32 <= V;  // false only in the last vocabulary tile
        if (!whole) {
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (col0 + j >= V) v[j] = -INFINITY;
        }
        float cmax = v[0];
#pragma unroll
        for (int j = 1; j < 32; ++j) cmax = fmaxf(cmax, v[j]);
        if (cmax == INFINITY) bad = true;  // NaN reaches S and U and is flagged there
        const float tm = cmax * L2E;
        if (tm > m) {
          const float dl = m - tm, f = ex2(dl);
          const float2 f2 = make_float2(f, f), dl2 = make_float2(dl, dl);
          U2 = __fmul2_rn(f2, __ffma2_rn(dl2, S2, U2));
          S2 = __fmul2_rn(S2, f2);
          m = tm;
        }
        const float2 nm = make_float2(-m, -m), l2e = make_float2(L2E, L2E);
        const float2 lo2 = make_float2(-1e30f, -1e30f);
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
          float2 dd = __ffma2_rn(make_float2(v[j], v[j + 1]), l2e, nm);
          if (!whole) dd = make_float2(fmaxf(dd.x, lo2.x), fmaxf(dd.y, lo2.y));  // -inf -> 0 weight
          const float2 e = make_float2(ex2(dd.x), ex2(dd.y));
          S2 = __fadd2_rn(S2, e);
          U2 = __ffma2_rn(e, dd, U2);
        }
        // chosen token: one chunk of the whole sweep holds it
        const uint32_t yo = (uint32_t)(y - col0);
        if (yo < 32u && (int32_t)yo + col0 < V) {
          xy = lm_pick(v, yo);
          has_y = true;
        }
        // top-KC: only chunks whose maximum reaches the list's threshold
        if (cmax >= thr) {
          uint32_t mask = 0u;
#pragma unroll
          for (int j = 0; j < 32; ++j) mask |= (v[j] >= thr && col0 + j < V ? 1u : 0u) << j;
          while (mask) {
            const uint32_t j = (uint32_t)__ffs(mask) - 1u;
            mask &= mask - 1u;
            const uint64_t k = make_key(lm_pick(v, j), (uint32_t)(col0 + (int32_t)j));
            if (k > L[KC - 1]) {
              lm_insert<KC>(L, k);
              if (L[KC - 1] != 0ull) thr = key_val(L[KC - 1]);
            }
          }
        }
      }
      lm_fence_before();
      __syncwarp();
      if (lane == 0) lm_mbar_arrive(tempty);
    }
    const float S = S2.x + S2.y, U = U2.x + U2.y;
    if (live) {
      LmPart* p = a.parts + (int64_t)split * a.n_rows + row;
      p->m = m;
      p->S = S;
      p->U = U;
      p->xy = xy;
      p->bad = bad ? 1u : 0u;
      p->has_y = has_y ? 1u : 0u;
#pragma unroll
      for (int j = 0; j < 32; ++j) p->top[j] = j < KC ? L[j] : 0ull;
    }
  }
  __syncthreads();
  if (clustered) lm_cluster_sync();  // no CTA leaves while others may still write into it
  if (warp == 1) {
    lm_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(LM_TMEM_COLS)
                 : "memory");
  }
}

// one warp per row: merge the splits in order, then the verifier's row
// finalisation (features, top-2 indices, flags)
__global__ void __launch_bounds__(256) lm_merge(const Args a, const LmPart* __restrict__ parts,
                                                int nsplit) {
  const int lane = threadIdx.x & 31;
  const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  if (row >= a.n_rows) return;
  float m = M2_INIT, S = 0.f, U = 0.f, xy = NAN;
  bool bad = false;
  uint64_t E = 0ull;
  for (int s = 0; s < nsplit; ++s) {
    const LmPart& p = parts[(int64_t)s * a.n_rows + row];
    lse_merge(m, S, U, p.m, p.S, p.U);
    bad |= p.bad != 0u;
    if (p.has_y) xy = p.xy;
    E = warp_merge_desc<uint64_t>(E, p.top[lane], lane);
  }
  RowPre pre;
  pre.y = a.chosen[row];
  pre.xy = (pre.y >= 0 && (int64_t)pre.y < a.vocab) ? xy : NAN;
  pre.r = -1;
  pre.lo = pre.hi = 0;
  pre.eos = 0;
  if (a.offsets) {
    pre.r = find_request(a.offsets, a.n_req, row, lane);
    if (pre.r >= 0) {
      pre.lo = __ldg(a.offsets + pre.r);
      pre.hi = __ldg(a.offsets + pre.r + 1);
    }
  }
  row_finish<float, MODE_FEATURES>(a, row, m, S, U, bad, lane < a.kc ? E : 0ull, pre, lane);
}

}  // namespace prk
