// LM head fused with the verifier's row reduction (Pro-Router, Section 3.1:
// the features need nothing the small model's decoding does not compute): the
// logits x = W h of a batch of hidden states are produced on the tensor cores
// and reduced to the Eq. 3 row state in the epilogue, so they never reach
// device memory.
//
//   lm_fused   2 x (row pairs x vocabulary splits) CTAs in thread-block
//              clusters of two along x, 320 threads; a pair (256 rows, one
//              split) per cluster, in bands of row pairs: a wave streams few
//              splits' W tiles past one band's H rows, both held in L2.
//              The pair shares one tcgen05.mma of M = 256 (cta_group::2):
//              the CTA of rank r holds rows 128 r .. of the pair's 256 rows
//              of H and rows 128 r .. of each 256-row tile of W, and its TMEM
//              receives its own 128 rows of the 256 x 256 logit tile.
//              warp 0   (both CTAs) TMA producer: K blocks of 128 (two boxes
//                       of 64 with the 128-byte swizzle) of its H rows and W
//                       half tile, a 3-stage ring of 64 KB stages; every load
//                       completes on the rank-0 CTA's stage barrier, which
//                       expects the bytes of both CTAs;
//              warp 1   owns the pair's TMEM (allocated by both CTAs
//                       together); in the rank-0 CTA it issues the MMAs (bf16
//                       in, fp32 accumulate, K = 16 each, 8 per stage) into
//                       one of two 256-column accumulators, so tile i + 1
//                       accumulates while the epilogue reads tile i, and
//                       releases stages and finished tiles to both CTAs by a
//                       multicast tcgen05.commit;
//              warps 2-9 (both CTAs) epilogue: warp w reads TMEM lanes 32 (w %
//                       4) .. and one 128-column half of the tile, one row per
//                       thread, folded into the row's online (max, sum of 2^t,
//                       sum of t 2^t) state, an exact running top-KC list and
//                       the chosen token's logit; each warp reports a read
//                       accumulator to the rank-0 CTA; at the end the two
//                       halves' states of a row are merged (through the idle
//                       stage ring) into one state per (row, split) in a small
//                       buffer.
//              A W block is read from L2 once per 256 rows, an H block once
//              per 256 vocabulary columns.
//   lm_merge   merges each row's partial states in a fixed order and runs
//              the verifier's own row finalisation (row_finish): the feature
//              record, or the fold into the row's decode slot.
// Every mbarrier wait is bounded (2 s of %globaltimer); a wait that runs out
// sets an error flag and stops that role's loop; the roles of the other CTA
// then run out of their own waits, the rank-0 producer waits (bounded) for
// the copies in flight, the MMA issuer for its own MMAs, and both CTAs free
// the pair's TMEM together before they exit.
#pragma once

#include <cuda.h>

#include "pr_device.cuh"
#include "pr_kernels.cuh"

namespace prk {

constexpr int LM_BM = 128;                             // rows of H per CTA (256 per pair)
constexpr int LM_BN = 256;                             // vocabulary columns per tile (MMA N)
constexpr int LM_BK = 128;                             // K per stage: two 64-wide swizzle boxes
constexpr int LM_STAGES = 3;
constexpr int LM_A_BYTES = LM_BM * LM_BK * 2;          // 32 KB: this CTA's rows of H
constexpr int LM_B_BYTES = (LM_BN / 2) * LM_BK * 2;    // 32 KB: this CTA's half of the W tile
constexpr int LM_BOX_K = 64;                           // box width: one 128-byte swizzle row
constexpr int LM_BOX_BYTES = 128 * LM_BOX_K * 2;       // one 128-row box
constexpr int LM_STAGE_BYTES = LM_A_BYTES + LM_B_BYTES;
constexpr int LM_NT = 320;
constexpr int LM_EPI_WARPS = 8;
constexpr int LM_HALVES = 2;                           // column halves of a tile (epilogue)
constexpr int LM_TMEM_COLS = 512;                      // two 256-column fp32 accumulators
constexpr size_t LM_SMEM = (size_t)LM_STAGES * LM_STAGE_BYTES + 1024 + 256;
constexpr uint64_t LM_WAIT_NS = 2000000000ull;         // a wait gives up after 2 s
constexpr uint32_t LM_ERR_TIMEOUT = 32u;                 // PR_FLAG_TIMEOUT in the context flag word

// instruction descriptor of tcgen05.mma kind::f16: fp32 accumulator (bits
// 4-5 = 1), bf16 A and B (bits 7-9, 10-12 = 1), both K-major (bits 15, 16 =
// 0), N / 8 in bits 17-22, M / 16 in bits 24-28 (M = 256: the pair's rows)
constexpr uint32_t LM_IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                              ((uint32_t)(LM_BN >> 3) << 17) | ((uint32_t)((2 * LM_BM) >> 4) << 24);

struct LmPart {            // one row's state over one vocabulary split
  float m, S, U, xy;       // base-2 (m, S, U); the chosen token's logit if in range
  uint32_t bad, has_y, pad0, pad1;
  uint64_t top[32];        // descending keys (value, lower index first); 0 = empty
};

struct LmArgs {
  int64_t n_rows, vocab;
  int32_t d, kblocks, ntiles;
  int32_t tiles_per_split;  // the last split stops at the last tile
  int32_t nsplit, npairs;   // vocabulary splits; 256-row pairs (CTA pairs per split)
  int32_t band;             // row pairs per band of the launch order
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
                                        uint32_t* err, uint64_t limit_ns = LM_WAIT_NS) {
  if (lm_mbar_test(b, parity)) return true;
  const uint64_t t0 = lm_clock();
  for (uint32_t i = 1;; ++i) {
    if (lm_mbar_test(b, parity)) return true;
    if ((i & 255u) == 0u) {
      if (*abort_) return false;
      if (lm_clock() - t0 > limit_ns) break;
    }
  }
  *abort_ = 1u;
  atomicOr(err, LM_ERR_TIMEOUT);
  return false;
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

__device__ __forceinline__ void lm_cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ uint32_t lm_cluster_x() {
  uint32_t v;
  asm volatile("mov.u32 %0, %%cluster_ctaid.x;" : "=r"(v));
  return v;
}

__device__ __forceinline__ void lm_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void lm_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// ---- CTA-pair forms (tcgen05 cta_group::2)

// shared::cluster address of the same variable in the CTA of the given rank
__device__ __forceinline__ uint32_t lm_mapa(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(lm_smem(p)), "r"(rank));
  return r;
}
// 2-D TMA load into this CTA's shared memory whose completion is counted on an
// mbarrier of either CTA of the pair (a shared::cluster address)
__device__ __forceinline__ void lm_tma_load_pair(const CUtensorMap* map, void* dst, uint32_t bar,
                                                 int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(lm_smem(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// arrive on an mbarrier of another CTA of the cluster (release at cluster scope)
__device__ __forceinline__ void lm_arrive_remote(uint32_t bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar)
               : "memory");
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

// insert (ov, col) into the list (Lv, Li) sorted by descending value code;
// the caller has checked ov > Lv[KC-1].  Columns reach a thread in increasing
// order, so a new entry goes after every kept entry of equal value: that is
// the order of the keys (value, lower index first).  All comparisons are
// against the old list, so the KC steps are independent: gt[j] = ov > Lv[j] is
// false then true along the list, and entry j becomes entry j-1 where
// gt[j-1], the new one where gt[j] alone, else stays.
template <int KC>
__device__ __forceinline__ void lm_insert(uint32_t (&Lv)[KC], uint32_t (&Li)[KC], uint32_t ov,
                                          uint32_t col) {
  bool gt[KC];
#pragma unroll
  for (int j = 0; j < KC; ++j) gt[j] = ov > Lv[j];
#pragma unroll
  for (int j = KC - 1; j > 0; --j) {
    Lv[j] = gt[j - 1] ? Lv[j - 1] : (gt[j] ? ov : Lv[j]);
    Li[j] = gt[j - 1] ? Li[j - 1] : (gt[j] ? col : Li[j]);
  }
  Lv[0] = gt[0] ? ov : Lv[0];
  Li[0] = gt[0] ? col : Li[0];
}

// One row's running state over the columns an epilogue thread folds in:
// online base-2 (m, S, U) with S and U kept as even / odd column pairs, the
// chosen token's logit, and the exact top-KC entries as order-preserving value
// codes (0 = empty) with their columns.
template <int KC>
struct LmRow {
  float m, xy, thr;  // thr: value of the KC-th entry kept (-inf while the list is not full)
  float2 S2, U2;
  bool bad, has_y;
  uint32_t Lv[KC], Li[KC];

  __device__ __forceinline__ void init() {
    m = M2_INIT;
    xy = NAN;
    thr = -INFINITY;
    S2 = make_float2(0.f, 0.f);
    U2 = make_float2(0.f, 0.f);
    bad = has_y = false;
#pragma unroll
    for (int j = 0; j < KC; ++j) Lv[j] = Li[j] = 0u;
  }

  // fold 32 consecutive logits v of columns col0 .. col0 + 31 (those >= V are
  // outside the vocabulary); y is the row's chosen token
  __device__ __forceinline__ void chunk(float (&v)[32], int32_t col0, int32_t V, int32_t y) {
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
      for (int j = 0; j < 32; ++j) mask |= (v[j] >= thr ? 1u : 0u) << j;
      if (!whole) {  // columns < V only (0 <= V - col0 < 32 here, or none)
        const int32_t nv = V - col0;
        mask &= nv > 0 ? (1u << nv) - 1u : 0u;
      }
      while (mask) {
        const uint32_t j = (uint32_t)__ffs(mask) - 1u;
        mask &= mask - 1u;
        const uint32_t ov = ord(lm_pick(v, j));
        if (ov > Lv[KC - 1]) {
          lm_insert<KC>(Lv, Li, ov, (uint32_t)col0 + j);
          if (Lv[KC - 1] != 0u) thr = unord(Lv[KC - 1]);
        }
      }
    }
  }

  __device__ __forceinline__ void store(LmPart* p) const {
    p->m = m;
    p->S = S2.x + S2.y;
    p->U = U2.x + U2.y;
    p->xy = xy;
    p->bad = bad ? 1u : 0u;
    p->has_y = has_y ? 1u : 0u;
#pragma unroll
    for (int j = 0; j < 32; ++j)  // the keys of make_key
      p->top[j] = (j < KC && Lv[j] != 0u)
                      ? ((uint64_t)Lv[j] << 32) | (uint64_t)(0xffffffffu - Li[j])
                      : 0ull;
  }
};

// out = the merge of the two column halves' states of one row: the online
// sums merged, the top-32 keys of the union (both lists descending, 0 =
// empty), the chosen token's logit from the half that holds it
__device__ __forceinline__ void lm_merge_halves(const LmPart& x, const LmPart& y, LmPart* out) {
  float m = x.m, S = x.S, U = x.U;
  lse_merge(m, S, U, y.m, y.S, y.U);
  out->m = m;
  out->S = S;
  out->U = U;
  out->xy = x.has_y ? x.xy : y.xy;
  out->bad = x.bad | y.bad;
  out->has_y = x.has_y | y.has_y;
  int i0 = 0, i1 = 0;
  for (int j = 0; j < 32; ++j) {
    const uint64_t k0 = i0 < 32 ? x.top[i0] : 0ull, k1 = i1 < 32 ? y.top[i1] : 0ull;
    if (k0 >= k1) {
      out->top[j] = k0;
      ++i0;
    } else {
      out->top[j] = k1;
      ++i1;
    }
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
  uint64_t* tfull = empty + LM_STAGES;   // [2] accumulator b holds a finished tile
  uint64_t* tempty = tfull + 2;          // [2] (rank 0) both epilogues have read accumulator b
  uint64_t* mdone = tempty + 2;          // (rank 0) the MMA issuer's own completion
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mdone + 1);
  volatile uint32_t* abort_ = tmem_slot + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = lm_cluster_x();
  const bool lead = rank == 0u;
  // launch order: bands of `band` row pairs; within a band all its pairs of
  // one split, then the next split; the last band may be shorter
  int split, pr;
  {
    const int u = (int)(blockIdx.x >> 1), G = a.band, per_band = G * a.nsplit;
    const int full_bands = a.npairs / G, b = u / per_band;
    if (b < full_bands) {
      const int r = u - b * per_band;
      split = r / G;
      pr = b * G + (r - split * G);
    } else {
      const int rem = a.npairs - full_bands * G, r = u - full_bands * per_band;
      split = r / rem;
      pr = full_bands * G + (r - split * rem);
    }
  }
  const int mt = 2 * pr + (int)rank;
  const int t0 = split * a.tiles_per_split;
  const int t1 = min(t0 + a.tiles_per_split, a.ntiles);

  if (threadIdx.x == 0) {
    for (int s = 0; s < LM_STAGES; ++s) {
      lm_mbar_init(full + s, 1);
      lm_mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      lm_mbar_init(tfull + b, 1);
      lm_mbar_init(tempty + b, 2 * LM_EPI_WARPS);  // every epilogue warp of both CTAs
    }
    lm_mbar_init(mdone, 1);
    *abort_ = 0u;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     lm_smem(tmem_slot)),
                 "r"(LM_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  __syncthreads();
  lm_cluster_sync();  // both CTAs' barriers and TMEM exist before any remote use
  lm_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t full0 = lm_mapa(full, 0u), tempty0 = lm_mapa(tempty, 0u);

  if (warp == 0) {
    if (lane == 0) {  // ---- TMA producer (both CTAs)
      int it = 0;
      for (int t = t0; t < t1 && !*abort_; ++t)
        for (int kb = 0; kb < a.kblocks; ++kb, ++it) {
          const int s = it % LM_STAGES;
          const uint32_t ph = (uint32_t)(it / LM_STAGES) & 1u;
          if (!lm_wait(empty + s, ph ^ 1u, abort_, a.err)) {
            t = t1;
            break;
          }
          uint8_t* st = sm + s * LM_STAGE_BYTES;
          if (lead) lm_mbar_expect(full + s, 2 * LM_STAGE_BYTES);  // both CTAs' bytes
          for (int hk = 0; hk < LM_BK / LM_BOX_K; ++hk) {  // boxes, 16 KB apart
            const int x = kb * LM_BK + LM_BOX_K * hk;
            lm_tma_load_pair(&tmA, st + hk * LM_BOX_BYTES, full0 + 8u * (uint32_t)s, x,
                             mt * LM_BM);
            lm_tma_load_pair(&tmB, st + LM_A_BYTES + hk * LM_BOX_BYTES, full0 + 8u * (uint32_t)s,
                             x, t * LM_BN + (int)rank * (LM_BN / 2));
          }
        }
      // rank 0's stage barriers count both CTAs' copies: it waits, bounded,
      // for the last stages, so no copy is in flight when the pair exits
      if (lead)
        for (int j = it - 1; j >= 0 && j >= it - LM_STAGES; --j) {
          volatile uint32_t no_abort = 0u;
          lm_wait(full + j % LM_STAGES, (uint32_t)(j / LM_STAGES) & 1u, &no_abort, a.err);
        }
    }
  } else if (warp == 1) {
    if (lane == 0 && lead) {  // ---- MMA issuer (rank 0)
      int it = 0;
      for (int i = 0, t = t0; t < t1 && !*abort_; ++t, ++i) {
        const int b = i & 1;
        if (!lm_wait(tempty + b, (((uint32_t)i >> 1) & 1u) ^ 1u, abort_, a.err)) break;
        lm_fence_after();
        const uint32_t dt = tmem + (uint32_t)(b * LM_BN);
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
          for (int k = 0; k < LM_BK / 16; ++k) {  // K = 16: 32 bytes along a box row
            const uint32_t ko = (uint32_t)((k / (LM_BOX_K / 16)) * LM_BOX_BYTES +
                                           32 * (k % (LM_BOX_K / 16)));
            asm volatile(
                "{\n\t.reg .pred p;\n\t"
                "setp.ne.b32 p, %4, 0;\n\t"
                "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(dt),
                "l"(lm_sdesc(sa + ko)), "l"(lm_sdesc(sb + ko)), "r"(LM_IDESC),
                "r"((kb | k) != 0 ? 1u : 0u)
                : "memory");
          }
          // stage s is free in both CTAs once these MMAs have read it
          asm volatile(
              "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::"
              "cluster.b64 [%0], %1;" ::"r"(lm_smem(empty + s)),
              "h"((uint16_t)3)
              : "memory");
        }
        if (!ok) break;
        asm volatile(
            "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::"
            "cluster.b64 [%0], %1;" ::"r"(lm_smem(tfull + b)),
            "h"((uint16_t)3)
            : "memory");
      }
      asm volatile(
          "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::"
          "cluster.b64 [%0], %1;" ::"r"(lm_smem(mdone)),
          "h"((uint16_t)1)
          : "memory");
      volatile uint32_t no_abort = 0u;
      lm_wait(mdone, 0u, &no_abort, a.err);
    }
  } else {  // ---- epilogue (both CTAs): TMEM lanes 32 (warp % 4) .., column half hc
    const int q = warp & 3, hc = (warp - 2) >> 2;
    const int64_t row = (int64_t)mt * LM_BM + 32 * q + lane;
    const bool live = row < a.n_rows;
    const int32_t y = live ? a.chosen[row] : -1;
    const int32_t V = (int32_t)a.vocab;
    LmRow<KC> st;
    st.init();
    for (int i = 0, t = t0; t < t1; ++t, ++i) {
      const int b = i & 1;
      int ok = 1;
      if (lane == 0) ok = lm_wait(tfull + b, ((uint32_t)i >> 1) & 1u, abort_, a.err) ? 1 : 0;
      ok = __shfl_sync(FULL, ok, 0);
      if (!ok) break;
      lm_fence_after();
      const int hw = LM_BN / LM_HALVES;
      const uint32_t tbase =
          tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * LM_BN + hc * hw);
      for (int c = 0; c < hw / 32; ++c) {
        float v[32];
        lm_tmem_ld32(tbase + 32 * c, v);
        st.chunk(v, t * LM_BN + hc * hw + 32 * c, V, y);
      }
      lm_fence_before();
      __syncwarp();
      if (lane == 0) lm_arrive_remote(tempty0 + 8u * (uint32_t)b);
    }
    // both column halves of each row go to shared memory (the stage ring is
    // idle once the last tile has been read); after the barrier below the
    // half-0 thread of the row merges them into the row's part of this split
    st.store(reinterpret_cast<LmPart*>(sm) + hc * LM_BM + 32 * q + lane);
  }
  __syncthreads();
  if (warp >= 2) {
    const int q = warp & 3, hc = (warp - 2) >> 2, lr = 32 * q + lane;
    const int64_t row = (int64_t)mt * LM_BM + lr;
    if (hc == 0 && row < a.n_rows) {
      const LmPart* ex = reinterpret_cast<const LmPart*>(sm);
      lm_merge_halves(ex[lr], ex[LM_BM + lr], a.parts + (int64_t)split * a.n_rows + row);
    }
  }
  lm_cluster_sync();  // the MMAs into both TMEMs are complete; no remote arrival is pending
  if (warp == 1) {
    lm_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(LM_TMEM_COLS)
                 : "memory");
  }
}

// The bounded wait on an mbarrier that nothing completes, with the given
// limit: *completed = 0 and PR_FLAG_TIMEOUT in *err once it runs out (one
// thread; the failure path of lm_fused's waits, exercised without a stall).
__global__ void lm_wait_probe(uint32_t* err, uint64_t limit_ns, int32_t* completed) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t abort_flag;
  lm_mbar_init(&bar, 1);
  abort_flag = 0u;
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  *completed = lm_wait(&bar, 0u, &abort_flag, err, limit_ns) ? 1 : 0;
}

// wpr warps per row (1, 2, 4 or 8; 8 / wpr rows per CTA): warp w of a row
// merges the row's parts (splits x column halves) w, w + wpr, ... in order,
// the row's first warp then merges the wpr results in warp order (with wpr =
// 1 simply all parts in order), then the verifier's row finalisation: the
// feature record (MODE_FEATURES) or the fold into the row's decode slot
// (MODE_DECODE).  Many parts per row (a small batch split over many
// vocabulary splits) take more warps per row.
template <int MODE>
__global__ void __launch_bounds__(256) lm_merge(const Args a, const LmPart* __restrict__ parts,
                                                int nparts, int wpr) {
  __shared__ float s_m[8], s_S[8], s_U[8], s_xy[8];
  __shared__ uint32_t s_fl[8];  // bit 0: a non-finite logit, bit 1: holds the chosen token
  __shared__ uint64_t s_top[8][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = warp / wpr, w = warp - g * wpr;
  const int64_t row = (int64_t)blockIdx.x * (8 / wpr) + g;
  const bool live = row < a.n_rows;
  float m = M2_INIT, S = 0.f, U = 0.f, xy = NAN;
  bool bad = false, has_y = false;
  uint64_t E = 0ull;
  if (live)
    for (int s = w; s < nparts; s += wpr) {
      const LmPart& p = parts[(int64_t)s * a.n_rows + row];
      lse_merge(m, S, U, p.m, p.S, p.U);
      bad |= p.bad != 0u;
      if (p.has_y) {
        xy = p.xy;
        has_y = true;
      }
      E = warp_merge_desc<uint64_t>(E, p.top[lane], lane);
    }
  if (wpr > 1) {
    if (lane == 0) {
      s_m[warp] = m;
      s_S[warp] = S;
      s_U[warp] = U;
      s_xy[warp] = xy;
      s_fl[warp] = (bad ? 1u : 0u) | (has_y ? 2u : 0u);
    }
    s_top[warp][lane] = E;
    __syncthreads();
    if (w != 0 || !live) return;
    m = M2_INIT;
    S = U = 0.f;
    xy = NAN;
    bad = false;
    E = 0ull;
    for (int v = warp; v < warp + wpr; ++v) {
      lse_merge(m, S, U, s_m[v], s_S[v], s_U[v]);
      bad |= (s_fl[v] & 1u) != 0u;
      if (s_fl[v] & 2u) xy = s_xy[v];
      E = warp_merge_desc<uint64_t>(E, s_top[v][lane], lane);
    }
  } else if (!live) {
    return;
  }
  RowPre pre;
  pre.y = a.chosen[row];
  pre.xy = (pre.y >= 0 && (int64_t)pre.y < a.vocab) ? xy : NAN;
  pre.r = -1;
  pre.lo = pre.hi = 0;
  pre.eos = 0;
  if (MODE == MODE_DECODE) {
    pre.r = a.slot[row];
    pre.eos = a.eos[row];
  } else if (a.offsets) {
    pre.r = find_request(a.offsets, a.n_req, row, lane);
    if (pre.r >= 0) {
      pre.lo = __ldg(a.offsets + pre.r);
      pre.hi = __ldg(a.offsets + pre.r + 1);
    }
  }
  row_finish<float, MODE>(a, row, m, S, U, bad, lane < a.kc ? E : 0ull, pre, lane);
}

}  // namespace prk
