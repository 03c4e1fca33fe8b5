// Kernels of the verifier data path: the row kernels (Eq. 3 features, with a
// fused pooling / scoring / ship-rule epilogue in route and decode modes) and
// the standalone pooling kernel.  Algorithm notes are in pr_device.cuh.
//   verify_rows_ws  persistent, warp-specialised: one CTA streams one row at a
//                   time (used whenever a row needs no split)
//   verify_rows     one thread-block cluster of C CTAs per row (C = 2, 4, 8:
//                   batches too small to fill the GPU, e.g. decode steps)
#pragma once

#include "pr_device.cuh"

namespace prk {

// A scattered 16-byte re-read of a row already streamed: without the 256-byte
// L2 prefetch of ld_stream, a load that misses L2 fetches one 32-byte sector
// from DRAM instead of a 256-byte block.
__device__ __forceinline__ uint4 ld_reread(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// ---- pooling, scoring, ship rule (Section 3.1) -------------------------------------

struct Pooled {
  float agg[NAGG];
  float score;
  uint8_t ship;
  uint32_t flags;
};

// Warp-parallel pool of rows [lo, hi) of a [rows][8] feature array.  Lane j
// sums rows lo + j, lo + j + 32, ... in order, then a fixed butterfly combines
// the lanes, so the result depends only on T.  All lanes return the result.
__device__ __forceinline__ Pooled pool_rows(const float* feat, const uint32_t* flags, int64_t lo,
                                            int64_t hi, const float* w, float b, float zthr,
                                            int lane) {
  float s[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
  float mn[5] = {INFINITY, INFINITY, INFINITY, INFINITY, INFINITY};
  uint32_t fl = 0;
#pragma unroll 4
  for (int64_t i = lo + lane; i < hi; i += 32) {
    const float4 a = __ldcg(reinterpret_cast<const float4*>(feat + i * NFEAT));
    const float4 c = __ldcg(reinterpret_cast<const float4*>(feat + i * NFEAT + 4));
    const float v[5] = {a.x, a.y, a.z, -a.w, c.x};  // l, m, margin, -H, h
#pragma unroll
    for (int f = 0; f < 5; ++f) {
      s[f] += v[f];
      mn[f] = fminf(mn[f], v[f]);
    }
    if (flags) fl |= __ldcg(flags + i);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
    for (int f = 0; f < 5; ++f) {
      s[f] += __shfl_xor_sync(FULL, s[f], o);
      mn[f] = fminf(mn[f], __shfl_xor_sync(FULL, mn[f], o));
    }
    fl |= __shfl_xor_sync(FULL, fl, o);
  }
  Pooled p;
  const int64_t T = hi - lo;
  p.flags = fl;
  if (fl & (FLAG_NONFINITE | FLAG_BAD_CHOSEN)) {
#pragma unroll
    for (int j = 0; j < NAGG; ++j) p.agg[j] = NAN;
    p.score = NAN;
    p.ship = 0;
    return p;
  }
  const float Tf = (float)T;
#pragma unroll
  for (int f = 0; f < 5; ++f) {
    p.agg[2 * f] = s[f] / Tf;
    p.agg[2 * f + 1] = mn[f];
  }
  p.agg[10] = (float)(T + 1) / (float)(2 * T);  // mean of t/T over t = 1..T
  float z = b;
#pragma unroll
  for (int j = 0; j < NAGG; ++j) z = fmaf(__ldg(w + j), p.agg[j], z);
  p.score = 1.f / (1.f + expf(-z));
  p.ship = (z >= zthr) ? 1 : 0;
  return p;
}

__device__ __forceinline__ void write_pooled(const Pooled& p, int64_t r, float* agg, float* score,
                                             uint8_t* ship, uint32_t* req_flags, int lane) {
  if (agg && lane < NAGG) {
    float v = p.agg[0];
#pragma unroll
    for (int j = 1; j < NAGG; ++j)
      if (lane == j) v = p.agg[j];
    agg[r * NAGG + lane] = v;
  }
  if (lane == 0) {
    score[r] = p.score;
    ship[r] = p.ship;
    req_flags[r] = p.flags;
  }
}

__device__ __forceinline__ void write_special(int64_t r, float sc, uint32_t fl, float* agg,
                                              float* score, uint8_t* ship, uint32_t* req_flags) {
  if (agg)
    for (int j = 0; j < NAGG; ++j) agg[r * NAGG + j] = NAN;
  score[r] = sc;
  ship[r] = 0;
  req_flags[r] = fl;
}

// Request that owns global row gr: the r with offsets[r] <= gr < offsets[r+1],
// by a 32-way search (two dependent loads for up to 1,024 requests).
// Returns -1 when the offsets are inconsistent with gr.  Whole warp.
__device__ __forceinline__ int32_t find_request(const int64_t* off, int32_t n_req, int64_t gr,
                                                int lane) {
  if (n_req <= 0) return -1;
  int64_t lo = 0, hi = n_req - 1;  // answer: largest r in [lo, hi] with off[r] <= gr
  while (hi > lo) {
    const int64_t step = (hi - lo + 32) / 32;
    const int64_t pos = lo + (int64_t)lane * step;
    const bool ok = pos <= hi && __ldg(off + pos) <= gr;
    const unsigned bal = __ballot_sync(FULL, ok);
    if (bal == 0) return -1;
    const int L = 31 - __clz(bal);
    lo = lo + (int64_t)L * step;
    hi = min(hi, lo + step - 1);
  }
  const int64_t a = __ldg(off + lo), c = __ldg(off + lo + 1);
  return (a <= gr && gr < c) ? (int32_t)lo : -1;
}

// Route mode: whether request r's rows [lo, hi) are inconsistent with the
// batch.  A whole-batch call also needs the last request to end at the last row.
__device__ __forceinline__ bool route_bad_request(const Args& a, int64_t r, int64_t lo,
                                                  int64_t hi) {
  return lo < 0 || hi < lo || hi > a.max_rows ||
         (a.whole && r == (int64_t)a.n_req - 1 && hi != a.max_rows);
}

// Route mode: the results of empty requests touching this launch's row range
// and of requests whose offsets are inconsistent (requests start, start +
// stride, ...).  Written by every launch; idempotent.
__device__ __forceinline__ void route_special_requests(const Args& a, int64_t start,
                                                       int64_t stride) {
  for (int64_t r = start; r < a.n_req; r += stride) {
    const int64_t lo = a.offsets[r], hi = a.offsets[r + 1];
    if (route_bad_request(a, r, lo, hi)) {
      write_special(r, NAN, FLAG_BAD_OFFSETS, a.agg, a.score, a.ship, a.req_flags);
      atomicOr(a.ctx_flags, FLAG_BAD_OFFSETS);
    } else if (lo == hi && lo >= a.row_base && lo <= a.row_base + a.n_rows) {
      write_special(r, 0.f, FLAG_EMPTY_REQ, a.agg, a.score, a.ship, a.req_flags);
    }
  }
}


// ---- cluster helpers ------------------------------------------------------------------

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ uint32_t dsmem_addr(const void* p, uint32_t rank) {
  uint32_t local = (uint32_t)__cvta_generic_to_shared(p), remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(rank));
  return remote;
}
__device__ __forceinline__ float dsmem_ld_f32(uint32_t a) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ int dsmem_ld_s32(uint32_t a) {
  int v;
  asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ uint64_t dsmem_ld_u64(uint32_t a) {
  uint64_t v;
  asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(a) : "memory");
  return v;
}

// ---- block reduction of the (m, S, U, bad) state ------------------------------------

__device__ __forceinline__ void block_reduce_state(Smem& sm, float& m, float& S, float& U,
                                                   bool& bad, int warp, int lane) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float mo = __shfl_xor_sync(FULL, m, o);
    const float So = __shfl_xor_sync(FULL, S, o);
    const float Uo = __shfl_xor_sync(FULL, U, o);
    lse_merge(m, S, U, mo, So, Uo);
  }
  bad = __any_sync(FULL, bad);
  if (lane == 0) {
    sm.pm[warp] = m;
    sm.pS[warp] = S;
    sm.pU[warp] = U;
    sm.pbad[warp] = bad;
  }
  __syncthreads();
  if (warp == 0) {
    m = lane < NWARP ? sm.pm[lane] : M2_INIT;
    S = lane < NWARP ? sm.pS[lane] : 0.f;
    U = lane < NWARP ? sm.pU[lane] : 0.f;
    bad = lane < NWARP ? (sm.pbad[lane] != 0) : false;
#pragma unroll
    for (int o = NWARP / 2; o > 0; o >>= 1) {
      const float mo = __shfl_xor_sync(FULL, m, o);
      const float So = __shfl_xor_sync(FULL, S, o);
      const float Uo = __shfl_xor_sync(FULL, U, o);
      lse_merge(m, S, U, mo, So, Uo);
    }
    bad = __any_sync(FULL, bad);
    // only lanes 0..NWARP-1 took part in the last butterfly: give every lane the total
    m = __shfl_sync(FULL, m, 0);
    S = __shfl_sync(FULL, S, 0);
    U = __shfl_sync(FULL, U, 0);
  }
}

// ---- one row's features and the mode's epilogue (one warp) ------------------------------

// What a row's epilogue needs that does not depend on the reduction: the
// emitted token and its logit, and the row's request (rows, from the CSR
// offsets) or decode slot.  The persistent kernel loads it for the next row
// while it waits for that row's stream, off the critical path.
struct RowPre {
  int32_t y;       // emitted token id
  float xy;        // its logit (NaN when y is outside [0, V))
  int32_t r;       // request (features with offsets, route) or decode slot; -1 if none
  int64_t lo, hi;  // rows of the request
  int eos;         // decode: the request ends with this row
};

// Whole warp (the request search is warp-collective).
template <typename T, int MODE>
__device__ __forceinline__ RowPre load_pre(const Args& a, int64_t row, const char* rowp, int lane) {
  using Tr = Traits<T>;
  RowPre p;
  p.y = a.chosen[row];
  p.xy = (p.y >= 0 && (int64_t)p.y < a.vocab) ? Tr::elem(rowp, p.y) : NAN;
  p.r = -1;
  p.lo = p.hi = 0;
  p.eos = 0;
  if (MODE == MODE_FEATURES && a.offsets) {
    p.r = find_request(a.offsets, a.n_req, row, lane);
  } else if (MODE == MODE_ROUTE) {
    p.r = find_request(a.offsets, a.n_req, a.row_base + row, lane);
  } else if (MODE == MODE_DECODE) {
    p.r = a.slot[row];
    p.eos = a.eos[row];
  }
  if (MODE != MODE_DECODE && p.r >= 0) {
    p.lo = __ldg(a.offsets + p.r);
    p.hi = __ldg(a.offsets + p.r + 1);
  }
  return p;
}

__device__ __forceinline__ int atom_add_acq_rel(int* p, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

// Eq. 3 features of the row from its (m, S, U) state and its top-32 element keys
// E (lane 0 = largest), then, by mode: write the record; or fold it into the
// request and, for the request's last row, pool / score / threshold; or fold it
// into its decode slot.  Whole warp.
template <typename T, int MODE>
__device__ __forceinline__ void row_finish(const Args& a, int64_t row, float m, float S, float U,
                                           bool bad, uint64_t E, const RowPre& pre, int lane) {
  const int64_t V = a.vocab;
  const int kc = a.kc, K = a.topk;
  const int32_t y = pre.y;
  uint32_t flags = 0;
  if (y < 0 || (int64_t)y >= V) flags |= FLAG_BAD_CHOSEN;
  const bool nonfinite = bad || !(S > 0.f) || !isfinite(S) || !isfinite(U);
  if (nonfinite) flags |= FLAG_NONFINITE;

  const float log2S = log2f(S);
  const bool hasE = lane < kc && E != 0ull;
  const float xk = hasE ? key_val(E) : -INFINITY;
  const float lp2 = fmaf(xk, L2E, -m) - log2S;  // log2 p of this lane's token
  const float pk = hasE ? exp2f(lp2) : 0.f;
  float term = (lane < K && pk > 0.f) ? pk * lp2 : 0.f;
  float pmass = lane < K ? pk : 0.f;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    term += __shfl_xor_sync(FULL, term, o);
    pmass += __shfl_xor_sync(FULL, pmass, o);
  }
  const float hraw = term * LN2;  // sum over top-K of p ln p = -H^K
  const float h = a.renorm ? (pmass > 0.f ? hraw / pmass - logf(pmass) : 0.f) : hraw;
  const float x1 = __shfl_sync(FULL, xk, 0);
  const float p1 = __shfl_sync(FULL, pk, 0);
  const float p2 = V >= 2 ? __shfl_sync(FULL, pk, 1) : 0.f;
  const uint64_t e1 = shfl64(E, 0), e2 = shfl64(E, 1);
  float logp = NAN;
  if (!(flags & FLAG_BAD_CHOSEN)) logp = (fmaf(pre.xy, L2E, -m) - log2S) * LN2;
  float fv[NFEAT];
  fv[0] = logp;
  fv[1] = p1;
  fv[2] = p1 - p2;
  fv[3] = (log2S - U / S) * LN2;
  fv[4] = h;
  fv[5] = 0.f;
  fv[6] = (m + log2S) * LN2;
  fv[7] = x1;
  int32_t i1 = (int32_t)key_idx(e1), i2 = V >= 2 ? (int32_t)key_idx(e2) : -1;
  if (nonfinite) {
#pragma unroll
    for (int j = 0; j < NFEAT; ++j) fv[j] = NAN;
    i1 = i2 = -1;
  }

  if (MODE == MODE_FEATURES) {
    if (a.offsets && !nonfinite && pre.r >= 0)
      fv[5] = (float)(row - pre.lo + 1) / (float)(pre.hi - pre.lo);
    if (lane < NFEAT) {
      float v = fv[0];
#pragma unroll
      for (int j = 1; j < NFEAT; ++j)
        if (lane == j) v = fv[j];
      a.feat[row * NFEAT + lane] = v;
    }
    if (lane == 0) {
      a.top2[2 * row] = i1;
      a.top2[2 * row + 1] = i2;
      a.row_flags[row] = flags;
    }
    return;
  }

  if (MODE == MODE_ROUTE) {
    const int64_t gr = a.row_base + row;
    const int32_t r = pre.r;
    const int64_t lo = pre.lo, hi = pre.hi;
    if (r < 0 || route_bad_request(a, r, lo, hi)) {
      if (lane == 0) atomicOr(a.ctx_flags, FLAG_BAD_OFFSETS);
      return;
    }
    if (!nonfinite) fv[5] = (float)(gr - lo + 1) / (float)(hi - lo);
    int last = 0;
    if (lane == 0) {
      // the record, then one acquire-release increment: the request's last row
      // sees every other row's record
      float4* rp = reinterpret_cast<float4*>(a.rec + gr * NFEAT);
      rp[0] = make_float4(fv[0], fv[1], fv[2], fv[3]);
      rp[1] = make_float4(fv[4], fv[5], fv[6], fv[7]);
      a.rec_flags[gr] = flags;
      last = (atom_add_acq_rel(a.req_cnt + r, 1) == (int)(hi - lo) - 1);
    }
    last = __shfl_sync(FULL, last, 0);
    if (last) {
      const Pooled p = pool_rows(a.rec, a.rec_flags, lo, hi, a.w, a.b, a.zthr, lane);
      write_pooled(p, r, a.agg, a.score, a.ship, a.req_flags, lane);
      if (lane == 0) a.req_cnt[r] = 0;
    }
    return;
  }

  if (MODE == MODE_DECODE) {
    if (lane != 0) return;
    const int32_t s = pre.r;
    if (s < 0 || s >= a.n_slots) {
      atomicOr(a.ctx_flags, FLAG_BAD_SLOT);
      return;
    }
    float* A = a.acc + (int64_t)s * ACC_WORDS;
    const int32_t n = __float_as_int(A[0]) + 1;
    const uint32_t fl = __float_as_uint(A[1]) | flags;
    const float v[5] = {fv[0], fv[1], fv[2], -fv[3], fv[4]};
#pragma unroll
    for (int f = 0; f < 5; ++f) {
      if (n == 1) {
        A[2 + f] = v[f];
        A[7 + f] = 0.f;
        A[12 + f] = v[f];
      } else {
        // compensated (Kahan) running sum in step order
        const float sum = A[2 + f], comp = A[7 + f];
        const float yv = v[f] - comp;
        const float tsum = sum + yv;
        A[7 + f] = (tsum - sum) - yv;
        A[2 + f] = tsum;
        A[12 + f] = fminf(A[12 + f], v[f]);
      }
    }
    if (!pre.eos) {
      A[0] = __int_as_float(n);
      A[1] = __uint_as_float(fl);
      return;
    }
    // the request ends with this row: pool, score, ship rule, clear the slot
    float ag[NAGG];
    float sc;
    uint8_t sh;
    if (fl & (FLAG_NONFINITE | FLAG_BAD_CHOSEN)) {
      for (int j = 0; j < NAGG; ++j) ag[j] = NAN;
      sc = NAN;
      sh = 0;
    } else {
      const float Tf = (float)n;
      for (int f = 0; f < 5; ++f) {
        ag[2 * f] = A[2 + f] / Tf;
        ag[2 * f + 1] = A[12 + f];
      }
      ag[10] = (float)(n + 1) / (float)(2 * n);
      float z = a.b;
      for (int j = 0; j < NAGG; ++j) z = fmaf(__ldg(a.w + j), ag[j], z);
      sc = 1.f / (1.f + expf(-z));
      sh = (z >= a.zthr) ? 1 : 0;
    }
    if (a.agg)
      for (int j = 0; j < NAGG; ++j) a.agg[(int64_t)s * NAGG + j] = ag[j];
    a.score[s] = sc;
    a.ship[s] = sh;
    a.req_flags[s] = fl;
    for (int j = 0; j < ACC_WORDS; ++j) A[j] = 0.f;
  }
}

// ---- the row kernel for split rows: one thread-block cluster of C CTAs per row ----------------

// Resident CTAs per SM the compiler sizes registers for: five for fp32 rows
// (48 registers), four for bf16.  Measured in CUDA graphs with one CTA per
// row: 354-row batches of V = 32,000 fp32 10.0 us per batch with five
// against 11.5 us with four (two consecutive launches then fit on the GPU
// together), 256-row decode steps of V = 151,936 bf16 11.1 against 10.7 us.
template <typename T>
constexpr int rows_min_blocks() {
  return sizeof(T) == 4 ? 5 : 4;
}

template <typename T, int MODE, bool ALIGNED>
__global__ void __launch_bounds__(NT, rows_min_blocks<T>()) verify_rows(const Args a) {
  __shared__ Smem sm;
  using Tr = Traits<T>;
  constexpr int VEC = Tr::VEC;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t C, rank, cid;
  asm("mov.u32 %0, %%cluster_nctarank;" : "=r"(C));
  asm("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  asm("mov.u32 %0, %%clusterid.x;" : "=r"(cid));
  const int64_t row = cid;

  pdl_trigger();  // a dependent launch may start streaming while this one finishes

  const char* rowp = reinterpret_cast<const char*>(a.logits) + row * a.row_stride * (int64_t)sizeof(T);
  const uint4* vp = reinterpret_cast<const uint4*>(rowp);
  const int64_t V = a.vocab;
  const int32_t gfull = (int32_t)(V / VEC);  // full 16-byte groups
  const bool has_tail = (V % VEC) != 0;      // the partial last group, index gfull
  const int32_t g0 = (int32_t)((int64_t)gfull * rank / C);
  const int32_t g1 = (int32_t)((int64_t)gfull * (rank + 1) / C);
  const int32_t ng = g1 - g0;
  const int32_t nfull = ng / TILE, rem = ng - nfull * TILE;
  const int32_t ntiles = nfull + (rem > 0 ? 1 : 0);
  int shift = 0;
  while (((ntiles + (1 << shift) - 1) >> shift) > MAX_SLOTS) ++shift;
  const int32_t smask = (1 << shift) - 1;
  const int32_t nslots = (ntiles + smask) >> shift;
  const uint4 NEG = make_uint4(Tr::NEG_WORD, Tr::NEG_WORD, Tr::NEG_WORD, Tr::NEG_WORD);

  if (tid == 0) {
    sm.ncand = 0;
    sm.nelem = 0;
    sm.tail_max = -INFINITY;
  }

  float m = M2_INIT;
  float2 S2 = make_float2(0.f, 0.f), U2 = make_float2(0.f, 0.f);
  float thr_max = -INFINITY, racc = -INFINITY;
  bool bad = false;

  // ---- stream the groups [g0, g1): tile t holds groups t*TILE + k*NT + tid ------------
  {
    auto load = [&](int32_t gi) -> uint4 {
      return ALIGNED ? ld_stream(vp + g0 + gi) : Tr::load_elems(rowp, (int64_t)(g0 + gi));
    };
    // one CTA per row: one thread keeps the tiles PF_TILES ahead on their way
    // into L2 (bulk prefetches need no registers, so the CTA has more bytes in
    // flight than its two register tiles; measured on 256-row decode steps:
    // 24.9 us isolated and 11.2 us in a CUDA graph against 27.0 and 12.8 us
    // without; with clusters, whose CTAs already keep HBM busy, it slowed
    // the step)
    auto prefetch_tile = [&](int32_t t) {
      if (PF_TILES > 0 && ALIGNED && C == 1 && tid == 0 && t < ntiles) {
        const int32_t gs = t * TILE;
        prefetch_l2(vp + g0 + gs, (uint32_t)min(TILE, ng - gs) * 16u);
      }
    };
#pragma unroll
    for (int32_t p = 1; p <= PF_TILES; ++p) prefetch_tile(p);
    uint4 cur[UNR], nxt[UNR];
    if (nfull > 0) {
#pragma unroll
      for (int k = 0; k < UNR; ++k) cur[k] = load(k * NT + tid);
    } else {
#pragma unroll
      for (int k = 0; k < UNR; ++k) cur[k] = (k * NT + tid < rem) ? load(k * NT + tid) : NEG;
    }
    for (int32_t t = 0; t < ntiles; ++t) {
      const int32_t nb = (t + 1) * TILE;
      prefetch_tile(t + 1 + PF_TILES);
      if (t + 1 < nfull) {
#pragma unroll
        for (int k = 0; k < UNR; ++k) nxt[k] = load(nb + k * NT + tid);
      } else if (t + 1 < ntiles) {
#pragma unroll
        for (int k = 0; k < UNR; ++k) nxt[k] = (k * NT + tid < rem) ? load(nb + k * NT + tid) : NEG;
      }
      const float tmax = Tr::tile_max(cur);
      thr_max = fmaxf(thr_max, tmax);
      racc = fmaxf(racc, tmax);
      if ((t & smask) == smask || t == ntiles - 1) {
        sm.tm[t >> shift][tid] = racc;
        racc = -INFINITY;
      }
      // online rescale, branch-free (a no-op when the maximum did not move)
      const float mn = fmaxf(m, tmax * L2E);
      const float dl = m - mn;
      const float f = ex2(dl);
      U2 = __fmul2_rn(make_float2(f, f), __ffma2_rn(make_float2(dl, dl), S2, U2));
      S2 = __fmul2_rn(make_float2(f, f), S2);
      m = mn;
      const float2 nm = make_float2(-m, -m);
      if (t < nfull) {
#pragma unroll
        for (int k = 0; k < UNR; ++k) Tr::accum(cur[k], nm, S2, U2);
      } else {
#pragma unroll
        for (int k = 0; k < UNR; ++k)
          if (k * NT + tid < rem) Tr::accum(cur[k], nm, S2, U2);
      }
#pragma unroll
      for (int k = 0; k < UNR; ++k) cur[k] = nxt[k];
    }
  }
  float S = S2.x + S2.y, U = U2.x + U2.y;

  // ---- the partial last group (fewer than VEC elements): cluster rank 0, thread 0
  if (has_tail && rank == 0 && tid == 0) {
    float tmx = -INFINITY;
    for (int64_t v = (int64_t)gfull * VEC; v < V; ++v) {
      const float x = Tr::elem(rowp, v);
      careful_add(x, m, S, U, bad);
      if (!isnan(x)) tmx = fmaxf(tmx, x);
    }
    sm.tail_max = tmx;
    thr_max = fmaxf(thr_max, tmx);
  }

  // ---- theta1: the kc-th largest per-thread maximum (a lower bound of the kc-th element)
  const int kc = a.kc;
  sm.wl[warp][lane] = warp_sort_desc<uint32_t>(ord(thr_max), lane);
  block_reduce_state(sm, m, S, U, bad, warp, lane);  // ends with a __syncthreads
  if (warp == 0) {
    uint32_t L = sm.wl[0][lane];
#pragma unroll 1
    for (int w2 = 1; w2 < NWARP; ++w2) L = warp_merge_desc<uint32_t>(L, sm.wl[w2][lane], lane);
    const float th1 = unord(__shfl_sync(FULL, L, kc - 1));
    if (lane == 0) {
      sm.theta1 = th1;
      sm.fallback = !(th1 > -INFINITY);
      // a masked (-inf), NaN or infinite logit made the CTA's fast
      // accumulators non-finite: it re-streams its range with guards (the
      // row's merged state is non-finite exactly when a CTA's is)
      sm.careful = (!bad && !(isfinite(S) && isfinite(U))) ? 1 : 0;
    }
  }
  if (tid < 32) sm.top[tid] = 0ull;
  __syncthreads();
  if (sm.careful) {
    float cm = M2_INIT, cS = 0.f, cU = 0.f;
    bool cbad = false;
    const int64_t e1 = (int64_t)g1 * VEC;
    for (int64_t v = (int64_t)g0 * VEC + tid; v < e1; v += NT)
      careful_add(Tr::elem(rowp, v), cm, cS, cU, cbad);
    if (has_tail && rank == 0)
      for (int64_t v = (int64_t)gfull * VEC + tid; v < V; v += NT)
        careful_add(Tr::elem(rowp, v), cm, cS, cU, cbad);
    block_reduce_state(sm, cm, cS, cU, cbad, warp, lane);  // warp 0 holds the CTA's state
    m = cm;
    S = cS;
    U = cU;
    bad = cbad;
  }

  // ---- candidate super-groups: stored tile maxima >= theta1
  const float th1 = sm.theta1;
  if (!sm.fallback) {
    for (int32_t s = 0; s < nslots; ++s) {
      const float v = sm.tm[s][tid];
      if (v >= th1) {
        const int i = atomicAdd(&sm.ncand, 1);
        if (i < CCAP) {
          sm.cand_v[i] = v;
          sm.cand_id[i] = ((uint32_t)s << 8) | (uint32_t)tid;
        }
      }
    }
    if (tid == 0 && has_tail && rank == 0 && sm.tail_max >= th1) {
      const int i = atomicAdd(&sm.ncand, 1);
      if (i < CCAP) {
        sm.cand_v[i] = sm.tail_max;
        sm.cand_id[i] = TAIL_ID;
      }
    }
  }
  __syncthreads();

  // ---- re-read the candidates; their elements >= theta1 become keys (kc
  // distinct elements reach theta1, so the CTA's top kc are among them)
  const int ncand = sm.ncand;
  const bool fb_cand = sm.fallback || ncand > CCAP;
  if (!fb_cand) {
    const float th = th1;
    const int n = ncand;
    const int gpc = UNR << shift;  // groups per super-group
    for (int i = tid; i < n * gpc; i += NT) {
      const int c = i / gpc, j = i - c * gpc;
      const uint32_t id = sm.cand_id[c];
      if (id == TAIL_ID) {
        if (j != 0) continue;
        for (int64_t v = (int64_t)gfull * VEC; v < V; ++v) {
          const float x = Tr::elem(rowp, v);
          if (x >= th) {
            const int e = atomicAdd(&sm.nelem, 1);
            if (e < ECAP) sm.ebuf[e] = make_key(x, (uint32_t)v);
          }
        }
        continue;
      }
      const int32_t t = (int32_t)((id >> 8) << shift) + j / UNR;
      const int32_t gi = t * TILE + (j % UNR) * NT + (int32_t)(id & 255u);
      if (t >= ntiles || gi >= ng) continue;
      const int32_t g = g0 + gi;
      const uint4 wv = ALIGNED ? ld_reread(vp + g) : Tr::load_elems(rowp, (int64_t)g);
#pragma unroll
      for (int e2 = 0; e2 < VEC; ++e2) {
        const float x = Tr::at(wv, e2);
        if (x >= th) {
          const int e = atomicAdd(&sm.nelem, 1);
          if (e < ECAP) sm.ebuf[e] = make_key(x, (uint32_t)(g * VEC + e2));
        }
      }
    }
  }
  __syncthreads();

  // ---- what the row's epilogue needs besides the reduction (cluster rank 0,
  // warp 0), fetched now so that its latency overlaps the selection
  RowPre pre;
  if (rank == 0 && warp == 0) {
    pre = load_pre<T, MODE>(a, row, rowp, lane);
    if (C == 1) {
      pdl_wait();
      if (MODE == MODE_DECODE && lane == 0 && pre.r >= 0 && pre.r < a.n_slots) {
        const float* A = a.acc + (int64_t)pre.r * ACC_WORDS;  // into L1 for row_finish
        asm volatile("prefetch.global.L1 [%0];" ::"l"(A));
        asm volatile("prefetch.global.L1 [%0];" ::"l"(A + 16));
      }
    }
  }

  // ---- the CTA's exact top-32 elements: up to NT candidate keys are ranked
  // by counting (keys are distinct: the index is part of the key), more by
  // warp 0's sorting network; the exact scan when the buffers overflowed
  uint64_t E = 0ull;
  const int ne = sm.nelem;
  const bool fb = fb_cand || ne > ECAP;
  if (!fb && ne <= NT) {
    if (tid < ne) {
      const uint64_t key = sm.ebuf[tid];
      int rk = 0;
      for (int q = 0; q < ne; ++q) rk += sm.ebuf[q] > key ? 1 : 0;
      if (rk < 32) sm.top[rk] = key;
    }
    __syncthreads();
    if (warp == 0) E = sm.top[lane];
  } else if (warp == 0) {
    const int n = ne;
    if (!fb) {
      for (int b0 = 0; b0 < n; b0 += 32) {
        uint64_t k = b0 + lane < n ? sm.ebuf[b0 + lane] : 0ull;
        k = warp_sort_desc<uint64_t>(k, lane);
        E = warp_merge_desc<uint64_t>(E, k, lane);
      }
    } else {
      // exact scan of the whole range (rows whose ties overflow the buffers)
      const float thr = th1;
      WarpTopK ek;
      ek.buf = sm.ebuf;
      ek.cnt = 0;
      ek.list = 0ull;
      for (int32_t gb = 0; gb < ng; gb += 32) {
        const int32_t gi = gb + lane;
        const bool in = gi < ng;
        uint4 wv = NEG;
        if (in) wv = ALIGNED ? ld_stream(vp + g0 + gi) : Tr::load_elems(rowp, (int64_t)(g0 + gi));
#pragma unroll 1
        for (int e2 = 0; e2 < VEC; ++e2) {
          const float x = Tr::at(wv, e2);
          const bool c = in && x >= thr;
          ek.push(c, c ? make_key(x, (uint32_t)((g0 + gi) * VEC + e2)) : 0ull, lane);
          ek.drain(lane);
        }
      }
      if (has_tail && rank == 0) {
        for (int64_t v0 = (int64_t)gfull * VEC; v0 < V; v0 += 32) {
          const int64_t v = v0 + lane;
          const bool in = v < V;
          const float x = in ? Tr::elem(rowp, v) : -INFINITY;
          const bool c = in && x >= thr;
          ek.push(c, c ? make_key(x, (uint32_t)v) : 0ull, lane);
          ek.drain(lane);
        }
      }
      ek.drain_all(lane);
      E = ek.list;
    }
  }

  // ---- split-vocab merge across the cluster (distributed shared memory)
  if (C > 1) {
    if (warp == 0) {
      if (lane == 0) {
        sm.fm = m;
        sm.fS = S;
        sm.fU = U;
        sm.fbad = bad;
      }
      sm.flist[lane] = E;
    }
    cluster_sync_all();
    if (rank == 0 && warp == 0) {
      for (uint32_t r = 1; r < C; ++r) {
        const float mo = dsmem_ld_f32(dsmem_addr(&sm.fm, r));
        const float So = dsmem_ld_f32(dsmem_addr(&sm.fS, r));
        const float Uo = dsmem_ld_f32(dsmem_addr(&sm.fU, r));
        const int bo = dsmem_ld_s32(dsmem_addr(&sm.fbad, r));
        lse_merge(m, S, U, mo, So, Uo);
        bad = bad || bo;
        const uint64_t peer = dsmem_ld_u64(dsmem_addr(&sm.flist[lane], r));
        E = warp_merge_desc<uint64_t>(E, peer, lane);
      }
    }
    cluster_sync_all();
    if (rank != 0) return;
  }

  if (warp != 0) return;

  pdl_wait();
  if (MODE == MODE_ROUTE) {
    const int64_t nclusters = gridDim.x / C;
    route_special_requests(a, (int64_t)cid * 32 + lane, nclusters * 32);
  }
  row_finish<T, MODE>(a, row, m, S, U, bad, E, pre, lane);
}

// ---- the persistent, warp-specialised row kernel (one CTA per row at a time) -----------------
//
// NWARP streaming warps read rows blockIdx.x, blockIdx.x + gridDim.x, ...; they
// never wait on the per-row selection: at the end of a row they leave its tile
// maxima, per-warp (m, S, U), sorted per-thread maxima and each thread's best
// tile in one of two shared buffers, signal the finaliser warp with a named
// barrier and go on (the next
// row's first tile is already in flight).  The finaliser warp turns a buffer
// into the row's exact top-K, features and epilogue, then hands the buffer
// back.  Named barriers (bar.arrive / bar.sync with NT + 32 threads) are the
// only synchronisation; every thread reaches each of them a known number of
// times, so no wait depends on data.

constexpr int NT_WS = NT + 32;
constexpr int BAR_FULL = 1;   // ids 1, 2: buffer b holds a streamed row
constexpr int BAR_EMPTY = 3;  // ids 3, 4: buffer b may be overwritten

__device__ __forceinline__ void named_bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
__device__ __forceinline__ void named_bar_arrive(int id, int n) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(n) : "memory");
}

struct SmemWS {
  float4 tinfo[2][NT];          // per thread: best, second and third tile maxima, and
                                //   (best tile | second tile << 16); two row buffers
  uint32_t wl[2][NWARP][32];    // per-warp sorted per-thread maxima, ord() encoded
  float pm[2][NWARP], pS[2][NWARP], pU[2][NWARP];
  float cand_v[CCAP];           // finaliser: candidate tiles (value,
  uint32_t cand_id[CCAP];       //   tile << 8 | thread, | BEST_BIT for a thread's best tile)
  uint64_t ebuf[ECAP];          // finaliser: candidate element keys
  uint4 best[2][UNR][NT];       // per thread: the groups of its best tile, as streamed
};

// A candidate that is its thread's best tile: the finaliser reads its groups
// from SmemWS::best instead of re-reading the row (tile indices stay below 2^16).
constexpr uint32_t BEST_BIT = 0x80000000u;

// Row geometry shared by the streaming warps and the finaliser (C = 1).
struct RowGeom {
  int32_t gfull, nfull, rem, ntiles;
  bool has_tail;
  __device__ __forceinline__ RowGeom(int64_t V, int vec) {
    gfull = (int32_t)(V / vec);
    has_tail = (V % vec) != 0;
    nfull = gfull / TILE;
    rem = gfull - nfull * TILE;
    ntiles = nfull + (rem > 0 ? 1 : 0);
  }
};

// The finaliser warp's work for one streamed row held in buffer b.
//
// Every streaming thread reports its best and second-best tile (value and
// index) and its third-best tile value.  theta1 = the kc-th largest thread
// maximum.  Candidate tiles are the best / second-best tiles >= theta1; a
// thread whose third-best value also reaches theta1 contributes all its
// tiles, and then theta stays theta1 (exact, if slower).  Otherwise theta =
// the kc-th largest candidate value.  Elements >= theta of the candidate
// tiles are the only ones that can be among the top kc.  A best tile is read
// from the copy the streaming thread left in shared memory; the other
// candidate tiles are re-read from the row, which may have left L2 by then.
template <typename T, int MODE, bool ALIGNED>
__device__ __noinline__ void finalize_ws(const Args& a, SmemWS& sm, int b, int64_t row,
                                         const RowGeom& geo, const RowPre& pre, int lane) {
  using Tr = Traits<T>;
  constexpr int VEC = Tr::VEC;
  const int64_t V = a.vocab;
  const int kc = a.kc;
  const char* rowp = reinterpret_cast<const char*>(a.logits) + row * a.row_stride * (int64_t)sizeof(T);
  const uint4* vp = reinterpret_cast<const uint4*>(rowp);
  const uint4 NEG = make_uint4(Tr::NEG_WORD, Tr::NEG_WORD, Tr::NEG_WORD, Tr::NEG_WORD);
  const unsigned lt = (1u << lane) - 1u;

  // ---- the row's (m, S, U) from the streaming warps' partials
  float m = lane < NWARP ? sm.pm[b][lane] : M2_INIT;
  float S = lane < NWARP ? sm.pS[b][lane] : 0.f;
  float U = lane < NWARP ? sm.pU[b][lane] : 0.f;
#pragma unroll
  for (int o = NWARP / 2; o > 0; o >>= 1) {
    const float mo = __shfl_xor_sync(FULL, m, o);
    const float So = __shfl_xor_sync(FULL, S, o);
    const float Uo = __shfl_xor_sync(FULL, U, o);
    lse_merge(m, S, U, mo, So, Uo);
  }
  m = __shfl_sync(FULL, m, 0);
  S = __shfl_sync(FULL, S, 0);
  U = __shfl_sync(FULL, U, 0);
  bool bad = false;

  // ---- the partial last group (fewer than VEC elements)
  float tail_max = -INFINITY;
  if (geo.has_tail) {
    if (lane == 0) {
      for (int64_t v = (int64_t)geo.gfull * VEC; v < V; ++v) {
        const float x = Tr::elem(rowp, v);
        careful_add(x, m, S, U, bad);
        if (!isnan(x)) tail_max = fmaxf(tail_max, x);
      }
    }
    m = __shfl_sync(FULL, m, 0);
    S = __shfl_sync(FULL, S, 0);
    U = __shfl_sync(FULL, U, 0);
    bad = __shfl_sync(FULL, (int)bad, 0) != 0;
    tail_max = __shfl_sync(FULL, tail_max, 0);
  }

  // ---- theta1: the kc-th largest per-thread maximum (a merge tree over the
  // eight per-warp sorted lists; independent merges interleave)
  uint32_t L0 = warp_merge_desc<uint32_t>(sm.wl[b][0][lane], sm.wl[b][1][lane], lane);
  uint32_t L1 = warp_merge_desc<uint32_t>(sm.wl[b][2][lane], sm.wl[b][3][lane], lane);
  uint32_t L2 = warp_merge_desc<uint32_t>(sm.wl[b][4][lane], sm.wl[b][5][lane], lane);
  uint32_t L3 = warp_merge_desc<uint32_t>(sm.wl[b][6][lane], sm.wl[b][7][lane], lane);
  L0 = warp_merge_desc<uint32_t>(L0, L1, lane);
  L2 = warp_merge_desc<uint32_t>(L2, L3, lane);
  uint32_t L = warp_merge_desc<uint32_t>(L0, L2, lane);
  if (geo.has_tail) L = warp_merge_desc<uint32_t>(L, lane == 0 ? ord(tail_max) : 0u, lane);
  const float th1 = unord(__shfl_sync(FULL, L, kc - 1));
  bool fb = !(th1 > -INFINITY);

  // ---- candidate tiles
  int n = 0;            // candidate tiles
  bool all3 = false;    // some thread has three tiles >= theta1
  if (!fb) {
#pragma unroll 2
    for (int j = 0; j < NT / 32; ++j) {
      const uint32_t t = (uint32_t)(j * 32 + lane);
      const float4 inf = sm.tinfo[b][t];
      const uint32_t ids = __float_as_uint(inf.w);
      const bool c1 = inf.x >= th1, c2 = inf.y >= th1, c3 = inf.z >= th1;
      all3 = all3 || c3;
      // the best and second-best tiles
      const unsigned b1 = __ballot_sync(FULL, c1);
      const unsigned b2 = __ballot_sync(FULL, c2 && !c3);
      const int p1 = n + __popc(b1 & lt);
      const int p2 = n + __popc(b1) + __popc(b2 & lt);
      if (c1 && p1 < CCAP) {
        sm.cand_v[p1] = inf.x;
        sm.cand_id[p1] = BEST_BIT | ((ids & 0xffffu) << 8) | t;
      }
      if (c2 && !c3 && p2 < CCAP) {
        sm.cand_v[p2] = inf.y;
        sm.cand_id[p2] = ((ids >> 16) << 8) | t;
      }
      n += __popc(b1) + __popc(b2);
      // a thread with a third tile >= theta1: every other tile of it
      unsigned b3 = __ballot_sync(FULL, c3);
      while (b3) {
        const int src = __ffs(b3) - 1;
        b3 &= b3 - 1;
        const uint32_t ts = (uint32_t)(j * 32 + src);
        const uint32_t ids_s = __shfl_sync(FULL, ids, src);
        const uint32_t ti1 = ids_s & 0xffffu;
        for (int t0 = 0; t0 < geo.ntiles; t0 += 32) {
          const int tt = t0 + lane;
          const bool c = tt < geo.ntiles && (uint32_t)tt != ti1;
          const unsigned bb = __ballot_sync(FULL, c);
          const int pos = n + __popc(bb & lt);
          if (c && pos < CCAP) {
            sm.cand_v[pos] = th1;
            sm.cand_id[pos] = ((uint32_t)tt << 8) | ts;
          }
          n += __popc(bb);
        }
      }
    }
    all3 = __any_sync(FULL, all3);
    // the partial last group is a candidate too (its elements are read below)
    if (geo.has_tail && tail_max >= th1) {
      if (lane == 0 && n < CCAP) {
        sm.cand_v[n] = tail_max;
        sm.cand_id[n] = TAIL_ID;
      }
      ++n;
    }
    if (n > CCAP) fb = true;
  }
  __syncwarp();

  // ---- the candidate tiles' groups: a thread's best tile from shared
  // memory, the others re-read from the row (issued first, so that sorting
  // the candidates for theta overlaps the loads); then keep elements >= theta
  const int total = fb ? 0 : n * UNR;
  // group `it` of the candidates (UNR per candidate tile): its index in the
  // row (or -1: none, or the partial last group) and its 16 bytes
  auto cand_group = [&](int it, int32_t& gsel_q, uint4& w) {
    gsel_q = -1;
    w = NEG;
    const uint32_t id = sm.cand_id[it >> 2];
    if (id == TAIL_ID) return;
    const int k = it & (UNR - 1), t = (int)(id & 255u);
    const int32_t gi = (int32_t)((id & ~BEST_BIT) >> 8) * TILE + k * NT + t;
    if (gi >= geo.gfull) return;
    gsel_q = gi;
    if (id & BEST_BIT) w = sm.best[b][k][t];
    else w = ALIGNED ? ld_reread(vp + gi) : Tr::load_elems(rowp, gi);
  };
  uint4 wv[4];
  int32_t gsel[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int it = q * 32 + lane;
    gsel[q] = -1;
    wv[q] = NEG;
    if (it < total) cand_group(it, gsel[q], wv[q]);
  }

  // ---- theta: the exact kc-th largest candidate value (theta1 if a thread
  // contributed all its tiles)
  float th = th1;
  if (!fb && !all3) {
    uint32_t Lc = 0u;
#pragma unroll 1
    for (int b0 = 0; b0 < n; b0 += 32) {
      uint32_t k = b0 + lane < n ? ord(sm.cand_v[b0 + lane]) : 0u;
      k = warp_sort_desc<uint32_t>(k, lane);
      Lc = warp_merge_desc<uint32_t>(Lc, k, lane);
    }
    const uint32_t kth = __shfl_sync(FULL, Lc, kc - 1);
    if (kth != 0u) th = unord(kth);  // (there are always kc candidates; kept as a guard)
  }

  int ne = 0;
  if (!fb) {
    for (int i0 = 0; i0 < total; i0 += 128) {
      if (i0 > 0) {
        // more than 128 candidate groups: the next batch of loads
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int it = i0 + q * 32 + lane;
          gsel[q] = -1;
          wv[q] = NEG;
          if (it < total && sm.cand_v[it >> 2] >= th) cand_group(it, gsel[q], wv[q]);
        }
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
#pragma unroll
        for (int e2 = 0; e2 < VEC; ++e2) {
          const float x = Tr::at(wv[q], e2);
          const bool c = gsel[q] >= 0 && x >= th;
          const unsigned bal = __ballot_sync(FULL, c);
          const int pos = ne + __popc(bal & lt);
          if (c && pos < ECAP) sm.ebuf[pos] = make_key(x, (uint32_t)(gsel[q] * VEC + e2));
          ne += __popc(bal);
        }
      }
    }
    if (geo.has_tail && tail_max >= th) {
      const int64_t v = (int64_t)geo.gfull * VEC + lane;
      const float x = v < V ? Tr::elem(rowp, v) : -INFINITY;
      const bool c = v < V && x >= th;
      const unsigned bal = __ballot_sync(FULL, c);
      const int pos = ne + __popc(bal & lt);
      if (c && pos < ECAP) sm.ebuf[pos] = make_key(x, (uint32_t)v);
      ne += __popc(bal);
    }
    if (ne > ECAP) fb = true;
  }
  __syncwarp();

  // ---- the row's exact top-32 elements
  uint64_t E = 0ull;
  if (!fb) {
#pragma unroll 1
    for (int b0 = 0; b0 < ne; b0 += 32) {
      uint64_t k = b0 + lane < ne ? sm.ebuf[b0 + lane] : 0ull;
      k = warp_sort_desc<uint64_t>(k, lane);
      E = warp_merge_desc<uint64_t>(E, k, lane);
    }
  } else {
    // exact scan of the whole row (rows whose ties overflow the buffers)
    WarpTopK ek;
    ek.buf = sm.ebuf;
    ek.cnt = 0;
    ek.list = 0ull;
#pragma unroll 1
    for (int32_t g0 = 0; g0 < geo.gfull; g0 += 32) {
      const int32_t g = g0 + lane;
      const bool in = g < geo.gfull;
      uint4 w4 = NEG;
      if (in) w4 = ALIGNED ? ld_stream(vp + g) : Tr::load_elems(rowp, g);
#pragma unroll 1
      for (int e2 = 0; e2 < VEC; ++e2) {
        const float x = Tr::at(w4, e2);
        const bool c = in && x >= th1;
        ek.push(c, c ? make_key(x, (uint32_t)(g * VEC + e2)) : 0ull, lane);
        ek.drain(lane);
      }
    }
    if (geo.has_tail) {
      const int64_t v = (int64_t)geo.gfull * VEC + lane;
      const bool in = v < V;
      const float x = in ? Tr::elem(rowp, v) : -INFINITY;
      const bool c = in && x >= th1;
      ek.push(c, c ? make_key(x, (uint32_t)v) : 0ull, lane);
      ek.drain(lane);
    }
    ek.drain_all(lane);
    E = ek.list;
  }

  // ---- rows that made the fast accumulators non-finite: re-stream with guards
  if (!bad && !(isfinite(S) && isfinite(U))) {
    float cm = M2_INIT, cS = 0.f, cU = 0.f;
    bool cbad = false;
#pragma unroll 1
    for (int64_t v = lane; v < V; v += 32) careful_add(Tr::elem(rowp, v), cm, cS, cU, cbad);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float mo = __shfl_xor_sync(FULL, cm, o);
      const float So = __shfl_xor_sync(FULL, cS, o);
      const float Uo = __shfl_xor_sync(FULL, cU, o);
      lse_merge(cm, cS, cU, mo, So, Uo);
    }
    m = __shfl_sync(FULL, cm, 0);
    S = __shfl_sync(FULL, cS, 0);
    U = __shfl_sync(FULL, cU, 0);
    bad = __any_sync(FULL, cbad);
  }

  row_finish<T, MODE>(a, row, m, S, U, bad, E, pre, lane);
}

template <typename T, int MODE, bool ALIGNED>
__global__ void __launch_bounds__(NT_WS, 3) verify_rows_ws(const Args a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  SmemWS& sm = *reinterpret_cast<SmemWS*>(smem_raw);
  using Tr = Traits<T>;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t G = gridDim.x;

  pdl_trigger();  // a dependent launch may start streaming while this one finishes

  const RowGeom geo(a.vocab, Tr::VEC);

  if (warp == NWARP) {
    // ---- the finaliser warp: the next row's inputs are fetched while its
    // stream is still running
    auto rowp_of = [&](int64_t r) {
      return reinterpret_cast<const char*>(a.logits) + r * a.row_stride * (int64_t)sizeof(T);
    };
    int i = 0;
    int64_t row = blockIdx.x;
    RowPre pre = load_pre<T, MODE>(a, row, rowp_of(row), lane);
    pdl_wait();
    if (MODE == MODE_ROUTE) route_special_requests(a, (int64_t)blockIdx.x * 32 + lane, G * 32);
    for (; row < a.n_rows; row += G, ++i) {
      const int b = i & 1;
      named_bar_sync(BAR_FULL + b, NT_WS);
      finalize_ws<T, MODE, ALIGNED>(a, sm, b, row, geo, pre, lane);
      if (row + 2 * G < a.n_rows) {
        __syncwarp();
        __threadfence_block();
        named_bar_arrive(BAR_EMPTY + b, NT_WS);
      }
      if (row + G < a.n_rows) pre = load_pre<T, MODE>(a, row + G, rowp_of(row + G), lane);
    }
    return;
  }

  // ---- the streaming warps
  const uint4 NEG = make_uint4(Tr::NEG_WORD, Tr::NEG_WORD, Tr::NEG_WORD, Tr::NEG_WORD);
  auto load_tile = [&](uint4 (&dst)[UNR], int64_t r, int32_t t) {
    const char* rp = reinterpret_cast<const char*>(a.logits) + r * a.row_stride * (int64_t)sizeof(T);
    const uint4* vp = reinterpret_cast<const uint4*>(rp);
    const int32_t base = t * TILE + tid;
    if (t < geo.nfull) {
#pragma unroll
      for (int k = 0; k < UNR; ++k)
        dst[k] = ALIGNED ? ld_stream(vp + base + k * NT) : Tr::load_elems(rp, base + k * NT);
    } else {
#pragma unroll
      for (int k = 0; k < UNR; ++k)
        dst[k] = (k * NT + tid < geo.rem)
                     ? (ALIGNED ? ld_stream(vp + base + k * NT) : Tr::load_elems(rp, base + k * NT))
                     : NEG;
    }
  };

  uint4 cur[UNR], nxt[UNR];
  int64_t row = blockIdx.x;
  if (row < a.n_rows && geo.ntiles > 0) load_tile(cur, row, 0);
  int i = 0;
  while (row < a.n_rows) {
    const int b = i & 1;
    if (i >= 2) named_bar_sync(BAR_EMPTY + b, NT_WS);
    const int64_t next = row + G;
    float m = M2_INIT;
    float2 S2 = make_float2(0.f, 0.f), U2 = make_float2(0.f, 0.f);
    // this thread's best, second and third tile maxima and the first two tiles
    float v1 = -INFINITY, v2 = -INFINITY, v3 = -INFINITY;
    uint32_t i1 = 0, i2 = 0;
    for (int32_t t = 0; t < geo.ntiles; ++t) {
      if (t + 1 < geo.ntiles) load_tile(nxt, row, t + 1);
      else if (next < a.n_rows) load_tile(nxt, next, 0);
      const float tmax = Tr::tile_max(cur);
      {
        const bool c1 = tmax > v1, c2 = tmax > v2;
        if (c1) {  // a new best tile: keep its groups for the finaliser
#pragma unroll
          for (int k = 0; k < UNR; ++k) sm.best[b][k][tid] = cur[k];
        }
        v3 = fmaxf(v3, fminf(tmax, v2));
        const float nv2 = c1 ? v1 : (c2 ? tmax : v2);
        const uint32_t ni2 = c1 ? i1 : (c2 ? (uint32_t)t : i2);
        v1 = c1 ? tmax : v1;
        i1 = c1 ? (uint32_t)t : i1;
        v2 = nv2;
        i2 = ni2;
      }
      const float mn = fmaxf(m, tmax * L2E);
      const float dl = m - mn;
      const float f = ex2(dl);
      U2 = __fmul2_rn(make_float2(f, f), __ffma2_rn(make_float2(dl, dl), S2, U2));
      S2 = __fmul2_rn(make_float2(f, f), S2);
      m = mn;
      const float2 nm = make_float2(-m, -m);
      if (t < geo.nfull) {
#pragma unroll
        for (int k = 0; k < UNR; ++k) Tr::accum(cur[k], nm, S2, U2);
      } else {
#pragma unroll
        for (int k = 0; k < UNR; ++k)
          if (k * NT + tid < geo.rem) Tr::accum(cur[k], nm, S2, U2);
      }
#pragma unroll
      for (int k = 0; k < UNR; ++k) cur[k] = nxt[k];
    }
    // the warp's partial state, its sorted per-thread maxima, the tile report
    float S = S2.x + S2.y, U = U2.x + U2.y;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float mo = __shfl_xor_sync(FULL, m, o);
      const float So = __shfl_xor_sync(FULL, S, o);
      const float Uo = __shfl_xor_sync(FULL, U, o);
      lse_merge(m, S, U, mo, So, Uo);
    }
    if (lane == 0) {
      sm.pm[b][warp] = m;
      sm.pS[b][warp] = S;
      sm.pU[b][warp] = U;
    }
    sm.wl[b][warp][lane] = warp_sort_desc<uint32_t>(ord(v1), lane);
    sm.tinfo[b][tid] = make_float4(v1, v2, v3, __uint_as_float(i1 | (i2 << 16)));
    __syncwarp();
    __threadfence_block();
    named_bar_arrive(BAR_FULL + b, NT_WS);
    row = next;
    ++i;
  }
}

// ---- standalone pooling kernel: one warp per request ----------------------------------

struct AggArgs {
  const float* feat;
  const uint32_t* row_flags;
  int64_t n_rows;
  const int64_t* offsets;
  int32_t n_req;
  const float* w;
  float b, zthr;
  float* agg;
  float* score;
  uint8_t* ship;
  uint32_t* req_flags;
  uint32_t* ctx_flags;
};

// internal linkage: the header is included by more than one translation unit
static __global__ void __launch_bounds__(NT) pool_requests(const AggArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t r = (int64_t)blockIdx.x * NWARP + (threadIdx.x >> 5);
  if (r >= a.n_req) return;
  const int64_t lo = a.offsets[r], hi = a.offsets[r + 1];
  if (lo < 0 || hi < lo || hi > a.n_rows) {
    if (lane == 0) {
      write_special(r, NAN, FLAG_BAD_OFFSETS, a.agg, a.score, a.ship, a.req_flags);
      atomicOr(a.ctx_flags, FLAG_BAD_OFFSETS);
    }
    return;
  }
  if (lo == hi) {
    if (lane == 0) write_special(r, 0.f, FLAG_EMPTY_REQ, a.agg, a.score, a.ship, a.req_flags);
    return;
  }
  const Pooled p = pool_rows(a.feat, a.row_flags, lo, hi, a.w, a.b, a.zthr, lane);
  write_pooled(p, r, a.agg, a.score, a.ship, a.req_flags, lane);
}

}  // namespace prk
