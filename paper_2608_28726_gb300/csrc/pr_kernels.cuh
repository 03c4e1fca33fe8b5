// Kernels of the verifier data path: the row kernel (Eq. 3 features, with a
// fused pooling / scoring / ship-rule epilogue in route and decode modes) and
// the standalone pooling kernel.  Algorithm notes are in pr_device.cuh.
#pragma once

#include "pr_device.cuh"

namespace prk {

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

// ---- the row kernel ------------------------------------------------------------------------

template <typename T, int MODE, bool ALIGNED>
__global__ void __launch_bounds__(NT) verify_rows(const Args a) {
  __shared__ Smem sm;
  using Tr = Traits<T>;
  constexpr int VEC = Tr::VEC;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t C, rank, cid;
  asm("mov.u32 %0, %%cluster_nctarank;" : "=r"(C));
  asm("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  asm("mov.u32 %0, %%clusterid.x;" : "=r"(cid));
  const int64_t row = cid;

  // Route mode: every launch writes the results of empty requests touching its
  // row range and of requests whose offsets are inconsistent.
  if (MODE == MODE_ROUTE) {
    for (int64_t r = (int64_t)blockIdx.x * NT + tid; r < a.n_req; r += (int64_t)gridDim.x * NT) {
      const int64_t lo = a.offsets[r], hi = a.offsets[r + 1];
      if (lo < 0 || hi < lo || hi > a.max_rows) {
        write_special(r, NAN, FLAG_BAD_OFFSETS, a.agg, a.score, a.ship, a.req_flags);
        atomicOr(a.ctx_flags, FLAG_BAD_OFFSETS);
      } else if (lo == hi && lo >= a.row_base && lo <= a.row_base + a.n_rows) {
        write_special(r, 0.f, FLAG_EMPTY_REQ, a.agg, a.score, a.ship, a.req_flags);
      }
    }
  }

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
  const int kc = a.kc, K = a.topk;
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
    }
  }
  __syncthreads();

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

  // ---- theta: the exact kc-th largest candidate value (warp 0)
  if (warp == 0 && !sm.fallback) {
    const int n = sm.ncand;
    if (n > CCAP) {
      if (lane == 0) sm.fallback = 1;
    } else {
      uint32_t L = 0u;
      for (int b0 = 0; b0 < n; b0 += 32) {
        uint32_t k = b0 + lane < n ? ord(sm.cand_v[b0 + lane]) : 0u;
        k = warp_sort_desc<uint32_t>(k, lane);
        L = warp_merge_desc<uint32_t>(L, k, lane);
      }
      const float th = unord(__shfl_sync(FULL, L, kc - 1));
      if (lane == 0) sm.theta = th;
    }
  }
  __syncthreads();

  // ---- re-read the candidates >= theta; elements >= theta become keys
  if (!sm.fallback) {
    const float th = sm.theta;
    const int n = sm.ncand;
    const int gpc = UNR << shift;  // groups per super-group
    for (int i = tid; i < n * gpc; i += NT) {
      const int c = i / gpc, j = i - c * gpc;
      if (!(sm.cand_v[c] >= th)) continue;
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
      const uint4 wv = ALIGNED ? ld_stream(vp + g) : Tr::load_elems(rowp, (int64_t)g);
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

  // ---- the CTA's exact top-32 elements (warp 0)
  uint64_t E = 0ull;
  if (warp == 0) {
    const int n = sm.nelem;
    if (!sm.fallback && n <= ECAP) {
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

  // ---- rows that made the fast accumulators non-finite: re-stream with guards
  if (warp == 0 && lane == 0) sm.careful = (!bad && !(isfinite(S) && isfinite(U))) ? 1 : 0;
  __syncthreads();
  if (sm.careful) {
    float cm = M2_INIT, cS = 0.f, cU = 0.f;
    bool cbad = false;
    for (int64_t v = tid; v < V; v += NT) careful_add(Tr::elem(rowp, v), cm, cS, cU, cbad);
    block_reduce_state(sm, cm, cS, cU, cbad, warp, lane);
    m = cm;
    S = cS;
    U = cU;
    bad = cbad;
  }
  if (warp != 0) return;

  // ---- finalize the row's record
  const int32_t y = a.chosen[row];
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
  if (!(flags & FLAG_BAD_CHOSEN)) {
    const float xy = Tr::elem(rowp, y);
    logp = (fmaf(xy, L2E, -m) - log2S) * LN2;
  }
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
    if (a.offsets && !nonfinite) {
      const int32_t r = find_request(a.offsets, a.n_req, row, lane);
      if (r >= 0) {
        const int64_t lo = __ldg(a.offsets + r), hi = __ldg(a.offsets + r + 1);
        fv[5] = (float)(row - lo + 1) / (float)(hi - lo);
      }
    }
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
    const int32_t r = find_request(a.offsets, a.n_req, gr, lane);
    const int64_t lo = r >= 0 ? __ldg(a.offsets + r) : 0, hi = r >= 0 ? __ldg(a.offsets + r + 1) : 0;
    if (r < 0 || lo < 0 || hi > a.max_rows) {
      if (lane == 0) atomicOr(a.ctx_flags, FLAG_BAD_OFFSETS);
      return;
    }
    if (!nonfinite) fv[5] = (float)(gr - lo + 1) / (float)(hi - lo);
    if (lane < NFEAT) {
      float v = fv[0];
#pragma unroll
      for (int j = 1; j < NFEAT; ++j)
        if (lane == j) v = fv[j];
      a.rec[gr * NFEAT + lane] = v;
    }
    if (lane == 0) a.rec_flags[gr] = flags;
    __threadfence();
    __syncwarp();
    int last = 0;
    if (lane == 0) last = (atomicAdd(a.req_cnt + r, 1) == (int)(hi - lo) - 1);
    last = __shfl_sync(FULL, last, 0);
    if (last) {
      __threadfence();
      const Pooled p = pool_rows(a.rec, a.rec_flags, lo, hi, a.w, a.b, a.zthr, lane);
      write_pooled(p, r, a.agg, a.score, a.ship, a.req_flags, lane);
      if (lane == 0) a.req_cnt[r] = 0;
    }
    return;
  }

  if (MODE == MODE_DECODE) {
    if (lane != 0) return;
    const int32_t s = a.slot[row];
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
    if (!a.eos[row]) {
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

__global__ void __launch_bounds__(NT) pool_requests(const AggArgs a) {
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
