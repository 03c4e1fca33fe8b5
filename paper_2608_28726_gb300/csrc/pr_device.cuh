// Device code of the verifier data path (Pro-Router, Section 3.1, Eq. 3).
//
// One kernel streams each logit row once from HBM and reduces it to the
// per-token features of Eq. 3; the same kernel, in its epilogue, pools finished
// requests, scores them and applies the ship rule "score >= tau".
//
// Row reduction (one CTA per row, or a thread-block cluster of C CTAs that
// split the row and merge through distributed shared memory):
//   * online log-sum-exp and entropy in base 2: with t_v = x_v log2(e) and a
//     running maximum m (itself some rounded x log2(e)), each thread keeps
//     S = sum 2^(t_v - m) and U = sum 2^(t_v - m) (t_v - m).  Then
//     LSE = ln2 (m + log2 S) and H = ln2 (log2 S - U / S).  Partial states
//     merge as S = sum_i S_i 2^(m_i - M), U = sum_i 2^(m_i - M)(U_i + (m_i - M) S_i).
//     The row is read in tiles of 4 x 16 bytes per thread; the tile maximum is
//     a packed max tree, the per-element work one packed FMA, one ex2, one
//     packed add and one packed FMA per two elements (f32x2 of sm_100+).
//   * exact top-K (and the first two tokens, lower index first on ties) at
//     almost no streaming cost: each thread only stores the maximum of each of
//     its tiles in shared memory.  After the stream, theta1 = the K-th largest
//     per-thread maximum is a lower bound of the K-th largest element (K
//     distinct elements reach it); the stored tile maxima >= theta1 are the
//     candidate "super-groups"; theta = the K-th largest candidate value is a
//     tighter bound, and every element >= theta lies in a candidate >= theta
//     (an element below theta has K strictly larger elements, the maxima of K
//     candidates).  Those few super-groups are re-read and their elements
//     >= theta sorted by (value, lower index first) with warp bitonic networks.
//     Ties never lose an element; rows whose ties swamp the buffers fall back
//     to an exact scan of the whole row.
//   * rows with -inf (masked tokens), NaN or +inf make the fast accumulators
//     non-finite; such rows are re-streamed with per-element guards, which
//     classify them exactly.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace prk {

constexpr int NT = 256;            // threads per CTA
constexpr int NWARP = NT / 32;     // warps per CTA
constexpr int UNR = 4;             // 16-byte groups per thread per tile
constexpr int TILE = NT * UNR;     // groups per CTA tile
constexpr int PF_TILES = 2;        // one CTA per row: tiles prefetched into L2 ahead of the loads
constexpr int MAX_SLOTS = 24;      // stored tile maxima per thread (tiles are merged beyond)
constexpr int CCAP = 256;          // candidate super-groups
constexpr int ECAP = 512;          // candidate elements
constexpr int MAXC = 8;            // largest cluster (CTAs per row)
constexpr int NFEAT = 8;
constexpr int NAGG = 11;
constexpr int ACC_WORDS = 20;      // decode slot: n, flags, 5 sums, 5 compensations, 5 minima, pad
constexpr float L2E = 1.4426950408889634f;
constexpr float LN2 = 0.6931471805599453f;
constexpr float M2_INIT = -1e30f;  // finite "no maximum yet" so that 2^(m - m') is 0, never NaN
constexpr unsigned FULL = 0xffffffffu;
constexpr uint32_t TAIL_ID = 0xffffffffu;  // candidate id of the partial last group

constexpr uint32_t FLAG_NONFINITE = 1u;
constexpr uint32_t FLAG_BAD_CHOSEN = 2u;
constexpr uint32_t FLAG_EMPTY_REQ = 4u;
constexpr uint32_t FLAG_BAD_OFFSETS = 8u;
constexpr uint32_t FLAG_BAD_SLOT = 16u;

enum Mode { MODE_FEATURES = 0, MODE_ROUTE = 1, MODE_DECODE = 2 };

struct Args {
  const void* logits;
  int64_t n_rows, vocab, row_stride;  // row_stride in elements
  const int32_t* chosen;
  int32_t topk, kc, renorm, aligned;  // kc = max(topk, 2)
  // features
  const int64_t* offsets;
  int32_t n_req;
  int64_t row_base;
  float* feat;
  int32_t* top2;
  uint32_t* row_flags;
  // route
  float* rec;
  uint32_t* rec_flags;
  int32_t* req_cnt;
  int64_t max_rows;
  const float* w;
  float b, zthr;
  float* score;
  uint8_t* ship;
  uint32_t* req_flags;
  float* agg;
  // decode
  const int32_t* slot;
  const uint8_t* eos;
  float* acc;
  int32_t n_slots;
  // route, whole batch per call: offsets[n_req] must equal n_rows, else the
  // last request is reported as inconsistent (rows past it have no request)
  int32_t whole;
  uint32_t* ctx_flags;
};

// ---- small helpers --------------------------------------------------------------

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// bulk prefetch of [p, p + bytes) into L2 (16-byte aligned, a multiple of 16 bytes)
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

__device__ __forceinline__ uint32_t hmax2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// order-preserving map float -> uint32 (larger float -> larger integer)
__device__ __forceinline__ uint32_t ord(float f) {
  uint32_t u = __float_as_uint(f);
  return u ^ ((uint32_t)((int32_t)u >> 31) | 0x80000000u);
}
__device__ __forceinline__ float unord(uint32_t o) {
  uint32_t u = (o & 0x80000000u) ? (o ^ 0x80000000u) : ~o;
  return __uint_as_float(u);
}
// key: value first, then the lower index first; never 0 for a real entry
__device__ __forceinline__ uint64_t make_key(float v, uint32_t index) {
  return ((uint64_t)ord(v) << 32) | (uint64_t)(0xffffffffu - index);
}
__device__ __forceinline__ float key_val(uint64_t k) { return unord((uint32_t)(k >> 32)); }
__device__ __forceinline__ uint32_t key_idx(uint64_t k) { return 0xffffffffu - (uint32_t)k; }

__device__ __forceinline__ uint64_t shfl_xor64(uint64_t v, int m) {
  uint32_t lo = (uint32_t)v, hi = (uint32_t)(v >> 32);
  lo = __shfl_xor_sync(FULL, lo, m);
  hi = __shfl_xor_sync(FULL, hi, m);
  return ((uint64_t)hi << 32) | lo;
}
__device__ __forceinline__ uint64_t shfl64(uint64_t v, int src) {
  uint32_t lo = (uint32_t)v, hi = (uint32_t)(v >> 32);
  lo = __shfl_sync(FULL, lo, src);
  hi = __shfl_sync(FULL, hi, src);
  return ((uint64_t)hi << 32) | lo;
}

// bitonic sort of one key per lane, descending (lane 0 = largest)
template <typename K>
__device__ __forceinline__ K warp_sort_desc(K k, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
    const bool desc = (lane & size) == 0;
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      K o;
      if constexpr (sizeof(K) == 8) o = shfl_xor64(k, stride);
      else o = __shfl_xor_sync(FULL, k, stride);
      const bool keep_max = (((lane & stride) == 0) == desc);
      k = keep_max ? (k > o ? k : o) : (k < o ? k : o);
    }
  }
  return k;
}

// a, b sorted descending across lanes -> the 32 largest of a U b, descending
template <typename K>
__device__ __forceinline__ K warp_merge_desc(K a, K b, int lane) {
  K br;
  if constexpr (sizeof(K) == 8) br = shfl64(b, 31 - lane);
  else br = __shfl_sync(FULL, b, 31 - lane);
  K t = a > br ? a : br;
#pragma unroll
  for (int stride = 16; stride > 0; stride >>= 1) {
    K o;
    if constexpr (sizeof(K) == 8) o = shfl_xor64(t, stride);
    else o = __shfl_xor_sync(FULL, t, stride);
    t = ((lane & stride) == 0) ? (t > o ? t : o) : (t < o ? t : o);
  }
  return t;
}

// (m, S, U) merge of two partial log-sum-exp / entropy states (base 2)
__device__ __forceinline__ void lse_merge(float& m, float& S, float& U, float mo, float So,
                                          float Uo) {
  if (So == 0.f) return;
  if (S == 0.f) {
    m = mo;
    S = So;
    U = Uo;
    return;
  }
  const float M = fmaxf(m, mo);
  const float da = m - M, db = mo - M;
  const float fa = ex2(da), fb = ex2(db);
  const float Sn = fa * S + fb * So;
  const float Un = fa * fmaf(da, S, U) + fb * fmaf(db, So, Uo);
  m = M;
  S = Sn;
  U = Un;
}

// one element with full guards: NaN / +inf mark the row, -inf is a masked token
__device__ __forceinline__ void careful_add(float x, float& m, float& S, float& U, bool& bad) {
  if (isnan(x) || x == INFINITY) {
    bad = true;
    return;
  }
  if (x == -INFINITY) return;
  const float t = x * L2E;
  if (t > m) {
    if (S != 0.f) {
      const float dl = m - t;
      const float f = ex2(dl);
      U = f * fmaf(dl, S, U);
      S *= f;
    }
    m = t;
  }
  const float d = fmaf(x, L2E, -m);
  const float e = ex2(d);
  if (e != 0.f) {
    S += e;
    U = fmaf(e, d, U);
  }
}

// ---- dtype traits ------------------------------------------------------------------

template <typename T>
struct Traits;

template <>
struct Traits<__nv_bfloat16> {
  static constexpr int VEC = 8;                       // elements per 16-byte group
  static constexpr uint32_t NEG_WORD = 0xff80ff80u;   // two bf16 -inf
  static __device__ __forceinline__ float elem(const void* row, int64_t v) {
    const uint16_t h = reinterpret_cast<const uint16_t*>(row)[v];
    return __uint_as_float((uint32_t)h << 16);
  }
  // a full group by element loads (rows that are not 16-byte aligned)
  static __device__ __forceinline__ uint4 load_elems(const void* row, int64_t g) {
    const uint16_t* h = reinterpret_cast<const uint16_t*>(row) + g * VEC;
    uint4 r;
    r.x = (uint32_t)h[0] | ((uint32_t)h[1] << 16);
    r.y = (uint32_t)h[2] | ((uint32_t)h[3] << 16);
    r.z = (uint32_t)h[4] | ((uint32_t)h[5] << 16);
    r.w = (uint32_t)h[6] | ((uint32_t)h[7] << 16);
    return r;
  }
  static __device__ __forceinline__ uint32_t wmax(const uint4& w) {
    return hmax2(hmax2(w.x, w.y), hmax2(w.z, w.w));
  }
  static __device__ __forceinline__ float wfinal(uint32_t u) {
    return fmaxf(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
  }
  // maximum of the UNR groups of a tile (NaN ignored unless all are NaN)
  static __device__ __forceinline__ float tile_max(const uint4 (&c)[UNR]) {
    uint32_t m0 = hmax2(wmax(c[0]), wmax(c[1]));
    uint32_t m1 = hmax2(wmax(c[2]), wmax(c[3]));
    return wfinal(hmax2(m0, m1));
  }
  static __device__ __forceinline__ float gmax(const uint4& w) { return wfinal(wmax(w)); }
  // accumulate the 8 elements of one group into the packed (S, U) state
  static __device__ __forceinline__ void accum(const uint4& w, float2 nm, float2& S, float2& U) {
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 x = make_float2(__uint_as_float(ws[j] << 16), __uint_as_float(ws[j] & 0xffff0000u));
      const float2 d = __ffma2_rn(x, make_float2(L2E, L2E), nm);
      const float2 e = make_float2(ex2(d.x), ex2(d.y));
      S = __fadd2_rn(S, e);
      U = __ffma2_rn(e, d, U);
    }
  }
  static __device__ __forceinline__ float at(const uint4& w, int j) {
    const int q = j >> 1;
    const uint32_t u = q == 0 ? w.x : (q == 1 ? w.y : (q == 2 ? w.z : w.w));
    return __uint_as_float((j & 1) ? (u & 0xffff0000u) : (u << 16));
  }
};

template <>
struct Traits<float> {
  static constexpr int VEC = 4;
  static constexpr uint32_t NEG_WORD = 0xff800000u;  // fp32 -inf
  static __device__ __forceinline__ float elem(const void* row, int64_t v) {
    return reinterpret_cast<const float*>(row)[v];
  }
  static __device__ __forceinline__ uint4 load_elems(const void* row, int64_t g) {
    const uint32_t* f = reinterpret_cast<const uint32_t*>(row) + g * VEC;
    return make_uint4(f[0], f[1], f[2], f[3]);
  }
  static __device__ __forceinline__ float gmax(const uint4& w) {
    return fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
                 fmaxf(__uint_as_float(w.z), __uint_as_float(w.w)));
  }
  static __device__ __forceinline__ float tile_max(const uint4 (&c)[UNR]) {
    return fmaxf(fmaxf(gmax(c[0]), gmax(c[1])), fmaxf(gmax(c[2]), gmax(c[3])));
  }
  static __device__ __forceinline__ void accum(const uint4& w, float2 nm, float2& S, float2& U) {
    const float2 x0 = make_float2(__uint_as_float(w.x), __uint_as_float(w.y));
    const float2 x1 = make_float2(__uint_as_float(w.z), __uint_as_float(w.w));
    const float2 d0 = __ffma2_rn(x0, make_float2(L2E, L2E), nm);
    const float2 d1 = __ffma2_rn(x1, make_float2(L2E, L2E), nm);
    const float2 e0 = make_float2(ex2(d0.x), ex2(d0.y));
    const float2 e1 = make_float2(ex2(d1.x), ex2(d1.y));
    S = __fadd2_rn(S, e0);
    U = __ffma2_rn(e0, d0, U);
    S = __fadd2_rn(S, e1);
    U = __ffma2_rn(e1, d1, U);
  }
  static __device__ __forceinline__ float at(const uint4& w, int j) {
    return __uint_as_float(j == 0 ? w.x : (j == 1 ? w.y : (j == 2 ? w.z : w.w)));
  }
};

// ---- shared state of one CTA ------------------------------------------------------

struct Smem {
  float tm[MAX_SLOTS][NT];    // per-thread tile (super-group) maxima
  uint32_t wl[NWARP][32];     // per-warp sorted thread maxima, ord() encoded
  float cand_v[CCAP];         // candidate super-groups: value
  uint32_t cand_id[CCAP];     //   and (slot << 8 | thread), or TAIL_ID
  uint64_t ebuf[ECAP];        // candidate element keys
  float pm[NWARP], pS[NWARP], pU[NWARP];
  int pbad[NWARP];
  int ncand, nelem, nsel;
  float theta1, theta;
  float tail_max;             // maximum of the partial last group (cluster rank 0)
  // the CTA's merged partial state, read by cluster rank 0 through DSMEM
  float fm, fS, fU;
  int fbad;
  uint64_t flist[32];
  uint64_t top[32];           // the CTA's top-32 keys, ranked by counting
  int careful, fallback;
};

// ---- warp-level top-32 of pushed keys ---------------------------------------------

struct WarpTopK {
  uint64_t* buf;  // at least 64 entries
  int cnt;        // warp-uniform
  uint64_t list;  // this lane's entry of the sorted list (lane 0 = best)

  __device__ __forceinline__ void push(bool c, uint64_t key, int lane) {
    const unsigned bal = __ballot_sync(FULL, c);
    if (c) buf[cnt + __popc(bal & ((1u << lane) - 1u))] = key;
    cnt += __popc(bal);
  }
  // merge every full batch of 32 keys into the list
  __device__ __forceinline__ void drain(int lane) {
    while (cnt >= 32) {
      __syncwarp();
      uint64_t k = buf[cnt - 32 + lane];
      cnt -= 32;
      __syncwarp();
      k = warp_sort_desc(k, lane);
      list = warp_merge_desc(list, k, lane);
    }
  }
  // merge whatever is left (fewer than 32)
  __device__ __forceinline__ void drain_all(int lane) {
    drain(lane);
    if (cnt > 0) {
      __syncwarp();
      uint64_t k = lane < cnt ? buf[lane] : 0ull;
      cnt = 0;
      __syncwarp();
      k = warp_sort_desc(k, lane);
      list = warp_merge_desc(list, k, lane);
    }
  }
};

// Programmatic dependent launch.  A launch made with programmatic stream serialization may
// start while the previous kernel on its stream is still running: every CTA
// allows its own dependents at once, reads only its inputs before
// pdl_wait(), and waits there before its first global write and before any
// read of context state (counters, decode slots) the previous launch may
// still update.  Without the option both are no-ops.
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

}  // namespace prk
