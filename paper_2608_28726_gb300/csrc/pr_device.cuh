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
//     The per-element work is one packed FMA, one ex2, one packed add and one
//     packed FMA per two elements (f32x2 instructions of sm_100+).
//   * exact top-K (and top-2 with the lowest-index tie rule) without touching
//     elements individually: the row is cut into 16-byte groups (8 bf16 or 4
//     fp32 elements).  Ordering groups by (group max, lower group index first),
//     the K largest elements under (value, lower index first) all lie in the K
//     largest groups.  So the stream only tracks group maxima: a warp keeps the
//     32 best group keys in a register-resident sorted list and pushes groups
//     whose maximum reaches its current K-th key into a shared-memory buffer,
//     merged 32 at a time with warp bitonic networks.  After the stream the K
//     winning groups (K * 16 bytes) are re-read and their elements sorted.
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
constexpr int LIST = 32;           // group keys kept per warp
constexpr int BUF = 32 + 32 * UNR; // candidate buffer per warp
constexpr int MAXC = 8;            // largest cluster (CTAs per row)
constexpr int NFEAT = 8;
constexpr int NAGG = 11;
constexpr int ACC_WORDS = 20;      // decode slot: n, flags, 5 sums, 5 compensations, 5 minima, pad
constexpr float L2E = 1.4426950408889634f;
constexpr float LN2 = 0.6931471805599453f;
constexpr float M2_INIT = -1e30f;  // finite "no maximum yet" so that 2^(m - m') is 0, never NaN
constexpr unsigned FULL = 0xffffffffu;

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

// bitonic sort of one 64-bit key per lane, descending (lane 0 = largest)
__device__ __forceinline__ uint64_t warp_sort_desc(uint64_t k, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
    const bool desc = (lane & size) == 0;
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      uint64_t o = shfl_xor64(k, stride);
      const bool keep_max = (((lane & stride) == 0) == desc);
      k = keep_max ? (k > o ? k : o) : (k < o ? k : o);
    }
  }
  return k;
}

// a, b sorted descending across lanes -> the 32 largest of a U b, descending
__device__ __forceinline__ uint64_t warp_merge_desc(uint64_t a, uint64_t b, int lane) {
  uint64_t br = shfl64(b, 31 - lane);
  uint64_t t = a > br ? a : br;
#pragma unroll
  for (int stride = 16; stride > 0; stride >>= 1) {
    uint64_t o = shfl_xor64(t, stride);
    t = ((lane & stride) == 0) ? (t > o ? t : o) : (t < o ? t : o);
  }
  return t;
}

__device__ __forceinline__ uint32_t warp_sort_desc32(uint32_t k, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
    const bool desc = (lane & size) == 0;
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      uint32_t o = __shfl_xor_sync(FULL, k, stride);
      const bool keep_max = (((lane & stride) == 0) == desc);
      k = keep_max ? max(k, o) : min(k, o);
    }
  }
  return k;
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
  static constexpr int VEC = 8;  // elements per 16-byte group
  static __device__ __forceinline__ float elem(const void* row, int64_t v) {
    const uint16_t h = reinterpret_cast<const uint16_t*>(row)[v];
    return __uint_as_float((uint32_t)h << 16);
  }
  // group maximum (NaN ignored unless every element is NaN)
  static __device__ __forceinline__ float gmax(const uint4& w) {
    __nv_bfloat162 a = __hmax2(*reinterpret_cast<const __nv_bfloat162*>(&w.x),
                               *reinterpret_cast<const __nv_bfloat162*>(&w.y));
    __nv_bfloat162 b = __hmax2(*reinterpret_cast<const __nv_bfloat162*>(&w.z),
                               *reinterpret_cast<const __nv_bfloat162*>(&w.w));
    __nv_bfloat162 c = __hmax2(a, b);
    const uint32_t u = *reinterpret_cast<const uint32_t*>(&c);
    return fmaxf(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
  }
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
  static __device__ __forceinline__ float elem(const void* row, int64_t v) {
    return reinterpret_cast<const float*>(row)[v];
  }
  static __device__ __forceinline__ float gmax(const uint4& w) {
    return fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
                 fmaxf(__uint_as_float(w.z), __uint_as_float(w.w)));
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
  uint64_t buf[NWARP][BUF];   // candidate group keys per warp
  uint64_t list[NWARP][LIST]; // per-warp sorted group lists at the end of the stream
  float pm[NWARP], pS[NWARP], pU[NWARP];
  int pbad[NWARP];
  unsigned long long theta;   // CTA-wide group-key threshold (monotone)
  unsigned int thval;         // CTA-wide value threshold, ord() encoded (monotone)
  // the CTA's merged partial state, read by cluster rank 0 through DSMEM
  float fm, fS, fU;
  int fbad;
  uint64_t flist[LIST];
  // decisions broadcast by warp 0
  int careful;
};

// ---- warp-level candidate buffer ---------------------------------------------------

struct WarpTopK {
  uint64_t* buf;
  int cnt;        // warp-uniform
  uint64_t list;  // this lane's entry of the sorted list (lane 0 = best)
  uint64_t thk;   // warp-uniform key threshold
  float thv;      // warp-uniform value threshold

  __device__ __forceinline__ void push(bool c, uint64_t key, int lane) {
    const unsigned bal = __ballot_sync(FULL, c);
    if (c) buf[cnt + __popc(bal & ((1u << lane) - 1u))] = key;
    cnt += __popc(bal);
  }
  // merge every full batch of 32 candidates into the list
  __device__ __forceinline__ bool drain(int lane) {
    bool merged = false;
    while (cnt >= 32) {
      __syncwarp();
      uint64_t k = buf[cnt - 32 + lane];
      cnt -= 32;
      __syncwarp();
      k = warp_sort_desc(k, lane);
      list = warp_merge_desc(list, k, lane);
      merged = true;
    }
    return merged;
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

}  // namespace prk
