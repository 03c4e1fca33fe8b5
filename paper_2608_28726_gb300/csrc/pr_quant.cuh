// The quantile-summary + MLP aggregator on the GPU (Pro-Router, Section 4.2,
// Table 2: the verifier-architecture ablation's alternative to the
// transformer head).  Per request: for each of the four Eq. 3 features (l, m,
// h, rho) over its T rows, the quantiles at levels a/b (q_level_a / q_level_b; linear
// interpolation between order statistics), a 28-number summary, then a
// 28 -> 64 -> 64 -> 1 ReLU MLP and a sigmoid.
//
// One CTA per request.  Up to Q_SMALL rows two warps per feature sort its
// column's order-preserving 32-bit keys (padded to 256) in registers, four
// per lane (a bitonic network inside the lanes, across them by shfl.xor, and
// one stage between the two warps).  Up to Q_CAP rows the
// four columns are bitonic-sorted together: up to 1,024 rows each thread
// holds a run of keys in registers (register and warp-shuffle stages, one
// stage through shared memory), above that in shared memory; longer requests
// find each needed order statistic by radix selection (four 8-bit passes of
// shared histograms over the request's rows in global memory).  All three
// give the exact order statistics.  The MLP runs in the same CTA with
// fixed-order sums (four threads per hidden unit, quarters added in a fixed
// butterfly).
#pragma once

#include "pr_device.cuh"

namespace prk {

constexpr int Q_NT = 256;
constexpr int Q_NQ = 7;             // quantile levels
constexpr int Q_NS = 4 * Q_NQ;      // summary length
constexpr int Q_H = 64;             // hidden width
constexpr int Q_CAP = 2048;         // rows sorted in shared memory
constexpr int Q_SMALL = 256;        // rows ranked by counting (one per thread)
__constant__ int32_t q_level_a[Q_NQ] = {0, 1, 1, 1, 3, 9, 1};
__constant__ int32_t q_level_b[Q_NQ] = {1, 10, 4, 2, 4, 10, 1};

// weight offsets (floats)
constexpr int QW_W1 = 0, QW_B1 = QW_W1 + Q_H * Q_NS, QW_W2 = QW_B1 + Q_H,
              QW_B2 = QW_W2 + Q_H * Q_H, QW_W3 = QW_B2 + Q_H, QW_B3 = QW_W3 + Q_H,
              QW_SIZE = QW_B3 + 1;

// the MLP's weights in shared memory once the keys are done with (they reuse
// the key buffer): rows padded to an odd stride, so that the 64 threads of a
// layer, one output each, read 64 different banks
constexpr int QS_W1 = 0, QS_B1 = Q_H * (Q_NS + 1), QS_W2 = QS_B1 + Q_H,
              QS_B2 = QS_W2 + Q_H * (Q_H + 1), QS_W3 = QS_B2 + Q_H, QS_B3 = QS_W3 + Q_H,
              QS_SIZE = QS_B3 + 1;
constexpr int QW_PER_T = (QW_SIZE + Q_NT - 1) / Q_NT;  // weights each thread fetches
static_assert(QS_SIZE <= 4 * Q_CAP, "the weights fit in the key buffer");
static_assert(4 * Q_SMALL + QS_SIZE <= 4 * Q_CAP, "beside the keys of a short request too");
static_assert(Q_SMALL == 256 && Q_NT == 256, "two warps per column sort 256 keys");
static_assert(Q_NT == 4 * Q_H && Q_NS % 4 == 0 && Q_H % 4 == 0, "four threads per hidden unit");

// shared-memory position of flat weight g
__device__ __forceinline__ int q_wpos(int g) {
  if (g < QW_B1) return QS_W1 + (g / Q_NS) * (Q_NS + 1) + g % Q_NS;
  if (g < QW_W2) return QS_B1 + (g - QW_B1);
  if (g < QW_B2) return QS_W2 + ((g - QW_W2) / Q_H) * (Q_H + 1) + (g - QW_W2) % Q_H;
  if (g < QW_W3) return QS_B2 + (g - QW_B2);
  if (g < QW_B3) return QS_W3 + (g - QW_W3);
  return QS_B3;
}

struct QArgs {
  const float* feat;
  const uint32_t* row_flags;
  int64_t n_rows;
  const int64_t* offsets;
  int32_t n_req;
  const float* w;
  float zthr;
  float* summary;  // [n_req][28] or null
  float* score;
  uint8_t* ship;
  uint32_t* req_flags;
  uint32_t* ctx_flags;
};

__device__ __forceinline__ uint32_t q_key(float x) {
  const uint32_t u = __float_as_uint(x);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float q_unkey(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// record slot of feature f: l, m, h, rho
__device__ __forceinline__ int q_slot(int f) { return f == 0 ? 0 : f == 1 ? 1 : f == 2 ? 4 : 5; }

// Key of rank r (0-based, ascending) among the keys of feature f in rows
// [lo, lo + T), by radix selection over global memory.  Whole CTA.
__device__ uint32_t q_select(const float* __restrict__ feat, int64_t lo, int T, int f, int r,
                             uint32_t* hist, uint32_t* bcast) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t prefix = 0, mask = 0;
  uint32_t rank = (uint32_t)r;
  const int slot = q_slot(f);
  for (int shift = 24; shift >= 0; shift -= 8) {
    if (tid < 256) hist[tid] = 0;
    __syncthreads();
    for (int t = tid; t < T; t += Q_NT) {
      const uint32_t k = q_key(feat[(lo + t) * NFEAT + slot]);
      if ((k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 0xff], 1u);
    }
    __syncthreads();
    if (warp == 0) {  // the digit whose cumulative count passes `rank`
      uint32_t c[8], s = 0;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        c[e] = hist[lane * 8 + e];
        s += c[e];
      }
      uint32_t x = s;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(FULL, x, o);
        if (lane >= o) x += y;
      }
      const unsigned hit = __ballot_sync(FULL, x > rank);
      const int L = __ffs(hit) - 1;  // first lane whose inclusive count passes rank
      if (lane == L) {
        uint32_t cum = x - s;
        int d = lane * 8;
        for (int e = 0; e < 8; ++e, ++d) {
          if (rank < cum + c[e]) break;
          cum += c[e];
        }
        bcast[0] = (uint32_t)d;
        bcast[1] = rank - cum;
      }
    }
    __syncthreads();
    prefix |= bcast[0] << shift;
    mask |= 0xffu << shift;
    rank = bcast[1];
    __syncthreads();
  }
  return prefix;
}

// Ascending bitonic sort of the 256 keys of one column held by two warps:
// lane l of warp `half` holds keys c = 128 half + 4 l .. + 3 in v.  Stages of
// partner distance below 4 run inside the lane's registers, 4..64 between
// lanes (shfl.xor), 128 between the two warps through xbuf (128 keys per
// warp) and the named barrier `bar` of the pair's 64 threads.
__device__ __forceinline__ void q_sort256_pair(uint32_t (&v)[4], int half, int lane,
                                               uint32_t* xbuf, int bar) {
#pragma unroll
  for (int k = 2; k <= 256; k <<= 1) {
    if (k == 256) {  // partner distance 128: the other warp
#pragma unroll
      for (int e = 0; e < 4; ++e) xbuf[half * 128 + lane * 4 + e] = v[e];
      asm volatile("bar.sync %0, 64;" ::"r"(bar) : "memory");
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const uint32_t p = xbuf[(half ^ 1) * 128 + lane * 4 + e];
        v[e] = half == 0 ? min(v[e], p) : max(v[e], p);  // one ascending block
      }
    }
#pragma unroll
    for (int j = (k >> 1) < 64 ? (k >> 1) : 64; j >= 4; j >>= 1) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int c = half * 128 + lane * 4 + e;
        const uint32_t p = __shfl_xor_sync(FULL, v[e], j >> 2);
        const bool keep_min = ((c & j) == 0) == ((c & k) == 0);
        v[e] = keep_min ? min(v[e], p) : max(v[e], p);
      }
    }
#pragma unroll
    for (int j = (k >> 1) < 2 ? (k >> 1) : 2; j >= 1; j >>= 1) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if ((e & j) == 0) {
          const uint32_t x = v[e], y = v[e + j];
          const bool up = ((half * 128 + lane * 4 + e) & k) == 0;
          const uint32_t lo = min(x, y), hi = max(x, y);
          v[e] = up ? lo : hi;
          v[e + j] = up ? hi : lo;
        }
      }
    }
  }
}

// Ascending bitonic sort of the four columns col f = qs + (f << ln2) of n2 =
// 2^ln2 keys each, n2 = 64 E (512 or 1,024), by the whole CTA: thread t
// holds the E consecutive keys c0 .. c0 + E - 1 of one column (two warps per
// column).  A compare-exchange stage of partner distance j runs in registers
// for j < E, between the lanes of a warp (shfl.xor) for j < 32 E, and through
// shared memory only for j = n2 / 2.
template <int E>
__device__ void q_bitonic(uint32_t* qs, int ln2) {
  const int n2 = 1 << ln2, tid = threadIdx.x;
  const int per_col = n2 / E;  // threads per column
  const int c0 = (tid % per_col) * E;
  uint32_t* col = qs + ((tid / per_col) << ln2);
  uint32_t v[E];
#pragma unroll
  for (int e = 0; e < E; ++e) v[e] = col[c0 + e];
  for (int k = 2; k <= n2; k <<= 1) {
    for (int j = k >> 1; j >= E; j >>= 1) {
      if (j >= 32 * E) {  // the other warp of the column
        __syncthreads();
#pragma unroll
        for (int e = 0; e < E; ++e) col[c0 + e] = v[e];
        __syncthreads();
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int c = c0 + e;
          const uint32_t p = col[c ^ j];
          const bool keep_min = ((c & j) == 0) == ((c & k) == 0);
          v[e] = keep_min ? min(v[e], p) : max(v[e], p);
        }
      } else {
        const int lm = j / E;  // lane distance
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int c = c0 + e;
          const uint32_t p = __shfl_xor_sync(FULL, v[e], lm);
          const bool keep_min = ((c & j) == 0) == ((c & k) == 0);
          v[e] = keep_min ? min(v[e], p) : max(v[e], p);
        }
      }
    }
#pragma unroll
    for (int jj = E / 2; jj >= 1; jj >>= 1) {  // inside the thread's keys
      if (jj < k) {
#pragma unroll
        for (int e = 0; e < E; ++e) {
          if ((e & jj) == 0) {
            const uint32_t x = v[e], y = v[e + jj];
            const bool up = ((c0 + e) & k) == 0;
            const uint32_t lo = min(x, y), hi = max(x, y);
            v[e] = up ? lo : hi;
            v[e + jj] = up ? hi : lo;
          }
        }
      }
    }
  }
  __syncthreads();
#pragma unroll
  for (int e = 0; e < E; ++e) col[c0 + e] = v[e];
}

__global__ void __launch_bounds__(Q_NT, 3) qmlp_requests(const QArgs a) {
  extern __shared__ __align__(16) uint32_t qs[];  // [4][n2] keys (shared-memory path)
  __shared__ float qv[Q_NS];
  __shared__ float h1[Q_H], h2[Q_H];
  __shared__ uint32_t hist[256], bcast[2], wfl[Q_NT / 32];
  __shared__ uint32_t qx[4][Q_SMALL];  // exchange between the two warps of a column
  __shared__ float zpart[2];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r = blockIdx.x;
  const int64_t lo = a.offsets[r], hi = a.offsets[r + 1];
  if (lo < 0 || hi < lo || hi > a.n_rows) {
    if (tid == 0) {
      a.score[r] = NAN;
      a.ship[r] = 0;
      a.req_flags[r] = FLAG_BAD_OFFSETS;
      atomicOr(a.ctx_flags, FLAG_BAD_OFFSETS);
    }
    return;
  }
  const int T = (int)(hi - lo);
  // the MLP's weights, fetched now (coalesced) so that their latency overlaps
  // the key loads and the sort
  float wr[QW_PER_T];
#pragma unroll
  for (int i = 0; i < QW_PER_T; ++i) {
    const int g = tid + i * Q_NT;
    wr[i] = g < QW_SIZE ? __ldg(a.w + g) : 0.f;
  }
  if (T == 0) {
    if (tid == 0) {
      a.score[r] = 0.f;
      a.ship[r] = 0;
      a.req_flags[r] = FLAG_EMPTY_REQ;
    }
    return;
  }
  // the rows' flags: read now, decided after the order statistics (a flagged
  // request is rare, and its loads then overlap the key loads)
  uint32_t fl = 0;
  if (a.row_flags)
    for (int t = tid; t < T; t += Q_NT) fl |= a.row_flags[lo + t];
  fl = __reduce_or_sync(FULL, fl);
  if (lane == 0) wfl[warp] = fl;

  float* W = reinterpret_cast<float*>(qs);  // the MLP's weights in shared memory
  if (T <= Q_SMALL) {
    // the weights go beside the keys at once (their loads were issued at the
    // top), so that staging them is off the request's critical path
    W = reinterpret_cast<float*>(qs + 4 * Q_SMALL);
#pragma unroll
    for (int i = 0; i < QW_PER_T; ++i) {
      const int g = tid + i * Q_NT;
      if (g < QW_SIZE) W[q_wpos(g)] = wr[i];
    }
    // two warps per feature column: its keys (padded with the largest key to
    // 256) sorted in registers, then stored in order for the interpolation
    {
      const int f = warp >> 1, half = warp & 1;
      const int slot = q_slot(f);
      uint32_t v[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int t = half * 128 + lane * 4 + e;
        v[e] = t < T ? q_key(__ldg(a.feat + (lo + t) * NFEAT + slot)) : 0xffffffffu;
      }
      q_sort256_pair(v, half, lane, qx[f], 1 + f);
#pragma unroll
      for (int e = 0; e < 4; ++e) qs[f * Q_SMALL + half * 128 + lane * 4 + e] = v[e];
    }
    __syncthreads();
    if (tid < Q_NS) {
      const int f = tid / Q_NQ, lv = tid - f * Q_NQ;
      const uint32_t num = (uint32_t)q_level_a[lv] * (uint32_t)(T - 1);  // T <= 256
      const uint32_t b = (uint32_t)q_level_b[lv];
      const uint32_t lo_i = num / b, rem = num - lo_i * b;
      const uint32_t* col = qs + f * Q_SMALL;
      const float xl = q_unkey(col[lo_i]);
      float q = xl;
      if (rem) q = xl + ((float)rem / (float)b) * (q_unkey(col[lo_i + 1]) - xl);
      qv[tid] = q;
    }
  } else if (T <= Q_CAP) {
    int ln2 = 9;  // n2 = 2^ln2 >= T, at least 512
    while ((1 << ln2) < T) ++ln2;
    const int n2 = 1 << ln2;
    // each thread reads whole records (two 16-byte loads give the four
    // features), several rows in flight at once
#pragma unroll 4
    for (int t = tid; t < n2; t += Q_NT) {
      uint32_t k0 = 0xffffffffu, k1 = 0xffffffffu, k2 = 0xffffffffu, k3 = 0xffffffffu;
      if (t < T) {
        const float4* rec = reinterpret_cast<const float4*>(a.feat + (lo + t) * NFEAT);
        const float4 r0 = __ldg(rec), r1 = __ldg(rec + 1);
        k0 = q_key(r0.x);  // l
        k1 = q_key(r0.y);  // m
        k2 = q_key(r1.x);  // h
        k3 = q_key(r1.y);  // rho
      }
      qs[t] = k0;
      qs[n2 + t] = k1;
      qs[2 * n2 + t] = k2;
      qs[3 * n2 + t] = k3;
    }
    __syncthreads();
    if (ln2 == 9) {
      q_bitonic<8>(qs, 9);
    } else if (ln2 == 10) {
      q_bitonic<16>(qs, 10);
    } else {  // 2,048 keys per column: shared-memory stages (32 keys per thread
              // would take the registers that the other requests' CTAs need)
      const int half = n2 >> 1, lh = ln2 - 1;
      for (int k = 2; k <= n2; k <<= 1) {
        for (int j = k >> 1; j > 0; j >>= 1) {
          for (int idx = tid; idx < 4 * half; idx += Q_NT) {
            const int f = idx >> lh, t = idx & (half - 1);
            const int i = ((t & ~(j - 1)) << 1) | (t & (j - 1));
            const int l = i + j;
            uint32_t* col = qs + (f << ln2);
            const uint32_t x = col[i], y = col[l];
            const bool up = (i & k) == 0;
            if ((x > y) == up) {
              col[i] = y;
              col[l] = x;
            }
          }
          __syncthreads();
        }
      }
    }
    __syncthreads();
    if (tid < Q_NS) {
      const int f = tid / Q_NQ, j = tid - f * Q_NQ;
      const int64_t num = (int64_t)q_level_a[j] * (T - 1);
      const int b = q_level_b[j];
      const int lo_i = (int)(num / b), rem = (int)(num - (int64_t)lo_i * b);
      const uint32_t* col = qs + (f << ln2);
      const float xl = q_unkey(col[lo_i]);
      float q = xl;
      if (rem) {
        const float xh = q_unkey(col[min(lo_i + 1, T - 1)]);
        q = xl + ((float)rem / (float)b) * (xh - xl);
      }
      qv[tid] = q;
    }
  } else {
    for (int f = 0; f < 4; ++f)
      for (int j = 0; j < Q_NQ; ++j) {
        const int64_t num = (int64_t)q_level_a[j] * (T - 1);
        const int b = q_level_b[j];
        const int lo_i = (int)(num / b), rem = (int)(num - (int64_t)lo_i * b);
        const float xl = q_unkey(q_select(a.feat, lo, T, f, lo_i, hist, bcast));
        float q = xl;
        if (rem) {
          const float xh = q_unkey(q_select(a.feat, lo, T, f, min(lo_i + 1, T - 1), hist, bcast));
          q = xl + ((float)rem / (float)b) * (xh - xl);
        }
        if (tid == 0) qv[f * Q_NQ + j] = q;
      }
  }
  __syncthreads();

  fl = 0;
#pragma unroll
  for (int w2 = 0; w2 < Q_NT / 32; ++w2) fl |= wfl[w2];
  if (fl & (FLAG_NONFINITE | FLAG_BAD_CHOSEN)) {
    if (tid == 0) {
      a.score[r] = NAN;
      a.ship[r] = 0;
      a.req_flags[r] = fl;
    }
    return;
  }

  // MLP 28 -> 64 -> 64 -> 1, weights from shared memory (longer requests
  // stage them now, in the key buffer)
  if (T > Q_SMALL) {
#pragma unroll
    for (int i = 0; i < QW_PER_T; ++i) {
      const int g = tid + i * Q_NT;
      if (g < QW_SIZE) W[q_wpos(g)] = wr[i];
    }
  }
  __syncthreads();
  // four threads per hidden unit: each sums a quarter of the inputs in order,
  // then the quarters are added in a fixed butterfly (lanes 4o .. 4o + 3)
  {
    const int o = tid >> 2, part = tid & 3;
    constexpr int P1 = Q_NS / 4, P2 = Q_H / 4;
    float s1 = 0.f;
#pragma unroll
    for (int i = 0; i < P1; ++i)
      s1 = fmaf(W[QS_W1 + o * (Q_NS + 1) + part * P1 + i], qv[part * P1 + i], s1);
    s1 += __shfl_xor_sync(FULL, s1, 1);
    s1 += __shfl_xor_sync(FULL, s1, 2);
    if (part == 0) h1[o] = fmaxf(s1 + W[QS_B1 + o], 0.f);
    __syncthreads();
    float s2 = 0.f;
#pragma unroll
    for (int i = 0; i < P2; ++i)
      s2 = fmaf(W[QS_W2 + o * (Q_H + 1) + part * P2 + i], h1[part * P2 + i], s2);
    s2 += __shfl_xor_sync(FULL, s2, 1);
    s2 += __shfl_xor_sync(FULL, s2, 2);
    if (part == 0) h2[o] = fmaxf(s2 + W[QS_B2 + o], 0.f);
  }
  __syncthreads();
  if (warp < 2) {
    float z = W[QS_W3 + tid] * h2[tid];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(FULL, z, o);
    if (lane == 0) zpart[warp] = z;
  }
  if (a.summary && tid < Q_NS) a.summary[r * Q_NS + tid] = qv[tid];
  __syncthreads();
  if (tid == 0) {
    const float z = (zpart[0] + zpart[1]) + W[QS_B3];
    a.score[r] = 1.f / (1.f + expf(-z));
    a.ship[r] = (z >= a.zthr) ? 1 : 0;
    a.req_flags[r] = fl;
  }
}

}  // namespace prk
