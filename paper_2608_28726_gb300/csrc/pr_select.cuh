// Operating-point calibration and selective-prediction metrics on the GPU
// (Pro-Router, Section 3.1: tau fixed on a validation pool; Section 4.1: the
// coverage rule with ship fraction q, AUROC and AUARC, the area under the
// accuracy of what ships against the fraction shipped).
//
// Everything follows from one ascending sort of the scores: a stable LSD radix
// sort of 32-bit order-preserving keys carrying the 0/1 label, 8 bits per pass
// (per-tile digit histograms, a per-digit scan over tiles, a scatter that
// ranks equal digits inside a warp with match.any, keeping the order of equal
// keys, and writes each digit's run contiguously).  Non-finite scores map to the largest key and sort last; the
// metrics use the n_f finite ones.  In the sorted array a tie group is a run
// of equal keys; a prefix count of labels gives every group's correct and
// incorrect counts, from which
//   AUROC  = sum over correct items of (incorrect below + 1/2 incorrect tied)
//            / (P N), summed exactly in integers (twice the numerator),
//   AUARC  = (1/n_f) sum over descending ranks k of C_k / k, C_k spreading a
//            tie group's correct answers evenly over its ranks; each term as
//            a float pair (about 44 bits), summed with compensation per
//            thread, then in fp64 in a fixed order (per tile, over tiles),
//   tau    = the k-th largest finite score, k = min(floor(q n + 1/2), n_f).
#pragma once

#include "pr_device.cuh"

namespace prk {

constexpr int SEL_NT = 256;                 // threads per CTA
constexpr int SEL_IPT = 8;                  // items per thread
constexpr int SEL_TILE = SEL_NT * SEL_IPT;  // items per tile
constexpr int SR_IPT = 16;                  // items per thread in the radix passes: longer
constexpr int SR_TILE = SEL_NT * SR_IPT;    // digit runs per tile, half the tile counts
constexpr int SEL_RADIX = 256;
constexpr int SEL_FEW_DIGITS = 16;          // a pass with at most this many digits ranks by match.any
constexpr uint32_t SEL_NONFINITE = 0xffffffffu;

struct SelResult {        // written by sel_finish, copied to the host
  float tau;
  int32_t pad;
  int64_t n_finite, k, n_ship, n_pos;
  double auroc, auarc, acc_shipped;
};

// finite score -> order-preserving key (-0 and +0 share one key)
__device__ __forceinline__ uint32_t sel_key(float s) {
  if (!isfinite(s)) return SEL_NONFINITE;
  const uint32_t u = __float_as_uint(s + 0.0f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float sel_unkey(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// keys, labels and the count of finite scores (one atomic per CTA); a thread
// takes 4 consecutive scores per step, vector loads when the pointers allow
__global__ void __launch_bounds__(SEL_NT) sel_init(const float* __restrict__ scores,
                                                   const uint8_t* __restrict__ labels, int64_t n,
                                                   uint32_t* __restrict__ key,
                                                   uint8_t* __restrict__ val,
                                                   unsigned long long* n_finite) {
  __shared__ uint32_t wsum[SEL_NT / 32];
  const int64_t base = (int64_t)blockIdx.x * SEL_TILE;
  const bool vec = ((reinterpret_cast<uintptr_t>(scores) | reinterpret_cast<uintptr_t>(labels)) &
                    15u) == 0;
  uint32_t fin = 0;
#pragma unroll
  for (int j = 0; j < SEL_IPT / 4; ++j) {
    const int64_t i = base + 4 * ((int64_t)j * SEL_NT + threadIdx.x);
    if (i + 3 < n && vec) {
      const float4 f = *reinterpret_cast<const float4*>(scores + i);
      uint32_t lab = 0;
      if (labels) lab = *reinterpret_cast<const uint32_t*>(labels + i);
      const uint4 k = make_uint4(sel_key(f.x), sel_key(f.y), sel_key(f.z), sel_key(f.w));
      *reinterpret_cast<uint4*>(key + i) = k;
      const uint32_t v = (lab & 0x000000ffu ? 1u : 0u) | (lab & 0x0000ff00u ? 0x100u : 0u) |
                         (lab & 0x00ff0000u ? 0x10000u : 0u) | (lab & 0xff000000u ? 0x1000000u : 0u);
      *reinterpret_cast<uint32_t*>(val + i) = v;
      fin += (k.x != SEL_NONFINITE) + (k.y != SEL_NONFINITE) + (k.z != SEL_NONFINITE) +
             (k.w != SEL_NONFINITE);
    } else {
      for (int e = 0; e < 4; ++e)
        if (i + e < n) {
          const uint32_t k = sel_key(scores[i + e]);
          key[i + e] = k;
          val[i + e] = labels ? (labels[i + e] != 0) : 0;
          fin += k != SEL_NONFINITE;
        }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) fin += __shfl_xor_sync(FULL, fin, o);
  if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = fin;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t t = 0;
    for (int w = 0; w < SEL_NT / 32; ++w) t += wsum[w];
    if (t) atomicAdd(n_finite, (unsigned long long)t);
  }
}

// counts[d * ntiles + tile] = items of `tile` whose digit at `shift` is d
// (per-warp sub-histograms keep the shared-memory atomics apart)
__global__ void __launch_bounds__(SEL_NT) sel_hist(const uint32_t* __restrict__ key, int64_t n,
                                                   int shift, uint32_t* __restrict__ counts,
                                                   int64_t ntiles) {
  __shared__ uint32_t h[SEL_NT / 32][SEL_RADIX];
  const int warp = threadIdx.x >> 5;
#pragma unroll
  for (int w = 0; w < SEL_NT / 32; ++w) h[w][threadIdx.x] = 0;
  __syncthreads();
  const int64_t base = (int64_t)blockIdx.x * SR_TILE;
#pragma unroll
  for (int j = 0; j < SR_IPT / 4; ++j) {
    const int64_t i = base + 4 * ((int64_t)j * SEL_NT + threadIdx.x);
    if (i + 3 < n) {
      const uint4 k = *reinterpret_cast<const uint4*>(key + i);
      atomicAdd(&h[warp][(k.x >> shift) & 0xff], 1u);
      atomicAdd(&h[warp][(k.y >> shift) & 0xff], 1u);
      atomicAdd(&h[warp][(k.z >> shift) & 0xff], 1u);
      atomicAdd(&h[warp][(k.w >> shift) & 0xff], 1u);
    } else {
      for (int e = 0; e < 4; ++e)
        if (i + e < n) atomicAdd(&h[warp][(key[i + e] >> shift) & 0xff], 1u);
    }
  }
  __syncthreads();
  uint32_t c = 0;
#pragma unroll
  for (int w = 0; w < SEL_NT / 32; ++w) c += h[w][threadIdx.x];
  counts[(int64_t)threadIdx.x * ntiles + blockIdx.x] = c;
}

// CTA d: exclusive scan of counts[d][0 .. ntiles) in place; total[d] = the sum.
// Windows of 8,192 counts are staged in shared memory with coalesced loads
// (one padding word per 32 so that a thread's 32 consecutive counts sit in 32
// banks); thread t scans counts [32 t, 32 t + 32) of the window, one block scan
// gives every thread its start, and the prefixes go back with coalesced
// stores.
constexpr int SEL_SCAN_W = SEL_NT * 32;  // counts per window

__global__ void __launch_bounds__(SEL_NT) sel_scan_digit(uint32_t* __restrict__ counts,
                                                         int64_t ntiles,
                                                         uint32_t* __restrict__ total) {
  __shared__ uint32_t buf[SEL_SCAN_W + SEL_SCAN_W / 32];
  __shared__ uint32_t ws[SEL_NT / 32];
  uint32_t* c = counts + (int64_t)blockIdx.x * ntiles;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t carry = 0;
  for (int64_t w0 = 0; w0 < ntiles; w0 += SEL_SCAN_W) {
    const int m = ntiles - w0 < SEL_SCAN_W ? (int)(ntiles - w0) : SEL_SCAN_W;
#pragma unroll 8
    for (int i = 0; i < 32; ++i) {
      const int idx = i * SEL_NT + tid;
      buf[idx + (idx >> 5)] = idx < m ? c[w0 + idx] : 0u;
    }
    __syncthreads();
    uint32_t* mine = buf + tid * 33;
    uint32_t sum = 0;
#pragma unroll
    for (int j = 0; j < 32; ++j) sum += mine[j];
    uint32_t x = sum;  // inclusive scan of the thread sums
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(FULL, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) ws[warp] = x;
    __syncthreads();
    uint32_t run = carry + x - sum, all = 0;
#pragma unroll
    for (int w = 0; w < SEL_NT / 32; ++w) {
      if (w < warp) run += ws[w];
      all += ws[w];
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const uint32_t v = mine[j];
      mine[j] = run;
      run += v;
    }
    __syncthreads();
#pragma unroll 8
    for (int i = 0; i < 32; ++i) {
      const int idx = i * SEL_NT + tid;
      if (idx < m) c[w0 + idx] = buf[idx + (idx >> 5)];
    }
    carry += all;
    __syncthreads();  // buf and ws are reused by the next window
  }
  if (tid == 0) total[blockIdx.x] = carry;
}

// Stable scatter of the tiles by the digit at `shift`.  Persistent: CTA b
// takes tiles b, b + grid, b + 2 grid, ..., and loads the next tile's keys,
// labels and offsets while it ranks and writes the current one.  Warp w owns
// items [w * 512, (w + 1) * 512) of a tile in 16 rounds of 32 consecutive
// items; the lanes holding the same digit in a round are found (with
// match.any, or with eight ballots, see sel_scatter) and ranked by lane,
// rounds in order, so the tile order of equal digits is kept.  The tile is then laid out in shared memory in digit order
// and written out in that order: each digit's run goes to consecutive
// addresses.  Indices are 32-bit (n < 2^31).
struct SelScatterSmem {
  uint32_t wcnt[SEL_NT / 32][SEL_RADIX];
  uint32_t gbase[SEL_RADIX];  // global position of the tile's first item of digit d,
                              // minus the digit's offset inside the tile
  uint32_t toff[SEL_RADIX];   // offset of digit d inside the tile
  uint32_t ws[SEL_NT / 32], ws2[SEL_NT / 32];
  uint32_t sk[SR_TILE];
  uint8_t sv[SR_TILE];
};

template <bool BALLOT>
__device__ __forceinline__ void sel_scatter_body(const uint32_t* __restrict__ key_in,
                                                      const uint8_t* __restrict__ val_in,
                                                      int64_t n64, int shift,
                                                      const uint32_t* __restrict__ counts,
                                                      int64_t ntiles64,
                                                      const uint32_t* __restrict__ total,
                                                      uint32_t* __restrict__ key_out,
                                                      uint8_t* __restrict__ val_out,
                                                      SelScatterSmem& sh) {
  auto& wcnt = sh.wcnt;
  auto& gbase = sh.gbase;
  auto& toff = sh.toff;
  auto& ws = sh.ws;
  auto& ws2 = sh.ws2;
  auto& sk = sh.sk;
  auto& sv = sh.sv;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t n = (uint32_t)n64, ntiles = (uint32_t)ntiles64;
  constexpr int PER_WARP = SR_TILE / (SEL_NT / 32);
  const unsigned lt = (1u << lane) - 1u;
  const uint32_t tv = total[tid];
  uint32_t k[SR_IPT];
  uint8_t v[SR_IPT];
  uint32_t bt = 0;  // items of digit tid in the tiles before the current one
  auto fetch = [&](uint32_t t, uint32_t (&kk)[SR_IPT], uint8_t (&vv)[SR_IPT], uint32_t& b) {
    const uint32_t base = t * (uint32_t)SR_TILE + (uint32_t)warp * PER_WARP;
#pragma unroll
    for (int r = 0; r < SR_IPT; ++r) {
      const uint32_t i = base + r * 32 + lane;
      kk[r] = i < n ? key_in[i] : 0u;
      vv[r] = i < n ? val_in[i] : 0;
    }
    b = counts[(size_t)tid * ntiles + t];
  };
  uint32_t tile = blockIdx.x;
  if (tile < ntiles) fetch(tile, k, v, bt);
  for (; tile < ntiles; tile += gridDim.x) {
    const uint32_t next = tile + gridDim.x;
    uint32_t kn[SR_IPT];
    uint8_t vn[SR_IPT];
    uint32_t btn = 0;
    if (next < ntiles) fetch(next, kn, vn, btn);  // in flight while this tile is done
#pragma unroll
    for (int w = 0; w < SEL_NT / 32; ++w) wcnt[w][tid] = 0;
    __syncthreads();
    const uint32_t tile0 = tile * (uint32_t)SR_TILE;
    const uint32_t base = tile0 + (uint32_t)warp * PER_WARP;
    const uint32_t nt = n - tile0 < (uint32_t)SR_TILE ? n - tile0 : (uint32_t)SR_TILE;
    uint32_t pos[SR_IPT];
#pragma unroll
    for (int r = 0; r < SR_IPT; ++r) {
      const bool ok = base + r * 32 + lane < n;
      const uint32_t d = (k[r] >> shift) & 0xff;
      unsigned peers;  // the lanes holding digit d (lanes without an item group apart)
      if (!BALLOT) {
        peers = __match_any_sync(FULL, ok ? d : SEL_RADIX);  // SEL_RADIX: no item
      } else {
        peers = __ballot_sync(FULL, ok);
        if (!ok) peers = ~peers;
#pragma unroll
        for (int bit = 0; bit < 8; ++bit) {
          const unsigned bal = __ballot_sync(FULL, (d >> bit) & 1u);
          peers &= ((d >> bit) & 1u) ? bal : ~bal;
        }
      }
      const uint32_t rank = __popc(peers & lt);
      const uint32_t before = ok ? wcnt[warp][d] : 0u;
      __syncwarp();
      if (ok && rank == 0) wcnt[warp][d] = before + __popc(peers);
      __syncwarp();
      pos[r] = before + rank;
    }
    __syncthreads();
    {
      // per digit (thread tid = digit): exclusive prefix over the warps, and
      // the tile's count of the digit
      uint32_t run = 0;
#pragma unroll
      for (int w = 0; w < SEL_NT / 32; ++w) {
        const uint32_t c = wcnt[w][tid];
        wcnt[w][tid] = run;
        run += c;
      }
      // exclusive scans over digits: of the tile's counts, and of the totals
      uint32_t x = run, y = tv;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t xx = __shfl_up_sync(FULL, x, o), yy = __shfl_up_sync(FULL, y, o);
        if (lane >= o) {
          x += xx;
          y += yy;
        }
      }
      if (lane == 31) {
        ws[warp] = x;
        ws2[warp] = y;
      }
      __syncthreads();
      uint32_t xb = 0, yb = 0;
      for (int w = 0; w < warp; ++w) {
        xb += ws[w];
        yb += ws2[w];
      }
      const uint32_t tile_off_d = xb + x - run;
      toff[tid] = tile_off_d;
      gbase[tid] = (yb + y - tv) + bt - tile_off_d;
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < SR_IPT; ++r) {
      const uint32_t i = base + r * 32 + lane;
      if (i < n) {
        const uint32_t d = (k[r] >> shift) & 0xff;
        const uint32_t p = toff[d] + wcnt[warp][d] + pos[r];
        sk[p] = k[r];
        sv[p] = v[r];
      }
    }
    __syncthreads();
    for (uint32_t j = tid; j < nt; j += SEL_NT) {
      const uint32_t kk = sk[j];
      const uint32_t o = gbase[(kk >> shift) & 0xff] + j;
      key_out[o] = kk;
      val_out[o] = sv[j];
    }
    __syncthreads();  // sk, sv, gbase, toff and wcnt are free for the next tile
#pragma unroll
    for (int r = 0; r < SR_IPT; ++r) {
      k[r] = kn[r];
      v[r] = vn[r];
    }
    bt = btn;
  }
}

// The warp ranking's method: match.any costs more the more distinct digits a
// warp holds, eight ballots (one per digit bit) cost the same for any mix.
// A pass whose keys hold few digits (the top byte of scores that share an
// exponent range) takes match.any, the others the ballots; the choice is one
// branch around the whole body, so each method compiles on its own.
__global__ void __launch_bounds__(SEL_NT) sel_scatter(const uint32_t* __restrict__ key_in,
                                                      const uint8_t* __restrict__ val_in,
                                                      int64_t n64, int shift,
                                                      const uint32_t* __restrict__ counts,
                                                      int64_t ntiles64,
                                                      const uint32_t* __restrict__ total,
                                                      uint32_t* __restrict__ key_out,
                                                      uint8_t* __restrict__ val_out) {
  __shared__ SelScatterSmem sh;
  if (__syncthreads_count(total[threadIdx.x] != 0u) <= SEL_FEW_DIGITS)
    sel_scatter_body<false>(key_in, val_in, n64, shift, counts, ntiles64, total, key_out, val_out,
                            sh);
  else
    sel_scatter_body<true>(key_in, val_in, n64, shift, counts, ntiles64, total, key_out, val_out,
                           sh);
}

// per tile: inclusive prefix of the labels inside the tile (first n_f items)
// and the tile's total.  Thread t owns items 8 t .. 8 t + 7 of the tile: one
// 8-byte load of labels, two 16-byte stores of prefixes.
__global__ void __launch_bounds__(SEL_NT) sel_label_prefix(const uint8_t* __restrict__ val,
                                                           const unsigned long long* n_finite,
                                                           uint32_t* __restrict__ pre,
                                                           uint32_t* __restrict__ tile_sum) {
  static_assert(SEL_IPT == 8, "one 8-byte vector of labels per thread");
  __shared__ uint32_t ws[SEL_NT / 32];
  const int64_t nf = (int64_t)*n_finite;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t base = (int64_t)blockIdx.x * SEL_TILE + (int64_t)tid * SEL_IPT;  // blocked
  uint32_t lab[2] = {0u, 0u};
  if (base + SEL_IPT <= nf) {
    const uint2 q = *reinterpret_cast<const uint2*>(val + base);
    lab[0] = q.x;
    lab[1] = q.y;
  } else {
    for (int j = 0; j < SEL_IPT; ++j)
      if (base + j < nf) lab[j >> 2] |= (uint32_t)val[base + j] << (8 * (j & 3));
  }
  uint32_t c[SEL_IPT], run = 0;
#pragma unroll
  for (int j = 0; j < SEL_IPT; ++j) {
    run += (lab[j >> 2] >> (8 * (j & 3))) & 0xffu;
    c[j] = run;
  }
  uint32_t x = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(FULL, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) ws[warp] = x;
  __syncthreads();
  uint32_t wbase = 0, all = 0;
#pragma unroll
  for (int w = 0; w < SEL_NT / 32; ++w) {
    if (w < warp) wbase += ws[w];
    all += ws[w];
  }
  const uint32_t off = wbase + x - run;
  if (base + SEL_IPT <= nf) {
#pragma unroll
    for (int q = 0; q < 2; ++q)
      *reinterpret_cast<uint4*>(pre + base + 4 * q) =
          make_uint4(off + c[4 * q], off + c[4 * q + 1], off + c[4 * q + 2], off + c[4 * q + 3]);
  } else {
    for (int j = 0; j < SEL_IPT; ++j)
      if (base + j < nf) pre[base + j] = off + c[j];
  }
  if (tid == 0) tile_sum[blockIdx.x] = all;
}

// exclusive scan of the tile sums (one CTA; the total goes to tile_off[ntiles])
__global__ void __launch_bounds__(1024) sel_scan_tiles(uint32_t* __restrict__ tile_sum,
                                                       int64_t ntiles,
                                                       uint32_t* __restrict__ tile_off) {
  __shared__ uint32_t ws[32];
  __shared__ uint32_t carry;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int64_t t0 = 0; t0 < ntiles; t0 += 1024) {
    const int64_t t = t0 + threadIdx.x;
    const uint32_t v = t < ntiles ? tile_sum[t] : 0u;
    uint32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(FULL, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) ws[warp] = x;
    __syncthreads();
    uint32_t wbase = 0, all = 0;
    for (int w = 0; w < 32; ++w) {
      if (w < warp) wbase += ws[w];
      all += ws[w];
    }
    const uint32_t c0 = carry;
    if (t < ntiles) tile_off[t] = c0 + wbase + x - v;
    __syncthreads();
    if (threadIdx.x == 0) carry = c0 + all;
    __syncthreads();
  }
  if (threadIdx.x == 0) tile_off[ntiles] = carry;
}

// Indices and counts below are 32-bit (n < 2^31): 64-bit integer arithmetic
// and 64-bit integer <-> float conversions run on the fp64 pipe, which is
// narrow on this GPU.
struct SelView {
  const uint32_t* key;  // sorted keys
  const uint32_t* pre;  // in-tile inclusive label prefix
  const uint32_t* tile_off;
  uint32_t nf;
};

// correct answers among the first x sorted items
__device__ __forceinline__ uint32_t sel_P(const SelView& s, uint32_t x) {
  if (x == 0) return 0;
  const uint32_t i = x - 1;
  return s.tile_off[i / SEL_TILE] + s.pre[i];
}

// [a, b): the run of keys equal to key[i]: up to 8 neighbours each way,
// then a binary search for long runs
__device__ __forceinline__ void sel_group(const SelView& s, uint32_t i, uint32_t& a, uint32_t& b) {
  const uint32_t k = s.key[i];
  a = i;
  int steps = 0;
  while (a > 0 && s.key[a - 1] == k && steps < 8) {
    --a;
    ++steps;
  }
  if (a > 0 && s.key[a - 1] == k) {  // first index in [0, a) with key == k
    uint32_t lo = 0, hi = a - 1;
    while (lo < hi) {
      const uint32_t mid = lo + ((hi - lo) >> 1);
      if (s.key[mid] < k) lo = mid + 1; else hi = mid;
    }
    a = lo;
  }
  b = i + 1;
  steps = 0;
  while (b < s.nf && s.key[b] == k && steps < 8) {
    ++b;
    ++steps;
  }
  if (b < s.nf && s.key[b] == k) {  // first index in (b, nf) with key > k
    uint32_t lo = b + 1, hi = s.nf;
    while (lo < hi) {
      const uint32_t mid = lo + ((hi - lo) >> 1);
      if (s.key[mid] <= k) lo = mid + 1; else hi = mid;
    }
    b = lo;
  }
}

// C / k for integers 0 <= C < 2^31, 1 <= k < 2^31 as an unevaluated sum hi + lo of two
// floats (about 44 correct bits) without fp64: C and k are split by bit masks
// into parts that floats hold exactly, a correctly rounded fp32 reciprocal
// gives the first quotient q, fmaf gives the remainder C - q k with single
// roundings, and the remainder times the reciprocal is the correction.
__device__ __forceinline__ float2 sel_ratio(uint32_t C, uint32_t k) {
  const float kh = (float)(k & ~0xffu), kl = (float)(k & 0xffu);
  const float ch = (float)(C & ~0xffu), cl = (float)(C & 0xffu);
  const float r = __frcp_rn((float)k);
  const float q = (ch + cl) * r;
  const float rem = fmaf(-q, kh, ch) + fmaf(-q, kl, cl);
  return make_float2(q, rem * r);
}

// Per tile: twice the AUROC numerator (integers) and the AUARC sum of its
// finite items: per thread a compensated float-float sum in item order (no
// fp64 in the loop), then fp64 over a fixed-order block tree.
__global__ void __launch_bounds__(SEL_NT) sel_metrics(const uint32_t* __restrict__ key,
                                                      const uint8_t* __restrict__ val,
                                                      const uint32_t* __restrict__ pre,
                                                      const uint32_t* __restrict__ tile_off,
                                                      const unsigned long long* n_finite,
                                                      int64_t ntiles,
                                                      unsigned long long* __restrict__ part_roc,
                                                      double* __restrict__ part_arc) {
  __shared__ double sd[SEL_NT];
  __shared__ unsigned long long su[SEL_NT];
  SelView s{key, pre, tile_off, (uint32_t)*n_finite};
  const uint32_t Ptot = tile_off[ntiles];
  const int tid = threadIdx.x;
  float fs = 0.f, fc = 0.f;  // compensated float-float sum of the thread's terms
  unsigned long long roc2 = 0;
  const uint32_t base = blockIdx.x * (uint32_t)SEL_TILE + (uint32_t)tid;
#pragma unroll 2
  for (int j = 0; j < SEL_IPT; ++j) {
    const uint32_t i = base + (uint32_t)j * SEL_NT;
    if (i < s.nf) {
      uint32_t a, b;
      sel_group(s, i, a, b);
      const uint32_t Pa = sel_P(s, a), Pb = sel_P(s, b);
      const uint32_t pos_g = Pb - Pa, n_g = b - a;
      if (val[i]) roc2 += 2ull * (a - Pa) + (n_g - pos_g);
      const uint32_t k = s.nf - i;      // descending rank, 1-based
      const uint32_t above = s.nf - b;  // items ranked before the group
      // C_k / k = (correct answers above the group) / k + (m / n_g)(pos_g / k)
      // with m = k - above members of the group shipped: float-float ratios
      // and one float-float product, the roundings carried into fc (a plain
      // fp32 term would round the same way for every k of a long tie group)
      float th, tl;
      if (n_g == 1) {
        const float2 t = sel_ratio(Ptot - Pb + pos_g, k);
        th = t.x;
        tl = t.y;
      } else {
        const float2 t1 = sel_ratio(Ptot - Pb, k);
        const float2 u1 = sel_ratio(k - above, n_g), u2 = sel_ratio(pos_g, k);
        const float p = u1.x * u2.x;
        const float pl = fmaf(u1.x, u2.x, -p) + fmaf(u1.x, u2.y, u1.y * u2.x);
        th = t1.x + p;  // two-sum of the high parts
        const float bv = th - t1.x;
        tl = ((t1.x - (th - bv)) + (p - bv)) + (t1.y + pl);
      }
      const float u = fs + th;  // two-sum into the running pair (fs, fc)
      const float bv = u - fs;
      fc += ((fs - (u - bv)) + (th - bv)) + tl;
      fs = u;
    }
  }
  sd[tid] = (double)fs + (double)fc;
  su[tid] = roc2;
  __syncthreads();
  for (int h = SEL_NT / 2; h > 0; h >>= 1) {
    if (tid < h) {
      sd[tid] += sd[tid + h];
      su[tid] += su[tid + h];
    }
    __syncthreads();
  }
  if (tid == 0) {
    part_arc[blockIdx.x] = sd[0];
    part_roc[blockIdx.x] = su[0];
  }
}

// One CTA: sums of the tile partials in tile order, then tau and the counts.
__global__ void __launch_bounds__(SEL_NT) sel_finish(const uint32_t* __restrict__ key,
                                                     const uint32_t* __restrict__ pre,
                                                     const uint32_t* __restrict__ tile_off,
                                                     const unsigned long long* n_finite,
                                                     int64_t n, int64_t ntiles, double q,
                                                     int has_labels,
                                                     const unsigned long long* part_roc,
                                                     const double* part_arc,
                                                     SelResult* __restrict__ out) {
  __shared__ double sd[SEL_NT];
  __shared__ unsigned long long su[SEL_NT];
  const int tid = threadIdx.x;
  const int64_t nf = (int64_t)*n_finite;
  const int64_t nt_used = (nf + SEL_TILE - 1) / SEL_TILE;
  double arc = 0.0;
  unsigned long long roc2 = 0;
  if (has_labels)
    for (int64_t t = tid; t < nt_used; t += SEL_NT) {  // each thread in tile order
      arc += part_arc[t];
      roc2 += part_roc[t];
    }
  sd[tid] = arc;
  su[tid] = roc2;
  __syncthreads();
  for (int h = SEL_NT / 2; h > 0; h >>= 1) {
    if (tid < h) {
      sd[tid] += sd[tid + h];
      su[tid] += su[tid + h];
    }
    __syncthreads();
  }
  if (tid != 0) return;
  SelView s{key, pre, tile_off, (uint32_t)nf};
  SelResult r;
  r.pad = 0;
  r.n_finite = nf;
  r.n_pos = has_labels ? (int64_t)tile_off[ntiles] : 0;
  int64_t k = (int64_t)floor(q * (double)n + 0.5);
  k = k < 0 ? 0 : (k > nf ? nf : k);
  r.k = k;
  const double nan = __longlong_as_double(0x7ff8000000000000ll);
  if (k == 0) {
    r.tau = __int_as_float(0x7f800000);  // +inf: nothing ships
    r.n_ship = 0;
    r.acc_shipped = nan;
  } else {
    const uint32_t i = (uint32_t)(nf - k);
    uint32_t a, b;
    sel_group(s, i, a, b);
    r.tau = sel_unkey(key[i]);
    r.n_ship = nf - a;
    r.acc_shipped = has_labels ? (double)(r.n_pos - sel_P(s, a)) / (double)r.n_ship : nan;
  }
  const int64_t P = r.n_pos, N = nf - P;
  r.auroc = (has_labels && P > 0 && N > 0) ? (double)su[0] / (2.0 * (double)P * (double)N) : nan;
  r.auarc = (has_labels && nf > 0) ? sd[0] / (double)nf : nan;
  *out = r;
}

}  // namespace prk
