// The verifier's scorer head on the GPU (Pro-Router, Section 3.1): the T x 4
// feature sequence x_t = (l_t, m_t, h_t, rho_t) of a request goes through a
// linear projection plus sinusoidal positional encoding, L post-norm
// transformer encoder layers (d = 64, 4 heads of 16, feed-forward 128, ReLU,
// LayerNorm eps 1e-5), a mean pool over t and a sigmoid layer.
//
// One CTA (256 threads) per request.  The request's activations live in a
// per-row scratch in device memory (L2-resident while the request runs):
// H [T][64] and QKV [T][192]; the attention output overwrites Q.  Every
// linear layer is a GEMM over chunks of 32 rows with the layer's weights
// staged in shared memory (rows padded by one float, so the column-parallel
// reads hit distinct banks) and 2 x (N / 16) register tiles per thread.
// Attention gives each lane one query and streams the keys with an online
// softmax.  All arithmetic is fp32 and every sum runs in a fixed order.
#pragma once

#include "pr_device.cuh"

namespace prk {

constexpr int HD = 64;            // model width
constexpr int HHEADS = 4;         // attention heads
constexpr int HDH = HD / HHEADS;  // width of a head
constexpr int HFF = 128;          // feed-forward width
constexpr int HIN = 4;            // input features
constexpr int HCH = 32;           // rows per GEMM chunk
constexpr int HSCR = 4 * HD;      // scratch floats per row: H (64) + QKV (192)
constexpr int HMAXL = 8;          // largest number of encoder layers accepted
constexpr float HLN_EPS = 1e-5f;

// offsets (in floats) inside one encoder layer's weights
constexpr int HL_WQKV = 0;
constexpr int HL_BQKV = HL_WQKV + 3 * HD * HD;
constexpr int HL_WO = HL_BQKV + 3 * HD;
constexpr int HL_BO = HL_WO + HD * HD;
constexpr int HL_G1 = HL_BO + HD;
constexpr int HL_BE1 = HL_G1 + HD;
constexpr int HL_W1 = HL_BE1 + HD;
constexpr int HL_B1 = HL_W1 + HFF * HD;
constexpr int HL_W2 = HL_B1 + HFF;
constexpr int HL_B2 = HL_W2 + HD * HFF;
constexpr int HL_G2 = HL_B2 + HD;
constexpr int HL_BE2 = HL_G2 + HD;
constexpr int HL_SIZE = HL_BE2 + HD;
constexpr int H_PRE = HD * HIN + HD;  // W_in, b_in

__host__ __device__ constexpr int64_t head_param_count(int n_layers) {
  return (int64_t)H_PRE + (int64_t)n_layers * HL_SIZE + HD + 1;
}

struct HeadArgs {
  const float* feat;          // [n_rows][8] row records
  const uint32_t* row_flags;  // [n_rows] or null
  int64_t n_rows;
  const int64_t* offsets;
  int32_t n_req;
  const float* w;             // head_param_count(n_layers) floats
  int32_t n_layers;
  float zthr;
  float* scratch;             // [n_rows][HSCR]
  float* score;
  uint8_t* ship;
  uint32_t* req_flags;
  uint32_t* ctx_flags;
};

constexpr int HWT = HFF * (HD + 1) + HD * (HFF + 1);  // W_1 and W_2 padded (the largest pair)
constexpr int HXA = HCH * (HD + 1);                   // a 32 x 64 chunk
constexpr int HXB = HCH * (HFF + 1);                  // a 32 x 128 chunk

// shared memory of one CTA (dynamic)
struct HeadSmem {
  float wt[HWT];        // staged weights
  float xa[HXA];        // GEMM input chunk / FFN output
  float xb[HXB];        // FFN hidden chunk / attention projection output
  float red[4][HD];     // partial sums of the mean pool
  float2 pe_g[HD / 2];  // encoding frequencies in half-turns, as float pairs
  uint32_t fl[NWARP];
};
static_assert(3 * HD * (HD + 1) <= HWT, "QKV weights must fit the staging buffer");

// out[r][c] = sum_k A[r][k] * Wt[c][k] + bias[c] for r < rows (<= 32), c < N.
// A: shared, row stride lda; Wt: shared, N x (K + 1).  Thread (rb, cb) =
// (tid / 16, tid % 16) computes rows 2 rb, 2 rb + 1 and columns cb + 16 j.
template <int N, int K, typename Store>
__device__ __forceinline__ void head_mm(const float* A, int lda, const float* Wt,
                                        const float* __restrict__ bias, int rows, Store store) {
  constexpr int CPT = N / 16;
  const int tid = threadIdx.x;
  const int rb = tid >> 4, cb = tid & 15;
  const int r0 = 2 * rb, r1 = 2 * rb + 1;
  float acc0[CPT], acc1[CPT];
#pragma unroll
  for (int j = 0; j < CPT; ++j) acc0[j] = acc1[j] = 0.f;
  const float* a0 = A + r0 * lda;
  const float* a1 = A + r1 * lda;
#pragma unroll 4
  for (int k = 0; k < K; ++k) {
    const float x0 = a0[k], x1 = a1[k];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
      const float wv = Wt[(cb + 16 * j) * (K + 1) + k];
      acc0[j] = fmaf(x0, wv, acc0[j]);
      acc1[j] = fmaf(x1, wv, acc1[j]);
    }
  }
#pragma unroll
  for (int j = 0; j < CPT; ++j) {
    const int c = cb + 16 * j;
    const float bc = __ldg(bias + c);
    if (r0 < rows) store(r0, c, acc0[j] + bc);
    if (r1 < rows) store(r1, c, acc1[j] + bc);
  }
}

// stage an N x K row-major weight matrix into shared memory, rows padded to K + 1
template <int N, int K>
__device__ __forceinline__ void head_stage(float* dst, const float* __restrict__ src) {
  for (int i = threadIdx.x; i < N * K; i += NT) {
    const int r = i / K, k = i - r * K;
    dst[r * (K + 1) + k] = __ldg(src + i);
  }
}

// rows [0, rows) of a 64-wide slice of the scratch (stride HSCR) into xa;
// the rows beyond are zero
__device__ __forceinline__ void head_load_chunk(float* xa, const float* src, int rows) {
  for (int i = threadIdx.x; i < HCH * HD; i += NT) {
    const int t = i / HD, k = i - t * HD;
    xa[t * (HD + 1) + k] = t < rows ? src[t * HSCR + k] : 0.f;
  }
}

// H[t] = LayerNorm(H[t] + D[t]) * g + be for the rows of a chunk; one warp per row
__device__ __forceinline__ void head_add_norm(float* H, const float* Dsm, int ldd, int rows,
                                              const float* __restrict__ g,
                                              const float* __restrict__ be) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int r = warp; r < rows; r += NWARP) {
    const float v0 = H[r * HSCR + lane] + Dsm[r * ldd + lane];
    const float v1 = H[r * HSCR + lane + 32] + Dsm[r * ldd + lane + 32];
    float s = v0 + v1;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(FULL, s, o);
    const float mu = s * (1.f / HD);
    const float d0 = v0 - mu, d1 = v1 - mu;
    float q = d0 * d0 + d1 * d1;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(FULL, q, o);
    const float inv = 1.f / sqrtf(q * (1.f / HD) + HLN_EPS);
    H[r * HSCR + lane] = d0 * inv * __ldg(g + lane) + __ldg(be + lane);
    H[r * HSCR + lane + 32] = d1 * inv * __ldg(g + lane + 32) + __ldg(be + lane + 32);
  }
}

// Sinusoidal encoding of position t, column j: sin(t f) for even j, cos(t f)
// for odd j, f = 10000^(-(j & ~1) / 64).  The angle is kept in half-turns,
// t g with g = f / pi held as a float pair (hi, lo): t * hi is split into its
// rounded value p and its exact error (fmaf), the even integer nearest p is
// removed exactly, and sinpi / cospi see an argument in [-1, 1] accurate to a
// few 1e-8 for every t < 2^24.
__device__ __forceinline__ float head_pe(int t, int j, float2 g) {
  const float tf = (float)t;
  const float p = tf * g.x;
  const float pe = fmaf(tf, g.x, -p);
  const float k2 = 2.f * rintf(0.5f * p);
  const float r = (p - k2) + (pe + tf * g.y);
  return (j & 1) ? cospif(r) : sinpif(r);
}

__global__ void __launch_bounds__(NT) head_requests(const HeadArgs a) {
  extern __shared__ __align__(16) unsigned char hsm_raw[];
  HeadSmem& sm = *reinterpret_cast<HeadSmem*>(hsm_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r = blockIdx.x;
  if (r >= a.n_req) return;
  const int64_t lo = a.offsets[r], hi = a.offsets[r + 1];
  // hi >= lo for every request makes the offsets non-decreasing, so the row
  // ranges (and the scratch rows) of different requests never overlap
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
  if (T == 0) {
    if (tid == 0) {
      a.score[r] = 0.f;
      a.ship[r] = 0;
      a.req_flags[r] = FLAG_EMPTY_REQ;
    }
    return;
  }
  // a flagged row escalates the request without running the head
  uint32_t fl = 0;
  if (a.row_flags)
    for (int t = tid; t < T; t += NT) fl |= a.row_flags[lo + t];
  fl = __reduce_or_sync(FULL, fl);
  if (lane == 0) sm.fl[warp] = fl;
  if (tid < HD / 2) {
    const double g = exp(-(double)(2 * tid) * (9.210340371976184 / HD)) * 0.3183098861837907;
    const float ghi = (float)g;
    sm.pe_g[tid] = make_float2(ghi, (float)(g - (double)ghi));
  }
  __syncthreads();
  fl = 0;
#pragma unroll
  for (int w2 = 0; w2 < NWARP; ++w2) fl |= sm.fl[w2];
  if (fl & (FLAG_NONFINITE | FLAG_BAD_CHOSEN)) {
    if (tid == 0) {
      a.score[r] = NAN;
      a.ship[r] = 0;
      a.req_flags[r] = fl;
    }
    return;
  }

  float* scr = a.scratch + lo * HSCR;  // row t: H at [t HSCR, +64), QKV at [+64, +256)
  const float* W = a.w;

  // ---- input projection + positional encoding
  for (int i = tid; i < T * HD; i += NT) {
    const int t = i / HD, j = i - t * HD;
    const float* f = a.feat + (lo + t) * NFEAT;
    const float x0 = f[0], x1 = f[1], x2 = f[4], x3 = f[5];  // l, m, h, rho
    float v = __ldg(W + HD * HIN + j);
    v = fmaf(__ldg(W + j * HIN + 0), x0, v);
    v = fmaf(__ldg(W + j * HIN + 1), x1, v);
    v = fmaf(__ldg(W + j * HIN + 2), x2, v);
    v = fmaf(__ldg(W + j * HIN + 3), x3, v);
    scr[t * HSCR + j] = v + head_pe(t, j, sm.pe_g[j >> 1]);
  }
  __syncthreads();

  constexpr float QSCALE = 0.25f;  // 1 / sqrt(16)
  for (int l = 0; l < a.n_layers; ++l) {
    const float* L = W + H_PRE + (int64_t)l * HL_SIZE;

    // ---- QKV = H W_qkv^T + b_qkv
    head_stage<3 * HD, HD>(sm.wt, L + HL_WQKV);
    for (int c0 = 0; c0 < T; c0 += HCH) {
      const int rows = min(HCH, T - c0);
      __syncthreads();
      head_load_chunk(sm.xa, scr + c0 * HSCR, rows);
      __syncthreads();
      float* dst = scr + c0 * HSCR + HD;
      head_mm<3 * HD, HD>(sm.xa, HD + 1, sm.wt, L + HL_BQKV, rows,
                          [&](int t, int c, float v) { dst[t * HSCR + c] = v; });
    }
    __syncthreads();

    // ---- attention: a warp takes 32 queries of one head, a lane one query;
    // keys and values are streamed with an online softmax.  The output
    // overwrites the lane's own Q (no other warp reads Q of that head and
    // block); K and V stay untouched.
    const int nqb = (T + 31) / 32;
    for (int task = warp; task < nqb * HHEADS; task += NWARP) {
      const int hq = task % HHEADS, qb = task / HHEADS;
      const int t = qb * 32 + lane;
      const bool on = t < T;
      float q[HDH], acc[HDH];
      const float* qrow = scr + (on ? t : 0) * HSCR + HD + hq * HDH;
#pragma unroll
      for (int d = 0; d < HDH; d += 4) {
        const float4 v4 = *reinterpret_cast<const float4*>(qrow + d);
        q[d] = v4.x * QSCALE;
        q[d + 1] = v4.y * QSCALE;
        q[d + 2] = v4.z * QSCALE;
        q[d + 3] = v4.w * QSCALE;
      }
#pragma unroll
      for (int d = 0; d < HDH; ++d) acc[d] = 0.f;
      float mx = -INFINITY, sum = 0.f;
      const float* kv = scr + 2 * HD + hq * HDH;
      for (int u = 0; u < T; ++u, kv += HSCR) {
        float kk[HDH], vv[HDH];
#pragma unroll
        for (int d = 0; d < HDH; d += 4) {
          const float4 k4 = *reinterpret_cast<const float4*>(kv + d);
          const float4 v4 = *reinterpret_cast<const float4*>(kv + HD + d);
          kk[d] = k4.x; kk[d + 1] = k4.y; kk[d + 2] = k4.z; kk[d + 3] = k4.w;
          vv[d] = v4.x; vv[d + 1] = v4.y; vv[d + 2] = v4.z; vv[d + 3] = v4.w;
        }
        float s = 0.f;
#pragma unroll
        for (int d = 0; d < HDH; ++d) s = fmaf(q[d], kk[d], s);
        if (s > mx) {
          const float f = __expf(mx - s);
          sum *= f;
#pragma unroll
          for (int d = 0; d < HDH; ++d) acc[d] *= f;
          mx = s;
        }
        const float p = __expf(s - mx);
        sum += p;
#pragma unroll
        for (int d = 0; d < HDH; ++d) acc[d] = fmaf(p, vv[d], acc[d]);
      }
      if (on) {
        const float inv = 1.f / sum;
        float* orow = scr + t * HSCR + HD + hq * HDH;
#pragma unroll
        for (int d = 0; d < HDH; d += 4)
          *reinterpret_cast<float4*>(orow + d) =
              make_float4(acc[d] * inv, acc[d + 1] * inv, acc[d + 2] * inv, acc[d + 3] * inv);
      }
    }
    __syncthreads();

    // ---- H = LN1(H + O), O = attention W_o^T + b_o
    head_stage<HD, HD>(sm.wt, L + HL_WO);
    for (int c0 = 0; c0 < T; c0 += HCH) {
      const int rows = min(HCH, T - c0);
      __syncthreads();
      head_load_chunk(sm.xa, scr + c0 * HSCR + HD, rows);
      __syncthreads();
      head_mm<HD, HD>(sm.xa, HD + 1, sm.wt, L + HL_BO, rows,
                      [&](int t, int c, float v) { sm.xb[t * (HD + 1) + c] = v; });
      __syncthreads();
      head_add_norm(scr + c0 * HSCR, sm.xb, HD + 1, rows, L + HL_G1, L + HL_BE1);
    }
    __syncthreads();

    // ---- H = LN2(H + W_2 ReLU(W_1 H + b_1) + b_2)
    head_stage<HFF, HD>(sm.wt, L + HL_W1);
    head_stage<HD, HFF>(sm.wt + HFF * (HD + 1), L + HL_W2);
    for (int c0 = 0; c0 < T; c0 += HCH) {
      const int rows = min(HCH, T - c0);
      __syncthreads();
      head_load_chunk(sm.xa, scr + c0 * HSCR, rows);
      __syncthreads();
      head_mm<HFF, HD>(sm.xa, HD + 1, sm.wt, L + HL_B1, rows,
                       [&](int t, int c, float v) { sm.xb[t * (HFF + 1) + c] = fmaxf(v, 0.f); });
      __syncthreads();
      head_mm<HD, HFF>(sm.xb, HFF + 1, sm.wt + HFF * (HD + 1), L + HL_B2, rows,
                       [&](int t, int c, float v) { sm.xa[t * (HD + 1) + c] = v; });
      __syncthreads();
      head_add_norm(scr + c0 * HSCR, sm.xa, HD + 1, rows, L + HL_G2, L + HL_BE2);
    }
    __syncthreads();
  }

  // ---- mean pool (fixed order), sigmoid layer, shipping rule
  {
    const int j = tid & (HD - 1), part = tid >> 6;  // 4 partial sums per column
    float s = 0.f;
    for (int t = part; t < T; t += 4) s += scr[t * HSCR + j];
    sm.red[part][j] = s;
  }
  __syncthreads();
  if (warp == 0) {
    const float* wout = W + H_PRE + (int64_t)a.n_layers * HL_SIZE;
    const float invT = 1.f / (float)T;
    float z = 0.f;
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
      const int j = lane + 32 * h2;
      const float pooled = ((sm.red[0][j] + sm.red[1][j]) + (sm.red[2][j] + sm.red[3][j])) * invT;
      z = fmaf(__ldg(wout + j), pooled, z);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(FULL, z, o);
    z += __ldg(wout + HD);
    if (lane == 0) {
      a.score[r] = 1.f / (1.f + expf(-z));
      a.ship[r] = (z >= a.zthr) ? 1 : 0;
      a.req_flags[r] = fl;
    }
  }
}

}  // namespace prk
