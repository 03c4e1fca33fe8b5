// The verifier's scorer head on the GPU (Pro-Router, Section 3.1): the T x 4
// feature sequence x_t = (l_t, m_t, h_t, rho_t) of a request goes through a
// linear projection plus sinusoidal positional encoding, L post-norm
// transformer encoder layers (d = 64, 4 heads of 16, feed-forward 128, ReLU,
// LayerNorm eps 1e-5), a mean pool over t and a sigmoid layer.
//
// The batch runs layer by layer, so that every step spreads over all SMs
// whatever the mix of request lengths:
//   head_embed   one CTA per request: H = W_in x_t + b_in + PE(t)
//   head_rows    persistent CTAs over 64-row tiles of the whole batch: all the
//                row-local work between two attentions, fused per tile --
//                O = A W_o^T + b_o, H = LN1(H + O), F = W_2 ReLU(W_1 H + b_1) + b_2,
//                H = LN2(H + F), then the next layer's QKV = H W_qkv^T + b_qkv
//   head_attn    one CTA per (request, head): softmax(Q K^T / 4) V with the
//                keys and values staged in shared memory, online softmax
//   head_pool    one CTA per request: fixed-order mean over t, sigmoid layer
// Activations live in a scratch of 256 floats per row (H | Q | K | V; the
// attention output overwrites Q), which stays in L2 for batches of tens of
// MB.  All arithmetic is fp32 on the CUDA cores (fp32 FMA, no tensor-core
// rounding) and every sum runs in a fixed order, so results are reproducible
// bit for bit.
#pragma once

#include "pr_device.cuh"

namespace prk {

constexpr int HD = 64;            // model width
constexpr int HHEADS = 4;         // attention heads
constexpr int HDH = HD / HHEADS;  // width of a head
constexpr int HFF = 128;          // feed-forward width
constexpr int HIN = 4;            // input features
constexpr int HSCR = 4 * HD;      // scratch floats per row: H | Q | K | V
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
  // head_rows: the layer whose attention output is consumed (null for the
  // QKV-only launch) and the layer whose QKV is produced (null for the last)
  const float* lcur;
  const float* lnext;
};

// ---- shared-memory layout of head_rows (floats) ---------------------------------------
constexpr int HTR = 64;                 // rows per tile
constexpr int LDA64 = HD + 4;           // padded row of a 64-wide operand
constexpr int LDA128 = HFF + 4;         // padded row of a 128-wide operand
constexpr int HS_WQKV = 0;                             // W_qkv [192][68]
constexpr int HS_VEC = HS_WQKV + 3 * HD * LDA64;       // b_qkv | b_o g1 be1 | b_1 | b_2 g2 be2
constexpr int HS_VEC_N = 3 * HD + 3 * HD + HFF + 3 * HD;
constexpr int HS_X0 = HS_VEC + HS_VEC_N;               // activation tile [64][68]
constexpr int HS_X1 = HS_X0 + HTR * LDA64;             // activation tile [64][68]
constexpr int HS_QKV_END = HS_X1 + HTR * LDA64;        // end of the QKV-only layout
constexpr int HS_WO = HS_QKV_END;                      // W_o [64][68]
constexpr int HS_W1 = HS_WO + HD * LDA64;              // W_1 [128][68]
constexpr int HS_W2 = HS_W1 + HFF * LDA64;             // W_2 [64][132]
constexpr int HS_HID = HS_W2 + HD * LDA128;            // hidden tile [64][132]
constexpr int HS_END = HS_HID + HTR * LDA128;
constexpr size_t HEAD_ROWS_SMEM_QKV = (size_t)HS_QKV_END * sizeof(float);
constexpr size_t HEAD_ROWS_SMEM_FULL = (size_t)HS_END * sizeof(float);
static_assert(HEAD_ROWS_SMEM_FULL <= 227 * 1024, "head_rows shared memory");
// vector offsets inside HS_VEC
constexpr int HV_BQKV = 0, HV_BO = 192, HV_G1 = 256, HV_BE1 = 320, HV_B1 = 384, HV_B2 = 512,
              HV_G2 = 576, HV_BE2 = 640;

constexpr int HR_QKV = 0, HR_MID = 1, HR_LAST = 2;

// ---- small helpers ------------------------------------------------------------------------

__device__ __forceinline__ void cp_async16(float* dst_smem, const float* src, bool valid) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst_smem);
  const int n = valid ? 16 : 0;  // 0: the 16 bytes are zero-filled, nothing is read
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(n)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// copy an N x K row-major matrix into shared rows of LD floats (16-byte pieces)
template <int N, int K, int LD>
__device__ __forceinline__ void stage_matrix(float* dst, const float* __restrict__ src) {
  constexpr int Q = K / 4;
  for (int c = threadIdx.x; c < N * Q; c += NT) {
    const int n = c / Q, q = c - n * Q;
    cp_async16(dst + n * LD + 4 * q, src + n * K + 4 * q, true);
  }
}

// rows [row0, row0 + 64) of scratch columns [col, col + 64) into a [64][68]
// tile; rows at or past n_rows are zero
__device__ __forceinline__ void load_tile(float* dst, const float* scr, int64_t row0,
                                          int64_t n_rows, int col) {
  for (int c = threadIdx.x; c < HTR * (HD / 4); c += NT) {
    const int r = c >> 4, q = c & 15;
    const bool ok = row0 + r < n_rows;
    const float* src = scr + (ok ? (row0 + r) : 0) * HSCR + col + 4 * q;
    cp_async16(dst + r * LDA64 + 4 * q, src, ok);
  }
}

// acc[i][j] = sum_k A[4 ty + i][k] * W[tx + 16 j][k] over k < K: thread
// (tx, ty) = (tid % 16, tid / 16) owns rows 4 ty .. 4 ty + 3 and columns
// tx + 16 j.  Operands are read as float4 along k; with rows padded by four
// floats both reads are free of bank conflicts.  Each output keeps two
// partial sums (even and odd k, in k order) in one packed fp32x2 FMA chain
// and adds them at the end.
template <int CPT, int K, int LDA, int LDW>
__device__ __forceinline__ void tile_mm(const float* A, const float* W, float (&acc)[4][CPT],
                                        int tx, int ty) {
  float2 acc2[4][CPT];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < CPT; ++j) acc2[i][j] = make_float2(0.f, 0.f);
  const float* a0 = A + 4 * ty * LDA;
  const float* w0 = W + tx * LDW;
#pragma unroll 2
  for (int k = 0; k < K; k += 4) {
    float4 a[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) a[i] = *reinterpret_cast<const float4*>(a0 + i * LDA + k);
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
      const float4 b = *reinterpret_cast<const float4*>(w0 + 16 * j * LDW + k);
      const float2 b01 = make_float2(b.x, b.y), b23 = make_float2(b.z, b.w);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        acc2[i][j] = __ffma2_rn(make_float2(a[i].x, a[i].y), b01, acc2[i][j]);
        acc2[i][j] = __ffma2_rn(make_float2(a[i].z, a[i].w), b23, acc2[i][j]);
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < CPT; ++j) acc[i][j] = acc2[i][j].x + acc2[i][j].y;
}

// LayerNorm of the thread's four rows held as v[i][j] (columns tx + 16 j); a
// row's 64 values sit in the 16 lanes of one half-warp
__device__ __forceinline__ void rows_layer_norm(float (&v)[4][4], const float* g,
                                                const float* be, int tx) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float s = (v[i][0] + v[i][1]) + (v[i][2] + v[i][3]);
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) s += __shfl_xor_sync(FULL, s, o);
    const float mu = s * (1.f / HD);
    float q = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      v[i][j] -= mu;
      q = fmaf(v[i][j], v[i][j], q);
    }
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) q += __shfl_xor_sync(FULL, q, o);
    const float inv = 1.f / sqrtf(q * (1.f / HD) + HLN_EPS);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c = tx + 16 * j;
      v[i][j] = fmaf(v[i][j] * inv, g[c], be[c]);
    }
  }
}

// Sinusoidal encoding of position t for the column pair (2i, 2i + 1):
// sin(t f) and cos(t f), f = 10000^(-2i / 64).  The angle is kept in
// half-turns, t g with g = f / pi held as a float pair (hi, lo): t * hi is
// split into its rounded value p and its exact error (fmaf), the even integer
// nearest p is removed exactly, and sincospi sees an argument in [-1, 1]
// accurate to a few 1e-8 for every t < 2^24.
__device__ __forceinline__ void head_pe_pair(int t, float2 g, float& sn, float& cs) {
  const float tf = (float)t;
  const float p = tf * g.x;
  const float pe = fmaf(tf, g.x, -p);
  const float k2 = 2.f * rintf(0.5f * p);
  const float r = (p - k2) + (pe + tf * g.y);
  sincospif(r, &sn, &cs);
}

// rows [lo, hi) of request r, or false for an empty or inconsistent request
__device__ __forceinline__ bool head_request(const HeadArgs& a, int64_t r, int64_t& lo,
                                             int64_t& hi) {
  lo = a.offsets[r];
  hi = a.offsets[r + 1];
  return lo >= 0 && hi > lo && hi <= a.n_rows;
}

// ---- kernels ---------------------------------------------------------------------------

// CTA (request, y) embeds rows t = y, y + 4, y + 8, ... of its request in
// chunks: the chunk's four input slots are staged in shared memory with one
// round of loads, then lane i of a warp writes columns 2i, 2i + 1 of a row
// (one sincospi per pair).
constexpr int HES = 4;          // CTAs per request
constexpr int HEMB_CHUNK = 256;

__global__ void __launch_bounds__(NT) head_embed(const HeadArgs a) {
  __shared__ float2 pe_g[HD / 2];
  __shared__ __align__(16) float4 xs[HEMB_CHUNK];
  pdl_trigger();
  pdl_wait();
  int64_t lo, hi;
  if (!head_request(a, blockIdx.x, lo, hi)) return;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid < HD / 2) {
    const double g = exp(-(double)(2 * tid) * (9.210340371976184 / HD)) * 0.3183098861837907;
    const float ghi = (float)g;
    pe_g[tid] = make_float2(ghi, (float)(g - (double)ghi));
  }
  const int T = (int)(hi - lo);
  const int y = blockIdx.y;
  const int nmine = T > y ? (T - y + HES - 1) / HES : 0;  // rows y + HES k < T
  const float* W = a.w;
  const int j0 = 2 * lane;
  const float4 wa = *reinterpret_cast<const float4*>(W + j0 * HIN);        // row 2i of W_in
  const float4 wb = *reinterpret_cast<const float4*>(W + (j0 + 1) * HIN);  // row 2i + 1
  const float2 bj = *reinterpret_cast<const float2*>(W + HD * HIN + j0);
  float* scr = a.scratch + lo * HSCR;
  for (int c0 = 0; c0 < nmine; c0 += HEMB_CHUNK) {
    const int n = min(HEMB_CHUNK, nmine - c0);
    __syncthreads();
    if (tid < n) {
      const int t = y + HES * (c0 + tid);
      const float4* f = reinterpret_cast<const float4*>(a.feat + (lo + t) * NFEAT);
      const float4 u = f[0], v = f[1];
      xs[tid] = make_float4(u.x, u.y, v.x, v.y);  // l, m, h, rho
    }
    __syncthreads();
    const float2 g = pe_g[lane];
    for (int r = warp; r < n; r += NWARP) {
      const float4 x = xs[r];
      const int t = y + HES * (c0 + r);
      float v0 = bj.x, v1 = bj.y;
      v0 = fmaf(wa.x, x.x, v0);
      v0 = fmaf(wa.y, x.y, v0);
      v0 = fmaf(wa.z, x.z, v0);
      v0 = fmaf(wa.w, x.w, v0);
      v1 = fmaf(wb.x, x.x, v1);
      v1 = fmaf(wb.y, x.y, v1);
      v1 = fmaf(wb.z, x.z, v1);
      v1 = fmaf(wb.w, x.w, v1);
      float sn, cs;
      head_pe_pair(t, g, sn, cs);
      *reinterpret_cast<float2*>(scr + (int64_t)t * HSCR + j0) = make_float2(v0 + sn, v1 + cs);
    }
  }
}

template <int MODE>
__global__ void __launch_bounds__(NT, MODE == HR_QKV ? 2 : 1) head_rows(const HeadArgs a) {
  extern __shared__ __align__(16) float hs[];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int64_t ntiles = (a.n_rows + HTR - 1) / HTR;
  float* sV = hs + HS_VEC;
  float* xin = hs + HS_X0;   // the tile's input (H for QKV-only, the attention output otherwise)
  float* xmid = hs + HS_X1;  // LN1 output; then the next tile's input
  const int in_col = (MODE == HR_QKV) ? 0 : HD;

  // The weights do not depend on the previous kernel: their copies start
  // before the dependency wait (with programmatic dependent launch they
  // overlap the previous kernel's tail); the first tile is loaded after it.
  pdl_trigger();
  if (MODE != HR_QKV) {
    stage_matrix<HD, HD, LDA64>(hs + HS_WO, a.lcur + HL_WO);
    stage_matrix<HFF, HD, LDA64>(hs + HS_W1, a.lcur + HL_W1);
    stage_matrix<HD, HFF, LDA128>(hs + HS_W2, a.lcur + HL_W2);
  }
  if (MODE != HR_LAST) stage_matrix<3 * HD, HD, LDA64>(hs + HS_WQKV, a.lnext + HL_WQKV);
  pdl_wait();
  load_tile(xin, a.scratch, (int64_t)blockIdx.x * HTR, a.n_rows, in_col);
  cp_async_commit();
  for (int i = tid; i < HS_VEC_N; i += NT) {
    float v = 0.f;
    if (i < 192) {
      if (MODE != HR_LAST) v = __ldg(a.lnext + HL_BQKV + i);
    } else if (MODE != HR_QKV) {
      const float* L = a.lcur;
      if (i < 256) v = __ldg(L + HL_BO + (i - 192));
      else if (i < 320) v = __ldg(L + HL_G1 + (i - 256));
      else if (i < 384) v = __ldg(L + HL_BE1 + (i - 320));
      else if (i < 512) v = __ldg(L + HL_B1 + (i - 384));
      else if (i < 576) v = __ldg(L + HL_B2 + (i - 512));
      else if (i < 640) v = __ldg(L + HL_G2 + (i - 576));
      else v = __ldg(L + HL_BE2 + (i - 640));
    }
    sV[i] = v;
  }

  for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
    const int64_t row0 = tile * HTR;
    const int64_t next = tile + gridDim.x;
    float h[4][4];
    if (MODE != HR_QKV) {
      // residual H of the thread's rows (issued early, used after GEMM_o)
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int64_t row = row0 + 4 * ty + i;
        const bool ok = row < a.n_rows;
        const float* src = a.scratch + (ok ? row : 0) * HSCR;
#pragma unroll
        for (int j = 0; j < 4; ++j) h[i][j] = ok ? src[tx + 16 * j] : 0.f;
      }
      cp_async_wait<0>();
      __syncthreads();

      // O = A W_o^T + b_o ; H = LN1(H + O)
      float acc[4][4];
      tile_mm<4, HD, LDA64, LDA64>(xin, hs + HS_WO, acc, tx, ty);
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) h[i][j] += acc[i][j] + sV[HV_BO + tx + 16 * j];
      rows_layer_norm(h, sV + HV_G1, sV + HV_BE1, tx);
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) xmid[(4 * ty + i) * LDA64 + tx + 16 * j] = h[i][j];
      __syncthreads();

      // hidden = ReLU(H W_1^T + b_1)
      {
        float acc1[4][8];
        tile_mm<8, HD, LDA64, LDA64>(xmid, hs + HS_W1, acc1, tx, ty);
        float* hid = hs + HS_HID;
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 8; ++j)
            hid[(4 * ty + i) * LDA128 + tx + 16 * j] =
                fmaxf(acc1[i][j] + sV[HV_B1 + tx + 16 * j], 0.f);
      }
      __syncthreads();
      // xmid is free: prefetch the next tile's input into it
      if (next < ntiles) load_tile(xmid, a.scratch, next * HTR, a.n_rows, in_col);
      cp_async_commit();

      // H = LN2(H + hidden W_2^T + b_2)
      float acc2[4][4];
      tile_mm<4, HFF, LDA128, LDA128>(hs + HS_HID, hs + HS_W2, acc2, tx, ty);
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) h[i][j] += acc2[i][j] + sV[HV_B2 + tx + 16 * j];
      rows_layer_norm(h, sV + HV_G2, sV + HV_BE2, tx);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int64_t row = row0 + 4 * ty + i;
        if (row < a.n_rows) {
          float* dst = a.scratch + row * HSCR;
#pragma unroll
          for (int j = 0; j < 4; ++j) dst[tx + 16 * j] = h[i][j];
        }
      }
      if (MODE == HR_MID) {
        // xin (consumed by GEMM_o two barriers ago) takes H for the QKV GEMM
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) xin[(4 * ty + i) * LDA64 + tx + 16 * j] = h[i][j];
        __syncthreads();
      }
    } else {
      cp_async_wait<0>();
      __syncthreads();
      // xmid is free (nothing in this mode writes it): prefetch the next tile
      if (next < ntiles) load_tile(xmid, a.scratch, next * HTR, a.n_rows, in_col);
      cp_async_commit();
    }

    if (MODE != HR_LAST) {
      // QKV = H W_qkv^T + b_qkv, written to scratch columns [64, 256), in two
      // halves of 96 columns
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        float acc3[4][6];
        tile_mm<6, HD, LDA64, LDA64>(xin, hs + HS_WQKV + half * 96 * LDA64, acc3, tx, ty);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int64_t row = row0 + 4 * ty + i;
          if (row < a.n_rows) {
            float* dst = a.scratch + row * HSCR + HD + half * 96;
#pragma unroll
            for (int j = 0; j < 6; ++j)
              dst[tx + 16 * j] = acc3[i][j] + sV[HV_BQKV + half * 96 + tx + 16 * j];
          }
        }
      }
    }
    __syncthreads();  // every read of xin is done before it becomes the prefetch buffer
    float* t_ = xin;
    xin = xmid;
    xmid = t_;
  }
  cp_async_wait<0>();
}

constexpr int HAW = 4;          // warps per head_attn CTA
constexpr int HKT = 32 * HAW;   // keys per shared-memory tile: 32 per warp
constexpr int HQS = 16;         // CTAs per (request, head)

// CTA (request, head, z) takes the 32-query blocks z, z + 8, z + 16, ...; a
// lane owns one query.  For each block all keys and values of the head pass
// through shared memory in tiles of 128; warp w scores keys 32 w .. 32 w + 31
// of every tile, 16 at a time, keeping a running maximum, sum and output (in
// base 2: the queries carry the factor log2(e) / 4).  The four warps' partial
// states are merged in warp order at the end of the block.
__global__ void __launch_bounds__(HAW * 32) head_attn(const HeadArgs a) {
  __shared__ __align__(16) float4 ks[HKT][HDH / 4];
  __shared__ __align__(16) float4 vs[HKT][HDH / 4];
  __shared__ float part[HAW][HDH + 2][32];
  pdl_trigger();
  pdl_wait();
  int64_t lo, hi;
  if (!head_request(a, blockIdx.x, lo, hi)) return;
  const int hh = blockIdx.y, z = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int T = (int)(hi - lo);
  float* scr = a.scratch + lo * HSCR;
  const int nqb = (T + 31) >> 5;
  constexpr float QSCALE = 0.25f * L2E;  // 1 / sqrt(16), in base 2

  for (int qb = z; qb < nqb; qb += HQS) {
    const int t = qb * 32 + lane;
    const bool on = t < T;
    float2 q2[HDH / 2], acc2[HDH / 2];  // (dimension 2e, 2e + 1) pairs
    {
      const float4* qp = reinterpret_cast<const float4*>(scr + (int64_t)(on ? t : 0) * HSCR + HD +
                                                         hh * HDH);
#pragma unroll
      for (int d = 0; d < HDH / 4; ++d) {
        const float4 v = qp[d];
        q2[2 * d] = make_float2(v.x * QSCALE, v.y * QSCALE);
        q2[2 * d + 1] = make_float2(v.z * QSCALE, v.w * QSCALE);
      }
    }
#pragma unroll
    for (int e = 0; e < HDH / 2; ++e) acc2[e] = make_float2(0.f, 0.f);
    float m = -INFINITY, l = 0.f;

    for (int k0 = 0; k0 < T; k0 += HKT) {
      const int nk = min(HKT, T - k0);
      __syncthreads();
      // the whole tile is written: rows past nk are zero, so the branch-free
      // loops below read finite values there (their scores are masked)
      for (int i = tid; i < HKT * 8; i += HAW * 32) {
        const int kr = i >> 3, pc = i & 7;  // pieces 0-3: K, 4-7: V
        const bool ok = kr < nk;
        const float* src = scr + (int64_t)(k0 + (ok ? kr : 0)) * HSCR + 2 * HD + hh * HDH;
        float4* dst = pc < 4 ? &ks[kr][pc] : &vs[kr][pc - 4];
        cp_async16(reinterpret_cast<float*>(dst), src + (pc < 4 ? 4 * pc : HD + 4 * (pc - 4)),
                   ok);
      }
      cp_async_commit();
      cp_async_wait<0>();
      __syncthreads();
      const int kb = 32 * warp, ke = min(nk, kb + 32);
      for (int j0 = kb; j0 < ke; j0 += 16) {
        const int jn = min(16, ke - j0);
        const float4(*kt)[HDH / 4] = ks + j0;
        const float4(*vt)[HDH / 4] = vs + j0;
        float sc[16];
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
          float2 d2 = make_float2(0.f, 0.f);  // even / odd dimensions
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const float4 k4 = kt[jj][p];
            d2 = __ffma2_rn(q2[2 * p], make_float2(k4.x, k4.y), d2);
            d2 = __ffma2_rn(q2[2 * p + 1], make_float2(k4.z, k4.w), d2);
          }
          sc[jj] = jj < jn ? d2.x + d2.y : -INFINITY;
        }
        float mt = sc[0];
#pragma unroll
        for (int jj = 1; jj < 16; ++jj) mt = fmaxf(mt, sc[jj]);
        const float mn = fmaxf(m, mt);
        const float f = ex2(m - mn);
        l *= f;
        const float2 f2 = make_float2(f, f);
#pragma unroll
        for (int e = 0; e < HDH / 2; ++e) acc2[e] = __fmul2_rn(acc2[e], f2);
        float pr[16];
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) pr[jj] = ex2(sc[jj] - mn);  // 0 for masked keys
        float ls = 0.f;
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) ls += pr[jj];
        l += ls;
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
          const float2 p2 = make_float2(pr[jj], pr[jj]);
#pragma unroll
          for (int pp = 0; pp < 4; ++pp) {
            const float4 v4 = vt[jj][pp];
            acc2[2 * pp] = __ffma2_rn(p2, make_float2(v4.x, v4.y), acc2[2 * pp]);
            acc2[2 * pp + 1] = __ffma2_rn(p2, make_float2(v4.z, v4.w), acc2[2 * pp + 1]);
          }
        }
        m = mn;
      }
    }
    // merge the four partial states (a warp that saw no key has m = -inf, l = 0)
    part[warp][0][lane] = m;
    part[warp][1][lane] = l;
#pragma unroll
    for (int e = 0; e < HDH / 2; ++e) {
      part[warp][2 + 2 * e][lane] = acc2[e].x;
      part[warp][3 + 2 * e][lane] = acc2[e].y;
    }
    __syncthreads();
    if (warp == 0 && on) {
      float M = part[0][0][lane];
#pragma unroll
      for (int w2 = 1; w2 < HAW; ++w2) M = fmaxf(M, part[w2][0][lane]);
      float fw[HAW], L = 0.f;
#pragma unroll
      for (int w2 = 0; w2 < HAW; ++w2) {
        fw[w2] = ex2(part[w2][0][lane] - M);
        L = fmaf(part[w2][1][lane], fw[w2], L);
      }
      const float inv = 1.f / L;
      float4* op = reinterpret_cast<float4*>(scr + (int64_t)t * HSCR + HD + hh * HDH);
#pragma unroll
      for (int d4 = 0; d4 < HDH / 4; ++d4) {
        float o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float v = 0.f;
#pragma unroll
          for (int w2 = 0; w2 < HAW; ++w2) v = fmaf(part[w2][2 + 4 * d4 + e][lane], fw[w2], v);
          o[e] = v * inv;
        }
        op[d4] = make_float4(o[0], o[1], o[2], o[3]);
      }
    }
  }
}

__global__ void __launch_bounds__(NT) head_pool(const HeadArgs a) {
  __shared__ __align__(16) float4 red[16][HD / 4];
  __shared__ uint32_t wfl[NWARP];
  __shared__ float zpart[2];
  pdl_trigger();
  pdl_wait();
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
  if (T == 0) {
    if (tid == 0) {
      a.score[r] = 0.f;
      a.ship[r] = 0;
      a.req_flags[r] = FLAG_EMPTY_REQ;
    }
    return;
  }
  uint32_t fl = 0;
  if (a.row_flags)
    for (int t = tid; t < T; t += NT) fl |= a.row_flags[lo + t];
  fl = __reduce_or_sync(FULL, fl);
  if (lane == 0) wfl[warp] = fl;
  // fixed-order partial sums: thread (rg, cg) adds rows rg, rg + 16, ... of columns 4 cg .. 4 cg + 3
  const int rg = tid >> 4, cg = tid & 15;
  float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
  const float* base = a.scratch + lo * HSCR + 4 * cg;
  for (int t = rg; t < T; t += 16) {
    const float4 v = *reinterpret_cast<const float4*>(base + (int64_t)t * HSCR);
    s.x += v.x;
    s.y += v.y;
    s.z += v.z;
    s.w += v.w;
  }
  red[rg][cg] = s;
  __syncthreads();
  fl = 0;
#pragma unroll
  for (int w2 = 0; w2 < NWARP; ++w2) fl |= wfl[w2];
  if (fl & (FLAG_NONFINITE | FLAG_BAD_CHOSEN)) {
    if (tid == 0) {
      a.score[r] = NAN;
      a.ship[r] = 0;
      a.req_flags[r] = fl;
    }
    return;
  }
  const float* wout = a.w + H_PRE + (int64_t)a.n_layers * HL_SIZE;
  if (warp < 2) {
    const int j = tid;  // column 0 .. 63
    const float* col = reinterpret_cast<const float*>(&red[0][0]) + j;
    float sum = 0.f;
#pragma unroll
    for (int g = 0; g < 16; ++g) sum += col[g * HD];
    float z = __ldg(wout + j) * (sum * (1.f / (float)T));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(FULL, z, o);
    if (lane == 0) zpart[warp] = z;
  }
  __syncthreads();
  if (tid == 0) {
    const float z = (zpart[0] + zpart[1]) + __ldg(wout + HD);
    a.score[r] = 1.f / (1.f + expf(-z));
    a.ship[r] = (z >= a.zthr) ? 1 : 0;
    a.req_flags[r] = fl;
  }
}

}  // namespace prk
