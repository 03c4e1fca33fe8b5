// The verifier's scorer head on the GPU (Pro-Router, Section 3.1): the T x 4
// feature sequence x_t = (l_t, m_t, h_t, rho_t) of a request goes through a
// linear projection plus sinusoidal positional encoding, L post-norm
// transformer encoder layers (d = 64, 4 heads of 16, feed-forward 128, ReLU,
// LayerNorm eps 1e-5), a mean pool over t and a sigmoid layer.
//
// The batch runs layer by layer, so that every step spreads over all SMs
// whatever the mix of request lengths:
//   head_embed   one CTA per request: H = W_in x_t + b_in + PE(t)
//   head_rows    one CTA per 128-row tile of the whole batch: all the row-local
//                work between two attentions, fused per tile --
//                O = A W_o^T + b_o, H = LN1(H + O), F = W_2 ReLU(W_1 H + b_1) + b_2,
//                H = LN2(H + F), then the next layer's QKV = H W_qkv^T + b_qkv
//   head_attn    one CTA per (request, head, 128-query block): softmax(Q K^T / 4) V,
//                online softmax over 64-key chunks
//   head_pool    one CTA per request: fixed-order mean over t, sigmoid layer
// Activations live in a scratch of 256 floats per row (H | Q | K | V; the
// attention output overwrites Q), which stays in L2 for batches of tens of
// MB.  Every contraction runs on the tensor cores with each fp32 operand split
// into two TF32 parts (three products per product), which keeps fp32-level
// accuracy; softmax, LayerNorm and the rest run in fp32 on the CUDA cores.
// Every sum runs in a fixed order, so results are reproducible bit for bit.
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

constexpr int HR_QKV = 0, HR_MID = 1, HR_LAST = 2;

// ---- small helpers ------------------------------------------------------------------------

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

// ---- head_attn: softmax(Q K^T / 4) V on the tensor cores ----------------------------
//
// CTA (request, head, z) takes the 128-query blocks z, z + gridDim.z, ... of
// its request; thread i owns query i of the block and TMEM lane i.  The keys pass
// in chunks of 64.  Per chunk two tcgen05.mma kind::tf32 contractions run with
// fp32 accumulators in TMEM: S = Q K^T (M = 128 queries, N = the chunk's keys
// rounded up to 16, K = 16) and O_c = P V (M = 128, K = the chunk's keys
// rounded up to 8).  Every fp32 operand x is split into x_hi = tf32(x) and
// x_lo = x - x_hi, and a product is taken as a_hi b_hi + a_hi b_lo +
// a_lo b_hi: the dropped a_lo b_lo and the tensor core's truncation of x_lo
// to TF32 are below 2^-21 of the product, so the contractions keep fp32-level
// accuracy on TF32 units.  The value operand is [V_hi | V_lo] side by side
// (N = 32), so each K step of P V is two MMAs, P_hi [V_hi | V_lo] and
// P_lo [V_hi | V_lo] (the P_lo V_lo half is never read), and O_c is the sum
// of the accumulator's two halves.
//
// Between the two contractions each thread reads its row of S, keeps the
// running maximum and sum (base 2, online over the chunks), writes P_hi back
// over S in TMEM (the A operand of the first MMA of a K step) and P_lo to
// shared memory (the second), and after P V folds O_c into its running
// output; the next chunk's keys and values are loaded while the P V MMAs
// run.  A CTA holds 128 TMEM columns and 50 KB of shared memory, so four run
// on an SM and one's MMAs overlap another's softmax.  One elected thread
// issues the MMAs; every wait on their completion is bounded.
//
// TMEM columns: S / P_hi 0-63, O_c 64-95, Q_hi 96-111, Q_lo 112-127.
// Shared memory: the key operand and P_lo in the K-major canonical layout
// without swizzle (core matrices of 8 rows x 16 bytes, consecutive along K at
// 128 bytes, 8-row groups at the stride byte offset); [V_hi | V_lo]^T in the
// 128-byte swizzled K-major layout (8 rows x 128 bytes per 1,024-byte atom,
// the 16-byte piece c of row r stored at piece c ^ r), so that the 32 lanes
// writing one dimension of 32 consecutive keys hit 32 different banks.
constexpr int HA_M = 128;                       // queries per block = TMEM lanes = threads
constexpr int HA_NC = 64;                       // keys per chunk
constexpr int HA_QZ_MIN = 4;                    // CTAs per (request, head): at least,
constexpr int HA_QZ_MAX = 16;                   //   and at most
constexpr uint32_t HA_TMEM_COLS = 128;
constexpr uint32_t HA_O_COL = HA_NC;            // O_c: [V_hi | V_lo] products, 32 columns
constexpr uint32_t HA_QH_COL = HA_O_COL + 2 * HDH;
constexpr uint32_t HA_QL_COL = HA_QH_COL + HDH;
constexpr int HA_K_SBO = (HDH / 4) * 128;       // key rows of 16 values: 4 core matrices
constexpr int HA_P_SBO = (HA_NC / 4) * 128;     // P_lo rows of 64 keys: 16 core matrices
constexpr int HA_VT_ROWS = 2 * HDH;             // [V_hi | V_lo]^T rows
constexpr int HA_VT_ATOM = HA_VT_ROWS * 128;    // 32 keys of all rows: 4 swizzle atoms
// shared memory (bytes from the 1,024-aligned base)
constexpr int HA_VT = 0;
constexpr int HA_K_HI = HA_VT + (HA_NC / 32) * HA_VT_ATOM;
constexpr int HA_K_LO = HA_K_HI + HA_NC * HDH * 4;
constexpr int HA_P_LO = HA_K_LO + HA_NC * HDH * 4;
constexpr int HA_BAR = HA_P_LO + HA_M * HA_NC * 4;  // mbarrier: MMA completion
constexpr int HA_TSLOT = HA_BAR + 8;                // TMEM base from tcgen05.alloc
constexpr size_t HA_SMEM = HA_TSLOT + 8 + 1024;     // + alignment of the base
constexpr int HA_CTAS_PER_SM = 4;
static_assert(HA_CTAS_PER_SM * (HA_SMEM + 1024) <= 233472, "shared memory of four CTAs");
static_assert(HA_CTAS_PER_SM * HA_TMEM_COLS <= 512 && HA_QL_COL + HDH <= HA_TMEM_COLS,
              "TMEM columns");
static_assert(HA_VT % 1024 == 0 && HA_VT_ATOM % 1024 == 0, "swizzle atoms are 1,024-aligned");
static_assert(HA_NC == 64, "a thread reads its scores in two groups of 32 columns");
// instruction descriptors of tcgen05.mma kind::tf32: fp32 accumulator (bits
// 4-5 = 1), TF32 A and B (bits 7-9, 10-12 = 2), both K-major (bits 15, 16 =
// 0), N / 8 in bits 17-22, M / 16 in bits 24-28
constexpr uint32_t HA_IDESC_S = (1u << 4) | (2u << 7) | (2u << 10) |
                                ((uint32_t)(HA_M >> 4) << 24);  // N (<= 64) set per chunk
constexpr uint32_t HA_IDESC_O = (1u << 4) | (2u << 7) | (2u << 10) |
                                ((uint32_t)(HA_VT_ROWS >> 3) << 17) | ((uint32_t)(HA_M >> 4) << 24);
constexpr uint64_t HA_WAIT_NS = 2000000000ull;  // a wait gives up after 2 s
constexpr uint32_t HA_ERR_TIMEOUT = 32u;        // PR_FLAG_TIMEOUT in the context flag word

__device__ __forceinline__ uint32_t ha_saddr(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
// byte offset of (row, 4-value piece j) in the canonical layout without swizzle
__device__ __forceinline__ uint32_t ha_kmaj(int row, int j, int sbo) {
  return (uint32_t)((row >> 3) * sbo + j * 128 + (row & 7) * 16);
}
// matrix descriptors: start >> 4 in bits 0-13, leading byte offset >> 4 in
// bits 16-29, stride byte offset >> 4 in bits 32-45, version 1 in bits
// 46-47, layout in bits 61-63 (0: no swizzle, 2: 128-byte swizzle)
__device__ __forceinline__ uint64_t ha_desc(uint32_t saddr, uint32_t sbo) {
  return (uint64_t)((saddr >> 4) & 0x3fffu) | ((uint64_t)(128u >> 4) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3fffu) << 32) | ((uint64_t)1 << 46);
}
__device__ __forceinline__ uint64_t ha_desc_sw128(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3fffu) | ((uint64_t)1 << 16) |
         ((uint64_t)(1024u >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
// tf32(x) rounded to nearest (ties away): the 13 low mantissa bits cleared
// after adding half of their range; exact for finite x, and x - tf32(x) is
// exact in fp32
__device__ __forceinline__ float ha_hi(float x) {
  return __uint_as_float((__float_as_uint(x) + 0x1000u) & 0xffffe000u);
}
__device__ __forceinline__ void ha_split(const float4 x, float4& h, float4& l) {
  h = make_float4(ha_hi(x.x), ha_hi(x.y), ha_hi(x.z), ha_hi(x.w));
  l = make_float4(x.x - h.x, x.y - h.y, x.z - h.z, x.w - h.w);
}
__device__ __forceinline__ void ha_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void ha_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// generic-proxy shared-memory writes become visible to the tensor cores
__device__ __forceinline__ void ha_fence_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// D (+)= A B^T, A and B from shared memory
__device__ __forceinline__ void ha_mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc,
                                       uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.u32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
// D (+)= A B^T, A from TMEM (lane = row, one column per K value)
__device__ __forceinline__ void ha_mma_ta(uint32_t d, uint32_t a, uint64_t b, uint32_t idesc,
                                          uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.u32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
      "r"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void ha_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   bar)
               : "memory");
}
__device__ __forceinline__ bool ha_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t ha_clock() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// bounded wait for the phase with the given parity: false once HA_WAIT_NS
// nanoseconds have passed without it
__device__ __forceinline__ bool ha_wait(uint32_t bar, uint32_t parity) {
  if (ha_try(bar, parity)) return true;
  const uint64_t t0 = ha_clock();
  for (uint32_t i = 1;; ++i) {
    if (ha_try(bar, parity)) return true;
    if ((i & 255u) == 0u && ha_clock() - t0 > HA_WAIT_NS) return false;
  }
}
// 32 consecutive fp32 columns of this warp's 32 TMEM lanes (lane = row)
__device__ __forceinline__ void ha_ld32(uint32_t taddr, float (&v)[32]) {
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
__device__ __forceinline__ void ha_st32(uint32_t taddr, const float (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(
          taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
}

__device__ __forceinline__ void ha_st16(uint32_t taddr, const float4 (&v)[4]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0].x)), "r"(__float_as_uint(v[0].y)), "r"(__float_as_uint(v[0].z)),
      "r"(__float_as_uint(v[0].w)), "r"(__float_as_uint(v[1].x)), "r"(__float_as_uint(v[1].y)),
      "r"(__float_as_uint(v[1].z)), "r"(__float_as_uint(v[1].w)), "r"(__float_as_uint(v[2].x)),
      "r"(__float_as_uint(v[2].y)), "r"(__float_as_uint(v[2].z)), "r"(__float_as_uint(v[2].w)),
      "r"(__float_as_uint(v[3].x)), "r"(__float_as_uint(v[3].y)), "r"(__float_as_uint(v[3].z)),
      "r"(__float_as_uint(v[3].w))
      : "memory");
}

// P = 2^(s QSCALE - mn) over 32 of this thread's score columns (col0 = the
// first one's index in the chunk): P_hi back into TMEM over S, P_lo into
// shared memory, the row sum into ls
template <bool FULL>
__device__ __forceinline__ void ha_softmax32(float (&v)[32], int col0, int nk, float qscale,
                                             float mn, float& ls, uint8_t* plo_row, int row,
                                             uint32_t taddr) {
#pragma unroll
  for (int j4 = 0; j4 < 8; ++j4) {
    float pl[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = 4 * j4 + e;
      float p = ex2(fmaf(v[j], qscale, -mn));
      if (!FULL) p = col0 + j < nk ? p : 0.f;
      ls += p;
      const float ph = ha_hi(p);
      v[j] = ph;
      pl[e] = p - ph;
    }
    *reinterpret_cast<float4*>(plo_row + ha_kmaj(row, (col0 >> 2) + j4, HA_P_SBO)) =
        make_float4(pl[0], pl[1], pl[2], pl[3]);
  }
  ha_st32(taddr, v);
}

__global__ void __launch_bounds__(HA_M, HA_CTAS_PER_SM) head_attn(const HeadArgs a) {
  extern __shared__ uint8_t ha_raw[];
  const int tid = threadIdx.x, warp = tid >> 5;
  int64_t lo, hi;
  // the offsets are inputs of the call, complete before its first kernel
  const int T = head_request(a, blockIdx.x, lo, hi) ? (int)(hi - lo) : 0;
  const int nqb = (T + HA_M - 1) / HA_M;
  if ((int)blockIdx.z >= nqb) {
    pdl_trigger();
    return;
  }
  const int hh = blockIdx.y;
  float* scr = a.scratch + lo * HSCR;
  // staging: key kr = tid % 64 of a chunk, its K (part 0) or V (part 1) row
  const int kr = tid & (HA_NC - 1), part = tid >> 6;
  const float* kv_src = scr + 2 * HD + part * HD + hh * HDH;
  float4 pre[HDH / 4];
  float4 qv[HDH / 4];
  auto load_row = [&](int k0) {
    const int k = k0 + kr;
    const bool on = k < T;  // rows past the request are zero; their scores are masked
    const float4* src = reinterpret_cast<const float4*>(kv_src + (int64_t)(on ? k : 0) * HSCR);
#pragma unroll
    for (int j = 0; j < HDH / 4; ++j) pre[j] = on ? src[j] : make_float4(0.f, 0.f, 0.f, 0.f);
  };
  auto load_q = [&](int qb) {
    const int q = qb * HA_M + tid;
    const bool on = q < T;
    const float4* src =
        reinterpret_cast<const float4*>(scr + (int64_t)(on ? q : 0) * HSCR + HD + hh * HDH);
#pragma unroll
    for (int j = 0; j < HDH / 4; ++j) qv[j] = on ? src[j] : make_float4(0.f, 0.f, 0.f, 0.f);
  };
  // the first block's loads are in flight while the CTA takes its TMEM
  pdl_wait();
  load_q(blockIdx.z);
  load_row(0);
  const uint32_t raw = ha_saddr(ha_raw);
  const uint32_t sb = (raw + 1023u) & ~1023u;  // swizzle atoms need a 1,024-aligned base
  uint8_t* sm = ha_raw + (sb - raw);
  const uint32_t bar = sb + HA_BAR;
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bar) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // TMEM is taken before the next kernel may start (the trigger below), so a
  // later kernel of the stream never holds the columns this CTA waits for
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     sb + HA_TSLOT),
                 "r"(HA_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  ha_fence_before();
  __syncthreads();
  ha_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(sm + HA_TSLOT);
  pdl_trigger();
  const uint32_t tq = tmem + ((uint32_t)(warp * 32) << 16);  // this warp's lane quarter
  constexpr float QSCALE = 0.25f * L2E;  // 1 / sqrt(16), in base 2
  uint32_t phase = 0;
  bool ok = true;

  auto store_row = [&]() {
    // the row index is re-read here so that the compiler does not keep the
    // 32 store addresses of the swizzled operand live across the chunk loop
    int rr;
    asm volatile("mov.b32 %0, %1;" : "=r"(rr) : "r"(kr));
    const uint32_t vbase = (uint32_t)((rr >> 5) * HA_VT_ATOM + (rr & 3) * 4);
    const uint32_t vc = (uint32_t)((rr >> 2) & 7);
#pragma unroll
    for (int j = 0; j < HDH / 4; ++j) {
      float4 h, l;
      ha_split(pre[j], h, l);
      if (part == 0) {
        *reinterpret_cast<float4*>(sm + HA_K_HI + ha_kmaj(rr, j, HA_K_SBO)) = h;
        *reinterpret_cast<float4*>(sm + HA_K_LO + ha_kmaj(rr, j, HA_K_SBO)) = l;
      } else {
        const float hv[4] = {h.x, h.y, h.z, h.w}, lv[4] = {l.x, l.y, l.z, l.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {  // rows d (V_hi) and 16 + d (V_lo), key rr
          const int d = 4 * j + e;
          const uint32_t off = vbase + (uint32_t)((d >> 3) * 1024 + (d & 7) * 128) +
                               ((vc ^ (uint32_t)(d & 7)) << 4);
          *reinterpret_cast<float*>(sm + HA_VT + off) = hv[e];
          *reinterpret_cast<float*>(sm + HA_VT + 2 * 1024 + off) = lv[e];
        }
      }
    }
  };

  for (int qb = blockIdx.z; qb < nqb && ok; qb += (int)gridDim.z) {
    const int q = qb * HA_M + tid;
    if (qb != (int)blockIdx.z) {
      load_q(qb);
      load_row(0);
    }
    {  // the block's queries into TMEM, split
      float4 qh[HDH / 4], ql[HDH / 4];
#pragma unroll
      for (int j = 0; j < HDH / 4; ++j) ha_split(qv[j], qh[j], ql[j]);
      ha_st16(tq + HA_QH_COL, qh);
      ha_st16(tq + HA_QL_COL, ql);
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    }
    store_row();
    float o[HDH];
#pragma unroll
    for (int d = 0; d < HDH; ++d) o[d] = 0.f;
    float m = -INFINITY, l = 0.f;

    for (int k0 = 0; k0 < T; k0 += HA_NC) {
      const int nk = min(HA_NC, T - k0);
      ha_fence_async();
      ha_fence_before();
      __syncthreads();
      ha_fence_after();
      if (tid == 0) {
        // S = Q K^T over the chunk's keys rounded up to 16 (N), K = 8 per instruction
        const uint32_t idesc = HA_IDESC_S | ((uint32_t)(((nk + 15) & ~15) >> 3) << 17);
        // descriptors of the first K step (a K step adds its byte offset >> 4)
        const uint64_t dk_hi = ha_desc(sb + HA_K_HI, HA_K_SBO);
        const uint64_t dk_lo = ha_desc(sb + HA_K_LO, HA_K_SBO);
#pragma unroll
        for (int s = 0; s < HDH / 8; ++s) {
          const uint64_t ko = (256u * s) >> 4;
          ha_mma_ta(tmem, tmem + HA_QH_COL + 8u * s, dk_hi + ko, idesc, s);
          ha_mma_ta(tmem, tmem + HA_QH_COL + 8u * s, dk_lo + ko, idesc, 1u);
          ha_mma_ta(tmem, tmem + HA_QL_COL + 8u * s, dk_hi + ko, idesc, 1u);
        }
        ha_commit(bar);
      }
      if (!__syncthreads_and(ha_wait(bar, phase))) {
        ok = false;  // the phase stays: the teardown waits for it again
        break;
      }
      phase ^= 1u;
      ha_fence_after();

      // this query's 64 scores in two groups of 32 columns; the second group
      // is skipped when the chunk has no key there (the P V MMAs below stop
      // at the chunk's keys too).  The first group is read twice (for the
      // maximum, then for P), so that only 32 scores are held at a time.
      float va[32], vb[32];
      const bool full = nk == HA_NC, gb = nk > 32;
      float mx = -INFINITY;
      ha_ld32(tq, va);
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (full || j < nk) mx = fmaxf(mx, va[j]);
      if (gb) {
        ha_ld32(tq + 32, vb);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (full || 32 + j < nk) mx = fmaxf(mx, vb[j]);
      }
      const float mn = fmaxf(m, mx * QSCALE);
      float ls = 0.f;
      if (full) {
        ha_softmax32<true>(vb, 32, nk, QSCALE, mn, ls, sm + HA_P_LO, tid, tq + 32);
        ha_ld32(tq, va);
        ha_softmax32<true>(va, 0, nk, QSCALE, mn, ls, sm + HA_P_LO, tid, tq);
      } else {
        if (gb) ha_softmax32<false>(vb, 32, nk, QSCALE, mn, ls, sm + HA_P_LO, tid, tq + 32);
        ha_ld32(tq, va);
        ha_softmax32<false>(va, 0, nk, QSCALE, mn, ls, sm + HA_P_LO, tid, tq);
      }
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      const float f = ex2(m - mn);  // 0 on the first chunk (m = -inf)
      l = fmaf(l, f, ls);
      m = mn;
      ha_fence_async();
      ha_fence_before();
      __syncthreads();
      ha_fence_after();
      if (tid == 0) {
        const int ns = (nk + 7) >> 3;  // K steps up to the chunk's last key
        const uint64_t dp_lo = ha_desc(sb + HA_P_LO, HA_P_SBO);
        const uint64_t dvt = ha_desc_sw128(sb + HA_VT);
#pragma unroll 4
        for (int s = 0; s < ns; ++s) {  // O_c = P [V_hi | V_lo], K = 8 keys per instruction
          const uint64_t vo = (uint64_t)((s >> 2) * HA_VT_ATOM + (s & 3) * 32) >> 4;
          const uint64_t po = (256u * s) >> 4;
          ha_mma_ta(tmem + HA_O_COL, tmem + 8u * s, dvt + vo, HA_IDESC_O, s);
          ha_mma(tmem + HA_O_COL, dp_lo + po, dvt + vo, HA_IDESC_O, 1u);
        }
        ha_commit(bar);
      }
      // the next chunk's rows are loaded while the P V MMAs run
      if (k0 + HA_NC < T) load_row(k0 + HA_NC);
      if (!__syncthreads_and(ha_wait(bar, phase))) {
        ok = false;
        break;
      }
      phase ^= 1u;
      ha_fence_after();
      {  // O = f O + O_c, O_c the sum of the [V_hi | V_lo] halves
        float oc[32];
        ha_ld32(tq + HA_O_COL, oc);
#pragma unroll
        for (int d = 0; d < HDH; ++d) o[d] = fmaf(o[d], f, oc[d] + oc[HDH + d]);
      }
      if (k0 + HA_NC < T) store_row();
    }
    if (ok && q < T) {
      const float inv = 1.f / l;
      float4* op = reinterpret_cast<float4*>(scr + (int64_t)q * HSCR + HD + hh * HDH);
#pragma unroll
      for (int j = 0; j < HDH / 4; ++j)
        op[j] = make_float4(o[4 * j] * inv, o[4 * j + 1] * inv, o[4 * j + 2] * inv,
                            o[4 * j + 3] * inv);
    }
  }
  if (!ok) {
    if (tid == 0) atomicOr(a.ctx_flags, HA_ERR_TIMEOUT);
    ha_wait(bar, phase);  // the MMAs still pending, bounded as well
  }
  ha_fence_before();
  __syncthreads();
  if (warp == 0) {
    ha_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(HA_TMEM_COLS)
                 : "memory");
  }
}

// ---- head_rows: the row-local block on the tensor cores -----------------------------
//
// CTA i takes the 128-row tile i of the whole batch; thread t owns row t and
// TMEM lane t.  The block's four GEMMs run as tcgen05.mma kind::tf32 with the
// same split as the attention (x = x_hi + x_lo, three products per product,
// fp32-level accuracy): the activations are the A operand in TMEM (one column
// per K value, written by their own row's thread), the weights the B operand
// in shared memory (K-major canonical layout without swizzle), fp32
// accumulators in TMEM.  Between the GEMMs each thread reads its row of the
// accumulator and does the row-local work in registers, LayerNorm included:
//   MID / LAST: O = A W_o^T (A: the attention output), H1 = LN1(H + O + b_o),
//               F = ReLU(H1 W_1^T + b_1), H2 = LN2(H1 + F W_2^T + b_2) -> H
//   MID / QKV:  QKV = H W_qkv^T + b_qkv -> Q, K, V (H = H2, or the embedding)
// The weights are split and staged by the threads before the dependency wait
// (they are inputs of the call), so with programmatic dependent launch they
// overlap the previous kernel; W_qkv of a MID launch is loaded into registers
// then and stored over W_o and W_1 once their GEMMs are done.  TMEM columns
// (512, one CTA per SM): A operands hi / lo at 0-63 / 64-127 (K = 64) or
// 0-127 / 128-255 (the hidden layer, K = 128); accumulators at 256 (W_1: 128
// columns; W_2: 64; W_qkv: 192) and 384 (W_o: 64); H1 kept at 448-511 for
// the second residual.  One elected thread issues the MMAs; every wait is
// bounded.
constexpr int HT_M = 128;                           // rows per tile = TMEM lanes
constexpr int HT_NT = 2 * HT_M;                     // threads: two per row (column halves)
constexpr uint32_t HT_TMEM_COLS = 512;
constexpr uint32_t HT_A_HI = 0, HT_A_LO = 64;       // K = 64 A operands
constexpr uint32_t HT_F_HI = 0, HT_F_LO = 128;      // the hidden layer (K = 128)
constexpr uint32_t HT_D = 256;                      // W_1, W_2, W_qkv accumulators
constexpr uint32_t HT_DO = 384;                     // W_o accumulator
constexpr uint32_t HT_H1 = 448;                     // H1, fp32
// shared memory (bytes): weights split in two, each matrix [N][K] hi then lo
constexpr int HT_WO = 0;                            // W_o, 2 x 16 KB
constexpr int HT_W1 = HT_WO + 2 * HD * HD * 4;      // W_1, 2 x 32 KB
constexpr int HT_W2 = HT_W1 + 2 * HFF * HD * 4;     // W_2, 2 x 32 KB
constexpr int HT_WEND = HT_W2 + 2 * HD * HFF * 4;   // 160 KB
constexpr int HT_WQKV = 0;                          // W_qkv, 2 x 48 KB, over W_o and W_1
static_assert(HT_WQKV + 2 * 3 * HD * HD * 4 <= HT_W2, "W_qkv fits over W_o and W_1");
constexpr int HT_VEC = HT_WEND;                     // b_qkv | b_o g1 be1 | b_1 | b_2 g2 be2
constexpr int HT_VEC_N = 3 * HD + 3 * HD + HFF + 3 * HD;
// the tile's 64-wide input / output rows, staged for coalesced global access
constexpr int HT_LDX = HD + 4;                      // padded row (floats): conflict-free per row
constexpr int HT_X = HT_VEC + HT_VEC_N * 4;
// the QKV output tile, staged over the weights once their GEMMs are done
constexpr int HT_LDQ = 3 * HD + 4;
constexpr int HT_Q = 0;
static_assert(HT_Q + HT_M * HT_LDQ * 4 <= HT_VEC, "the QKV tile fits over the weights");
constexpr int HT_XCH = HT_X + HT_M * HT_LDX * 4;    // row sums of the two halves [2][2][128]
constexpr int HT_BAR = HT_XCH + 4 * HT_M * 4;       // mbarrier: MMA completion
constexpr int HT_TSLOT = HT_BAR + 8;
constexpr size_t HT_SMEM = HT_TSLOT + 8;
static_assert(HT_SMEM <= 227 * 1024, "head_rows shared memory");
static_assert(HT_BAR % 8 == 0, "mbarrier alignment");
// vector offsets inside HT_VEC
constexpr int HV_BQKV = 0, HV_BO = 192, HV_G1 = 256, HV_BE1 = 320, HV_B1 = 384, HV_B2 = 512,
              HV_G2 = 576, HV_BE2 = 640;

// tf32 instruction descriptor for M = 128 and the given N
__host__ __device__ constexpr uint32_t ht_idesc(int n) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(HT_M >> 4) << 24);
}

// float4 piece c of an [N][K] weight matrix: source row n, values 4 j .. 4 j + 3,
// stored at float 4 c of the canonical layout (core matrices of 8 rows x 4
// values, consecutive along K, 8-row groups one after another)
template <int N, int K>
__device__ __forceinline__ void ht_piece_src(int c, int& n, int& j) {
  constexpr int Q = K / 4;
  const int g = c >> 3;
  n = ((g / Q) << 3) | (c & 7);
  j = g % Q;
}
// this thread's pieces of W, raw, into the matrix's lo half (cp.async: all in
// flight at once); ht_split_w then splits them in place once they have landed
template <int N, int K>
__device__ __forceinline__ void ht_copy_w(uint8_t* dst, const float* __restrict__ src) {
  constexpr int IT = N * K / 4 / HT_NT;
#pragma unroll
  for (int i = 0; i < IT; ++i) {
    const int c = threadIdx.x + i * HT_NT;
    int n, j;
    ht_piece_src<N, K>(c, n, j);
    const uint32_t d = ha_saddr(dst + N * K * 4 + 16 * c);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src + n * K + 4 * j)
                 : "memory");
  }
}
template <int N, int K>
__device__ __forceinline__ void ht_split_w(uint8_t* dst) {
  constexpr int IT = N * K / 4 / HT_NT;
#pragma unroll
  for (int i = 0; i < IT; ++i) {
    const int c = threadIdx.x + i * HT_NT;
    float4* lo = reinterpret_cast<float4*>(dst + N * K * 4) + c;
    float4 h, l;
    ha_split(*lo, h, l);
    reinterpret_cast<float4*>(dst)[c] = h;
    *lo = l;
  }
}

// D (+)= A B^T over K: A_hi / A_lo in TMEM columns, B = W (N rows, hi then lo)
// in shared memory; three products per K step of 8
template <int N, int K>
__device__ __forceinline__ void ht_gemm(uint32_t d, uint32_t a_hi, uint32_t a_lo, uint32_t w) {
  constexpr uint32_t SBO = (K / 4) * 128;
  const uint64_t bh = ha_desc(w, SBO), bl = ha_desc(w + N * K * 4, SBO);
#pragma unroll
  for (int s = 0; s < K / 8; ++s) {
    const uint64_t ko = (256u * s) >> 4;
    ha_mma_ta(d, a_hi + 8u * s, bh + ko, ht_idesc(N), s);
    ha_mma_ta(d, a_hi + 8u * s, bl + ko, ht_idesc(N), 1u);
    ha_mma_ta(d, a_lo + 8u * s, bh + ko, ht_idesc(N), 1u);
  }
}

// 32 values split in two and written to TMEM as A-operand columns
__device__ __forceinline__ void ht_put_split(uint32_t t_hi, uint32_t t_lo, const float* v) {
  float h[32], l[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    h[j] = ha_hi(v[j]);
    l[j] = v[j] - h[j];
  }
  ha_st32(t_hi, h);
  ha_st32(t_lo, l);
}

// LayerNorm of a row whose 64 values are held by two threads, 32 each (half
// hf holds columns 32 hf ..): the halves' partial sums meet in shared memory
// and are added in half order, so both threads see the same statistics
__device__ __forceinline__ void ht_layer_norm(float (&v)[32], const float* g, const float* be,
                                              float* xch, int r, int hf) {
  float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int j = 0; j < 32; ++j) s4[j & 3] += v[j];
  xch[hf * HT_M + r] = (s4[0] + s4[1]) + (s4[2] + s4[3]);
  __syncthreads();
  const float mu = (xch[r] + xch[HT_M + r]) * (1.f / HD);
  float q4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    v[j] -= mu;
    q4[j & 3] = fmaf(v[j], v[j], q4[j & 3]);
  }
  xch[(2 + hf) * HT_M + r] = (q4[0] + q4[1]) + (q4[2] + q4[3]);
  __syncthreads();
  const float inv =
      1.f / sqrtf((xch[2 * HT_M + r] + xch[3 * HT_M + r]) * (1.f / HD) + HLN_EPS);
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = fmaf(v[j] * inv, g[32 * hf + j], be[32 * hf + j]);
}

// rows [row0, row0 + 128) of scratch columns [col, col + 64) into the staging
// tile with cp.async, sixteen threads per row (coalesced); rows past the batch
// are zero-filled
__device__ __forceinline__ void ht_load_rows(uint8_t* sm, const float* scr, int64_t row0,
                                             int64_t n_rows, int col) {
#pragma unroll
  for (int i = 0; i < HT_M * (HD / 4) / HT_NT; ++i) {
    const int c = threadIdx.x + i * HT_NT;
    const int r = c >> 4, q = c & 15;
    const bool ok = row0 + r < n_rows;
    const float* src = scr + (ok ? row0 + r : 0) * HSCR + col + 4 * q;
    const uint32_t d = ha_saddr(sm + HT_X + (r * HT_LDX + 4 * q) * 4);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src),
                 "r"(ok ? 16 : 0)
                 : "memory");
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}
// the staging tile back to scratch columns [col, col + 64), coalesced
__device__ __forceinline__ void ht_store_rows(const uint8_t* sm, float* scr, int64_t row0,
                                              int64_t n_rows, int col) {
#pragma unroll
  for (int i = 0; i < HT_M * (HD / 4) / HT_NT; ++i) {
    const int c = threadIdx.x + i * HT_NT;
    const int r = c >> 4, q = c & 15;
    if (row0 + r < n_rows)
      *reinterpret_cast<float4*>(scr + (row0 + r) * HSCR + col + 4 * q) =
          *reinterpret_cast<const float4*>(sm + HT_X + (r * HT_LDX + 4 * q) * 4);
  }
}

template <int MODE>
__global__ void __launch_bounds__(HT_NT, 1) head_rows(const HeadArgs a) {
  extern __shared__ __align__(16) uint8_t ht_sm[];
  const int tid = threadIdx.x, warp = tid >> 5;
  const int r = tid & (HT_M - 1);  // the row (TMEM lane) ...
  const int hf = tid >> 7;         // ... and the half of its columns this thread takes
  const uint32_t sb = ha_saddr(ht_sm);
  const uint32_t bar = sb + HT_BAR;
  float* sV = reinterpret_cast<float*>(ht_sm + HT_VEC);
  float* xch = reinterpret_cast<float*>(ht_sm + HT_XCH);
  // this thread's half of its row in the staging tile (8 pieces of 16 bytes)
  float4* xrow = reinterpret_cast<float4*>(ht_sm + HT_X) + r * (HT_LDX / 4) + 8 * hf;
  const int64_t row0 = (int64_t)blockIdx.x * HT_M;

  // the weights and vectors are inputs of the call: staged before the wait,
  // their copies in flight while the CTA takes its TMEM
  constexpr int WQ_IT = 3 * HD * HD / 4 / HT_NT;
  float4 wq_hold[MODE == HR_MID ? WQ_IT : 1];
  if (MODE == HR_QKV) ht_copy_w<3 * HD, HD>(ht_sm + HT_WQKV, a.lnext + HL_WQKV);
  if (MODE != HR_QKV) {
    ht_copy_w<HD, HD>(ht_sm + HT_WO, a.lcur + HL_WO);
    ht_copy_w<HFF, HD>(ht_sm + HT_W1, a.lcur + HL_W1);
    ht_copy_w<HD, HFF>(ht_sm + HT_W2, a.lcur + HL_W2);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
  if (MODE == HR_MID) {  // W_qkv waits in registers until W_o and W_1 are done
#pragma unroll
    for (int i = 0; i < WQ_IT; ++i) {
      int n, j;
      ht_piece_src<3 * HD, HD>(tid + i * HT_NT, n, j);
      wq_hold[i] = __ldg(reinterpret_cast<const float4*>(a.lnext + HL_WQKV + n * HD) + j);
    }
  }
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bar) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // TMEM is taken before the next kernel may start (the trigger below), so a
  // later kernel of the stream never holds the columns this CTA waits for
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     sb + HT_TSLOT),
                 "r"(HT_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
#pragma unroll
  for (int k = 0; k < (HT_VEC_N + HT_NT - 1) / HT_NT; ++k) {
    const int i = tid + k * HT_NT;
    if (i >= HT_VEC_N) break;
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
  asm volatile("cp.async.wait_all;" ::: "memory");  // this thread's pieces, split in place
  if (MODE == HR_QKV) ht_split_w<3 * HD, HD>(ht_sm + HT_WQKV);
  if (MODE != HR_QKV) {
    ht_split_w<HD, HD>(ht_sm + HT_WO);
    ht_split_w<HFF, HD>(ht_sm + HT_W1);
    ht_split_w<HD, HFF>(ht_sm + HT_W2);
  }
  ha_fence_before();
  __syncthreads();
  ha_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(ht_sm + HT_TSLOT);
  const uint32_t tq = tmem + ((uint32_t)((warp & 3) * 32) << 16);  // this warp's lane quarter
  const uint32_t c32 = 32u * hf;                                    // this half's first column
  pdl_trigger();
  pdl_wait();

  // the tile's input rows (the attention output over Q for MID / LAST, H for
  // QKV), then this thread's half row as the first GEMM's A operand
  ht_load_rows(ht_sm, a.scratch, row0, a.n_rows, MODE == HR_QKV ? 0 : HD);
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();
  auto read_half = [&](float (&x)[32]) {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 v = xrow[j];
      x[4 * j] = v.x;
      x[4 * j + 1] = v.y;
      x[4 * j + 2] = v.z;
      x[4 * j + 3] = v.w;
    }
  };
  {
    float x[32];
    read_half(x);
    ht_put_split(tq + HT_A_HI + c32, tq + HT_A_LO + c32, x);
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
  }
  uint32_t phase = 0;
  bool ok = true;
  // all threads' operands written -> one thread issues the MMAs -> every
  // thread waits (bounded) for their completion; `during` runs meanwhile
  auto mma_step = [&](auto issue, auto during) -> bool {
    ha_fence_async();
    ha_fence_before();
    __syncthreads();
    ha_fence_after();
    if (tid == 0) {
      issue();
      ha_commit(bar);
    }
    during();
    if (!__syncthreads_and(ha_wait(bar, phase))) return false;
    phase ^= 1u;
    ha_fence_after();
    return true;
  };
  auto nothing = [] {};

  if (MODE != HR_QKV) {
    float h[32];
    // O = A W_o^T, while the residual H comes into the staging tile
    ok = mma_step(
        [&] { ht_gemm<HD, HD>(tmem + HT_DO, tmem + HT_A_HI, tmem + HT_A_LO, sb + HT_WO); },
        [&] { ht_load_rows(ht_sm, a.scratch, row0, a.n_rows, 0); });
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();
    if (ok) {
      // H1 = LN1(H + O + b_o): kept in TMEM for the second residual and split
      // as the A operand of W_1
      read_half(h);
      {
        float d[32];
        ha_ld32(tq + HT_DO + c32, d);
#pragma unroll
        for (int j = 0; j < 32; ++j) h[j] += d[j] + sV[HV_BO + c32 + j];
      }
      ht_layer_norm(h, sV + HV_G1, sV + HV_BE1, xch, r, hf);
      ha_st32(tq + HT_H1 + c32, h);
      ht_put_split(tq + HT_A_HI + c32, tq + HT_A_LO + c32, h);
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      ok = mma_step(
          [&] { ht_gemm<HFF, HD>(tmem + HT_D, tmem + HT_A_HI, tmem + HT_A_LO, sb + HT_W1); },
          nothing);
    }
    if (ok) {
      if (MODE == HR_MID) {  // W_o and W_1 are done: W_qkv over them
#pragma unroll
        for (int i = 0; i < WQ_IT; ++i) {
          float4 hh, ll;
          ha_split(wq_hold[i], hh, ll);
          reinterpret_cast<float4*>(ht_sm + HT_WQKV)[tid + i * HT_NT] = hh;
          reinterpret_cast<float4*>(ht_sm + HT_WQKV + 3 * HD * HD * 4)[tid + i * HT_NT] = ll;
        }
      }
      // F = ReLU(H1 W_1^T + b_1), split as the A operand of W_2 (64 columns a half)
#pragma unroll
      for (int c = 0; c < HFF / 64; ++c) {
        const uint32_t col = 64u * hf + 32u * c;
        float d[32];
        ha_ld32(tq + HT_D + col, d);
#pragma unroll
        for (int j = 0; j < 32; ++j) d[j] = fmaxf(d[j] + sV[HV_B1 + col + j], 0.f);
        ht_put_split(tq + HT_F_HI + col, tq + HT_F_LO + col, d);
      }
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      ok = mma_step(
          [&] { ht_gemm<HD, HFF>(tmem + HT_D, tmem + HT_F_HI, tmem + HT_F_LO, sb + HT_W2); },
          nothing);
    }
    if (ok) {
      // H2 = LN2(H1 + F W_2^T + b_2) -> H, through the staging tile
      {
        float d[32], rr[32];
        ha_ld32(tq + HT_D + c32, d);
        ha_ld32(tq + HT_H1 + c32, rr);
#pragma unroll
        for (int j = 0; j < 32; ++j) h[j] = rr[j] + (d[j] + sV[HV_B2 + c32 + j]);
      }
      ht_layer_norm(h, sV + HV_G2, sV + HV_BE2, xch, r, hf);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        xrow[j] = make_float4(h[4 * j], h[4 * j + 1], h[4 * j + 2], h[4 * j + 3]);
      if (MODE == HR_MID) {
        ht_put_split(tq + HT_A_HI + c32, tq + HT_A_LO + c32, h);
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      }
      __syncthreads();
      ht_store_rows(ht_sm, a.scratch, row0, a.n_rows, 0);
    }
  }
  if (MODE != HR_LAST && ok) {
    // QKV = H W_qkv^T + b_qkv -> scratch columns [64, 256), through a
    // staging tile over the weights (their MMAs are done); 96 columns a half
    ok = mma_step(
        [&] { ht_gemm<3 * HD, HD>(tmem + HT_D, tmem + HT_A_HI, tmem + HT_A_LO, sb + HT_WQKV); },
        nothing);
    if (ok) {
      float4* qrow = reinterpret_cast<float4*>(ht_sm + HT_Q) + r * (HT_LDQ / 4);
#pragma unroll
      for (int c = 0; c < 3; ++c) {
        const uint32_t col = 96u * hf + 32u * c;
        float d[32];
        ha_ld32(tq + HT_D + col, d);
#pragma unroll
        for (int j = 0; j < 8; ++j)
          qrow[col / 4 + j] = make_float4(d[4 * j] + sV[HV_BQKV + col + 4 * j],
                                          d[4 * j + 1] + sV[HV_BQKV + col + 4 * j + 1],
                                          d[4 * j + 2] + sV[HV_BQKV + col + 4 * j + 2],
                                          d[4 * j + 3] + sV[HV_BQKV + col + 4 * j + 3]);
      }
      __syncthreads();
#pragma unroll 4
      for (int i = 0; i < HT_M * (3 * HD / 4) / HT_NT; ++i) {  // 48 pieces of 16 bytes a row
        const int f = tid + i * HT_NT;
        const int rw = f / (3 * HD / 4), q = f - rw * (3 * HD / 4);
        if (row0 + rw < a.n_rows)
          *reinterpret_cast<float4*>(a.scratch + (row0 + rw) * HSCR + HD + 4 * q) =
              reinterpret_cast<const float4*>(ht_sm + HT_Q)[rw * (HT_LDQ / 4) + q];
      }
    }
  }
  if (!ok) {
    if (tid == 0) atomicOr(a.ctx_flags, HA_ERR_TIMEOUT);
    ha_wait(bar, phase);  // the MMAs still pending, bounded as well
  }
  ha_fence_before();
  __syncthreads();
  if (warp == 0) {
    ha_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(HT_TMEM_COLS)
                 : "memory");
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
