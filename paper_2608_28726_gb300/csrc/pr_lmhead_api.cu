// Host side of pr_lmhead_features: argument checks, the TMA tensor maps of the
// hidden states and the LM-head weights, the vocabulary split and the launches
// of the kernels in pr_lmhead.cuh.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>

#include "pr_ctx.h"
#include "pr_lmhead.cuh"

using namespace prh;

static_assert(prk::LM_ERR_TIMEOUT == PR_FLAG_TIMEOUT, "flag bit");
// the last tile's columns (and a chunk's end, col0 + 32) stay below 2^31
static_assert((PR_LMHEAD_MAX_VOCAB + prk::LM_BN - 1) / prk::LM_BN * prk::LM_BN <= 0x7fffffffLL,
              "vocabulary limit");

namespace {

typedef CUresult (*EncodeTiled)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// the driver's tensor-map encoder, looked up once through the runtime (no link
// against the driver library)
EncodeTiled encoder() {
  static EncodeTiled fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiled>(p);
  }
  return fn;
}

// row-major bf16 matrix [rows][d] read in boxes of LM_BOX_K = 64 columns x
// box_rows rows, 128-byte swizzle, zero fill outside the matrix
bool make_map(CUtensorMap* map, const void* base, int64_t rows, int64_t d, uint32_t box_rows) {
  EncodeTiled enc = encoder();
  if (!enc) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  const cuuint32_t box[2] = {(cuuint32_t)prk::LM_BOX_K, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
             box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

}  // namespace

// The first launch of both LM-head entry points: lm_fused over the batch into
// the context's state buffer.  On return *nparts is the number of partial
// states per row (one per vocabulary split; the kernel has already merged each
// row's two column halves).
static pr_status launch_lm_fused(pr_ctx* c, const void* hidden, const void* weight, int64_t n_rows,
                                 int64_t d, int64_t vocab, const int32_t* chosen, int kc,
                                 cudaStream_t s, int64_t* nparts_out) {
  if (!c->lm_ready) {
    PR_CUDA(cudaFuncSetAttribute(prk::lm_fused<20>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)prk::LM_SMEM));
    PR_CUDA(cudaFuncSetAttribute(prk::lm_fused<32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)prk::LM_SMEM));
    c->lm_ready = true;
  }
  const int64_t mtiles = (n_rows + prk::LM_BM - 1) / prk::LM_BM;
  const int64_t ntiles = (vocab + prk::LM_BN - 1) / prk::LM_BN;
  if (mtiles > 0x7fffffffLL) return PR_ERR_INVALID_ARG;
  const void* kern = kc <= 20 ? reinterpret_cast<const void*>(&prk::lm_fused<20>)
                              : reinterpret_cast<const void*>(&prk::lm_fused<32>);
  // Launch shape: nsplit vocabulary splits (around 12, or for a small batch as
  // many as fill one wave of one CTA per SM; among those the count with the
  // least idle tail in the last wave), CTA pairs of
  // 256 rows ordered in bands of `band` row pairs, whose H rows (256 d bf16
  // each) fill about a quarter of L2: a wave then holds one band's H plus the
  // W tiles of a few splits, each read from DRAM about once per wave.
  const int64_t mt_pad = (mtiles + 1) / 2 * 2;
  int64_t nsplit = 1;
  {
    double best = 1e30;
    const int64_t fill = std::max<int64_t>(1, c->num_sms / mt_pad);  // splits filling a wave
    const double target = std::max<double>(12.0, (double)fill);
    for (int64_t ns = 8; ns <= std::max<int64_t>(24, fill) && ns <= ntiles; ++ns) {
      const int64_t ctas = mt_pad * ns;
      const int64_t waves = (ctas + c->num_sms - 1) / c->num_sms;
      const double waste = (double)(waves * c->num_sms - ctas) / (double)(waves * c->num_sms);
      const double score = waste + 0.002 * std::abs((double)ns - target);
      if (score < best) {
        best = score;
        nsplit = ns;
      }
    }
    if (best == 1e30) nsplit = std::max<int64_t>(1, std::min<int64_t>(ntiles, c->num_sms / mt_pad));
  }
  const int64_t per_split = (ntiles + nsplit - 1) / nsplit;
  CUtensorMap ma, mb;  // boxes of 128 rows x 64 columns: a CTA's H rows, half a W tile
  if (!make_map(&ma, hidden, n_rows, d, (uint32_t)prk::LM_BM) ||
      !make_map(&mb, weight, vocab, d, (uint32_t)(prk::LM_BN / 2)))
    return PR_ERR_UNSUPPORTED;
  const int64_t nparts = nsplit;  // one state per (row, split)
  const size_t part_bytes = (size_t)nparts * (size_t)n_rows * sizeof(prk::LmPart);
  if (part_bytes > c->lm_parts_bytes) {
    PR_CUDA(cudaDeviceSynchronize());  // the old buffer may still be in use
    cudaFree(c->lm_parts);
    c->lm_parts = nullptr;
    c->lm_parts_bytes = 0;
    if (cudaMalloc(&c->lm_parts, part_bytes) != cudaSuccess) {
      cudaGetLastError();
      c->lm_parts = nullptr;
      return PR_ERR_NO_MEMORY;
    }
    c->lm_parts_bytes = part_bytes;
  }
  prk::LmArgs la;
  memset(&la, 0, sizeof la);
  la.n_rows = n_rows;
  la.vocab = vocab;
  la.d = (int32_t)d;
  la.kblocks = (int32_t)((d + prk::LM_BK - 1) / prk::LM_BK);
  la.ntiles = (int32_t)ntiles;
  la.tiles_per_split = (int32_t)per_split;
  la.nsplit = (int32_t)nsplit;
  la.npairs = (int32_t)(mt_pad / 2);
  {
    const int64_t h_pair = 256 * d * 2, budget = (int64_t)32 << 20;
    la.band = (int32_t)std::max<int64_t>(1, std::min<int64_t>(la.npairs, budget / h_pair));
  }
  la.chosen = chosen;
  la.parts = static_cast<prk::LmPart*>(c->lm_parts);
  la.err = c->flags;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  if (mt_pad * nsplit > 0x7fffffffLL) return PR_ERR_INVALID_ARG;
  cfg.gridDim = dim3((unsigned)(mt_pad * nsplit));
  cfg.blockDim = dim3(prk::LM_NT);
  cfg.dynamicSmemBytes = prk::LM_SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;  // a CTA pair lies along x
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void* kargs[] = {&ma, &mb, &la};
  PR_CUDA(cudaLaunchKernelExC(&cfg, kern, kargs));
  *nparts_out = nparts;
  return PR_OK;
}

// The merge launch: wpr warps per row, more for rows with many parts.
static void launch_lm_merge(const prk::Args& a, pr_ctx* c, int64_t nparts, int mode,
                            cudaStream_t s) {
  const int wpr = nparts >= 64 ? 8 : nparts >= 32 ? 4 : 1;
  const int64_t rows_per_cta = 8 / wpr;
  const unsigned grid = (unsigned)((a.n_rows + rows_per_cta - 1) / rows_per_cta);
  const prk::LmPart* parts = static_cast<const prk::LmPart*>(c->lm_parts);
  if (mode == prk::MODE_DECODE)
    prk::lm_merge<prk::MODE_DECODE><<<grid, 256, 0, s>>>(a, parts, (int)nparts, wpr);
  else
    prk::lm_merge<prk::MODE_FEATURES><<<grid, 256, 0, s>>>(a, parts, (int)nparts, wpr);
}

extern "C" {

pr_status pr_lmhead_features(pr_ctx* c, const void* hidden, const void* weight, int64_t n_rows,
                             int64_t d, int64_t vocab, const int32_t* chosen, int32_t topk,
                             const int64_t* offsets, int32_t n_req, float* feat, int32_t* top2,
                             uint32_t* row_flags, void* stream) {
  if (!c || n_rows < 0 || n_rows > 0x7fffffffLL || vocab <= 0 || vocab > PR_LMHEAD_MAX_VOCAB)
    return PR_ERR_INVALID_ARG;
  if (d <= 0 || d % 8 != 0 || d > (int64_t)1 << 20) return PR_ERR_INVALID_ARG;
  if (topk < 1 || topk > PR_MAX_TOPK || n_req < 0 || (offsets && n_req < 1))
    return PR_ERR_INVALID_ARG;
  if (n_rows == 0) return PR_OK;
  if (!hidden || !weight || !chosen || !feat || !top2 || !row_flags) return PR_ERR_INVALID_ARG;
  if (!aligned16(hidden) || !aligned16(weight)) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  const int kc = topk > 2 ? topk : 2;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((st = timing_begin(c, s)) != PR_OK) return st;
  int64_t nparts = 0;
  if ((st = launch_lm_fused(c, hidden, weight, n_rows, d, vocab, chosen, kc, s, &nparts)) != PR_OK)
    return st;
  if ((st = timing_mark(c, s)) != PR_OK) return st;
  prk::Args a;
  memset(&a, 0, sizeof a);
  a.n_rows = n_rows;
  a.vocab = vocab;
  a.chosen = chosen;
  a.topk = topk;
  a.kc = kc;
  a.renorm = c->renorm;
  a.offsets = offsets;
  a.n_req = offsets ? n_req : 0;
  a.feat = feat;
  a.top2 = top2;
  a.row_flags = row_flags;
  a.ctx_flags = c->flags;
  launch_lm_merge(a, c, nparts, prk::MODE_FEATURES, s);
  PR_CUDA(cudaGetLastError());
  g_launches.fetch_add(2, std::memory_order_relaxed);
  return timing_mark(c, s);
}

pr_status pr_lmhead_decode_step(pr_ctx* c, const void* hidden, const void* weight, int32_t n_live,
                                int64_t d, int64_t vocab, const int32_t* slot,
                                const int32_t* chosen, const uint8_t* eos, const float* w, float b,
                                float tau, float* score_out, uint8_t* ship_out,
                                uint32_t* slot_flags, float* agg_out, void* stream) {
  if (!c || n_live < 0 || vocab <= 0 || vocab > PR_LMHEAD_MAX_VOCAB) return PR_ERR_INVALID_ARG;
  if (d <= 0 || d % 8 != 0 || d > (int64_t)1 << 20) return PR_ERR_INVALID_ARG;
  if (n_live > c->max_requests) return PR_ERR_INVALID_ARG;
  if (n_live == 0) return PR_OK;
  if (!hidden || !weight || !slot || !chosen || !eos || !w || !score_out || !ship_out ||
      !slot_flags)
    return PR_ERR_INVALID_ARG;
  if (!aligned16(hidden) || !aligned16(weight)) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  const int kc = c->topk > 2 ? c->topk : 2;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((st = timing_begin(c, s)) != PR_OK) return st;
  int64_t nparts = 0;
  if ((st = launch_lm_fused(c, hidden, weight, n_live, d, vocab, chosen, kc, s, &nparts)) != PR_OK)
    return st;
  if ((st = timing_mark(c, s)) != PR_OK) return st;
  prk::Args a;
  memset(&a, 0, sizeof a);
  a.n_rows = n_live;
  a.vocab = vocab;
  a.chosen = chosen;
  a.topk = c->topk;
  a.kc = kc;
  a.renorm = c->renorm;
  a.slot = slot;
  a.eos = eos;
  a.acc = c->acc;
  a.n_slots = c->max_requests;
  a.w = w;
  a.b = b;
  a.zthr = zthreshold(tau);
  a.score = score_out;
  a.ship = ship_out;
  a.req_flags = slot_flags;
  a.agg = agg_out;
  a.ctx_flags = c->flags;
  launch_lm_merge(a, c, nparts, prk::MODE_DECODE, s);
  PR_CUDA(cudaGetLastError());
  g_launches.fetch_add(2, std::memory_order_relaxed);
  return timing_mark(c, s);
}

pr_status pr_selftest_wait(pr_ctx* c, int64_t limit_ns, int32_t* completed) {
  if (!c || !completed || limit_ns < 0 || limit_ns > 2000000000LL) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  int32_t* d = nullptr;
  PR_CUDA(cudaMalloc(&d, sizeof(int32_t)));
  prk::lm_wait_probe<<<1, 1>>>(c->flags, (uint64_t)limit_ns, d);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaMemcpy(completed, d, sizeof(int32_t), cudaMemcpyDeviceToHost);
  cudaFree(d);
  if (e != cudaSuccess) return cuda_fail(e, "pr_selftest_wait");
  g_launches.fetch_add(1, std::memory_order_relaxed);
  return PR_OK;
}

}  // extern "C"
