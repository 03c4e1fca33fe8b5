// Host side of the scorer head's C ABI entry points (pr_head_param_count,
// pr_head_score): argument checks, the context's activation scratch and the
// launch chain of the kernels in pr_head.cuh.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>

#include "pr_ctx.h"
#include "pr_head.cuh"

using namespace prh;

namespace {

// One kernel of the scorer head's chain; `pdl` lets it start while the
// previous kernel on the stream finishes (it waits before reading that
// kernel's results).
pr_status launch_head(pr_ctx* c, const void* kernel, dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                      bool pdl, const prk::HeadArgs& a) {
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  void* args[] = {const_cast<prk::HeadArgs*>(&a)};
  PR_CUDA(cudaLaunchKernelExC(&cfg, kernel, args));
  g_launches.fetch_add(1, std::memory_order_relaxed);
  return timing_mark(c, s);
}

}  // namespace

extern "C" {

int64_t pr_head_param_count(int32_t n_layers) {
  if (n_layers < 1 || n_layers > prk::HMAXL) return -1;
  return prk::head_param_count(n_layers);
}

pr_status pr_head_score(pr_ctx* c, const float* feat, const uint32_t* row_flags, int64_t n_rows,
                        const int64_t* offsets, int32_t n_req, const float* w, int32_t n_layers,
                        float tau, float* score, uint8_t* ship, uint32_t* req_flags,
                        void* stream) {
  if (!c || n_req < 0 || n_rows < 0) return PR_ERR_INVALID_ARG;
  if (n_layers < 1 || n_layers > prk::HMAXL) return PR_ERR_INVALID_ARG;
  if (n_rows > ((int64_t)1 << 30)) return PR_ERR_INVALID_ARG;
  if (n_req == 0) return PR_OK;
  if (!offsets || !w || !score || !ship || !req_flags) return PR_ERR_INVALID_ARG;
  if (n_rows > 0 && !feat) return PR_ERR_INVALID_ARG;
  if (!aligned16(w) || !aligned16(feat)) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  if (!c->head_ready) {
    PR_CUDA(cudaFuncSetAttribute(prk::head_rows<prk::HR_QKV>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)prk::HT_SMEM));
    PR_CUDA(cudaFuncSetAttribute(prk::head_rows<prk::HR_MID>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)prk::HT_SMEM));
    PR_CUDA(cudaFuncSetAttribute(prk::head_rows<prk::HR_LAST>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)prk::HT_SMEM));
    PR_CUDA(cudaFuncSetAttribute(prk::head_attn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)prk::HA_SMEM));
    c->head_ready = true;
  }
  if (n_rows > c->head_scr_rows) {
    // grow: wait for the kernels that may still use the old scratch
    PR_CUDA(cudaDeviceSynchronize());
    cudaFree(c->head_scr);
    c->head_scr = nullptr;
    c->head_scr_rows = 0;
    const size_t bytes = (size_t)n_rows * prk::HSCR * sizeof(float);
    if (cudaMalloc(&c->head_scr, bytes) != cudaSuccess) {
      cudaGetLastError();
      c->head_scr = nullptr;
      return PR_ERR_NO_MEMORY;
    }
    PR_CUDA(cudaMemset(c->head_scr, 0, bytes));
    c->head_scr_rows = n_rows;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((st = timing_begin(c, s)) != PR_OK) return st;
  prk::HeadArgs a;
  memset(&a, 0, sizeof a);
  a.feat = feat;
  a.row_flags = row_flags;
  a.n_rows = n_rows;
  a.offsets = offsets;
  a.n_req = n_req;
  a.w = w;
  a.n_layers = n_layers;
  a.zthr = zthreshold(tau);
  a.scratch = c->head_scr;
  a.score = score;
  a.ship = ship;
  a.req_flags = req_flags;
  a.ctx_flags = c->flags;
  const float* layer0 = w + prk::H_PRE;
  auto layer = [&](int l) { return layer0 + (int64_t)l * prk::HL_SIZE; };
  const dim3 blk(prk::NT);
  st = launch_head(c, reinterpret_cast<const void*>(&prk::head_embed),
                   dim3((unsigned)n_req, prk::HES), blk, 0, s, c->overlap != 0, a);
  if (st != PR_OK) return st;
  if (n_rows > 0) {
    // one CTA per 128-row tile (the row kernels hold all 512 TMEM columns of an SM)
    const unsigned ntiles = (unsigned)((n_rows + prk::HT_M - 1) / prk::HT_M);
    const dim3 rblk(prk::HT_NT);
    a.lcur = nullptr;
    a.lnext = layer(0);
    st = launch_head(c, reinterpret_cast<const void*>(&prk::head_rows<prk::HR_QKV>), dim3(ntiles),
                     rblk, prk::HT_SMEM, s, true, a);
    if (st != PR_OK) return st;
    // CTAs per (request, head): one per query block of a request of the mean
    // length, at least HA_QZ_MIN.  A CTA whose request has no block z exits at
    // once, but empty CTAs still slow the launch chain, and too few leave long
    // requests' blocks in sequence (two layers, back-to-back calls: 64 requests
    // of U{32..256} rows 72.3 us with 8 CTAs, 71.0 with 4; 1,024 lognormal
    // requests 1.12 ms with 8, 1.07 with 4; four requests of 2,100 and 1,300
    // rows 484 us with 8, 359 with 14).
    const int64_t mean_t = n_rows / n_req;
    const unsigned gz = (unsigned)std::min<int64_t>(
        prk::HA_QZ_MAX, std::max<int64_t>(prk::HA_QZ_MIN, (mean_t + prk::HA_M - 1) / prk::HA_M));
    for (int l = 0; l < n_layers; ++l) {
      st = launch_head(c, reinterpret_cast<const void*>(&prk::head_attn),
                       dim3((unsigned)n_req, prk::HHEADS, gz), dim3(prk::HA_M), prk::HA_SMEM, s,
                       true, a);
      if (st != PR_OK) return st;
      a.lcur = layer(l);
      const bool last = l + 1 == n_layers;
      a.lnext = last ? nullptr : layer(l + 1);
      const void* k = last ? reinterpret_cast<const void*>(&prk::head_rows<prk::HR_LAST>)
                           : reinterpret_cast<const void*>(&prk::head_rows<prk::HR_MID>);
      st = launch_head(c, k, dim3(ntiles), rblk, prk::HT_SMEM, s, true, a);
      if (st != PR_OK) return st;
    }
  }
  return launch_head(c, reinterpret_cast<const void*>(&prk::head_pool), dim3((unsigned)n_req), blk, 0,
                     s, true, a);
}

}  // extern "C"
