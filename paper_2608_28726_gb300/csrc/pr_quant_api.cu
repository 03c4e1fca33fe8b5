// Host side of pr_quantile_score: argument checks and the launch of the
// kernel in pr_quant.cuh.
#include <cuda_runtime.h>

#include <cstring>

#include "pr_ctx.h"
#include "pr_quant.cuh"

using namespace prh;

static_assert(prk::QW_SIZE == PR_QMLP_PARAMS, "weight layout");

extern "C" {

pr_status pr_quantile_score(pr_ctx* c, const float* feat, const uint32_t* row_flags,
                            int64_t n_rows, const int64_t* offsets, int32_t n_req, const float* w,
                            float tau, float* summary, float* score, uint8_t* ship,
                            uint32_t* req_flags, void* stream) {
  if (!c || n_req < 0 || n_rows < 0 || n_rows > 0x7fffffffLL) return PR_ERR_INVALID_ARG;
  if (n_req == 0) return PR_OK;
  if (!offsets || !w || !score || !ship || !req_flags) return PR_ERR_INVALID_ARG;
  if (n_rows > 0 && !feat) return PR_ERR_INVALID_ARG;
  if (!aligned16(feat)) return PR_ERR_INVALID_ARG;  // records are read as 16-byte words
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((st = timing_begin(c, s)) != PR_OK) return st;
  prk::QArgs a;
  memset(&a, 0, sizeof a);
  a.feat = feat;
  a.row_flags = row_flags;
  a.n_rows = n_rows;
  a.offsets = offsets;
  a.n_req = n_req;
  a.w = w;
  a.zthr = zthreshold(tau);
  a.summary = summary;
  a.score = score;
  a.ship = ship;
  a.req_flags = req_flags;
  a.ctx_flags = c->flags;
  prk::qmlp_requests<<<(unsigned)n_req, prk::Q_NT, 4 * prk::Q_CAP * sizeof(uint32_t), s>>>(a);
  PR_CUDA(cudaGetLastError());
  g_launches.fetch_add(1, std::memory_order_relaxed);
  return timing_mark(c, s);
}

}  // extern "C"
