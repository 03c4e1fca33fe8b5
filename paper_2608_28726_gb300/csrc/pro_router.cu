// Host side of the verifier's entry points in include/pro_router.h: argument
// checks, launch configuration of the row kernels, the host-memory pipeline
// and the allocation-free call.
#include <cuda_runtime.h>

#include <atomic>
#include <mutex>
#include <cmath>
#include <cstdio>
#include <algorithm>
#include <cstring>
#include <new>

#include "pr_ctx.h"
#include "pr_kernels.cuh"

using namespace prh;

namespace {

template <typename T, int MODE>
void* kernel_ptr(bool aligned) {
  return aligned ? reinterpret_cast<void*>(&prk::verify_rows<T, MODE, true>)
                 : reinterpret_cast<void*>(&prk::verify_rows<T, MODE, false>);
}

void* row_kernel(pr_dtype dt, int mode, bool aligned) {
  if (dt == PR_DTYPE_BF16) {
    if (mode == prk::MODE_FEATURES) return kernel_ptr<__nv_bfloat16, prk::MODE_FEATURES>(aligned);
    if (mode == prk::MODE_ROUTE) return kernel_ptr<__nv_bfloat16, prk::MODE_ROUTE>(aligned);
    return kernel_ptr<__nv_bfloat16, prk::MODE_DECODE>(aligned);
  }
  if (mode == prk::MODE_FEATURES) return kernel_ptr<float, prk::MODE_FEATURES>(aligned);
  if (mode == prk::MODE_ROUTE) return kernel_ptr<float, prk::MODE_ROUTE>(aligned);
  return kernel_ptr<float, prk::MODE_DECODE>(aligned);
}

int blocks_per_sm(pr_ctx* c, pr_dtype dt, int mode) {
  int& v = c->bps[dt == PR_DTYPE_BF16 ? 1 : 0][mode];
  if (v == 0) {
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, row_kernel(dt, mode, true), prk::NT, 0) !=
            cudaSuccess ||
        n <= 0)
      n = 1;
    v = n;
  }
  return v;
}

template <typename T, int MODE>
void* ws_kernel_ptr(bool aligned) {
  return aligned ? reinterpret_cast<void*>(&prk::verify_rows_ws<T, MODE, true>)
                 : reinterpret_cast<void*>(&prk::verify_rows_ws<T, MODE, false>);
}

void* ws_kernel(pr_dtype dt, int mode, bool aligned) {
  if (dt == PR_DTYPE_BF16) {
    if (mode == prk::MODE_FEATURES) return ws_kernel_ptr<__nv_bfloat16, prk::MODE_FEATURES>(aligned);
    if (mode == prk::MODE_ROUTE) return ws_kernel_ptr<__nv_bfloat16, prk::MODE_ROUTE>(aligned);
    return ws_kernel_ptr<__nv_bfloat16, prk::MODE_DECODE>(aligned);
  }
  if (mode == prk::MODE_FEATURES) return ws_kernel_ptr<float, prk::MODE_FEATURES>(aligned);
  if (mode == prk::MODE_ROUTE) return ws_kernel_ptr<float, prk::MODE_ROUTE>(aligned);
  return ws_kernel_ptr<float, prk::MODE_DECODE>(aligned);
}

// shared memory opt-in and residency of the persistent kernel, once per instantiation
pr_status ws_setup(pr_ctx* c, pr_dtype dt, int mode, bool aligned, int* bps) {
  int& v = c->ws_bps[dt == PR_DTYPE_BF16 ? 1 : 0][mode][aligned ? 1 : 0];
  if (v == 0) {
    void* f = ws_kernel(dt, mode, aligned);
    PR_CUDA(cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)sizeof(prk::SmemWS)));
    int n = 0;
    PR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, f, prk::NT_WS, sizeof(prk::SmemWS)));
    v = n > 0 ? n : 1;
  }
  *bps = v;
  return PR_OK;
}

// Launch shape of a batch: CTAs per row (C) and whether the persistent
// kernel runs it.
//  * the forced option: split 1 is the persistent kernel, 2 / 4 / 8 clusters;
//  * a batch with at least one row per SM that fits one wave of resident
//    CTAs: one CTA per row, without a cluster.  Such a launch leaves room for
//    the next one, so back-to-back calls overlap one launch's per-row
//    selection with the next one's stream (measured in CUDA graphs: 256 x
//    151,936 bf16 decode steps 12.8 us per step against 15.6 us with two-CTA
//    clusters, which fill 84% of the slots; 354 x 32,000 fp32 batches 12.0 us
//    against 13.9 us with the persistent kernel);
//  * fewer rows: the largest split (<= 8) whose CTAs still fit in one wave;
//  * more rows: the persistent kernel.
// The persistent kernel keeps a thread's best tile indices in 16 bits, so rows
// of more than 2^16 tiles (over 536 M bf16 or 268 M fp32 values) take one CTA
// per row instead, the forced split 1 included.
struct LaunchShape {
  int C;
  bool persistent;
};

LaunchShape choose_launch(pr_ctx* c, pr_dtype dt, int mode, int64_t n_rows, int64_t vocab) {
  const int64_t groups = vocab / (dt == PR_DTYPE_BF16 ? 8 : 4);
  const bool ws_fits = (groups + prk::TILE - 1) / prk::TILE <= 65536;
  if (c->split == 1) return {1, ws_fits};
  if (c->split == 2 || c->split == 4 || c->split == 8) return {c->split, false};
  const int64_t slots = (int64_t)c->num_sms * blocks_per_sm(c, dt, mode);
  if (n_rows >= c->num_sms && n_rows <= slots) return {1, false};
  int s = 1;
  while (s < prk::MAXC && n_rows * (s * 2) <= slots) s <<= 1;
  return {s, s == 1 && ws_fits};
}

pr_status launch_rows(pr_ctx* c, pr_dtype dt, int mode, const prk::Args& a, cudaStream_t st) {
  if (a.n_rows == 0) return PR_OK;
  const LaunchShape shape = choose_launch(c, dt, mode, a.n_rows, a.vocab);
  const int C = shape.C;
  if (shape.persistent) {
    // persistent warp-specialised kernel: every SM gets its resident CTAs
    int bps = 0;
    const pr_status s = ws_setup(c, dt, mode, a.aligned != 0, &bps);
    if (s != PR_OK) return s;
    const int64_t grid = std::min<int64_t>(a.n_rows, (int64_t)c->num_sms * bps);
    cudaLaunchConfig_t cfg;
    memset(&cfg, 0, sizeof cfg);
    cfg.gridDim = dim3((unsigned)grid, 1, 1);
    cfg.blockDim = dim3(prk::NT_WS, 1, 1);
    cfg.dynamicSmemBytes = sizeof(prk::SmemWS);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = c->overlap ? 1 : 0;
    void* args[] = {const_cast<prk::Args*>(&a)};
    PR_CUDA(cudaLaunchKernelExC(&cfg, ws_kernel(dt, mode, a.aligned != 0), args));
    g_launches.fetch_add(1, std::memory_order_relaxed);
    return PR_OK;
  }
  if (a.n_rows * C > 0x7fffffffLL) return PR_ERR_INVALID_ARG;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)(a.n_rows * C), 1, 1);
  cfg.blockDim = dim3(prk::NT, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (C > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = (unsigned)C;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  if (c->overlap) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  void* args[] = {const_cast<prk::Args*>(&a)};
  PR_CUDA(cudaLaunchKernelExC(&cfg, row_kernel(dt, mode, a.aligned != 0), args));
  g_launches.fetch_add(1, std::memory_order_relaxed);
  return PR_OK;
}


size_t esize(pr_dtype dt) { return dt == PR_DTYPE_BF16 ? 2 : 4; }

bool valid_dtype(pr_dtype dt) { return dt == PR_DTYPE_F32 || dt == PR_DTYPE_BF16; }

// the part of the row checks shared by every entry point
pr_status check_rows(pr_dtype dt, const void* logits, int64_t n_rows, int64_t vocab,
                     int64_t row_stride) {
  if (!valid_dtype(dt)) return PR_ERR_INVALID_ARG;
  if (n_rows < 0 || vocab <= 0 || vocab > 0x7fffffffLL || row_stride < vocab)
    return PR_ERR_INVALID_ARG;
  if (n_rows > 0 && !logits) return PR_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(logits) % esize(dt)) != 0) return PR_ERR_INVALID_ARG;
  return PR_OK;
}

void fill_row_args(prk::Args& a, const void* logits, pr_dtype dt, int64_t n_rows, int64_t vocab,
                   int64_t row_stride, const int32_t* chosen, int32_t topk, int32_t renorm) {
  memset(&a, 0, sizeof a);
  a.logits = logits;
  a.n_rows = n_rows;
  a.vocab = vocab;
  a.row_stride = row_stride;
  a.chosen = chosen;
  a.topk = topk;
  a.kc = topk > 2 ? topk : 2;
  a.renorm = renorm;
  a.aligned = aligned16(logits) && ((row_stride * (int64_t)esize(dt)) % 16) == 0;
}


}  // namespace

extern "C" {

pr_status pr_token_features(pr_ctx* c, const void* logits, pr_dtype dt, int64_t n_rows,
                            int64_t vocab, int64_t row_stride, const int32_t* chosen,
                            int32_t topk, const int64_t* offsets, int32_t n_req, float* feat,
                            int32_t* top2, uint32_t* row_flags, void* stream) {
  if (!c) return PR_ERR_INVALID_ARG;
  pr_status st = check_rows(dt, logits, n_rows, vocab, row_stride);
  if (st != PR_OK) return st;
  if (topk < 1 || topk > PR_MAX_TOPK || n_req < 0) return PR_ERR_INVALID_ARG;
  if (n_rows > 0 && (!chosen || !feat || !top2 || !row_flags)) return PR_ERR_INVALID_ARG;
  if (offsets && n_req < 1) return PR_ERR_INVALID_ARG;
  if ((st = set_device(c)) != PR_OK) return st;
  prk::Args a;
  fill_row_args(a, logits, dt, n_rows, vocab, row_stride, chosen, topk, c->renorm);
  a.offsets = offsets;
  a.n_req = offsets ? n_req : 0;
  a.feat = feat;
  a.top2 = top2;
  a.row_flags = row_flags;
  a.ctx_flags = c->flags;
  return launch_rows(c, dt, prk::MODE_FEATURES, a, reinterpret_cast<cudaStream_t>(stream));
}

pr_status pr_aggregate_score(pr_ctx* c, const float* feat, const uint32_t* row_flags,
                             int64_t n_rows, const int64_t* offsets, int32_t n_req,
                             const float* w, float b, float tau, float* agg, float* score,
                             uint8_t* ship, uint32_t* req_flags, void* stream) {
  if (!c || n_req < 0 || n_rows < 0) return PR_ERR_INVALID_ARG;
  if (n_req == 0) return PR_OK;
  if (!offsets || !w || !score || !ship || !req_flags) return PR_ERR_INVALID_ARG;
  if (n_rows > 0 && !feat) return PR_ERR_INVALID_ARG;
  if (!aligned16(feat)) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  prk::AggArgs a;
  memset(&a, 0, sizeof a);
  a.feat = feat;
  a.row_flags = row_flags;
  a.n_rows = n_rows;
  a.offsets = offsets;
  a.n_req = n_req;
  a.w = w;
  a.b = b;
  a.zthr = zthreshold(tau);
  a.agg = agg;
  a.score = score;
  a.ship = ship;
  a.req_flags = req_flags;
  a.ctx_flags = c->flags;
  const unsigned grid = (unsigned)((n_req + prk::NWARP - 1) / prk::NWARP);
  prk::pool_requests<<<grid, prk::NT, 0, reinterpret_cast<cudaStream_t>(stream)>>>(a);
  PR_CUDA(cudaGetLastError());
  g_launches.fetch_add(1, std::memory_order_relaxed);
  return PR_OK;
}

pr_status pr_route(pr_ctx* c, const void* logits, pr_dtype dt, int64_t row_base,
                   int64_t n_rows, int64_t vocab, int64_t row_stride, const int32_t* chosen,
                   const int64_t* offsets, int32_t n_req, const float* w, float b, float tau,
                   float* score, uint8_t* ship, uint32_t* req_flags, float* agg, void* stream) {
  if (!c) return PR_ERR_INVALID_ARG;
  pr_status st = check_rows(dt, logits, n_rows, vocab, row_stride);
  if (st != PR_OK) return st;
  if (n_req < 1 || n_req > c->max_requests || row_base < 0 || row_base + n_rows > c->max_rows)
    return PR_ERR_INVALID_ARG;
  if (!offsets || !w || !score || !ship || !req_flags || (n_rows > 0 && !chosen))
    return PR_ERR_INVALID_ARG;
  if ((st = set_device(c)) != PR_OK) return st;
  prk::Args a;
  fill_row_args(a, logits, dt, n_rows, vocab, row_stride, chosen, c->topk, c->renorm);
  a.offsets = offsets;
  a.n_req = n_req;
  a.row_base = row_base;
  a.rec = c->rec;
  a.rec_flags = c->rec_flags;
  a.req_cnt = c->req_cnt;
  a.max_rows = c->max_rows;
  a.w = w;
  a.b = b;
  a.zthr = zthreshold(tau);
  a.score = score;
  a.ship = ship;
  a.req_flags = req_flags;
  a.agg = agg;
  a.ctx_flags = c->flags;
  return launch_rows(c, dt, prk::MODE_ROUTE, a, reinterpret_cast<cudaStream_t>(stream));
}

pr_status pr_decode_step(pr_ctx* c, const void* logits, pr_dtype dt, int32_t n_live,
                         int64_t vocab, int64_t row_stride, const int32_t* slot,
                         const int32_t* chosen, const uint8_t* eos, const float* w, float b,
                         float tau, float* score_out, uint8_t* ship_out, uint32_t* slot_flags,
                         float* agg_out, void* stream) {
  if (!c) return PR_ERR_INVALID_ARG;
  pr_status st = check_rows(dt, logits, n_live, vocab, row_stride);
  if (st != PR_OK) return st;
  if (n_live > c->max_requests) return PR_ERR_INVALID_ARG;
  if (n_live > 0 && (!slot || !chosen || !eos || !w || !score_out || !ship_out || !slot_flags))
    return PR_ERR_INVALID_ARG;
  if ((st = set_device(c)) != PR_OK) return st;
  prk::Args a;
  fill_row_args(a, logits, dt, n_live, vocab, row_stride, chosen, c->topk, c->renorm);
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
  return launch_rows(c, dt, prk::MODE_DECODE, a, reinterpret_cast<cudaStream_t>(stream));
}

pr_status pr_route_host(pr_ctx* c, const void* logits, pr_dtype dt, int64_t n_rows,
                        int64_t vocab, int64_t row_stride, const int32_t* chosen,
                        const int64_t* offsets, int32_t n_req, const float* w, float b, float tau,
                        int64_t chunk_rows, float* score, uint8_t* ship, uint32_t* req_flags,
                        float* agg, void* stream) {
  if (!c) return PR_ERR_INVALID_ARG;
  pr_status st = check_rows(dt, logits, n_rows, vocab, row_stride);
  if (st != PR_OK) return st;
  if (n_req < 1 || n_req > c->max_requests || n_rows > c->max_rows || chunk_rows < 1)
    return PR_ERR_INVALID_ARG;
  if (!offsets || !w || !score || !ship || !req_flags || (n_rows > 0 && !chosen))
    return PR_ERR_INVALID_ARG;
  if ((st = set_device(c)) != PR_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const size_t row_bytes = (size_t)row_stride * esize(dt);
  // a chunk never holds more than the batch: the staging buffers are sized
  // from it (and chunk_rows * row_bytes then stays within the host buffer)
  chunk_rows = std::min<int64_t>(chunk_rows, std::max<int64_t>(n_rows, 1));

  // staging: two chunks of rows, token ids, the offsets, weights and outputs
  if (c->stage_rows < chunk_rows || c->stage_row_bytes != row_bytes) {
    for (int i = 0; i < 2; ++i) {
      cudaFree(c->stage[i]);
      cudaFree(c->stage_chosen[i]);
      c->stage[i] = nullptr;
      c->stage_chosen[i] = nullptr;
    }
    c->stage_rows = 0;
    for (int i = 0; i < 2; ++i) {
      if (cudaMalloc(&c->stage[i], (size_t)chunk_rows * row_bytes) != cudaSuccess ||
          cudaMalloc(reinterpret_cast<void**>(&c->stage_chosen[i]),
                     (size_t)chunk_rows * sizeof(int32_t)) != cudaSuccess) {
        cudaGetLastError();
        return PR_ERR_NO_MEMORY;
      }
    }
    c->stage_rows = chunk_rows;
    c->stage_row_bytes = row_bytes;
  }
  if (!c->copy_stream) {
    PR_CUDA(cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking));
    for (int i = 0; i < 2; ++i) {
      PR_CUDA(cudaEventCreateWithFlags(&c->ev_copied[i], cudaEventDisableTiming));
      PR_CUDA(cudaEventCreateWithFlags(&c->ev_free[i], cudaEventDisableTiming));
    }
  }
  if (c->h_offsets_cap < n_req + 1) {
    cudaFree(c->h_offsets_dev);
    c->h_offsets_dev = nullptr;
    c->h_offsets_cap = 0;
    if (cudaMalloc(reinterpret_cast<void**>(&c->h_offsets_dev), (size_t)(n_req + 1) * sizeof(int64_t)) !=
        cudaSuccess) {
      cudaGetLastError();
      return PR_ERR_NO_MEMORY;
    }
    c->h_offsets_cap = n_req + 1;
  }
  if (!c->h_w_dev) {
    bool ok = cudaMalloc(reinterpret_cast<void**>(&c->h_w_dev), prk::NAGG * sizeof(float)) == cudaSuccess &&
              cudaMalloc(reinterpret_cast<void**>(&c->h_out),
                         (size_t)(c->max_requests > 0 ? c->max_requests : 1) * (prk::NAGG + 1) *
                             sizeof(float)) == cudaSuccess &&
              cudaMalloc(reinterpret_cast<void**>(&c->h_ship_dev), (size_t)(c->max_requests + 1)) ==
                  cudaSuccess &&
              cudaMalloc(reinterpret_cast<void**>(&c->h_flags_dev),
                         (size_t)(c->max_requests + 1) * sizeof(uint32_t)) == cudaSuccess;
    if (!ok) {
      cudaGetLastError();
      return PR_ERR_NO_MEMORY;
    }
  }
  float* d_score = c->h_out;
  float* d_agg = c->h_out + c->max_requests;
  PR_CUDA(cudaMemcpyAsync(c->h_offsets_dev, offsets, (size_t)(n_req + 1) * sizeof(int64_t),
                          cudaMemcpyHostToDevice, s));
  PR_CUDA(cudaMemcpyAsync(c->h_w_dev, w, prk::NAGG * sizeof(float), cudaMemcpyHostToDevice, s));

  // chunk i: copy on copy_stream into buffer i % 2, route on s
  const int64_t nchunks = (n_rows + chunk_rows - 1) / chunk_rows;
  PR_CUDA(cudaEventRecord(c->ev_free[0], s));
  PR_CUDA(cudaEventRecord(c->ev_free[1], s));
  for (int64_t i = 0; i < nchunks; ++i) {
    const int j = (int)(i & 1);
    const int64_t r0 = i * chunk_rows;
    const int64_t nr = (r0 + chunk_rows <= n_rows) ? chunk_rows : n_rows - r0;
    PR_CUDA(cudaStreamWaitEvent(c->copy_stream, c->ev_free[j], 0));
    PR_CUDA(cudaMemcpyAsync(c->stage[j], static_cast<const char*>(logits) + (size_t)r0 * row_bytes,
                            (size_t)nr * row_bytes, cudaMemcpyHostToDevice, c->copy_stream));
    PR_CUDA(cudaMemcpyAsync(c->stage_chosen[j], chosen + r0, (size_t)nr * sizeof(int32_t),
                            cudaMemcpyHostToDevice, c->copy_stream));
    PR_CUDA(cudaEventRecord(c->ev_copied[j], c->copy_stream));
    PR_CUDA(cudaStreamWaitEvent(s, c->ev_copied[j], 0));
    st = pr_route(c, c->stage[j], dt, r0, nr, vocab, row_stride, c->stage_chosen[j],
                  c->h_offsets_dev, n_req, c->h_w_dev, b, tau, d_score, c->h_ship_dev,
                  c->h_flags_dev, agg ? d_agg : nullptr, stream);
    if (st != PR_OK) return st;
    PR_CUDA(cudaEventRecord(c->ev_free[j], s));
  }
  PR_CUDA(cudaMemcpyAsync(score, d_score, (size_t)n_req * sizeof(float), cudaMemcpyDeviceToHost, s));
  PR_CUDA(cudaMemcpyAsync(ship, c->h_ship_dev, (size_t)n_req, cudaMemcpyDeviceToHost, s));
  PR_CUDA(cudaMemcpyAsync(req_flags, c->h_flags_dev, (size_t)n_req * sizeof(uint32_t),
                          cudaMemcpyDeviceToHost, s));
  if (agg)
    PR_CUDA(cudaMemcpyAsync(agg, d_agg, (size_t)n_req * prk::NAGG * sizeof(float),
                            cudaMemcpyDeviceToHost, s));
  PR_CUDA(cudaStreamSynchronize(s));
  return PR_OK;
}

}  // extern "C"

// ---- verification without any allocation ---------------------------------------------
//
// Scratch of pr_route_noalloc: per-row records, per-request completion counters
// and a flag word, in one file-scope device array.  Every device that loads
// this library holds it (about 580 KB) until the process exits.

namespace {

constexpr size_t NA_REC_BYTES = (size_t)PR_NOALLOC_MAX_ROWS * prk::NFEAT * sizeof(float);
constexpr size_t NA_RFL_BYTES = (size_t)PR_NOALLOC_MAX_ROWS * sizeof(uint32_t);
constexpr size_t NA_CNT_BYTES = (size_t)PR_NOALLOC_MAX_REQUESTS * sizeof(int32_t);
constexpr size_t NA_OFF_RFL = NA_REC_BYTES;
constexpr size_t NA_OFF_CNT = NA_OFF_RFL + NA_RFL_BYTES;
constexpr size_t NA_OFF_FLAGS = NA_OFF_CNT + NA_CNT_BYTES;
constexpr size_t NA_BYTES = NA_OFF_FLAGS + 256;

static __device__ __align__(256) unsigned char g_noalloc_scratch[NA_BYTES];

constexpr int NA_MAX_DEVICES = 64;

struct NoAllocDevice {
  bool ready = false;
  unsigned char* scratch = nullptr;  // device address of g_noalloc_scratch on this device
  int num_sms = 0;
  int bps[2] = {0, 0};               // CTAs per SM of the route kernel, fp32 / bf16
};

std::mutex g_noalloc_mu;
NoAllocDevice g_noalloc_dev[NA_MAX_DEVICES];

// Once per device, with that device current: the scratch's device address
// (host code may not use the symbol itself) and the launch shape.
pr_status noalloc_setup(int dev, NoAllocDevice** out) {
  if (dev < 0 || dev >= NA_MAX_DEVICES) return PR_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  NoAllocDevice& d = g_noalloc_dev[dev];
  if (!d.ready) {
    void* p = nullptr;
    PR_CUDA(cudaGetSymbolAddress(&p, g_noalloc_scratch));
    PR_CUDA(cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev));
    for (int i = 0; i < 2; ++i) {
      const pr_dtype dt = i ? PR_DTYPE_BF16 : PR_DTYPE_F32;
      int n = 0;
      PR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(
          &n, row_kernel(dt, prk::MODE_ROUTE, true), prk::NT, 0));
      d.bps[i] = n > 0 ? n : 1;
    }
    d.scratch = static_cast<unsigned char*>(p);
    d.ready = true;
  }
  *out = &d;
  return PR_OK;
}

}  // namespace

extern "C" {

pr_status pr_route_noalloc(const void* logits, pr_dtype dt, int64_t n_rows, int64_t vocab,
                           int64_t row_stride, const int32_t* chosen, const int64_t* offsets,
                           int32_t n_req, const float* w, float b, float tau, float* score,
                           uint8_t* ship, uint32_t* req_flags, float* agg, void* stream) {
  pr_status st = check_rows(dt, logits, n_rows, vocab, row_stride);
  if (st != PR_OK) return st;
  if (n_rows > PR_NOALLOC_MAX_ROWS || n_req > PR_NOALLOC_MAX_REQUESTS) return PR_ERR_INVALID_ARG;
  if (n_rows < 1 || n_req < 1 || !offsets || !w || !score || !ship || !req_flags || !chosen)
    return PR_ERR_INVALID_ARG;
  int dev = 0;
  PR_CUDA(cudaGetDevice(&dev));
  NoAllocDevice* d = nullptr;
  if ((st = noalloc_setup(dev, &d)) != PR_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

  // the counters and the flag word start every call at zero
  PR_CUDA(cudaMemsetAsync(d->scratch + NA_OFF_CNT, 0, (size_t)n_req * sizeof(int32_t), s));
  PR_CUDA(cudaMemsetAsync(d->scratch + NA_OFF_FLAGS, 0, sizeof(uint32_t), s));

  prk::Args a;
  fill_row_args(a, logits, dt, n_rows, vocab, row_stride, chosen, 20, 0);
  a.offsets = offsets;
  a.n_req = n_req;
  a.row_base = 0;
  a.rec = reinterpret_cast<float*>(d->scratch);
  a.rec_flags = reinterpret_cast<uint32_t*>(d->scratch + NA_OFF_RFL);
  a.req_cnt = reinterpret_cast<int32_t*>(d->scratch + NA_OFF_CNT);
  a.max_rows = n_rows;
  a.w = w;
  a.b = b;
  a.zthr = zthreshold(tau);
  a.score = score;
  a.ship = ship;
  a.req_flags = req_flags;
  a.agg = agg;
  a.ctx_flags = reinterpret_cast<uint32_t*>(d->scratch + NA_OFF_FLAGS);
  a.whole = 1;  // no flag word the caller can read: report short offsets in the last request

  // CTAs per row (the cluster kernel only; no persistent-kernel set-up here):
  // double C, up to MAXC, while the batch's CTAs stay under two waves of
  // resident CTAs
  const int64_t slots = (int64_t)d->num_sms * d->bps[dt == PR_DTYPE_BF16 ? 1 : 0];
  int C = 1;
  while (C < prk::MAXC && n_rows * C < 2 * slots) C <<= 1;
  if (n_rows * C > 0x7fffffffLL) return PR_ERR_INVALID_ARG;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)(n_rows * C), 1, 1);
  cfg.blockDim = dim3(prk::NT, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = C > 1 ? 1 : 0;
  void* args[] = {&a};
  PR_CUDA(cudaLaunchKernelExC(&cfg, row_kernel(dt, prk::MODE_ROUTE, a.aligned != 0), args));
  g_launches.fetch_add(1, std::memory_order_relaxed);
  return PR_OK;
}

}  // extern "C"
