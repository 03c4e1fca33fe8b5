// Host side of the context and diagnostics entry points in
// include/pro_router.h: context creation and workspace, options, the flag
// word, per-kernel timing, decode-slot checkpoints, status strings; and the
// host helpers every translation unit of the library shares.
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>

#include "pr_ctx.h"
#include "pr_device.cuh"

namespace prh {

thread_local char g_cuda_err[256] = "";
std::atomic<uint64_t> g_launches{0};

pr_status cuda_fail(cudaError_t e, const char* what) {
  snprintf(g_cuda_err, sizeof g_cuda_err, "%s: %s", what, cudaGetErrorString(e));
  return PR_ERR_CUDA;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

float zthreshold(float tau) {
  const double t = (double)tau;
  if (!(t > 0.0)) return -INFINITY;
  if (!(t < 1.0)) return INFINITY;
  return (float)std::log(t / (1.0 - t));
}

pr_status set_device(pr_ctx* c) {
  PR_CUDA(cudaSetDevice(c->device));
  return PR_OK;
}

pr_status timing_begin(pr_ctx* c, cudaStream_t s) {
  c->tev_n = 0;
  if (!c->timing) return PR_OK;
  return timing_mark(c, s);
}

pr_status timing_mark(pr_ctx* c, cudaStream_t s) {
  if (!c->timing || c->tev_n > PR_MAX_TIMED) return PR_OK;
  cudaEvent_t& e = c->tev[c->tev_n];
  if (!e) PR_CUDA(cudaEventCreate(&e));
  PR_CUDA(cudaEventRecord(e, s));
  ++c->tev_n;
  return PR_OK;
}

}  // namespace prh

using namespace prh;

namespace {

constexpr uint32_t STATE_MAGIC = 0x50525354u;  // "PRST"
constexpr uint32_t STATE_VERSION = 1u;

}  // namespace

extern "C" {

const char* pr_status_string(pr_status s) {
  switch (s) {
    case PR_OK:
      return "ok";
    case PR_ERR_INVALID_ARG:
      return "invalid argument";
    case PR_ERR_UNSUPPORTED:
      return "unsupported";
    case PR_ERR_CUDA:
      return "CUDA error";
    case PR_ERR_NO_MEMORY:
      return "out of memory";
  }
  return "unknown status";
}

const char* pr_last_cuda_error(void) { return g_cuda_err; }

uint64_t pr_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

pr_status pr_ctx_create(pr_ctx** out, int device, int64_t max_rows, int32_t max_requests) {
  if (!out || max_rows < 0 || max_requests < 0) return PR_ERR_INVALID_ARG;
  *out = nullptr;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev)
    return PR_ERR_INVALID_ARG;
  pr_ctx* c = new (std::nothrow) pr_ctx();
  if (!c) return PR_ERR_NO_MEMORY;
  c->device = device;
  c->max_rows = max_rows;
  c->max_requests = max_requests;
  pr_status st = set_device(c);
  if (st != PR_OK) {
    delete c;
    return st;
  }
  cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, device);
  int major = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, device);
  if (major < 10) {
    delete c;
    return PR_ERR_UNSUPPORTED;
  }
  bool ok = true;
  auto alloc = [&](void** p, size_t bytes) {
    if (!ok) return;
    if (bytes == 0) bytes = 16;
    if (cudaMalloc(p, bytes) != cudaSuccess || cudaMemset(*p, 0, bytes) != cudaSuccess) ok = false;
  };
  alloc(reinterpret_cast<void**>(&c->rec), (size_t)max_rows * prk::NFEAT * sizeof(float));
  alloc(reinterpret_cast<void**>(&c->rec_flags), (size_t)max_rows * sizeof(uint32_t));
  alloc(reinterpret_cast<void**>(&c->req_cnt), (size_t)max_requests * sizeof(int32_t));
  alloc(reinterpret_cast<void**>(&c->acc), (size_t)max_requests * prk::ACC_WORDS * sizeof(float));
  alloc(reinterpret_cast<void**>(&c->flags), sizeof(uint32_t));
  if (!ok || cudaDeviceSynchronize() != cudaSuccess) {
    cudaGetLastError();
    pr_ctx_destroy(c);
    return PR_ERR_NO_MEMORY;
  }
  *out = c;
  return PR_OK;
}

pr_status pr_ctx_destroy(pr_ctx* c) {
  if (!c) return PR_ERR_INVALID_ARG;
  cudaSetDevice(c->device);
  cudaDeviceSynchronize();
  cudaFree(c->rec);
  cudaFree(c->rec_flags);
  cudaFree(c->req_cnt);
  cudaFree(c->acc);
  cudaFree(c->flags);
  for (int i = 0; i < 2; ++i) {
    cudaFree(c->stage[i]);
    cudaFree(c->stage_chosen[i]);
    if (c->ev_copied[i]) cudaEventDestroy(c->ev_copied[i]);
    if (c->ev_free[i]) cudaEventDestroy(c->ev_free[i]);
  }
  cudaFree(c->h_offsets_dev);
  cudaFree(c->h_w_dev);
  cudaFree(c->h_out);
  cudaFree(c->h_ship_dev);
  cudaFree(c->h_flags_dev);
  cudaFree(c->head_scr);
  cudaFree(c->sel_ws);
  cudaFree(c->lm_parts);
  for (cudaEvent_t e : c->tev)
    if (e) cudaEventDestroy(e);
  if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
  delete c;
  return PR_OK;
}

pr_status pr_ctx_reset(pr_ctx* c, void* stream) {
  if (!c) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PR_CUDA(cudaMemsetAsync(c->req_cnt, 0, (size_t)c->max_requests * sizeof(int32_t) + 0, s));
  PR_CUDA(cudaMemsetAsync(c->acc, 0, (size_t)c->max_requests * prk::ACC_WORDS * sizeof(float), s));
  PR_CUDA(cudaMemsetAsync(c->flags, 0, sizeof(uint32_t), s));
  return PR_OK;
}

pr_status pr_ctx_set_option(pr_ctx* c, int32_t option, int32_t value) {
  if (!c) return PR_ERR_INVALID_ARG;
  switch (option) {
    case PR_OPT_TOPK:
      if (value < 1 || value > PR_MAX_TOPK) return PR_ERR_INVALID_ARG;
      c->topk = value;
      return PR_OK;
    case PR_OPT_TOPK_RENORM:
      if (value != 0 && value != 1) return PR_ERR_INVALID_ARG;
      c->renorm = value;
      return PR_OK;
    case PR_OPT_SPLIT:
      if (value != 0 && value != 1 && value != 2 && value != 4 && value != 8)
        return PR_ERR_INVALID_ARG;
      c->split = value;
      return PR_OK;
    case PR_OPT_OVERLAP:
      if (value != 0 && value != 1) return PR_ERR_INVALID_ARG;
      c->overlap = value;
      return PR_OK;
    case PR_OPT_TIMING:
      if (value != 0 && value != 1) return PR_ERR_INVALID_ARG;
      c->timing = value;
      return PR_OK;
  }
  return PR_ERR_INVALID_ARG;
}

pr_status pr_ctx_flags(pr_ctx* c, void* stream, int32_t clear, uint32_t* flags) {
  if (!c || !flags) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint32_t v = 0;
  PR_CUDA(cudaMemcpyAsync(&v, c->flags, sizeof v, cudaMemcpyDeviceToHost, s));
  if (clear) PR_CUDA(cudaMemsetAsync(c->flags, 0, sizeof(uint32_t), s));
  PR_CUDA(cudaStreamSynchronize(s));
  *flags = v;
  return PR_OK;
}

pr_status pr_last_error(pr_ctx* c, uint32_t* flags) {
  if (!c || !flags) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  PR_CUDA(cudaDeviceSynchronize());
  return pr_ctx_flags(c, nullptr, 0, flags);
}

pr_status pr_ctx_kernel_times(pr_ctx* c, float* ms, int32_t cap, int32_t* n) {
  if (!c || !n || cap < 0 || (cap > 0 && !ms)) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  const int32_t k = c->tev_n > 0 ? c->tev_n - 1 : 0;
  *n = k;
  if (k == 0) return PR_OK;
  PR_CUDA(cudaEventSynchronize(c->tev[k]));
  for (int32_t i = 0; i < k && i < cap; ++i) PR_CUDA(cudaEventElapsedTime(&ms[i], c->tev[i], c->tev[i + 1]));
  return PR_OK;
}

pr_status pr_state_export(pr_ctx* c, void* host_buf, size_t* bytes) {
  if (!c || !bytes) return PR_ERR_INVALID_ARG;
  const size_t body = (size_t)c->max_requests * prk::ACC_WORDS * sizeof(float);
  const size_t need = 4 * sizeof(uint32_t) + body;
  if (!host_buf) {
    *bytes = need;
    return PR_OK;
  }
  if (*bytes < need) return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  PR_CUDA(cudaDeviceSynchronize());
  uint32_t hdr[4] = {STATE_MAGIC, STATE_VERSION, (uint32_t)c->max_requests,
                     (uint32_t)prk::ACC_WORDS};
  memcpy(host_buf, hdr, sizeof hdr);
  if (body) PR_CUDA(cudaMemcpy(static_cast<char*>(host_buf) + sizeof hdr, c->acc, body,
                               cudaMemcpyDeviceToHost));
  *bytes = need;
  return PR_OK;
}

pr_status pr_state_import(pr_ctx* c, const void* host_buf, size_t bytes) {
  if (!c || !host_buf) return PR_ERR_INVALID_ARG;
  const size_t body = (size_t)c->max_requests * prk::ACC_WORDS * sizeof(float);
  uint32_t hdr[4];
  if (bytes != sizeof hdr + body) return PR_ERR_INVALID_ARG;
  memcpy(hdr, host_buf, sizeof hdr);
  if (hdr[0] != STATE_MAGIC || hdr[1] != STATE_VERSION || hdr[2] != (uint32_t)c->max_requests ||
      hdr[3] != (uint32_t)prk::ACC_WORDS)
    return PR_ERR_INVALID_ARG;
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  PR_CUDA(cudaDeviceSynchronize());
  if (body) PR_CUDA(cudaMemcpy(c->acc, static_cast<const char*>(host_buf) + sizeof hdr, body,
                               cudaMemcpyHostToDevice));
  return PR_OK;
}

}  // extern "C"
