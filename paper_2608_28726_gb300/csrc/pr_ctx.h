// Internal to the library: the context structure and the host helpers shared
// by the translation units behind the C ABI.
#pragma once

#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>

#include "pro_router.h"

#define PR_MAX_TIMED 24  // kernels one call can time under PR_OPT_TIMING

struct pr_ctx {
  int device = 0;
  int num_sms = 0;
  int64_t max_rows = 0;
  int32_t max_requests = 0;
  // options
  int32_t topk = 20, renorm = 0, split = 0, overlap = 0;
  // workspace
  float* rec = nullptr;          // [max_rows][8] per-row records of pr_route
  uint32_t* rec_flags = nullptr; // [max_rows]
  int32_t* req_cnt = nullptr;    // [max_requests] completion counters
  float* acc = nullptr;          // [max_requests][ACC_WORDS] decode slots
  uint32_t* flags = nullptr;     // flag word
  // pr_route_host staging (allocated on first use)
  void* stage[2] = {nullptr, nullptr};
  int32_t* stage_chosen[2] = {nullptr, nullptr};
  int64_t stage_rows = 0;
  size_t stage_row_bytes = 0;
  int64_t* h_offsets_dev = nullptr;
  int32_t h_offsets_cap = 0;
  float* h_w_dev = nullptr;
  float* h_out = nullptr;        // [max_requests][NAGG + 1] scores and aggregates
  uint8_t* h_ship_dev = nullptr;
  uint32_t* h_flags_dev = nullptr;
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t ev_copied[2] = {nullptr, nullptr};
  cudaEvent_t ev_free[2] = {nullptr, nullptr};
  // occupancy cache per (dtype, mode)
  int bps[2][3] = {{0, 0, 0}, {0, 0, 0}};
  // persistent kernel: CTAs per SM per (dtype, mode, aligned); 0 = not set up yet
  int ws_bps[2][3][2] = {};
  // scorer head: activation scratch (rows x prk::HSCR floats), grown on demand
  float* head_scr = nullptr;
  int64_t head_scr_rows = 0;
  bool head_ready = false;
  // pr_selective_metrics: sort workspace for up to sel_cap scores, grown on demand
  void* sel_ws = nullptr;
  int64_t sel_cap = 0;
  // its persistent radix scatter: resident CTAs per SM; 0 = not set up yet
  int sel_scatter_bps = 0;
  // pr_lmhead_features: per-(row, split) states, grown on demand
  void* lm_parts = nullptr;
  size_t lm_parts_bytes = 0;
  bool lm_ready = false;
  // PR_OPT_TIMING: events after each kernel of the last multi-kernel call
  int32_t timing = 0;
  cudaEvent_t tev[PR_MAX_TIMED + 1] = {};
  int32_t tev_n = 0;
};

namespace prh {

extern thread_local char g_cuda_err[256];
extern std::atomic<uint64_t> g_launches;

// record the CUDA error text for pr_last_cuda_error and return PR_ERR_CUDA
pr_status cuda_fail(cudaError_t e, const char* what);
bool aligned16(const void* p);
// the ship threshold on z = logit(score): log(tau / (1 - tau)), +-inf outside (0, 1)
float zthreshold(float tau);
pr_status set_device(pr_ctx* c);
// PR_OPT_TIMING: start a timed call / mark the end of one of its kernels
pr_status timing_begin(pr_ctx* c, cudaStream_t s);
pr_status timing_mark(pr_ctx* c, cudaStream_t s);

}  // namespace prh

#define PR_CUDA(call)                                         \
  do {                                                        \
    cudaError_t e_ = (call);                                  \
    if (e_ != cudaSuccess) return prh::cuda_fail(e_, #call); \
  } while (0)
