// Host side of pr_selective_metrics: argument checks, the context's sort
// workspace and the launch sequence of the kernels in pr_select.cuh.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstddef>
#include <cstring>

#include "pr_ctx.h"
#include "pr_select.cuh"

using namespace prh;

static_assert(sizeof(prk::SelResult) == sizeof(pr_selective), "result layout");
static_assert(offsetof(prk::SelResult, n_finite) == offsetof(pr_selective, n_finite), "layout");
static_assert(offsetof(prk::SelResult, auroc) == offsetof(pr_selective, auroc), "layout");
static_assert(offsetof(prk::SelResult, acc_shipped) == offsetof(pr_selective, acc_shipped),
              "layout");

namespace {

size_t align256(size_t b) { return (b + 255) & ~(size_t)255; }

// byte offsets of the workspace pieces for capacity n
struct SelLayout {
  size_t key0, key1, val0, val1, pre, counts, total, tsum, toff, proc, parc, nf, out, bytes;
  explicit SelLayout(int64_t n) {
    const int64_t nt = (n + prk::SEL_TILE - 1) / prk::SEL_TILE;
    size_t o = 0;
    auto take = [&](size_t b) {
      const size_t at = o;
      o += align256(b);
      return at;
    };
    key0 = take((size_t)n * 4);
    key1 = take((size_t)n * 4);
    val0 = take((size_t)n);
    val1 = take((size_t)n);
    pre = take((size_t)n * 4);
    counts = take((size_t)nt * prk::SEL_RADIX * 4);
    total = take(prk::SEL_RADIX * 4);
    tsum = take((size_t)nt * 4);
    toff = take(((size_t)nt + 1) * 4);
    proc = take((size_t)nt * 8);
    parc = take((size_t)nt * 8);
    nf = take(8);
    out = take(sizeof(prk::SelResult));
    bytes = o;
  }
};

}  // namespace

extern "C" {

pr_status pr_selective_metrics(pr_ctx* c, const float* scores, const uint8_t* labels, int64_t n,
                               double q, pr_selective* out, void* stream) {
  if (!c || !out || n < 0 || n > 0x7fffffffLL) return PR_ERR_INVALID_ARG;
  if (!(q >= 0.0 && q <= 1.0)) return PR_ERR_INVALID_ARG;
  if (n > 0 && !scores) return PR_ERR_INVALID_ARG;
  const double nan = __builtin_nan("");
  if (n == 0) {
    memset(out, 0, sizeof *out);
    out->tau = __builtin_inff();
    out->auroc = out->auarc = out->acc_shipped = nan;
    return PR_OK;
  }
  pr_status st = set_device(c);
  if (st != PR_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (n > c->sel_cap) {
    PR_CUDA(cudaDeviceSynchronize());  // the old workspace may still be in use
    cudaFree(c->sel_ws);
    c->sel_ws = nullptr;
    c->sel_cap = 0;
    const SelLayout L(n);
    if (cudaMalloc(&c->sel_ws, L.bytes) != cudaSuccess) {
      cudaGetLastError();
      c->sel_ws = nullptr;
      return PR_ERR_NO_MEMORY;
    }
    c->sel_cap = n;
  }
  const SelLayout L(c->sel_cap);
  char* w = static_cast<char*>(c->sel_ws);
  uint32_t* key[2] = {reinterpret_cast<uint32_t*>(w + L.key0), reinterpret_cast<uint32_t*>(w + L.key1)};
  uint8_t* val[2] = {reinterpret_cast<uint8_t*>(w + L.val0), reinterpret_cast<uint8_t*>(w + L.val1)};
  uint32_t* pre = reinterpret_cast<uint32_t*>(w + L.pre);
  uint32_t* counts = reinterpret_cast<uint32_t*>(w + L.counts);
  uint32_t* total = reinterpret_cast<uint32_t*>(w + L.total);
  uint32_t* tsum = reinterpret_cast<uint32_t*>(w + L.tsum);
  uint32_t* toff = reinterpret_cast<uint32_t*>(w + L.toff);
  unsigned long long* proc = reinterpret_cast<unsigned long long*>(w + L.proc);
  double* parc = reinterpret_cast<double*>(w + L.parc);
  unsigned long long* nf = reinterpret_cast<unsigned long long*>(w + L.nf);
  prk::SelResult* res = reinterpret_cast<prk::SelResult*>(w + L.out);
  const int64_t ntiles = (n + prk::SEL_TILE - 1) / prk::SEL_TILE;
  const unsigned g_tiles = (unsigned)ntiles;
  // the scatter is persistent: one wave of resident CTAs
  if (c->sel_scatter_bps == 0) {
    int b = 0;
    PR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, prk::sel_scatter, prk::SEL_NT, 0));
    c->sel_scatter_bps = b > 0 ? b : 1;
  }
  const int64_t rtiles = (n + prk::SR_TILE - 1) / prk::SR_TILE;  // tiles of the radix passes
  const unsigned g_scatter =
      (unsigned)std::min<int64_t>(rtiles, (int64_t)c->num_sms * c->sel_scatter_bps);
  int launches = 0;
  // after each launch: count it, check it, and (PR_OPT_TIMING) record an event
  auto launched = [&]() -> pr_status {
    ++launches;
    PR_CUDA(cudaGetLastError());
    return timing_mark(c, s);
  };
#define PR_LAUNCHED()                        \
  do {                                       \
    if ((st = launched()) != PR_OK) return st; \
  } while (0)

  PR_CUDA(cudaMemsetAsync(nf, 0, sizeof *nf, s));
  if ((st = timing_begin(c, s)) != PR_OK) return st;
  prk::sel_init<<<g_tiles, prk::SEL_NT, 0, s>>>(scores, labels, n, key[0], val[0], nf);
  PR_LAUNCHED();
  for (int pass = 0; pass < 4; ++pass) {
    const int cur = pass & 1, nxt = cur ^ 1;
    prk::sel_hist<<<(unsigned)rtiles, prk::SEL_NT, 0, s>>>(key[cur], n, 8 * pass, counts, rtiles);
    PR_LAUNCHED();
    prk::sel_scan_digit<<<prk::SEL_RADIX, prk::SEL_NT, 0, s>>>(counts, rtiles, total);
    PR_LAUNCHED();
    prk::sel_scatter<<<g_scatter, prk::SEL_NT, 0, s>>>(key[cur], val[cur], n, 8 * pass, counts,
                                                       rtiles, total, key[nxt], val[nxt]);
    PR_LAUNCHED();
  }
  // four passes: the sorted arrays are back in key[0], val[0]
  prk::sel_label_prefix<<<g_tiles, prk::SEL_NT, 0, s>>>(val[0], nf, pre, tsum);
  PR_LAUNCHED();
  prk::sel_scan_tiles<<<1, 1024, 0, s>>>(tsum, ntiles, toff);
  PR_LAUNCHED();
  if (labels) {
    prk::sel_metrics<<<g_tiles, prk::SEL_NT, 0, s>>>(key[0], val[0], pre, toff, nf, ntiles, proc,
                                                    parc);
    PR_LAUNCHED();
  }
  prk::sel_finish<<<1, prk::SEL_NT, 0, s>>>(key[0], pre, toff, nf, n, ntiles, q, labels ? 1 : 0,
                                            proc, parc, res);
  PR_LAUNCHED();
#undef PR_LAUNCHED
  g_launches.fetch_add((uint64_t)launches, std::memory_order_relaxed);
  PR_CUDA(cudaMemcpyAsync(out, res, sizeof *out, cudaMemcpyDeviceToHost, s));
  PR_CUDA(cudaStreamSynchronize(s));
  return PR_OK;
}

}  // extern "C"
