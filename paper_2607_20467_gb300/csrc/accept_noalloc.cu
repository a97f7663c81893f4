// dcl_accept_noalloc: the block acceptance pass of dcl_accept for callers that cannot
// allocate device memory - e.g. code running inside another framework's memory pool
// or under an allocation-free real-time budget, where cudaMalloc is forbidden or may
// stall.  It needs no dcl_ctx (creating one allocates); its per-position scratch (the
// top-1 id and the top-1 / top-2 probabilities of every position) lives in the
// file-scope device array below instead, which every GPU that loads this library
// holds until the process exits.
#include <mutex>
#include <string>

#include "../../include/dcleap.h"
#include "common.cuh"

namespace {

constexpr int kMaxPositions = DCL_NOALLOC_MAX_POSITIONS;
constexpr int kMaxDevices = 64;

// For n = B*P positions of a call: n int32 top-1 ids, then n float top-1 probabilities,
// then n float top-2 probabilities (12 bytes per position).
static __device__ __align__(256) unsigned char g_accept_scratch[3 * 4 * kMaxPositions];

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once per device
// and kept for the life of the process: a cudaDeviceReset, which unloads this library's
// device code and frees the array, leaves the kept address stale, so the call is not to be
// used after one).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_addr[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_accept_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = ptr;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" dcl_status dcl_accept_noalloc(const void* logits_dev, int32_t B, int32_t P, int32_t V,
                                         const int32_t* committed_dev, int32_t* x_dev,
                                         const dcl_decode_config* cfg, int32_t* k_dev,
                                         void* cuda_stream) {
  if (!logits_dev || !committed_dev || !x_dev || !cfg || !k_dev) {
    dcl::set_thread_error("dcl_accept_noalloc: NULL argument");
    return DCL_ERR_INVALID_ARG;
  }
  if (B <= 0 || P <= 0 || V <= 1 || P > 4096 || (int64_t)B * P > kMaxPositions) {
    dcl::set_thread_error(("dcl_accept_noalloc: need P <= 4096 (as dcl_accept), B*P in [1, " +
                          std::to_string(kMaxPositions) + "] (the size of its static scratch) and V > 1")
                             .c_str());
    return DCL_ERR_INVALID_ARG;
  }
  if (cfg->max_window < 0 || cfg->min_commit < 0 || (cfg->confidence != 0 && cfg->confidence != 1) ||
      (cfg->acceptance != 0 && cfg->acceptance != 1)) {
    dcl::set_thread_error("dcl_accept_noalloc: bad decode config");
    return DCL_ERR_INVALID_ARG;
  }
  void* base = nullptr;
  cudaError_t e = scratch_address(&base);
  if (e != cudaSuccess) {
    dcl::set_thread_error((std::string("dcl_accept_noalloc: cudaGetSymbolAddress failed: ") +
                          cudaGetErrorString(e))
                             .c_str());
    return DCL_ERR_CUDA;
  }
  // Every position the commit pass reads is written by the statistics pass of the same
  // call, so the scratch left by an earlier call needs no clearing.
  const size_t n = (size_t)B * P;
  int32_t* ids = static_cast<int32_t*>(base);
  float* c1 = reinterpret_cast<float*>(ids + n);
  float* c2 = c1 + n;
  const int window = cfg->max_window > 0 ? cfg->max_window : (P / 2 > 0 ? P / 2 : 1);
  dcl::DcvParams prm{cfg->tau_commit, cfg->tau_draft, window, cfg->min_commit, cfg->contiguous_drafts,
                     cfg->acceptance, P};
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  e = dcl::accept_stats_launch(static_cast<const __nv_bfloat16*>(logits_dev), committed_dev, B, P, V, ids, c1,
                               c2, cfg->confidence, s);
  if (e == cudaSuccess) e = dcl::accept_commit_launch(committed_dev, ids, c1, x_dev, k_dev, B, P, prm, s);
  if (e != cudaSuccess) {
    dcl::set_thread_error((std::string("dcl_accept_noalloc: launch failed: ") + cudaGetErrorString(e)).c_str());
    return DCL_ERR_CUDA;
  }
  return DCL_OK;
}
