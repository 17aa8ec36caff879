// ps_lmhead_ppo_fwd_noalloc: the fused forward with its scratch in a static device array.
//
// Some callers cannot allocate device memory for a workspace: a plugin hosted by a
// framework that owns the GPU's memory (its pool is reserved up front and plugins may not
// call cudaMalloc), or a deployment whose device memory plan is fixed at start-up. For
// them this entry point runs exactly the work of ps_lmhead_ppo_fwd with the workspace
// taken from a file-scope __device__ array of kStaticScratchBytes, which every GPU that
// loads the library holds until the process exits. The function allocates nothing: no
// cudaMalloc, no cudaFree, no allocating library routine.
#include <cuda_runtime.h>

#include <mutex>

#include "psppo.h"

namespace {

constexpr size_t kStaticScratchBytes = 64ull << 20;  // 64 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_fwd_scratch[kStaticScratchBytes];

std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of this device's copy of g_fwd_scratch. In host code the symbol is only a
// host-side stand-in, so the address must come from cudaGetSymbolAddress, once per device,
// with that device current.
int scratch_for_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return PS_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_fwd_scratch) != cudaSuccess || p == nullptr) return PS_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return PS_OK;
}

}  // namespace

extern "C" int ps_lmhead_ppo_fwd_noalloc(int64_t N, int d, int V, int dtype, const void* Hpk, const void* W,
                                         const int32_t* tok, const float* oldlogp, const float* adv,
                                         const float* w, double eps, double loss_scale, double* loss, float* lse,
                                         float* logp, float* ratio, float* coef, float* row_loss,
                                         ps_stream_t stream) {
  if (ps_lmhead_ppo_fwd_workspace_size(N, d, V, dtype) == 0) return PS_ERR_INVALID_ARG;
  void* scratch = nullptr;
  const int rc = scratch_for_current_device(&scratch);
  if (rc != PS_OK) return rc;
  // The forward takes as many vocabulary partials as the 64 MiB hold; when not even one per row
  // fits it refuses the workspace before launching anything: the problem is too large for the
  // static scratch. The status word at the head of the scratch is cleared by the call itself.
  const int r = ps_lmhead_ppo_fwd(N, d, V, dtype, Hpk, W, tok, oldlogp, adv, w, eps, loss_scale, loss, lse, logp,
                                  ratio, coef, row_loss, scratch, kStaticScratchBytes, stream);
  return r == PS_ERR_WORKSPACE ? PS_ERR_UNSUPPORTED : r;
}
