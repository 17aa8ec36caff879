// ps_lmhead_ppo_fwd_noalloc: the fused forward with its scratch in a static device array.
//
// Some callers cannot allocate device memory for a workspace: a plugin hosted by a
// framework that owns the GPU's memory (its pool is reserved up front and plugins may not
// call cudaMalloc), or a deployment whose device memory plan is fixed at start-up. For
// them this entry point runs exactly the work of ps_lmhead_ppo_fwd with the workspace
// taken from a file-scope __device__ array of kStaticScratchBytes, which every GPU that
// loads the library holds until the process exits. The function allocates nothing: no
// cudaMalloc, no cudaFree, no allocating library routine.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "psppo.h"

namespace {

constexpr size_t kStaticScratchBytes = 64ull << 20;  // 64 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_fwd_scratch[kStaticScratchBytes];

std::mutex g_mu;

// The array's device address in one device context. A context that is destroyed and created
// again (cudaDeviceReset, then any runtime call) loads the module anew, possibly at another
// address, so the address is keyed on the context's process-unique id (cuCtxGetId).
struct ScratchSlot {
  void* ptr = nullptr;
  unsigned long long ctx_id = 0;
};
ScratchSlot g_slot[kMaxDevices];

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);
struct CtxFns {
  CtxGetCurrentFn get_current = nullptr;
  CtxGetIdFn get_id = nullptr;
};

// Driver entry points through the runtime (the library does not link libcuda itself).
const CtxFns& ctx_fns() {
  static CtxFns f;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f.get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f.get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  return f;
}

// Device address of the current context's copy of g_fwd_scratch. In host code the symbol is only
// a host-side stand-in, so the address comes from cudaGetSymbolAddress, with the device current,
// once per device context: on the first call, and again after the context has changed.
int scratch_for_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return PS_ERR_CUDA;
  const CtxFns& f = ctx_fns();
  if (f.get_current == nullptr || f.get_id == nullptr) return PS_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  void* p = nullptr;
  CUcontext ctx = nullptr;
  if (f.get_current(&ctx) != CUDA_SUCCESS) return PS_ERR_CUDA;
  if (ctx == nullptr) {
    // no context is current yet: the runtime creates the device's primary context (and makes it
    // current) on its first call that needs one, such as this lookup
    if (cudaGetSymbolAddress(&p, g_fwd_scratch) != cudaSuccess || p == nullptr) return PS_ERR_CUDA;
    if (f.get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return PS_ERR_CUDA;
  }
  unsigned long long id = 0;
  if (f.get_id(ctx, &id) != CUDA_SUCCESS) return PS_ERR_CUDA;
  ScratchSlot& slot = g_slot[dev];
  if (slot.ptr == nullptr || slot.ctx_id != id) {
    if (p == nullptr && (cudaGetSymbolAddress(&p, g_fwd_scratch) != cudaSuccess || p == nullptr)) return PS_ERR_CUDA;
    slot.ptr = p;
    slot.ctx_id = id;
  }
  *out = slot.ptr;
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
