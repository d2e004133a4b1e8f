// context.cu - identity of the current device's context, through driver entry
// points (no link-time dependency on libcuda).
#include <cuda.h>

#include <mutex>

#include "context.cuh"

namespace cover {
namespace {

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

CtxGetCurrentFn g_get_current = nullptr;
CtxGetIdFn g_get_id = nullptr;
std::once_flag g_once;

void load_entry_points() {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    g_get_current = reinterpret_cast<CtxGetCurrentFn>(p);
  p = nullptr;
  if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    g_get_id = reinterpret_cast<CtxGetIdFn>(p);
}

}  // namespace

bool current_device_ctx(int* dev, unsigned long long* ctx_id) {
  std::call_once(g_once, load_entry_points);
  if (g_get_current == nullptr || g_get_id == nullptr) return false;
  if (cudaGetDevice(dev) != cudaSuccess || *dev < 0 || *dev >= kMaxDevices) return false;
  CUcontext ctx = nullptr;
  if (g_get_current(&ctx) != CUDA_SUCCESS) return false;
  if (ctx == nullptr) {
    // nothing current yet: bind (and if needed create) the device's primary context
    if (cudaSetDevice(*dev) != cudaSuccess || g_get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return false;
  }
  return g_get_id(ctx, ctx_id) == CUDA_SUCCESS;
}

}  // namespace cover
