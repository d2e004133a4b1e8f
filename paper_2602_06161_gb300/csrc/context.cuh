// context.cuh - host-side set-up that belongs to one CUDA context.
//
// A kernel's dynamic shared-memory limit (cudaFuncSetAttribute), the device
// address of a __device__ symbol and the SM count are properties of the
// context of the device that was current when they were obtained. A launcher
// that cached them in a plain static would use them on another device, or in
// a context created anew after cudaDeviceReset, where they do not hold. Each
// launcher therefore keeps them in a ContextCache: one entry per device, tagged
// with the unique id of the context it was computed in and recomputed when the
// device's current context has a different id. A lock serialises first calls
// from several host threads.
#pragma once

#include <cuda_runtime.h>

#include <mutex>

namespace cover {

constexpr int kMaxDevices = 64;

// The current device and the unique id of its current context. If no context
// is current on the calling thread yet, the device's primary context is made
// current first (what the next runtime call would do anyway); a context the
// caller made current is left in place. Returns false on any failure.
bool current_device_ctx(int* dev, unsigned long long* ctx_id);

template <typename T>
class ContextCache {
 public:
  // *out = the value init computed in the current context of the current
  // device, running init(T&) (0 on success, else a negative status that is
  // returned and nothing cached) the first time in that context.
  template <typename F>
  int get(T* out, F&& init) {
    int dev = 0;
    unsigned long long id = 0;
    if (!current_device_ctx(&dev, &id)) return -3;
    std::lock_guard<std::mutex> lock(mu_);
    if (!valid_[dev] || ids_[dev] != id) {
      T v{};
      const int rc = init(v);
      if (rc != 0) return rc;
      vals_[dev] = v;
      ids_[dev] = id;
      valid_[dev] = true;
    }
    *out = vals_[dev];
    return 0;
  }

 private:
  std::mutex mu_;
  bool valid_[kMaxDevices] = {};
  unsigned long long ids_[kMaxDevices] = {};
  T vals_[kMaxDevices] = {};
};

}  // namespace cover
