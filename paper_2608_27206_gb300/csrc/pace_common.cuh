// Shared host-side plumbing of libpace: status codes, CUDA error capture, the
// per-device status word, and the sm_103 check.
#pragma once
#include <cuda_runtime.h>
#include <atomic>
#include <cstdint>
#include <cstddef>

#include "pace.h"

namespace pace {

// Kernel identifiers written to the device status word next to the error code.
enum KernelId : int {
  K_APC_PASS1 = 1,
  K_APC_PASS2 = 2,
  K_APC_TAIL = 3,
  K_APC_RESAMPLE = 4,
  K_ATTN_ROW_LSE = 5,
  K_ATTN_COLSUM = 6,
  K_ATTN_COMBINE = 7,
  K_ATTN_REDUCE = 8,
  K_DDAE_SELECT = 9,
  K_GATHER = 10,
  K_SELFTEST = 11,
  K_PRUNE_INDEX = 12,
  K_GATHER_MULTI = 13,
};

// Device status word layout: [0] = code (pace_status_t), [1] = kernel id.
// Records the first error only.
__device__ __forceinline__ void record_error(int* status, int code, int kernel) {
  if (status != nullptr && atomicCAS(&status[0], 0, code) == 0) atomicExch(&status[1], kernel);
}

// Wall-clock limit of every device-side wait (nanoseconds).
constexpr uint64_t kWaitLimitNs = 1000000000ull;

// Host helpers (implemented in pace_api.cu).
pace_status_t set_cuda_error(cudaError_t e);
pace_status_t check_device();              // current device is sm_103 and initialised
int* device_status_word();                 // status word of the current device
pace_status_t check_launch();              // cudaGetLastError -> status

// Generation of the library's per-device set-up.  pace_init(dev) advances it, so every cache
// built on DeviceOnce below (function attributes, symbol addresses) is filled again on the next
// call: after cudaDeviceReset the cached values belong to a destroyed context.
constexpr int kMaxDevices = 64;
uint32_t device_generation(int dev);

// Per-device one-time set-up tied to the generation: done(dev) is true once mark(dev) ran in
// the device's current generation.  Objects of this type live in static storage (zeroed).
class DeviceOnce {
 public:
  bool done(int dev) const {
    return dev >= 0 && dev < kMaxDevices &&
           flag_[dev].load(std::memory_order_acquire) == device_generation(dev) + 1u;
  }
  void mark(int dev) {
    if (dev >= 0 && dev < kMaxDevices) flag_[dev].store(device_generation(dev) + 1u, std::memory_order_release);
  }

 private:
  std::atomic<uint32_t> flag_[kMaxDevices];
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace pace

#define PACE_CHECK(expr)                             \
  do {                                               \
    pace_status_t _s = (expr);                       \
    if (_s != PACE_OK) return _s;                    \
  } while (0)

#define PACE_CUDA(expr)                              \
  do {                                               \
    cudaError_t _e = (expr);                         \
    if (_e != cudaSuccess) return pace::set_cuda_error(_e); \
  } while (0)
