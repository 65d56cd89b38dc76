// libpace host API: status strings, per-device initialisation (sm_103 check and
// device status word), budget helper and parameter defaults.
#include <atomic>
#include <cmath>
#include <mutex>

#include "pace_common.cuh"
#include "pace_ptx.cuh"

namespace pace {

namespace {
thread_local int t_last_cuda_error = 0;
std::atomic<uint64_t> g_launches{0};
std::mutex g_mutex;
// Per-device state: 0 = not checked yet, 1 = sm_103 and initialised, 2 = unsupported.
std::atomic<int> g_state[kMaxDevices];
int* g_status[kMaxDevices] = {};
std::atomic<uint32_t> g_generation[kMaxDevices];

// Status word of every device that loads the library: [code, kernel id].
__device__ int g_status_word[2];
}  // namespace

uint32_t device_generation(int dev) {
  return (dev >= 0 && dev < kMaxDevices) ? g_generation[dev].load(std::memory_order_acquire) : 0u;
}

pace_status_t set_cuda_error(cudaError_t e) {
  t_last_cuda_error = static_cast<int>(e);
  return PACE_ERR_CUDA;
}

static pace_status_t init_device_locked(int dev) {
  if (dev < 0 || dev >= kMaxDevices) return PACE_ERR_INVALID_ARG;
  const int st = g_state[dev].load(std::memory_order_acquire);
  if (st != 0) return st == 1 ? PACE_OK : PACE_ERR_UNSUPPORTED_ARCH;
  int major = 0, minor = 0;
  PACE_CUDA(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev));
  PACE_CUDA(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev));
  if (!(major == 10 && minor == 3)) {
    g_state[dev].store(2, std::memory_order_release);
    return PACE_ERR_UNSUPPORTED_ARCH;
  }
  int prev = -1;
  PACE_CUDA(cudaGetDevice(&prev));
  if (prev != dev) PACE_CUDA(cudaSetDevice(dev));
  void* p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_status_word);
  if (e == cudaSuccess) e = cudaMemset(p, 0, 2 * sizeof(int));
  if (prev != dev) cudaSetDevice(prev);
  if (e != cudaSuccess) return set_cuda_error(e);
  g_status[dev] = static_cast<int*>(p);
  g_state[dev].store(1, std::memory_order_release);
  return PACE_OK;
}

pace_status_t check_device() {
  int dev = -1;
  PACE_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < kMaxDevices) {
    const int st = g_state[dev].load(std::memory_order_acquire);
    if (st != 0) return st == 1 ? PACE_OK : PACE_ERR_UNSUPPORTED_ARCH;
  }
  std::lock_guard<std::mutex> lk(g_mutex);
  return init_device_locked(dev);
}

int* device_status_word() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  if (g_state[dev].load(std::memory_order_acquire) != 1) return nullptr;
  return g_status[dev];
}

pace_status_t check_launch() {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return set_cuda_error(e);
  g_launches.fetch_add(1, std::memory_order_relaxed);
  return PACE_OK;
}

// One CTA waits on an mbarrier that nothing ever arrives at: the bounded wait must give up
// after limit_ns and record PACE_ERR_TIMEOUT, leaving the context usable.
__global__ void selftest_wait_kernel(uint64_t limit_ns, int* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    ptx::mbar_init(ptx::smem_u32(&bar), 1);
    ptx::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !ptx::mbar_wait(ptx::smem_u32(&bar), 0, limit_ns))
    record_error(status, PACE_ERR_TIMEOUT, K_SELFTEST);
}

}  // namespace pace

extern "C" {

const char* pace_status_string(pace_status_t s) {
  switch (s) {
    case PACE_OK: return "PACE_OK";
    case PACE_ERR_INVALID_ARG: return "PACE_ERR_INVALID_ARG";
    case PACE_ERR_UNSUPPORTED_ARCH: return "PACE_ERR_UNSUPPORTED_ARCH";
    case PACE_ERR_WORKSPACE: return "PACE_ERR_WORKSPACE";
    case PACE_ERR_CUDA: return "PACE_ERR_CUDA";
    case PACE_ERR_TIMEOUT: return "PACE_ERR_TIMEOUT";
  }
  return "PACE_ERR_UNKNOWN";
}

int pace_last_cuda_error(void) { return pace::t_last_cuda_error; }

uint64_t pace_kernel_launch_count(void) { return pace::g_launches.load(std::memory_order_relaxed); }

pace_status_t pace_init(int device) {
  std::lock_guard<std::mutex> lk(pace::g_mutex);
  if (device < 0 || device >= pace::kMaxDevices) return PACE_ERR_INVALID_ARG;
  // Start a new set-up generation: the status word's address and every per-device cache of the
  // library are looked up again (they are stale after a cudaDeviceReset).
  pace::g_generation[device].fetch_add(1u, std::memory_order_acq_rel);
  pace::g_state[device].store(0, std::memory_order_release);
  return pace::init_device_locked(device);
}

pace_status_t pace_device_status(int* code, int* where, int clear) {
  PACE_CHECK(pace::check_device());
  int* w = pace::device_status_word();
  if (w == nullptr) return PACE_ERR_INVALID_ARG;
  int h[2] = {0, 0};
  PACE_CUDA(cudaDeviceSynchronize());
  PACE_CUDA(cudaMemcpy(h, w, sizeof(h), cudaMemcpyDeviceToHost));
  if (code) *code = h[0];
  if (where) *where = h[1];
  if (clear) PACE_CUDA(cudaMemset(w, 0, sizeof(h)));
  return PACE_OK;
}

pace_status_t pace_selftest_wait_timeout(uint32_t limit_us, pace_stream_t stream) {
  if (limit_us == 0 || limit_us > 1000000u) return PACE_ERR_INVALID_ARG;
  PACE_CHECK(pace::check_device());
  pace::selftest_wait_kernel<<<1, 32, 0, stream>>>(static_cast<uint64_t>(limit_us) * 1000ull,
                                                   pace::device_status_word());
  return pace::check_launch();
}

int32_t pace_budget_vanilla(int32_t n_vis_vanilla, int32_t n_vis_condensed, double frac) {
  if (n_vis_condensed <= 0) return 0;
  const int32_t k = pace_budget(n_vis_vanilla, frac);
  return k < n_vis_condensed ? k : n_vis_condensed;
}

int32_t pace_budget(int32_t n_vis, double frac) {
  if (n_vis <= 0 || !(frac > 0.0)) return 0;
  double k = std::floor(frac * static_cast<double>(n_vis) + 0.5);
  if (k > n_vis) k = n_vis;
  return static_cast<int32_t>(k);
}

void pace_apc_params_default(pace_apc_params* p) {
  if (!p) return;
  p->alpha = 0.6f;
  p->gamma = 1.5f;
  p->tail_frac = 0.10f;
  p->r_min = 0.0f;
  p->r_max = 1.0f;
  p->align = 28;
}

void pace_ddae_params_default(pace_ddae_params* p) {
  if (!p) return;
  p->tau = 0.5f;
  p->fusion = PACE_DDAE_ADAPTIVE;
}

}  // extern "C"
