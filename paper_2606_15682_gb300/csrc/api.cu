// Library-wide state and helpers: the per-device status word, the launch
// counter and the status strings.
#include <atomic>
#include <mutex>

#include "common.cuh"

namespace nvfp4 {
namespace {

// One status word per device that loads the library (a module-scope device
// variable, so nothing is allocated at run time).  Kernels record the first
// device-side error here with atomicCAS.
__device__ int g_status_word;

constexpr int kMaxDevices = 64;
std::atomic<uint64_t> g_launches{0};
std::mutex g_mu;
int* g_status_ptr[kMaxDevices] = {};
int g_sms[kMaxDevices] = {};

int current_device() {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return 0;
  return d;
}

}  // namespace

int* status_word_dev() {
  const int d = current_device();
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_status_ptr[d]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    g_status_ptr[d] = static_cast<int*>(p);
  }
  return g_status_ptr[d];
}

int sm_count() {
  const int d = current_device();
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_sms[d]) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, d) != cudaSuccess || n <= 0) n = 148;
    g_sms[d] = n;
  }
  return g_sms[d];
}

void count_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

std::atomic<int> g_fault{NVFP4_FAULT_NONE};

bool take_fault(int what) {
  int armed = what;
  return what != NVFP4_FAULT_NONE && g_fault.compare_exchange_strong(armed, NVFP4_FAULT_NONE);
}

}  // namespace nvfp4

using namespace nvfp4;

NVFP4_API nvfp4_status nvfp4_get_device_status(int32_t* status_host, void* stream) {
  NVFP4_TRACE("nvfp4_get_device_status");
  if (!status_host) return NVFP4_ERR_INVALID_ARG;
  int* p = status_word_dev();
  if (!p) return NVFP4_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int v = 0;
  if (cudaStreamSynchronize(s) != cudaSuccess) return NVFP4_ERR_CUDA;
  if (cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return NVFP4_ERR_CUDA;
  if (cudaMemset(p, 0, sizeof(int)) != cudaSuccess) return NVFP4_ERR_CUDA;
  *status_host = v;
  return NVFP4_OK;
}

NVFP4_API const char* nvfp4_status_string(nvfp4_status s) {
  switch (s) {
    case NVFP4_OK: return "ok";
    case NVFP4_ERR_INVALID_ARG: return "invalid argument";
    case NVFP4_ERR_SHAPE: return "unsupported or inconsistent shape";
    case NVFP4_ERR_ALIGN: return "misaligned pointer or leading dimension";
    case NVFP4_ERR_UNSUPPORTED: return "unsupported device";
    case NVFP4_ERR_CUDA: return "CUDA error";
    case NVFP4_ERR_TIMEOUT: return "bounded device wait timed out";
    case NVFP4_ERR_CAPACITY: return "KV cache capacity exceeded";
    case NVFP4_ERR_BOUNDS: return "store index out of bounds (bounds-checked build)";
  }
  return "unknown status";
}

NVFP4_API uint64_t nvfp4_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

NVFP4_API nvfp4_status nvfp4_debug_inject_fault(int what) {
  NVFP4_TRACE("nvfp4_debug_inject_fault");
  if (what != NVFP4_FAULT_NONE && what != NVFP4_FAULT_ATTN_SKIP_STAGE && what != NVFP4_FAULT_GEMM_SKIP_STAGE)
    return NVFP4_ERR_INVALID_ARG;
  g_fault.store(what);
  return NVFP4_OK;
}
