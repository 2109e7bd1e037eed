// Host-side helpers of libhsa: status strings, budget checks (Sec. 2.2), the
// caching-window margin (Sec. 2.5), |A_i| from group sizes, the noise
// schedule of the Euler solver (Sec. 2.1), and the per-device error word that
// kernels write instead of trapping.
#include <atomic>
#include <cmath>

#include "hsa_internal.cuh"

namespace {
// One word per device; kernels receive its address as an argument.
__device__ unsigned g_hsa_error_word;

constexpr int kMaxDevices = 64;
std::atomic<unsigned *> g_err_ptr[kMaxDevices];
std::atomic<int> g_sm_count[kMaxDevices];

int current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return -1;
  return dev;
}
}  // namespace

namespace hsa {

unsigned *device_error_word() {
  const int dev = current_device();
  if (dev < 0) return nullptr;
  unsigned *p = g_err_ptr[dev].load(std::memory_order_acquire);
  if (!p) {
    void *addr = nullptr;
    if (cudaGetSymbolAddress(&addr, g_hsa_error_word) != cudaSuccess) return nullptr;
    p = static_cast<unsigned *>(addr);
    g_err_ptr[dev].store(p, std::memory_order_release);
  }
  return p;
}

std::atomic<unsigned long long> g_launches{0};

void count_launches(int n) { g_launches.fetch_add((unsigned long long)n, std::memory_order_relaxed); }

int sm_count() {
  const int dev = current_device();
  if (dev < 0) return 1;
  int n = g_sm_count[dev].load(std::memory_order_relaxed);
  if (n <= 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 1;
    g_sm_count[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

}  // namespace hsa

extern "C" const char *hsa_status_string(int status) {
  switch (status) {
    case HSA_OK: return "ok";
    case HSA_ERR_INVALID_ARG: return "invalid argument";
    case HSA_ERR_NOT_DIVISOR: return "a step budget does not divide T";
    case HSA_ERR_BAD_COUNTS: return "group sizes negative or not summing to N";
    case HSA_ERR_UNSUPPORTED: return "unsupported shape";
    case HSA_ERR_NONFINITE: return "non-finite statistic";
    case HSA_ERR_INDEX: return "index or group id out of range";
    case HSA_ERR_TIMEOUT: return "bounded pipeline wait ran out";
    case HSA_ERR_CUDA: return "CUDA error";
    case HSA_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    default: return "unknown status";
  }
}

extern "C" int hsa_version(void) { return 1; }

extern "C" int hsa_check_budgets(int T, const int *budgets, const int *counts, int K, int N) {
  if (T < 1 || K < 1 || N < 0 || !budgets) return HSA_ERR_INVALID_ARG;
  for (int k = 0; k < K; ++k) {
    if (budgets[k] < 1 || budgets[k] > T) return HSA_ERR_INVALID_ARG;
    if (T % budgets[k]) return HSA_ERR_NOT_DIVISOR;
    if (k && budgets[k] > budgets[k - 1]) return HSA_ERR_INVALID_ARG;
  }
  if (budgets[0] != T) return HSA_ERR_INVALID_ARG;
  if (counts) {
    long long total = 0;
    for (int k = 0; k < K; ++k) {
      if (counts[k] < 0) return HSA_ERR_BAD_COUNTS;
      total += counts[k];
    }
    if (total != N) return HSA_ERR_BAD_COUNTS;
  }
  return HSA_OK;
}

extern "C" int hsa_window_margin(int T, int window_pct) {
  if (T < 1 || window_pct < 0 || window_pct > 100) return HSA_ERR_INVALID_ARG;
  return (int)(((long long)(100 - window_pct) * T) / 200);
}

extern "C" int hsa_active_count(const int *budgets, const int *counts, int K, int T, int iter,
                                int window_pct) {
  if (!counts) return HSA_ERR_INVALID_ARG;
  long long N = 0;
  for (int k = 0; k < K; ++k) N += counts[k];
  if (N > 0x7fffffffLL) return HSA_ERR_BAD_COUNTS;
  const int st = hsa_check_budgets(T, budgets, counts, K, (int)N);
  if (st != HSA_OK) return st;
  const int m = hsa_window_margin(T, window_pct);
  if (m < 0 || iter < 0 || iter >= T) return HSA_ERR_INVALID_ARG;
  const bool full = iter < m || iter > T - m - 1;
  long long n = 0;
  for (int k = 0; k < K; ++k)
    if (full || iter % (T / budgets[k]) == 0) n += counts[k];
  return (int)n;
}

extern "C" int hsa_sigma_schedule(int T, double shift, double *sigma) {
  if (T < 1 || !sigma || !(shift > 0.0) || !std::isfinite(shift)) return HSA_ERR_INVALID_ARG;
  for (int i = 0; i <= T; ++i) {
    const double t = (double)(T - i) / (double)T;
    sigma[i] = shift * t / (1.0 + (shift - 1.0) * t);
  }
  return HSA_OK;
}

extern "C" int hsa_get_device_error(hsa_stream_t stream) {
  unsigned *word = hsa::device_error_word();
  if (!word) return HSA_ERR_CUDA;
  cudaStream_t s = (cudaStream_t)stream;
  unsigned bits = 0;
  if (cudaMemcpyAsync(&bits, word, sizeof bits, cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return HSA_ERR_CUDA;
  if (cudaMemsetAsync(word, 0, sizeof bits, s) != cudaSuccess) return HSA_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return HSA_ERR_CUDA;
  if (bits & hsa::kErrTimeout) return HSA_ERR_TIMEOUT;
  if (bits & hsa::kErrNonfinite) return HSA_ERR_NONFINITE;
  if (bits & hsa::kErrIndex) return HSA_ERR_INDEX;
  return HSA_OK;
}

extern "C" unsigned long long hsa_launch_count(void) {
  return hsa::g_launches.load(std::memory_order_relaxed);
}
