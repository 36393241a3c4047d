// Per-device launch state: SM counts and raised shared-memory limits, kept for
// each GPU separately (a function attribute set on one device does not apply
// on another) and guarded for concurrent host threads.
#include <mutex>
#include <set>
#include <tuple>

#include "internal.h"

namespace tre {

namespace {
constexpr int kMaxDevices = 64;
int g_sms[kMaxDevices];                     // 0 = not looked up yet
std::mutex g_mu;
std::set<std::tuple<int, const void*, int, bool>> g_attr;   // (device, fn, bytes, carveout)

int current_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    dev = 0;
  }
  return dev;
}
}  // namespace

int device_sm_count() {
  const int dev = current_device();
  std::lock_guard<std::mutex> lk(g_mu);
  int* slot = dev >= 0 && dev < kMaxDevices ? &g_sms[dev] : nullptr;
  if (slot && *slot > 0) return *slot;
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  if (n <= 0) return 1;          // not cached: looked up again on the next call
  if (slot) *slot = n;
  return n;
}

cudaError_t func_smem_once(const void* fn, int bytes, bool max_carveout) {
  const int dev = current_device();
  std::lock_guard<std::mutex> lk(g_mu);
  const auto key = std::make_tuple(dev, fn, bytes, max_carveout);
  if (g_attr.count(key)) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (!e && max_carveout)
    e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  if (e) return e;
  g_attr.insert(key);
  return cudaSuccess;
}

}  // namespace tre
