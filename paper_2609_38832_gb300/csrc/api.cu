// api.cu -- shared host-side pieces of the C ABI: status strings, the per-device
// property cache, the driver tensor-map encoder and the RoPE frequency table.
#include <math.h>
#include <stdio.h>
#include <mutex>

#include "common.cuh"

namespace namoh {

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_info_mutex;
DeviceInfo g_info[kMaxDevices];
bool g_info_valid[kMaxDevices] = {};

std::once_flag g_encoder_once;
EncodeTiledFn g_encoder = nullptr;
}  // namespace

bool current_device_info(DeviceInfo* out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return false;
  if (dev < kMaxDevices) {
    std::lock_guard<std::mutex> lock(g_info_mutex);
    if (g_info_valid[dev]) {
      *out = g_info[dev];
      return true;
    }
  }
  DeviceInfo info{};
  info.device = dev;
  int optin = 0;
  if (cudaDeviceGetAttribute(&info.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return false;
  if (cudaDeviceGetAttribute(&info.major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) return false;
  if (cudaDeviceGetAttribute(&info.minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) return false;
  if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return false;
  info.max_smem_optin = (size_t)optin;
  if (dev < kMaxDevices) {
    std::lock_guard<std::mutex> lock(g_info_mutex);
    g_info[dev] = info;
    g_info_valid[dev] = true;
  }
  *out = info;
  return true;
}

namespace {
thread_local char g_last_error[160] = "no error";
}

int cuda_fail(cudaError_t e, const char* where) {
  snprintf(g_last_error, sizeof g_last_error, "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
  return NAMOH_ERR_CUDA;
}

int cuda_check_launch(const char* where) {
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? NAMOH_OK : cuda_fail(e, where);
}

const char* last_error_text() { return g_last_error; }

EncodeTiledFn tensor_map_encoder() {
  std::call_once(g_encoder_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess) {
      g_encoder = reinterpret_cast<EncodeTiledFn>(fn);
    }
  });
  return g_encoder;
}

void fill_rope_table(RopeTable* t, int d, double base) {
  for (int j = 0; j < 64; ++j) {
    double th = (j < d / 2) ? pow(base, -2.0 * (double)j / (double)d) : 0.0;
    float hi = (float)th;
    t->theta_hi[j] = hi;
    t->theta_lo[j] = (float)(th - (double)hi);
  }
  const double two_pi = 6.283185307179586476925286766559;
  float p0 = (float)two_pi;
  float p1 = (float)(two_pi - (double)p0);
  float p2 = (float)(two_pi - (double)p0 - (double)p1);
  t->two_pi[0] = p0;
  t->two_pi[1] = p1;
  t->two_pi[2] = p2;
  t->inv_two_pi = (float)(1.0 / two_pi);
}

}  // namespace namoh

extern "C" const char* namoh_status_string(int status) {
  switch (status) {
    case NAMOH_OK:
      return "ok";
    case NAMOH_ERR_INVALID_ARG:
      return "invalid argument";
    case NAMOH_ERR_UNSUPPORTED:
      return "unsupported configuration or device";
    case NAMOH_ERR_WORKSPACE:
      return "workspace missing, misaligned or too small";
    case NAMOH_ERR_CUDA:
      return "CUDA error";
    default:
      return "unknown status";
  }
}

extern "C" int namoh_version(void) { return (1 << 16) | 0; }

extern "C" const char* namoh_last_error_string(void) { return namoh::last_error_text(); }
