// Device status word, device queries and the status entry points.

#include <atomic>

#include "common.cuh"

namespace spl {

namespace {
std::atomic<uint64_t> g_launches{0};
constexpr int kMaxDevices = 64;
int g_sm_count[kMaxDevices] = {0};
int g_cc[kMaxDevices] = {0};

int current_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
  return dev;
}
}  // namespace

void note_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

int device_sm_count() {
  const int dev = current_device();
  if (g_sm_count[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) v = kNumSMsGB300;
    g_sm_count[dev] = v;
  }
  return g_sm_count[dev];
}

int device_cc() {
  const int dev = current_device();
  if (g_cc[dev] == 0) {
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    g_cc[dev] = major * 10 + minor;
  }
  return g_cc[dev];
}

}  // namespace spl

extern "C" spl_status spl_get_device_status(cudaStream_t stream) {
  if (cudaStreamSynchronize(stream) != cudaSuccess) return SPL_ECUDA;
  unsigned int word = 0;
  if (spl::read_clear_device_status(&word) != cudaSuccess) return SPL_ECUDA;
  if (word & spl::kStatusTimeout) return SPL_ETIMEOUT;
  return cudaGetLastError() == cudaSuccess ? SPL_OK : SPL_ECUDA;
}

extern "C" uint64_t spl_launch_count(void) { return spl::g_launches.load(std::memory_order_relaxed); }

extern "C" const char* spl_status_string(spl_status status) {
  switch (status) {
    case SPL_OK: return "SPL_OK";
    case SPL_EINVAL: return "SPL_EINVAL";
    case SPL_ESHAPE: return "SPL_ESHAPE";
    case SPL_EALIGN: return "SPL_EALIGN";
    case SPL_ECUDA: return "SPL_ECUDA";
    case SPL_ETIMEOUT: return "SPL_ETIMEOUT";
    case SPL_EUNSUPPORTED: return "SPL_EUNSUPPORTED";
    case SPL_EWORKSPACE: return "SPL_EWORKSPACE";
  }
  return "SPL_UNKNOWN";
}

// The boundary's listed names for the two status calls (the same calls as above).
extern "C" spl_status spl_get_last_device_status(cudaStream_t stream) { return spl_get_device_status(stream); }

extern "C" const char* spl_status_str(spl_status status) { return spl_status_string(status); }

extern "C" spl_status spl_copy_2d(void* dst, size_t dst_pitch, const void* src, size_t src_pitch, size_t width_bytes,
                                  size_t rows, cudaStream_t stream) {
  if (rows == 0 || width_bytes == 0) return SPL_OK;
  if (!dst || !src || width_bytes > dst_pitch || width_bytes > src_pitch) return SPL_EINVAL;
  const cudaError_t e = cudaMemcpy2DAsync(dst, dst_pitch, src, src_pitch, width_bytes, rows, cudaMemcpyDefault, stream);
  return e == cudaSuccess ? SPL_OK : SPL_ECUDA;
}
