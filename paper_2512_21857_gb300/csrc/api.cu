// Library-wide entry points: version, status names, the per-device error word.
#include <mutex>

#include "adt_common.cuh"

namespace {

// One error word per device that loads the library.  Kernels receive its
// device address as an argument and atomically OR ADT_DEVERR_* bits into it.
__device__ unsigned g_device_error_word;

constexpr int kMaxDevices = 64;
std::once_flag g_once[kMaxDevices];
adt::DeviceInfo g_info[kMaxDevices];
adt_status g_info_status[kMaxDevices];

void init_device(int dev) {
  adt::DeviceInfo info{};
  info.device = dev;
  g_info_status[dev] = ADT_ERR_CUDA;
  if (cudaDeviceGetAttribute(&info.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return;
  if (cudaDeviceGetAttribute(&info.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
      cudaSuccess)
    return;
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_device_error_word) != cudaSuccess) return;
  info.error_word = static_cast<unsigned*>(p);
  g_info[dev] = info;
  g_info_status[dev] = ADT_OK;
}

}  // namespace

namespace adt {

adt_status device_info(DeviceInfo* out) {
  int dev = 0;
  ADT_CUDA_TRY(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return ADT_ERR_UNSUPPORTED;
  std::call_once(g_once[dev], init_device, dev);
  if (g_info_status[dev] != ADT_OK) return g_info_status[dev];
  *out = g_info[dev];
  return ADT_OK;
}

}  // namespace adt

extern "C" {

int32_t adt_version(void) { return 100; }

const char* adt_status_string(adt_status s) {
  switch (s) {
    case ADT_OK: return "ADT_OK";
    case ADT_ERR_INVALID_ARG: return "ADT_ERR_INVALID_ARG";
    case ADT_ERR_UNSUPPORTED: return "ADT_ERR_UNSUPPORTED";
    case ADT_ERR_CUDA: return "ADT_ERR_CUDA";
    case ADT_ERR_TIMEOUT: return "ADT_ERR_TIMEOUT";
    case ADT_ERR_WORKSPACE: return "ADT_ERR_WORKSPACE";
    case ADT_ERR_DEVICE: return "ADT_ERR_DEVICE";
  }
  return "ADT_ERR_UNKNOWN";
}

adt_status adt_get_device_error(void* stream, uint32_t* bits) {
  adt::DeviceInfo info;
  adt_status st = adt::device_info(&info);
  if (st != ADT_OK) return st;
  cudaStream_t s = adt::as_stream(stream);
  unsigned host = 0;
  ADT_CUDA_TRY(cudaMemcpyAsync(&host, info.error_word, sizeof(unsigned), cudaMemcpyDeviceToHost, s));
  ADT_CUDA_TRY(cudaMemsetAsync(info.error_word, 0, sizeof(unsigned), s));
  ADT_CUDA_TRY(cudaStreamSynchronize(s));
  if (bits) *bits = host;
  if (host & ADT_DEVERR_TIMEOUT) return ADT_ERR_TIMEOUT;
  return host ? ADT_ERR_DEVICE : ADT_OK;
}

}  // extern "C"
