// Library-wide entry points: device error word, status names, version.
#include <cuda_runtime.h>

#include "common.cuh"

extern "C" __attribute__((visibility("hidden"))) unsigned int ipd_internal_take_attn_error();
extern "C" __attribute__((visibility("hidden"))) unsigned int ipd_internal_take_score_error();
extern "C" __attribute__((visibility("hidden"))) unsigned int ipd_internal_take_loss_error();
extern "C" __attribute__((visibility("hidden"))) unsigned int ipd_internal_take_kv_error();

extern "C" int ipd_get_device_error(uint32_t *code) {
  if (!code) return IPD_ERR_INVALID_ARG;
  if (cudaDeviceSynchronize() != cudaSuccess) return IPD_ERR_CUDA;
  const unsigned int a = ipd_internal_take_attn_error();
  const unsigned int b = ipd_internal_take_score_error();
  const unsigned int c = ipd_internal_take_loss_error();
  const unsigned int d = ipd_internal_take_kv_error();
  if (a == 0xffffffffu || b == 0xffffffffu || c == 0xffffffffu || d == 0xffffffffu)
    return IPD_ERR_CUDA;
  *code = a ? a : (b ? b : (c ? c : d));
  return IPD_OK;
}

extern "C" const char *ipd_status_string(int status) {
  switch (status) {
    case IPD_OK: return "IPD_OK";
    case IPD_ERR_INVALID_ARG: return "IPD_ERR_INVALID_ARG";
    case IPD_ERR_UNSUPPORTED: return "IPD_ERR_UNSUPPORTED";
    case IPD_ERR_WORKSPACE: return "IPD_ERR_WORKSPACE";
    case IPD_ERR_CUDA: return "IPD_ERR_CUDA";
    case IPD_ERR_TIMEOUT: return "IPD_ERR_TIMEOUT";
    case IPD_ERR_DEVICE: return "IPD_ERR_DEVICE";
    case IPD_ERR_CAPACITY: return "IPD_ERR_CAPACITY";
    default: return "IPD_ERR_UNKNOWN";
  }
}

extern "C" int ipd_version(void) { return 100; }

extern "C" int ipd_device_readable(const void *ptr, int *readable) {
  if (!readable) return IPD_ERR_INVALID_ARG;
  *readable = 0;
  if (!ptr) return IPD_OK;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    (void)cudaGetLastError();  // an unregistered host pointer is not an error state
    return IPD_OK;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return IPD_ERR_CUDA;
  if (a.type == cudaMemoryTypeDevice) *readable = a.device == dev;
  else if (a.type == cudaMemoryTypeManaged) *readable = 1;
  else if (a.type == cudaMemoryTypeHost) *readable = a.devicePointer == ptr;
  return IPD_OK;
}
