// Library-wide entry points of libsd.so: status names, version, and the
// device error word collected from every translation unit.
#include "common.cuh"

extern "C" const char* sd_status_str(sd_status s) {
  switch (s) {
    case SD_OK: return "SD_OK";
    case SD_ERR_INVALID_ARG: return "SD_ERR_INVALID_ARG";
    case SD_ERR_UNSUPPORTED: return "SD_ERR_UNSUPPORTED";
    case SD_ERR_WORKSPACE: return "SD_ERR_WORKSPACE";
    case SD_ERR_CUDA: return "SD_ERR_CUDA";
    case SD_ERR_DEVICE: return "SD_ERR_DEVICE";
    case SD_ERR_TIMEOUT: return "SD_ERR_TIMEOUT";
  }
  return "SD_ERR_UNKNOWN";
}

extern "C" const char* sd_version(void) { return "sd 0.1 sm_103a"; }

extern "C" sd_status sd_get_device_error(sd_stream_t stream, uint32_t* bits) {
  if (!bits) return SD_ERR_INVALID_ARG;
  *bits = 0;
  if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) {
    (void)cudaGetLastError();
    return SD_ERR_CUDA;
  }
  cudaError_t (*take[])(uint32_t*) = {sd_take_error_rope, sd_take_error_kv,
                                      sd_take_error_attention, sd_take_error_attention_tc,
                                      sd_take_error_greedy,
                                      sd_take_error_sample, sd_take_error_budget};
  for (auto fn : take) {
    if (fn(bits) != cudaSuccess) {
      (void)cudaGetLastError();
      return SD_ERR_CUDA;
    }
  }
  if (*bits & SD_DEVERR_TIMEOUT) return SD_ERR_TIMEOUT;
  return *bits ? SD_ERR_DEVICE : SD_OK;
}
