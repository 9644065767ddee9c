// status.cuh -- device-side error codes (same values as cer_status) and the
// first-error-wins record into the per-device status word.
#pragma once

namespace cer {

enum DeviceStatus : int {
  CER_DEV_OK = 0,
  CER_DEV_NAN = 5,       // CER_ERR_NAN
  CER_DEV_TIMEOUT = 7,   // CER_ERR_TIMEOUT
  CER_DEV_INDEX = 10,    // CER_ERR_INDEX
};

__device__ __forceinline__ void record_status(int* status, int code) {
  if (status != nullptr) atomicCAS(status, 0, code);
}

}  // namespace cer
