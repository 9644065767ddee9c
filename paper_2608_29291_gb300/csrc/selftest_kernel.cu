// selftest_kernel.cu -- a check of the bounded waits every kernel of this
// library relies on (no paper counterpart: failure detection of the library
// itself).
//
// One thread waits, through the same mbar_wait / flag_wait the GEMM,
// attention and stream-K code use, but with a caller-given limit of at most
// 100 ms, either for a global flag to hold a token or for an mbarrier phase
// that completes only if the thread arrived on it first.  When the wait gives
// up the kernel records CER_DEV_TIMEOUT in the status word and returns:
// nothing else is in flight (no copy, no MMA, no tensor memory), so the
// context stays usable and the caller reads CER_ERR_TIMEOUT from
// cer_sync_status.
#include "kernels.h"
#include "ptx.cuh"
#include "status.cuh"

namespace cer {

__global__ void bounded_wait_selftest_kernel(int kind, const unsigned long long* flag, unsigned long long token,
                                             int arrive, unsigned long long limit_ns, int* status) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  abort_flag = 0;
  if (kind == 0) {
    flag_wait(flag, token, &abort_flag, status, limit_ns);
  } else {
    mbar_init(&bar, 1);
    if (arrive) mbar_arrive(&bar);
    mbar_wait(&bar, 0, &abort_flag, status, limit_ns);
  }
}

cudaError_t launch_bounded_wait_selftest(int kind, const unsigned long long* flag, unsigned long long token,
                                         int arrive, unsigned long long limit_ns, int* status, cudaStream_t stream) {
  bounded_wait_selftest_kernel<<<1, 32, 0, stream>>>(kind, flag, token, arrive, limit_ns, status);
  return cudaGetLastError();
}

}  // namespace cer
