// noalloc.cu -- cer_score_static: the routing-logit scorer for callers that
// cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating routine) when they
// need the scores: a plug-in or custom-operator host that hands its operators
// no workspace and forbids device allocation once the model is loaded, or a
// real-time loop whose memory budget is frozen at start-up.  cer_score needs
// a caller-supplied workspace; this variant instead keeps the scorer's
// scratch (bias and output-weight tables plus the partial scores) in one
// file-scope static device array of kStaticScratchBytes.  That array exists
// on every GPU that loads this library, from module load until the process
// exits.
//
// The array's device address is looked up (cudaGetSymbolAddress) by the
// first call made on a device, with that device current, and again whenever
// the current context is no longer the one it was taken in (after a
// cudaDeviceReset the module is loaded afresh and the array moves).  The name
// of the array in host code is only a host-side stand-in and is never passed
// to a kernel.  Make the first call on a device before any stream capture.
//
// Every call shares the one array: calls whose work can overlap on the GPU
// (different streams, or different host threads) race on it; calls on one
// stream are ordered and safe.  The array keeps the last call's contents;
// nothing in it needs to start at zero, since every value the kernels read
// is written earlier in the same call.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/cer_api.h"
#include "kernels.h"

namespace {

constexpr size_t kStaticScratchBytes = size_t(4) << 20;  // 4 MiB

static __device__ __align__(256) unsigned char g_score_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices];
unsigned long long g_scratch_ctx[kMaxDevices];   // context the address was taken in

}  // namespace

extern "C" cer_status cer_score_static(const void* h, int B, int N, int d, const cer_scorer* core,
                                       const cer_scorer* exp, const float* t, int task, float* logits,
                                       float* probs, cudaStream_t stream) {
  if (core == nullptr) return cer::internal_fail(CER_ERR_NULL, "core scorer is NULL");
  const int exp_hidden = (task == CER_TASK_GEN && exp != nullptr) ? exp->hidden : 0;
  const size_t need = cer_score_workspace_size(B, N, core->hidden, exp_hidden, task);
  if (need > kStaticScratchBytes)
    return cer::internal_fail(CER_ERR_WORKSPACE,
                              "cer_score_static: these sizes need %zu bytes of scratch but the static scratch holds "
                              "%zu bytes; use cer_score with a caller-supplied workspace",
                              need, kStaticScratchBytes);
  // The device must be one whose module this library can load before the
  // array's address can be asked for.
  cer_status st = cer::require_supported_device();
  if (st != CER_OK) return st;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cer::internal_fail(CER_ERR_DEVICE, "cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return cer::internal_fail(CER_ERR_DEVICE, "device index %d out of range", dev);
  const unsigned long long ctx = cer::current_context_id();
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    if (g_scratch_addr[dev] == nullptr || ctx == 0 || ctx != g_scratch_ctx[dev]) {
      g_scratch_addr[dev] = nullptr;
      e = cudaGetSymbolAddress(&g_scratch_addr[dev], g_score_scratch);
      if (e != cudaSuccess) {
        g_scratch_addr[dev] = nullptr;
        return cer::internal_fail(CER_ERR_DEVICE, "cudaGetSymbolAddress(static scratch): %s", cudaGetErrorString(e));
      }
      g_scratch_ctx[dev] = cer::current_context_id();
    }
    scratch = g_scratch_addr[dev];
  }
  return cer_score(h, B, N, d, core, exp, t, task, logits, probs, scratch, kStaticScratchBytes, stream);
}
