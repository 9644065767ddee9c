// cer_api.cu -- the C ABI declared in include/cer_api.h: host-side argument
// checks, workspace carving, tensor-map encoding, per-device state (SM count,
// architecture check, the device status word) and the launch sequences.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <set>
#include <string>
#include <utility>

#include "../../include/cer_api.h"
#include "kernels.h"

namespace {

// ---------------------------------------------------------------- errors

thread_local std::string g_error;

cer_status fail(cer_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_error = buf;
  return s;
}

cer_status cuda_fail(cudaError_t e, const char* where) {
  return fail(e == cudaErrorLaunchFailure || e == cudaErrorInvalidConfiguration ? CER_ERR_LAUNCH : CER_ERR_DEVICE,
              "%s: %s", where, cudaGetErrorString(e));
}

// ---------------------------------------------------------------- per device

__device__ int g_status_word;  // first kernel-detected error on this device

constexpr int kMaxDevices = 64;

struct DeviceInfo {
  bool ready = false;
  bool supported = false;
  int n_sm = 0;
  int* status = nullptr;             // device address of g_status_word
  unsigned long long ctx = 0;        // the context that address belongs to
};

std::mutex g_dev_mu;
DeviceInfo g_dev[kMaxDevices];

cer_status device_info(DeviceInfo** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return fail(CER_ERR_DEVICE, "device index %d out of range", dev);
  const unsigned long long ctx = cer::current_context_id();
  std::lock_guard<std::mutex> lk(g_dev_mu);
  DeviceInfo& d = g_dev[dev];
  // The status word's address is looked up again whenever the context is not
  // the one it was taken in (or cannot be identified).
  if (!d.ready || (d.supported && (ctx == 0 || ctx != d.ctx))) {
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    d.supported = (major == 10 && minor == 3);
    cudaDeviceGetAttribute(&d.n_sm, cudaDevAttrMultiProcessorCount, dev);
    d.ready = false;
    if (d.supported) {
      e = cudaGetSymbolAddress(reinterpret_cast<void**>(&d.status), g_status_word);
      if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(status)");
      d.ctx = cer::current_context_id();
    }
    d.ready = true;
  }
  if (!d.supported) return fail(CER_ERR_DEVICE, "device %d is not an sm_103 GPU; this library holds sm_103a code only", dev);
  *out = &d;
  return CER_OK;
}

// ---------------------------------------------------------------- checks

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

// The GEMMs' stream-K region (partial accumulators, then flags), placed right
// after the act buffer of every FFN workspace.
size_t ffn_stream_k_bytes(long long M) {
  return M > 0 ? cer::kStreamKPartialBytes + cer::kStreamKFlagBytes : 0;
}
void carve_stream_k(char** ws, long long M, cer::FfnArgs* a) {
  if (M <= 0) return;
  a->sk.partial = reinterpret_cast<float*>(*ws);
  a->sk.flags = reinterpret_cast<unsigned long long*>(*ws + cer::kStreamKPartialBytes);
  *ws += ffn_stream_k_bytes(M);
}

#define CER_REQUIRE(cond, status, ...) \
  do {                                 \
    if (!(cond)) return fail(status, __VA_ARGS__); \
  } while (0)

#define CER_PTR(p) CER_REQUIRE((p) != nullptr, CER_ERR_NULL, "%s is NULL", #p)
// A pointer that may be NULL only when the tensor it stands for is empty.
#define CER_PTR_IF(p, nonempty) CER_REQUIRE(!(nonempty) || (p) != nullptr, CER_ERR_NULL, "%s is NULL", #p)
#define CER_ALIGN(p) CER_REQUIRE((p) == nullptr || aligned16(p), CER_ERR_ALIGN, "%s is not 16-byte aligned", #p)

struct ScoreShape {
  int Hc = 0, He = 0, gen = 0, max_partials = 0, Ht = 0;
};

cer_status check_scorer(const cer_scorer* s, const char* name, bool is_core, int* hidden) {
  if (s == nullptr) return fail(CER_ERR_NULL, "%s scorer is NULL", name);
  if (s->W1 == nullptr || s->w2 == nullptr) return fail(CER_ERR_NULL, "%s scorer W1/w2 is NULL", name);
  if (!aligned16(s->W1) || !aligned16(s->w2) || (s->b1 && !aligned16(s->b1)) || (s->U && !aligned16(s->U)))
    return fail(CER_ERR_ALIGN, "%s scorer tensors must be 16-byte aligned", name);
  if (s->hidden < 64 || s->hidden > 4096 || s->hidden % 64 != 0)
    return fail(CER_ERR_SHAPE, "%s scorer hidden=%d must be a multiple of 64 in [64, 4096]", name, s->hidden);
  if (s->n_segments < 1 || s->n_segments > 64)
    return fail(CER_ERR_SHAPE, "%s scorer n_segments=%d must be in [1, 64]", name, s->n_segments);
  if (is_core && (s->n_segments != 1 || s->U != nullptr))
    return fail(CER_ERR_SHAPE, "the core scorer is shared by all tasks: n_segments must be 1 and U NULL");
  if (s->U != nullptr && (s->emb_dim < 2 || s->emb_dim > 1024 || s->emb_dim % 2 != 0))
    return fail(CER_ERR_SHAPE, "%s scorer emb_dim=%d must be even in [2, 1024]", name, s->emb_dim);
  *hidden = s->hidden;
  return CER_OK;
}

cer_status check_score_args(const void* h, int B, int N, int d, const cer_scorer* core, const cer_scorer* exp,
                            const float* t, int task, ScoreShape* sh) {
  CER_PTR_IF(h, static_cast<long long>(B) * N > 0);
  CER_ALIGN(h);
  CER_ALIGN(t);
  CER_REQUIRE(task == CER_TASK_UND || task == CER_TASK_GEN, CER_ERR_RANGE, "task=%d is neither UND nor GEN", task);
  CER_REQUIRE(B >= 0 && N >= 0, CER_ERR_SHAPE, "B=%d N=%d must be >= 0", B, N);
  CER_REQUIRE(static_cast<long long>(B) * N < (1ll << 31), CER_ERR_SHAPE, "B*N too large");
  CER_REQUIRE(d >= 64 && d <= 16384 && d % 64 == 0, CER_ERR_SHAPE, "d=%d must be a multiple of 64 in [64, 16384]", d);
  cer_status s = check_scorer(core, "core", true, &sh->Hc);
  if (s != CER_OK) return s;
  sh->gen = (task == CER_TASK_GEN);
  if (sh->gen) {
    s = check_scorer(exp, "expansion", false, &sh->He);
    if (s != CER_OK) return s;
    CER_PTR_IF(t, B > 0);
  }
  sh->max_partials = cer::score_max_partials(sh->Hc, sh->He, sh->gen);
  CER_REQUIRE(sh->max_partials > 0, CER_ERR_SHAPE, "scorer hidden widths must be multiples of 64");
  sh->Ht = sh->Hc + (sh->gen ? sh->He : 0);
  return CER_OK;
}

size_t score_ws_bytes(int B, int N, const ScoreShape& sh) {
  return 2 * round256(static_cast<size_t>(B) * sh.Ht * sizeof(float)) +
         round256(static_cast<size_t>(sh.max_partials) * B * N * sizeof(float));
}

cer::ScoreWorkspace carve_score_ws(void* ws, int B, int N, const ScoreShape& sh) {
  char* p = static_cast<char*>(ws);
  cer::ScoreWorkspace w;
  const size_t tab = round256(static_cast<size_t>(B) * sh.Ht * sizeof(float));
  w.bias_tab = reinterpret_cast<float*>(p);
  w.w2_tab = reinterpret_cast<float*>(p + tab);
  w.partial = reinterpret_cast<float*>(p + 2 * tab);
  return w;
}

cer::ScoreArgs make_score_args(const void* h, int B, int N, int d, const cer_scorer* core, const cer_scorer* exp,
                               const float* t, const ScoreShape& sh, int* status) {
  cer::ScoreArgs a{};
  a.h = static_cast<const __nv_bfloat16*>(h);
  a.B = B;
  a.N = N;
  a.d = d;
  a.W1 = static_cast<const __nv_bfloat16*>(core->W1);
  a.b1 = core->b1;
  a.w2 = core->w2;
  a.Hc = sh.Hc;
  a.gen = sh.gen;
  a.t = t;
  a.S = 1;
  if (sh.gen) {
    a.W1e = static_cast<const __nv_bfloat16*>(exp->W1);
    a.b1e = exp->b1;
    a.w2e = exp->w2;
    a.U = static_cast<const __nv_bfloat16*>(exp->U);
    a.He = sh.He;
    a.E = exp->U ? exp->emb_dim : 0;
    a.S = exp->n_segments;
  }
  a.status = status;
  return a;
}

cer_status check_ffn_shape(int M, int d, int I, const int32_t* chan, int C) {
  CER_REQUIRE(M >= 0, CER_ERR_SHAPE, "M=%d must be >= 0", M);
  CER_REQUIRE(d >= 64 && d <= 16384 && d % 64 == 0, CER_ERR_SHAPE, "d=%d must be a multiple of 64 in [64, 16384]", d);
  CER_REQUIRE(I >= 1, CER_ERR_SHAPE, "I=%d must be >= 1", I);
  CER_REQUIRE(C >= 64 && C <= I && C % 64 == 0, CER_ERR_SHAPE, "C=%d must be a multiple of 64 in [64, I=%d]", C, I);
  CER_REQUIRE(chan != nullptr || C == I, CER_ERR_SHAPE, "chan == NULL requires C == I (C=%d, I=%d)", C, I);
  return CER_OK;
}

}  // namespace

// ---------------------------------------------------------------- internal helpers

namespace cer {

cer_status internal_fail(cer_status status, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_error = buf;
  return status;
}

static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return encode;
}

using PfnCtxGetCurrent = CUresult (*)(CUcontext*);
using PfnCtxGetId = CUresult (*)(CUcontext, unsigned long long*);

unsigned long long current_context_id() {
  static PfnCtxGetCurrent get_current = nullptr;
  static PfnCtxGetId get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fn, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<PfnCtxGetCurrent>(fn);
    fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<PfnCtxGetId>(fn);
  });
  if (get_current == nullptr || get_id == nullptr) return 0;
  CUcontext c = nullptr;
  if (get_current(&c) != CUDA_SUCCESS || c == nullptr) return 0;
  unsigned long long id = 0;
  if (get_id(c, &id) != CUDA_SUCCESS) return 0;
  return id;
}

cer_status require_supported_device() {
  DeviceInfo* d = nullptr;
  return device_info(&d);
}

bool encode_bf16_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_cols,
                    uint32_t box_rows) {
  const PFN_cuTensorMapEncodeTiled_v12000 encode = tensor_map_encoder();
  if (encode == nullptr || rows == 0 || cols == 0) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_bf16_col_blocks(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
                            uint32_t box_blocks) {
  const PFN_cuTensorMapEncodeTiled_v12000 encode = tensor_map_encoder();
  if (encode == nullptr || rows == 0 || cols == 0 || cols % 64 != 0) return false;
  // [cols / 64][rows][64]: element (r, 64 b + c) sits at coordinate (c, r, b).
  const cuuint64_t dims[3] = {64, rows, cols / 64};
  const cuuint64_t strides[2] = {cols * 2, 128};
  const cuuint32_t box[3] = {64, box_rows, box_blocks};
  const cuuint32_t estr[3] = {1, 1, 1};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

cudaError_t ensure_max_smem(const void* func, size_t bytes) {
  // A function attribute belongs to the context it was set in: remembered per
  // (context, function), and set on every call when the context cannot be
  // identified.
  static std::mutex mu;
  static std::set<std::pair<unsigned long long, const void*>> done;
  const unsigned long long ctx = current_context_id();
  std::lock_guard<std::mutex> lk(mu);
  if (ctx != 0 && done.count({ctx, func})) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
  if (e == cudaSuccess) {
    const unsigned long long now = current_context_id();
    if (now != 0) done.insert({now, func});
  }
  return e;
}

cudaError_t prefer_max_shared(const void* func) {
  static std::mutex mu;
  static std::set<std::pair<unsigned long long, const void*>> done;
  const unsigned long long ctx = current_context_id();
  std::lock_guard<std::mutex> lk(mu);
  if (ctx != 0 && done.count({ctx, func})) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(func, cudaFuncAttributePreferredSharedMemoryCarveout,
                                       static_cast<int>(cudaSharedmemCarveoutMaxShared));
  if (e == cudaSuccess) {
    const unsigned long long now = current_context_id();
    if (now != 0) done.insert({now, func});
  }
  return e;
}

}  // namespace cer

// ---------------------------------------------------------------- the ABI

extern "C" {

int cer_version(void) { return 1; }

const char* cer_get_error(void) { return g_error.c_str(); }

const char* cer_status_string(cer_status s) {
  switch (s) {
    case CER_OK: return "CER_OK";
    case CER_ERR_NULL: return "CER_ERR_NULL";
    case CER_ERR_SHAPE: return "CER_ERR_SHAPE";
    case CER_ERR_ALIGN: return "CER_ERR_ALIGN";
    case CER_ERR_RANGE: return "CER_ERR_RANGE";
    case CER_ERR_NAN: return "CER_ERR_NAN";
    case CER_ERR_DEVICE: return "CER_ERR_DEVICE";
    case CER_ERR_TIMEOUT: return "CER_ERR_TIMEOUT";
    case CER_ERR_LAUNCH: return "CER_ERR_LAUNCH";
    case CER_ERR_WORKSPACE: return "CER_ERR_WORKSPACE";
    case CER_ERR_INDEX: return "CER_ERR_INDEX";
  }
  return "CER_UNKNOWN";
}

cer_status cer_sync_status(cudaStream_t stream) {
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int v = 0;
  e = cudaMemcpy(&v, dev->status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "reading the status word");
  if (v != 0) {
    const int zero = 0;
    e = cudaMemcpy(dev->status, &zero, sizeof(int), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "clearing the status word");
    return fail(static_cast<cer_status>(v), "device reported %s", cer_status_string(static_cast<cer_status>(v)));
  }
  return CER_OK;
}

size_t cer_score_workspace_size(int B, int N, int core_hidden, int exp_hidden, int task) {
  ScoreShape sh;
  sh.Hc = core_hidden;
  sh.He = exp_hidden;
  sh.gen = (task == CER_TASK_GEN);
  sh.max_partials = cer::score_max_partials(sh.Hc, sh.He, sh.gen);
  if (sh.max_partials == 0 || B < 0 || N < 0) return 0;
  sh.Ht = sh.Hc + (sh.gen ? sh.He : 0);
  return score_ws_bytes(B, N, sh);
}

cer_status cer_score(const void* h, int B, int N, int d, const cer_scorer* core, const cer_scorer* exp,
                     const float* t, int task, float* logits, float* probs, void* workspace,
                     size_t workspace_bytes, cudaStream_t stream) {
  ScoreShape sh;
  cer_status s = check_score_args(h, B, N, d, core, exp, t, task, &sh);
  if (s != CER_OK) return s;
  CER_PTR_IF(logits, static_cast<long long>(B) * N > 0);
  CER_ALIGN(logits);
  CER_ALIGN(probs);
  CER_ALIGN(workspace);
  const size_t need = score_ws_bytes(B, N, sh);
  CER_REQUIRE(workspace != nullptr && workspace_bytes >= need, CER_ERR_WORKSPACE,
              "workspace of %zu bytes needed, %zu given", need, workspace_bytes);
  DeviceInfo* dev = nullptr;
  if ((s = device_info(&dev)) != CER_OK) return s;
  if (B == 0 || N == 0) return CER_OK;
  cer::ScoreWorkspace ws = carve_score_ws(workspace, B, N, sh);
  cer::ScoreArgs a = make_score_args(h, B, N, d, core, exp, t, sh, dev->status);
  int n_partials = 0;
  cudaError_t e = cer::launch_score(a, ws, nullptr, dev->n_sm, stream, &n_partials);
  if (e != cudaSuccess) return cuda_fail(e, "scorer launch");
  e = cer::launch_score_reduce(ws.partial, n_partials, static_cast<size_t>(B) * N, logits, probs, dev->n_sm,
                               stream);
  if (e != cudaSuccess) return cuda_fail(e, "score reduce launch");
  return CER_OK;
}

cer_status cer_select_topk(const float* logits, int B, int N, int r0, int r1, int K, int32_t* idx, uint8_t* mask,
                           cudaStream_t stream) {
  CER_PTR_IF(logits, static_cast<long long>(B) * N > 0);
  CER_PTR_IF(idx, static_cast<long long>(B) * (K + N - (r1 - r0)) > 0);
  CER_ALIGN(logits);
  CER_ALIGN(idx);
  CER_ALIGN(mask);
  CER_REQUIRE(B >= 0 && N >= 0 && N <= cer::kTopkMaxN, CER_ERR_SHAPE, "B=%d N=%d (N <= %d)", B, N, cer::kTopkMaxN);
  CER_REQUIRE(0 <= r0 && r0 <= r1 && r1 <= N, CER_ERR_RANGE, "routable range [%d, %d) not inside [0, %d]", r0, r1, N);
  CER_REQUIRE(0 <= K && K <= r1 - r0, CER_ERR_RANGE, "K=%d not in [0, N_r=%d]", K, r1 - r0);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cer::TopkArgs a{};
  a.src = logits;
  a.n_chunks = 1;
  a.chunk_stride = 0;
  a.B = B;
  a.N = N;
  a.r0 = r0;
  a.r1 = r1;
  a.K = K;
  a.idx = idx;
  a.mask = mask;
  a.status = dev->status;
  cudaError_t e = cer::launch_topk(a, stream);
  if (e != cudaSuccess) return cuda_fail(e, "top-K launch");
  return CER_OK;
}

cer_status cer_gather(const void* h, int B, int N, int d, const int32_t* idx, int k_tot, void* X,
                      cudaStream_t stream) {
  CER_PTR_IF(h, static_cast<long long>(B) * N > 0);
  CER_PTR_IF(idx, static_cast<long long>(B) * k_tot > 0);
  CER_PTR_IF(X, static_cast<long long>(B) * k_tot > 0);
  CER_ALIGN(h);
  CER_ALIGN(idx);
  CER_ALIGN(X);
  CER_REQUIRE(B >= 0 && N >= 0 && k_tot >= 0 && k_tot <= N, CER_ERR_SHAPE, "B=%d N=%d k_tot=%d", B, N, k_tot);
  CER_REQUIRE(d > 0 && d % 8 == 0, CER_ERR_SHAPE, "d=%d must be a positive multiple of 8", d);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cudaError_t e = cer::launch_gather(static_cast<const __nv_bfloat16*>(h), B, N, d, idx, k_tot,
                                     static_cast<__nv_bfloat16*>(X), dev->status, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "gather launch");
  return CER_OK;
}

cer_status cer_scatter_add(void* h, int B, int N, int d, const int32_t* idx, int k_tot, const void* Y,
                           cudaStream_t stream) {
  CER_PTR_IF(h, static_cast<long long>(B) * N > 0);
  CER_PTR_IF(idx, static_cast<long long>(B) * k_tot > 0);
  CER_PTR_IF(Y, static_cast<long long>(B) * k_tot > 0);
  CER_ALIGN(h);
  CER_ALIGN(idx);
  CER_ALIGN(Y);
  CER_REQUIRE(B >= 0 && N >= 0 && k_tot >= 0 && k_tot <= N, CER_ERR_SHAPE, "B=%d N=%d k_tot=%d", B, N, k_tot);
  CER_REQUIRE(d > 0 && d % 8 == 0, CER_ERR_SHAPE, "d=%d must be a positive multiple of 8", d);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cudaError_t e = cer::launch_scatter_add(static_cast<__nv_bfloat16*>(h), B, N, d, idx, k_tot,
                                          static_cast<const __nv_bfloat16*>(Y), dev->status, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "scatter-add launch");
  return CER_OK;
}

cer_status cer_scatter_add_checked(void* h, int B, int N, int d, const int32_t* idx, int k_tot, const void* Y,
                                   cudaStream_t stream) {
  CER_PTR_IF(h, static_cast<long long>(B) * N > 0);
  CER_PTR_IF(idx, static_cast<long long>(B) * k_tot > 0);
  CER_PTR_IF(Y, static_cast<long long>(B) * k_tot > 0);
  CER_ALIGN(h);
  CER_ALIGN(idx);
  CER_ALIGN(Y);
  CER_REQUIRE(B >= 0 && N >= 0 && k_tot >= 0 && k_tot <= N, CER_ERR_SHAPE, "B=%d N=%d k_tot=%d", B, N, k_tot);
  CER_REQUIRE(N <= cer::kScatterCheckedMaxN, CER_ERR_SHAPE, "N=%d exceeds %d for the checked scatter-add", N,
              cer::kScatterCheckedMaxN);
  CER_REQUIRE(d > 0 && d % 8 == 0, CER_ERR_SHAPE, "d=%d must be a positive multiple of 8", d);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cudaError_t e = cer::launch_scatter_add_checked(static_cast<__nv_bfloat16*>(h), B, N, d, idx, k_tot,
                                                  static_cast<const __nv_bfloat16*>(Y), dev->status, stream);
  if (e != cudaSuccess) return cuda_fail(e, "checked scatter-add launch");
  return CER_OK;
}

cer_status cer_selftest_bounded_wait(int kind, const unsigned long long* flag, unsigned long long token, int arrive,
                                     int limit_us, cudaStream_t stream) {
  CER_REQUIRE(kind == 0 || kind == 1, CER_ERR_RANGE, "kind=%d must be 0 (flag) or 1 (mbarrier)", kind);
  CER_REQUIRE(kind == 1 || flag != nullptr, CER_ERR_NULL, "flag is NULL");
  CER_REQUIRE(flag == nullptr || (reinterpret_cast<uintptr_t>(flag) & 7u) == 0, CER_ERR_ALIGN,
              "flag is not 8-byte aligned");
  CER_REQUIRE(limit_us >= 1 && limit_us <= 100000, CER_ERR_RANGE, "limit_us=%d must be in [1, 100000]", limit_us);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cudaError_t e = cer::launch_bounded_wait_selftest(kind, flag, token, arrive ? 1 : 0,
                                                    static_cast<unsigned long long>(limit_us) * 1000ull, dev->status,
                                                    stream);
  if (e != cudaSuccess) return cuda_fail(e, "bounded-wait self-test launch");
  return CER_OK;
}

cer_status cer_pack_ffn_weights(const void* Wg, const void* Wu, const void* WdT, int I, int d, const int32_t* chan,
                                int C, void* Wg_out, void* Wu_out, void* WdT_out, cudaStream_t stream) {
  CER_PTR(Wg);
  CER_PTR(Wu);
  CER_PTR(WdT);
  CER_PTR(chan);
  CER_PTR(Wg_out);
  CER_PTR(Wu_out);
  CER_PTR(WdT_out);
  CER_ALIGN(Wg);
  CER_ALIGN(Wu);
  CER_ALIGN(WdT);
  CER_ALIGN(chan);
  CER_ALIGN(Wg_out);
  CER_ALIGN(Wu_out);
  CER_ALIGN(WdT_out);
  CER_REQUIRE(d > 0 && d % 8 == 0, CER_ERR_SHAPE, "d=%d must be a positive multiple of 8", d);
  CER_REQUIRE(I >= 1 && C >= 1 && C <= I, CER_ERR_SHAPE, "C=%d must be in [1, I=%d]", C, I);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  const void* src[3] = {Wg, Wu, WdT};
  void* dst[3] = {Wg_out, Wu_out, WdT_out};
  for (int i = 0; i < 3; ++i) {
    cudaError_t e = cer::launch_gather(static_cast<const __nv_bfloat16*>(src[i]), 1, I, d, chan, C,
                                       static_cast<__nv_bfloat16*>(dst[i]), dev->status, dev->n_sm, stream);
    if (e != cudaSuccess) return cuda_fail(e, "weight pack launch");
  }
  return CER_OK;
}

size_t cer_routed_ffn_workspace_size(int M, int d, int C, int with_chan) {
  if (M < 0 || d < 0 || C < 0) return 0;
  size_t ws = round256(static_cast<size_t>(M) * C * 2) + ffn_stream_k_bytes(M);
  if (with_chan) ws += 3 * round256(static_cast<size_t>(C) * d * 2);
  return ws;
}

namespace {

// Kept-channel slices of the FFN weights: the given arrays when chan is NULL
// (they already hold exactly C channels), else packed into `ws`.
cer_status ffn_weight_slices(const void* Wg, const void* Wu, const void* WdT, int I, int d, const int32_t* chan,
                             int C, char** ws, const __nv_bfloat16* out[3], DeviceInfo* dev, cudaStream_t stream) {
  if (chan == nullptr) {
    out[0] = static_cast<const __nv_bfloat16*>(Wg);
    out[1] = static_cast<const __nv_bfloat16*>(Wu);
    out[2] = static_cast<const __nv_bfloat16*>(WdT);
    return CER_OK;
  }
  const void* src[3] = {Wg, Wu, WdT};
  const size_t slice = round256(static_cast<size_t>(C) * d * 2);
  for (int i = 0; i < 3; ++i) {
    __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(*ws);
    *ws += slice;
    cudaError_t e = cer::launch_gather(static_cast<const __nv_bfloat16*>(src[i]), 1, I, d, chan, C, dst, dev->status,
                                       dev->n_sm, stream);
    if (e != cudaSuccess) return cuda_fail(e, "weight pack launch");
    out[i] = dst;
  }
  return CER_OK;
}

}  // namespace

cer_status cer_routed_ffn(const void* X, int M, int d, const void* Wg, const void* Wu, const void* WdT, int I,
                          const int32_t* chan, int C, void* Y, void* workspace, size_t workspace_bytes,
                          cudaStream_t stream) {
  CER_PTR_IF(X, M > 0);
  CER_PTR(Wg);
  CER_PTR(Wu);
  CER_PTR(WdT);
  CER_PTR_IF(Y, M > 0);
  CER_ALIGN(X);
  CER_ALIGN(Wg);
  CER_ALIGN(Wu);
  CER_ALIGN(WdT);
  CER_ALIGN(chan);
  CER_ALIGN(Y);
  CER_ALIGN(workspace);
  cer_status s = check_ffn_shape(M, d, I, chan, C);
  if (s != CER_OK) return s;
  const size_t need = cer_routed_ffn_workspace_size(M, d, C, chan != nullptr);
  CER_REQUIRE(M == 0 || (workspace != nullptr && workspace_bytes >= need), CER_ERR_WORKSPACE,
              "workspace of %zu bytes needed, %zu given", need, workspace_bytes);
  DeviceInfo* dev = nullptr;
  if ((s = device_info(&dev)) != CER_OK) return s;
  if (M == 0) return CER_OK;
  char* ws = static_cast<char*>(workspace);
  cer::FfnArgs a{};
  a.act = reinterpret_cast<__nv_bfloat16*>(ws);
  ws += round256(static_cast<size_t>(M) * C * 2);
  carve_stream_k(&ws, M, &a);
  const __nv_bfloat16* w[3];
  if ((s = ffn_weight_slices(Wg, Wu, WdT, I, d, chan, C, &ws, w, dev, stream)) != CER_OK) return s;
  a.X = static_cast<const __nv_bfloat16*>(X);
  a.M = M;
  a.d = d;
  a.C = C;
  a.Wg = w[0];
  a.Wu = w[1];
  a.WdT = w[2];
  a.Y = static_cast<__nv_bfloat16*>(Y);
  a.scatter = 0;
  a.status = dev->status;
  cudaError_t e = cer::launch_ffn_gateup(a, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "gate/up GEMM launch");
  e = cer::launch_ffn_down(a, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "down GEMM launch");
  return CER_OK;
}

size_t cer_routed_block_workspace_size(int B, int N, int d, int core_hidden, int exp_hidden, int task, int r0,
                                       int r1, int K, int C, int with_chan) {
  const size_t sc = cer_score_workspace_size(B, N, core_hidden, exp_hidden, task);
  if (sc == 0) return 0;
  if (B < 0 || N < 0 || d < 0 || r0 < 0 || r1 < r0 || r1 > N || K < 0 || K > r1 - r0 || C < 0) return 0;
  const size_t k_tot = static_cast<size_t>(K) + (N - (r1 - r0));
  const size_t M = static_cast<size_t>(B) * k_tot;
  return sc + round256(M * sizeof(int32_t)) + round256(M * d * 2) + cer_routed_ffn_workspace_size(
                                                                          static_cast<int>(M), d, C, with_chan);
}

}  // extern "C"

namespace {

// The UCS FFN gate of the fused block (Sec. 3.4 (2)): the FFN weights hold
// all I channels with the C_keep kept ones first; the gate/up GEMM runs over
// all of them, Eq. 8 / Eq. 9 give the leakage of the pruned tail, and the
// down GEMM contracts C_keep or I channels accordingly.
struct GateArgs {
  int C_keep;
  const float* norms;
  float delta;
  float* saliency;
  float* leakage;
  uint8_t* use_pruned;
};

size_t gate_ws_bytes(long long M, int I) {
  const size_t n_parts = 2 * static_cast<size_t>((M + 127) / 128);
  return round256(n_parts * I * sizeof(float)) + round256(2 * static_cast<size_t>((I + 255) / 256) * sizeof(float)) +
         256;  // + leakage and decision when the caller passes NULL
}

cer_status check_gate(const GateArgs* g, int I, int C) {
  if (g == nullptr) return CER_OK;
  CER_PTR(g->norms);
  CER_ALIGN(g->norms);
  CER_ALIGN(g->saliency);
  CER_ALIGN(g->leakage);
  CER_REQUIRE(C == I, CER_ERR_SHAPE, "the gated FFN takes all I channels (C=%d, I=%d)", C, I);
  CER_REQUIRE(g->C_keep >= 64 && g->C_keep <= I && g->C_keep % 64 == 0, CER_ERR_SHAPE,
              "C_keep=%d must be a multiple of 64 in [64, I=%d]", g->C_keep, I);
  return CER_OK;
}

// Saliency, leakage and the decision from the gate/up GEMM's column sums; the
// decision flag then drives the down GEMM's contraction length (fa.use_small_k).
// gate_ws: colsum | per-block partial sums | leakage / decision fallbacks.
cer_status run_gate(const GateArgs& g, cer::FfnArgs& fa, char* gate_ws, cudaStream_t stream) {
  const int n_parts = 2 * ((fa.M + 127) / 128);
  char* p = gate_ws + round256(static_cast<size_t>(n_parts) * fa.C * sizeof(float));
  float* part_ws = reinterpret_cast<float*>(p);
  p += round256(2 * static_cast<size_t>((fa.C + 255) / 256) * sizeof(float));
  float* leak = g.leakage ? g.leakage : reinterpret_cast<float*>(p);
  uint8_t* flag = g.use_pruned ? g.use_pruned : reinterpret_cast<uint8_t*>(p + 16);
  cudaError_t e = cer::launch_ffn_gate(fa.colsum, n_parts, fa.M, fa.C, g.C_keep, g.norms, g.delta, g.saliency,
                                       part_ws, leak, flag, stream);
  if (e != cudaSuccess) return cuda_fail(e, "FFN gate launch");
  fa.use_small_k = flag;
  return CER_OK;
}

cer_status routed_block_impl(void* h, void* out, int B, int N, int d, const cer_scorer* core, const cer_scorer* exp,
                             const float* t, int task, int r0, int r1, int K, const void* Wg, const void* Wu,
                             const void* WdT, int I, const int32_t* chan, int C, float* logits, int32_t* idx,
                             uint8_t* mask, void* workspace, size_t workspace_bytes, cudaEvent_t* stage_events,
                             int n_stage_events, const GateArgs* gate, cudaStream_t stream) {
  ScoreShape sh;
  cer_status s = check_score_args(h, B, N, d, core, exp, t, task, &sh);
  if (s != CER_OK) return s;
  CER_PTR(Wg);
  CER_PTR(Wu);
  CER_PTR(WdT);
  CER_ALIGN(out);
  CER_ALIGN(Wg);
  CER_ALIGN(Wu);
  CER_ALIGN(WdT);
  CER_ALIGN(chan);
  CER_ALIGN(logits);
  CER_ALIGN(idx);
  CER_ALIGN(mask);
  CER_ALIGN(workspace);
  CER_REQUIRE(N <= cer::kTopkMaxN, CER_ERR_SHAPE, "N=%d exceeds %d", N, cer::kTopkMaxN);
  CER_REQUIRE(0 <= r0 && r0 <= r1 && r1 <= N, CER_ERR_RANGE, "routable range [%d, %d) not inside [0, %d]", r0, r1, N);
  CER_REQUIRE(0 <= K && K <= r1 - r0, CER_ERR_RANGE, "K=%d not in [0, N_r=%d]", K, r1 - r0);
  const int k_tot = K + N - (r1 - r0);
  const long long M64 = static_cast<long long>(B) * k_tot;
  CER_REQUIRE(M64 < (1ll << 31), CER_ERR_SHAPE, "too many kept rows");
  s = check_ffn_shape(static_cast<int>(M64), d, I, chan, C);
  if (s != CER_OK) return s;
  if ((s = check_gate(gate, I, C)) != CER_OK) return s;
  CER_REQUIRE(gate == nullptr || chan == nullptr, CER_ERR_RANGE, "the gated FFN takes packed weights (chan NULL)");
  CER_REQUIRE(stage_events == nullptr || n_stage_events == 6, CER_ERR_RANGE,
              "stage_events needs exactly 6 events (got %d)", n_stage_events);
  const size_t need = cer_routed_block_workspace_size(B, N, d, sh.Hc, sh.He, task, r0, r1, K, C, chan != nullptr) +
                      (gate ? gate_ws_bytes(M64, I) : 0);
  CER_REQUIRE(workspace != nullptr && workspace_bytes >= need, CER_ERR_WORKSPACE,
              "workspace of %zu bytes needed, %zu given", need, workspace_bytes);
  const bool in_place = (out == nullptr || out == h);
  const size_t hbytes = static_cast<size_t>(B) * N * d * 2;
  if (!in_place) {
    const char* a0 = static_cast<const char*>(h);
    const char* b0 = static_cast<const char*>(out);
    CER_REQUIRE(b0 + hbytes <= a0 || a0 + hbytes <= b0, CER_ERR_RANGE, "out overlaps h without being equal to it");
  }
  DeviceInfo* dev = nullptr;
  if ((s = device_info(&dev)) != CER_OK) return s;

  auto mark = [&](int i) -> cudaError_t {
    return stage_events ? cudaEventRecord(stage_events[i], stream) : cudaSuccess;
  };
  cudaError_t e = mark(0);
  if (e != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
  void* dst = in_place ? h : out;
  if (!in_place && hbytes) {
    e = cudaMemcpyAsync(out, h, hbytes, cudaMemcpyDeviceToDevice, stream);  // bypass rows
    if (e != cudaSuccess) return cuda_fail(e, "bypass copy");
  }
  if (B == 0 || N == 0) {
    for (int i = 1; i < 6; ++i) mark(i);
    return CER_OK;
  }
  char* ws = static_cast<char*>(workspace);
  cer::ScoreWorkspace sws = carve_score_ws(ws, B, N, sh);
  ws += score_ws_bytes(B, N, sh);
  int32_t* idx_buf = idx ? idx : reinterpret_cast<int32_t*>(ws);
  ws += round256(static_cast<size_t>(M64) * sizeof(int32_t));
  __nv_bfloat16* X = reinterpret_cast<__nv_bfloat16*>(ws);
  ws += round256(static_cast<size_t>(M64) * d * 2);
  __nv_bfloat16* act = reinterpret_cast<__nv_bfloat16*>(ws);
  ws += round256(static_cast<size_t>(M64) * C * 2);
  cer::FfnArgs fa{};
  carve_stream_k(&ws, M64, &fa);
  char* gate_ws = ws + (chan ? 3 * round256(static_cast<size_t>(C) * d * 2) : 0);

  // S1: scorer GEMM -> partial sums
  cer::ScoreArgs sa = make_score_args(h, B, N, d, core, exp, t, sh, dev->status);
  int n_partials = 0;
  e = cer::launch_score(sa, sws, M64 > 0 ? &fa.sk : nullptr, dev->n_sm, stream, &n_partials);
  if (e != cudaSuccess) return cuda_fail(e, "scorer launch");
  if ((e = mark(1)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");

  // S2: reduce partial sums + top-K keep list
  cer::TopkArgs ta{};
  ta.src = sws.partial;
  ta.n_chunks = n_partials;
  ta.chunk_stride = static_cast<size_t>(B) * N;
  ta.B = B;
  ta.N = N;
  ta.r0 = r0;
  ta.r1 = r1;
  ta.K = K;
  ta.logits_out = logits;
  ta.idx = idx_buf;
  ta.mask = mask;
  ta.status = dev->status;
  e = cer::launch_topk(ta, stream);
  if (e != cudaSuccess) return cuda_fail(e, "top-K launch");
  if ((e = mark(2)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");

  // S3: pack the kept rows (and, if a channel list is given, the kept weight rows)
  const __nv_bfloat16* w[3];
  if ((s = ffn_weight_slices(Wg, Wu, WdT, I, d, chan, C, &ws, w, dev, stream)) != CER_OK) return s;
  e = cer::launch_gather(static_cast<const __nv_bfloat16*>(h), B, N, d, idx_buf, k_tot, X, dev->status, dev->n_sm,
                         stream);
  if (e != cudaSuccess) return cuda_fail(e, "gather launch");
  if ((e = mark(3)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");

  // S4: gate/up GEMM with the SwiGLU epilogue
  fa.X = X;
  fa.M = static_cast<int>(M64);
  fa.d = d;
  fa.C = C;
  fa.Wg = w[0];
  fa.Wu = w[1];
  fa.WdT = w[2];
  fa.act = act;
  fa.h = static_cast<const __nv_bfloat16*>(h);
  fa.out = static_cast<__nv_bfloat16*>(dst);
  fa.idx = idx_buf;
  fa.N = N;
  fa.k_tot = k_tot;
  fa.scatter = 1;
  fa.status = dev->status;
  if (gate) {
    fa.colsum = reinterpret_cast<float*>(gate_ws);
    fa.C_small = gate->C_keep;
  }
  if (M64 > 0) {
    e = cer::launch_ffn_gateup(fa, dev->n_sm, stream);
    if (e != cudaSuccess) return cuda_fail(e, "gate/up GEMM launch");
  }
  if (gate) {
    if ((s = run_gate(*gate, fa, gate_ws, stream)) != CER_OK) return s;
  }
  if ((e = mark(4)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");

  // S4+S5: down GEMM with the unpack (scatter-add into the residual) fused
  if (M64 > 0) {
    e = cer::launch_ffn_down(fa, dev->n_sm, stream);
    if (e != cudaSuccess) return cuda_fail(e, "down GEMM launch");
  }
  if ((e = mark(5)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
  return CER_OK;
}

}  // namespace

extern "C" {

cer_status cer_routed_block(void* h, void* out, int B, int N, int d, const cer_scorer* core, const cer_scorer* exp,
                            const float* t, int task, int r0, int r1, int K, const void* Wg, const void* Wu,
                            const void* WdT, int I, const int32_t* chan, int C, float* logits, int32_t* idx,
                            uint8_t* mask, void* workspace, size_t workspace_bytes, cudaEvent_t* stage_events,
                            int n_stage_events, cudaStream_t stream) {
  return routed_block_impl(h, out, B, N, d, core, exp, t, task, r0, r1, K, Wg, Wu, WdT, I, chan, C, logits, idx,
                           mask, workspace, workspace_bytes, stage_events, n_stage_events, nullptr, stream);
}

size_t cer_routed_block_gated_workspace_size(int B, int N, int d, int core_hidden, int exp_hidden, int task, int r0,
                                             int r1, int K, int I) {
  const size_t base = cer_routed_block_workspace_size(B, N, d, core_hidden, exp_hidden, task, r0, r1, K, I, 0);
  if (base == 0) return 0;
  const long long M = static_cast<long long>(B) * (K + N - (r1 - r0));
  return base + gate_ws_bytes(M, I);
}

cer_status cer_routed_block_gated(void* h, void* out, int B, int N, int d, const cer_scorer* core,
                                  const cer_scorer* exp, const float* t, int task, int r0, int r1, int K,
                                  const void* Wg, const void* Wu, const void* WdT, int I, int C_keep,
                                  const float* norms, float delta, float* saliency, float* leakage,
                                  uint8_t* use_pruned, float* logits, int32_t* idx, uint8_t* mask, void* workspace,
                                  size_t workspace_bytes, cudaEvent_t* stage_events, int n_stage_events,
                                  cudaStream_t stream) {
  GateArgs g{C_keep, norms, delta, saliency, leakage, use_pruned};
  return routed_block_impl(h, out, B, N, d, core, exp, t, task, r0, r1, K, Wg, Wu, WdT, I, nullptr, I, logits, idx,
                           mask, workspace, workspace_bytes, stage_events, n_stage_events, &g, stream);
}

cer_status cer_ffn_channel_norms(const void* WdT, int I, int d, float* norms, cudaStream_t stream) {
  CER_PTR(WdT);
  CER_PTR(norms);
  CER_ALIGN(WdT);
  CER_ALIGN(norms);
  CER_REQUIRE(I >= 1 && d > 0 && d % 8 == 0, CER_ERR_SHAPE, "I=%d d=%d (d a positive multiple of 8)", I, d);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cudaError_t e = cer::launch_row_norms(static_cast<const __nv_bfloat16*>(WdT), I, d, norms, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "channel-norm launch");
  return CER_OK;
}

size_t cer_routed_ffn_gated_workspace_size(int M, int d, int I) {
  if (M < 0 || d < 0 || I < 0) return 0;
  return cer_routed_ffn_workspace_size(M, d, I, 0) + gate_ws_bytes(M, I);
}

cer_status cer_routed_ffn_gated(const void* X, int M, int d, const void* Wg, const void* Wu, const void* WdT, int I,
                                int C_keep, const float* norms, float delta, void* Y, float* saliency,
                                float* leakage, uint8_t* use_pruned, void* workspace, size_t workspace_bytes,
                                cudaStream_t stream) {
  CER_PTR_IF(X, M > 0);
  CER_PTR(Wg);
  CER_PTR(Wu);
  CER_PTR(WdT);
  CER_PTR_IF(Y, M > 0);
  CER_ALIGN(X);
  CER_ALIGN(Wg);
  CER_ALIGN(Wu);
  CER_ALIGN(WdT);
  CER_ALIGN(Y);
  CER_ALIGN(workspace);
  cer_status s = check_ffn_shape(M, d, I, nullptr, I);
  if (s != CER_OK) return s;
  GateArgs g{C_keep, norms, delta, saliency, leakage, use_pruned};
  if ((s = check_gate(&g, I, I)) != CER_OK) return s;
  const size_t need = cer_routed_ffn_gated_workspace_size(M, d, I);
  CER_REQUIRE(M == 0 || (workspace != nullptr && workspace_bytes >= need), CER_ERR_WORKSPACE,
              "workspace of %zu bytes needed, %zu given", need, workspace_bytes);
  DeviceInfo* dev = nullptr;
  if ((s = device_info(&dev)) != CER_OK) return s;
  if (M == 0) return CER_OK;
  char* ws = static_cast<char*>(workspace);
  cer::FfnArgs a{};
  a.act = reinterpret_cast<__nv_bfloat16*>(ws);
  ws += round256(static_cast<size_t>(M) * I * 2);
  carve_stream_k(&ws, M, &a);
  a.X = static_cast<const __nv_bfloat16*>(X);
  a.M = M;
  a.d = d;
  a.C = I;
  a.C_small = C_keep;
  a.Wg = static_cast<const __nv_bfloat16*>(Wg);
  a.Wu = static_cast<const __nv_bfloat16*>(Wu);
  a.WdT = static_cast<const __nv_bfloat16*>(WdT);
  a.Y = static_cast<__nv_bfloat16*>(Y);
  a.scatter = 0;
  a.colsum = reinterpret_cast<float*>(ws);
  a.status = dev->status;
  cudaError_t e = cer::launch_ffn_gateup(a, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "gate/up GEMM launch");
  if ((s = run_gate(g, a, ws, stream)) != CER_OK) return s;
  e = cer::launch_ffn_down(a, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "down GEMM launch");
  return CER_OK;
}

cer_status cer_drop_set_stats(const uint8_t* mask_t, const uint8_t* mask_ref, int B, int N, int r0, int r1,
                              float* jaccard, float* j_rand, float* rda, int32_t* counts, cudaStream_t stream) {
  const bool any = static_cast<long long>(B) * N > 0;
  CER_PTR_IF(mask_t, any);
  CER_PTR_IF(mask_ref, any);
  CER_PTR_IF(jaccard, B > 0);
  CER_ALIGN(mask_t);
  CER_ALIGN(mask_ref);
  CER_ALIGN(jaccard);
  CER_ALIGN(j_rand);
  CER_ALIGN(rda);
  CER_ALIGN(counts);
  CER_REQUIRE(B >= 0 && N >= 0, CER_ERR_SHAPE, "B=%d N=%d must be >= 0", B, N);
  CER_REQUIRE(0 <= r0 && r0 <= r1 && r1 <= N, CER_ERR_RANGE, "routable range [%d, %d) not inside [0, %d]", r0, r1, N);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cudaError_t e = cer::launch_drop_stats(mask_t, mask_ref, B, N, r0, r1, jaccard, j_rand, rda, counts, stream);
  if (e != cudaSuccess) return cuda_fail(e, "drop-set statistics launch");
  return CER_OK;
}

size_t cer_redundancy_gap_workspace_size(int B, int N) {
  if (B < 0 || N < 0) return 0;
  return round256(static_cast<size_t>(B) * N * sizeof(float));
}

cer_status cer_redundancy_gap(const void* h_in, const void* h_out, const uint8_t* mask, int B, int N, int d,
                              float delta, float* gap, uint8_t* skip, void* workspace, size_t workspace_bytes,
                              cudaStream_t stream) {
  const bool any = static_cast<long long>(B) * N > 0;
  CER_PTR_IF(h_in, any);
  CER_PTR_IF(h_out, any);
  CER_PTR_IF(mask, any);
  CER_PTR_IF(gap, B > 0);
  CER_ALIGN(h_in);
  CER_ALIGN(h_out);
  CER_ALIGN(mask);
  CER_ALIGN(gap);
  CER_ALIGN(skip);
  CER_ALIGN(workspace);
  CER_REQUIRE(B >= 0 && N >= 0, CER_ERR_SHAPE, "B=%d N=%d must be >= 0", B, N);
  CER_REQUIRE(d > 0 && d % 8 == 0, CER_ERR_SHAPE, "d=%d must be a positive multiple of 8", d);
  const size_t need = cer_redundancy_gap_workspace_size(B, N);
  CER_REQUIRE(!any || (workspace != nullptr && workspace_bytes >= need), CER_ERR_WORKSPACE,
              "workspace of %zu bytes needed, %zu given", need, workspace_bytes);
  DeviceInfo* dev = nullptr;
  cer_status s = device_info(&dev);
  if (s != CER_OK) return s;
  cudaError_t e = cer::launch_redundancy_gap(static_cast<const __nv_bfloat16*>(h_in),
                                             static_cast<const __nv_bfloat16*>(h_out), mask, B, N, d, delta, gap,
                                             skip, static_cast<float*>(workspace), dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "redundancy-gap launch");
  return CER_OK;
}

namespace {

cer_status check_qkv(int B, int L, int Hq, int Hkv) {
  CER_REQUIRE(B >= 0 && L >= 0, CER_ERR_SHAPE, "B=%d L=%d must be >= 0", B, L);
  CER_REQUIRE(Hq >= 1 && Hkv >= 1 && Hq % Hkv == 0 && Hq + 2 * Hkv <= 1024, CER_ERR_SHAPE,
              "Hq=%d, Hkv=%d: need Hq, Hkv >= 1, Hq a multiple of Hkv, Hq + 2 Hkv <= 1024", Hq, Hkv);
  CER_REQUIRE(static_cast<long long>(B) * L < (1LL << 31), CER_ERR_SHAPE, "B*L=%lld rows exceed 2^31",
              static_cast<long long>(B) * L);
  return CER_OK;
}

}  // namespace

cer_status cer_rope_packed(void* qkv, int B, int L, int Hq, int Hkv, const int32_t* pos, double base,
                           cudaStream_t stream) {
  const bool any = static_cast<long long>(B) * L > 0;
  CER_PTR_IF(qkv, any);
  CER_PTR_IF(pos, any);
  CER_ALIGN(qkv);
  CER_ALIGN(pos);
  cer_status s = check_qkv(B, L, Hq, Hkv);
  if (s != CER_OK) return s;
  CER_REQUIRE(base > 1.0 && std::isfinite(base), CER_ERR_RANGE, "rotary base %g must be finite and > 1", base);
  DeviceInfo* dev = nullptr;
  if ((s = device_info(&dev)) != CER_OK) return s;
  if (!any) return CER_OK;
  cer::RopeFreqTable ft;
  for (int j = 0; j < cer::kHeadDim / 2; ++j)
    ft.g[j] = std::pow(base, -2.0 * j / cer::kHeadDim) / (2.0 * M_PI);
  cudaError_t e = cer::launch_rope(static_cast<__nv_bfloat16*>(qkv), static_cast<long long>(B) * L, Hq, Hkv, pos,
                                   ft, dev->status, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "rotary embedding launch");
  return CER_OK;
}

cer_status cer_packed_attention(const void* qkv, int B, int L, int Hq, int Hkv, int causal, void* out,
                                cudaStream_t stream) {
  const bool any = static_cast<long long>(B) * L > 0;
  CER_PTR_IF(qkv, any);
  CER_PTR_IF(out, any);
  CER_ALIGN(qkv);
  CER_ALIGN(out);
  cer_status s = check_qkv(B, L, Hq, Hkv);
  if (s != CER_OK) return s;
  CER_REQUIRE(causal == 0 || causal == 1, CER_ERR_RANGE, "causal=%d must be 0 or 1", causal);
  DeviceInfo* dev = nullptr;
  if ((s = device_info(&dev)) != CER_OK) return s;
  if (!any) return CER_OK;
  cudaError_t e = cer::launch_packed_attention(static_cast<const __nv_bfloat16*>(qkv), B, L, Hq, Hkv, causal,
                                               static_cast<__nv_bfloat16*>(out), dev->status, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "packed attention launch");
  return CER_OK;
}

size_t cer_routed_attention_workspace_size(int B, int L, int d, int Hq, int Hkv) {
  if (B < 0 || L < 0 || d < 0 || Hq < 1 || Hkv < 1) return 0;
  const long long M = static_cast<long long>(B) * L;
  const size_t width = static_cast<size_t>(Hq + 2 * Hkv) * cer::kHeadDim;
  return round256(static_cast<size_t>(M) * d * 2) + round256(static_cast<size_t>(M) * width * 2) +
         round256(static_cast<size_t>(M) * Hq * cer::kHeadDim * 2) +
         round256(static_cast<size_t>(M) * (cer::kHeadDim / 2) * sizeof(float2)) + ffn_stream_k_bytes(M);
}

cer_status cer_routed_attention(void* h, void* out, int B, int N, int d, const int32_t* idx, int L,
                                const void* WqkvT, const void* WoT, int Hq, int Hkv, int causal, double base,
                                void* qkv, void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  const long long M64 = static_cast<long long>(B) * L;
  const bool any_h = static_cast<long long>(B) * N > 0;
  CER_PTR_IF(h, any_h);
  CER_PTR_IF(idx, M64 > 0);
  CER_PTR(WqkvT);
  CER_PTR(WoT);
  CER_ALIGN(h);
  CER_ALIGN(out);
  CER_ALIGN(idx);
  CER_ALIGN(WqkvT);
  CER_ALIGN(WoT);
  CER_ALIGN(qkv);
  CER_ALIGN(workspace);
  cer_status s = check_qkv(B, L, Hq, Hkv);
  if (s != CER_OK) return s;
  CER_REQUIRE(N >= 0 && L <= N, CER_ERR_SHAPE, "L=%d must be in [0, N=%d]", L, N);
  CER_REQUIRE(d >= 64 && d <= 16384 && d % 64 == 0, CER_ERR_SHAPE, "d=%d must be a multiple of 64 in [64, 16384]", d);
  CER_REQUIRE(causal == 0 || causal == 1, CER_ERR_RANGE, "causal=%d must be 0 or 1", causal);
  CER_REQUIRE(base > 1.0 && std::isfinite(base), CER_ERR_RANGE, "rotary base %g must be finite and > 1", base);
  const size_t need = cer_routed_attention_workspace_size(B, L, d, Hq, Hkv);
  CER_REQUIRE(M64 == 0 || (workspace != nullptr && workspace_bytes >= need), CER_ERR_WORKSPACE,
              "workspace of %zu bytes needed, %zu given", need, workspace_bytes);
  const bool in_place = (out == nullptr || out == h);
  const size_t hbytes = static_cast<size_t>(B) * N * d * 2;
  if (!in_place) {
    CER_PTR_IF(out, any_h);
    const char* a0 = static_cast<const char*>(h);
    const char* b0 = static_cast<const char*>(out);
    CER_REQUIRE(b0 + hbytes <= a0 || a0 + hbytes <= b0, CER_ERR_RANGE, "out overlaps h without being equal to it");
  }
  DeviceInfo* dev = nullptr;
  if ((s = device_info(&dev)) != CER_OK) return s;
  void* dst = in_place ? h : out;
  cudaError_t e;
  if (!in_place && hbytes) {
    e = cudaMemcpyAsync(out, h, hbytes, cudaMemcpyDeviceToDevice, stream);   // bypass rows
    if (e != cudaSuccess) return cuda_fail(e, "bypass copy");
  }
  if (M64 == 0) return CER_OK;
  const int M = static_cast<int>(M64);
  const int width = (Hq + 2 * Hkv) * cer::kHeadDim;
  char* ws = static_cast<char*>(workspace);
  __nv_bfloat16* X = reinterpret_cast<__nv_bfloat16*>(ws);
  ws += round256(static_cast<size_t>(M) * d * 2);
  __nv_bfloat16* qkv_ws = reinterpret_cast<__nv_bfloat16*>(ws);
  ws += round256(static_cast<size_t>(M) * width * 2);
  __nv_bfloat16* attn = reinterpret_cast<__nv_bfloat16*>(ws);
  ws += round256(static_cast<size_t>(M) * Hq * cer::kHeadDim * 2);
  float2* rope_cs = reinterpret_cast<float2*>(ws);
  ws += round256(static_cast<size_t>(M) * (cer::kHeadDim / 2) * sizeof(float2));
  cer::FfnArgs proj{};
  carve_stream_k(&ws, M, &proj);
  __nv_bfloat16* qkv_rows = qkv ? static_cast<__nv_bfloat16*>(qkv) : qkv_ws;

  // pack R, with the rotary (cos, sin) of every packed row's original position
  cer::RopeFreqTable ft;
  for (int j = 0; j < cer::kHeadDim / 2; ++j)
    ft.g[j] = std::pow(base, -2.0 * j / cer::kHeadDim) / (2.0 * M_PI);
  e = cer::launch_gather_rope(static_cast<const __nv_bfloat16*>(h), B, N, d, idx, L, X, rope_cs, ft, dev->status,
                              dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "gather launch");
  // qkv = X WqkvT: the down-projection GEMM in plain-output mode (K = d,
  // N = width), the query and key heads rotated in its epilogue
  cer::FfnArgs q = proj;
  q.act = X;
  q.M = M;
  q.C = d;
  q.d = width;
  q.WdT = static_cast<const __nv_bfloat16*>(WqkvT);
  q.Y = qkv_rows;
  q.scatter = 0;
  q.rope_cs = rope_cs;
  q.rope_heads = Hq + Hkv;
  q.status = dev->status;
  e = cer::launch_ffn_down(q, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "QKV projection launch");
  // attention on the packed rows
  e = cer::launch_packed_attention(qkv_rows, B, L, Hq, Hkv, causal, attn, dev->status, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "packed attention launch");
  // out[b, idx] = bf16(h + A WoT): the down-projection GEMM with its fused unpack
  cer::FfnArgs o = proj;
  o.act = attn;
  o.M = M;
  o.C = Hq * cer::kHeadDim;
  o.d = d;
  o.WdT = static_cast<const __nv_bfloat16*>(WoT);
  o.h = static_cast<const __nv_bfloat16*>(h);
  o.out = static_cast<__nv_bfloat16*>(dst);
  o.idx = idx;
  o.N = N;
  o.k_tot = L;
  o.scatter = 1;
  o.status = dev->status;
  e = cer::launch_ffn_down(o, dev->n_sm, stream);
  if (e != cudaSuccess) return cuda_fail(e, "output projection launch");
  return CER_OK;
}

}  // extern "C"
