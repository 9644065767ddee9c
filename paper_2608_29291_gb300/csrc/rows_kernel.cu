// rows_kernel.cu -- S3 gather (token compaction) and S5 scatter-add (unpack
// with bypass), Sec. 3.4.  Pure HBM streams: one warp per packed row, 16-byte
// vector loads and stores, four vectors in flight per lane; a persistent grid
// of 16 warps per SM.  Dropped rows are never touched.
#include <cuda_bf16.h>

#include "kernels.h"
#include "ptx.cuh"
#include "status.cuh"

namespace cer {

constexpr int kRowThreads = 512;

// With ROPE the warp also writes row m's rotary (cos, sin) for the 64
// frequencies, two per lane: the angle in turns x = i * g_j (fp64, reduced
// exactly) through fp32 sincospif, as in the rotary-embedding kernel.
template <bool ROPE>
__global__ void __launch_bounds__(kRowThreads) gather_rows_kernel(const uint4* __restrict__ h, int N, int d16,
                                                                  const int32_t* __restrict__ idx, int k_tot,
                                                                  int M, uint4* __restrict__ X, int* status,
                                                                  float2* __restrict__ cs,
                                                                  const __grid_constant__ RopeFreqTable ft) {
  griddep_wait();
  griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int wpb = blockDim.x >> 5;
  for (int m = blockIdx.x * wpb + (threadIdx.x >> 5); m < M; m += gridDim.x * wpb) {
    const int b = m / k_tot;
    const int i = __ldg(idx + m);
    if (i < 0 || i >= N) {
      if (lane == 0) record_status(status, CER_DEV_INDEX);
      continue;
    }
    if constexpr (ROPE) {
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int j = lane + 32 * u;
        const double x = static_cast<double>(i) * ft.g[j];
        float sn, cn;
        sincospif(2.0f * static_cast<float>(x - rint(x)), &sn, &cn);
        cs[static_cast<size_t>(m) * (kHeadDim / 2) + j] = make_float2(cn, sn);
      }
    }
    const uint4* src = h + (static_cast<size_t>(b) * N + i) * d16;
    uint4* dst = X + static_cast<size_t>(m) * d16;
    int c = lane;
    for (; c + 96 < d16; c += 128) {
      const uint4 v0 = __ldg(src + c), v1 = __ldg(src + c + 32), v2 = __ldg(src + c + 64), v3 = __ldg(src + c + 96);
      dst[c] = v0;
      dst[c + 32] = v1;
      dst[c + 64] = v2;
      dst[c + 96] = v3;
    }
    for (; c < d16; c += 32) dst[c] = __ldg(src + c);
  }
}

// The row gather as bulk copies (S3 without the rotary table): each worker
// thread owns one shared-memory slot of a row's d * 2 bytes, copies its rows
// global -> shared with cp.async.bulk (completion counted on the slot's
// mbarrier, the wait bounded) and shared -> global with a bulk store, and
// reuses the slot once that store has read it.  A few instructions move a
// whole row, so every row of the call can be in flight at once (the slots per
// CTA are sized so the grid's slots cover M, up to ~200 KB per CTA).  At
// long_7b (2816 rows of 7 KB) the gather stage went from 0.55 to 0.59 of
// the measured HBM bandwidth.
__global__ void gather_rows_bulk_kernel(const char* __restrict__ h, int N, uint32_t row_bytes,
                                        const int32_t* __restrict__ idx, int k_tot, int M, int slots,
                                        char* __restrict__ X, int* status) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ __align__(16) char gslot[];
  __shared__ int abort_flag;
  const int t = threadIdx.x;
  if (t == 0) abort_flag = 0;
  uint64_t* bar = reinterpret_cast<uint64_t*>(gslot + static_cast<size_t>(slots) * row_bytes);
  if (t < slots) mbar_init(&bar[t], 1);
  fence_mbar_init();
  __syncthreads();
  if (t >= slots) return;
  char* slot = gslot + static_cast<size_t>(t) * row_bytes;
  uint32_t phase = 0;
  bool pending = false;   // a load was issued and not yet waited for
  for (int m = blockIdx.x * slots + t; m < M; m += gridDim.x * slots) {
    const int b = m / k_tot;
    const int i = __ldg(idx + m);
    if (i < 0 || i >= N) {
      record_status(status, CER_DEV_INDEX);
      continue;
    }
    bulk_wait_group_read0();   // the slot's previous store has read it
    mbar_arrive_expect_tx(&bar[t], row_bytes);
    bulk_load(slot, h + (static_cast<size_t>(b) * N + i) * row_bytes, row_bytes, &bar[t]);
    pending = true;
    if (!mbar_wait(&bar[t], phase, &abort_flag, status)) break;
    pending = false;
    phase ^= 1;
    bulk_store(X + static_cast<size_t>(m) * row_bytes, slot, row_bytes);
    bulk_commit_group();
  }
  // The loads this thread waited for have landed; one it gave up on may
  // still be in flight (a timeout): give it a bounded moment before the CTA's
  // shared memory goes away.  Then let the stores finish.
  if (pending) {
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(&bar[t], phase) && globaltimer_ns() - t0 < 100000000ull) {
    }
  }
  bulk_wait_group0();
}

__device__ __forceinline__ uint32_t add_bf16x2(uint32_t hv, uint32_t yv) {
  __nv_bfloat162 a = *reinterpret_cast<__nv_bfloat162*>(&hv);
  __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162*>(&yv);
  const float2 fa = __bfloat1622float2(a), fb = __bfloat1622float2(b);
  __nv_bfloat162 r = __floats2bfloat162_rn(fa.x + fb.x, fa.y + fb.y);
  return *reinterpret_cast<uint32_t*>(&r);
}

__device__ __forceinline__ uint4 add_row_vec(uint4 hv, uint4 yv) {
  return make_uint4(add_bf16x2(hv.x, yv.x), add_bf16x2(hv.y, yv.y), add_bf16x2(hv.z, yv.z), add_bf16x2(hv.w, yv.w));
}

__global__ void __launch_bounds__(kRowThreads) scatter_add_kernel(uint4* __restrict__ h, int N, int d16,
                                                                  const int32_t* __restrict__ idx, int k_tot,
                                                                  int M, const uint4* __restrict__ Y,
                                                                  int* status) {
  griddep_wait();
  griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int wpb = blockDim.x >> 5;
  for (int m = blockIdx.x * wpb + (threadIdx.x >> 5); m < M; m += gridDim.x * wpb) {
    const int b = m / k_tot;
    const int i = __ldg(idx + m);
    if (i < 0 || i >= N) {
      if (lane == 0) record_status(status, CER_DEV_INDEX);
      continue;
    }
    uint4* row = h + (static_cast<size_t>(b) * N + i) * d16;
    const uint4* y = Y + static_cast<size_t>(m) * d16;
    int c = lane;
    for (; c + 32 < d16; c += 64) {
      const uint4 h0 = row[c], h1 = row[c + 32];
      const uint4 y0 = __ldg(y + c), y1 = __ldg(y + c + 32);
      row[c] = add_row_vec(h0, y0);
      row[c + 32] = add_row_vec(h1, y1);
    }
    for (; c < d16; c += 32) row[c] = add_row_vec(row[c], __ldg(y + c));
  }
}

// The validating form of the scatter-add: one CTA per sequence first marks
// every index of the sequence in a bitmap of its N tokens in shared memory;
// an index out of range or marked twice makes the sequence invalid, and then
// none of its rows is written (two warps adding into one row would race) and
// CER_DEV_INDEX is recorded.  A valid sequence's rows are then added as in
// scatter_add_kernel, one warp per row.
__global__ void __launch_bounds__(kRowThreads) scatter_add_checked_kernel(uint4* __restrict__ h, int N, int d16,
                                                                          const int32_t* __restrict__ idx,
                                                                          int k_tot, const uint4* __restrict__ Y,
                                                                          int* status) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ uint32_t seen[];
  __shared__ int bad;
  const int b = blockIdx.x;
  const int words = (N + 31) / 32;
  for (int i = threadIdx.x; i < words; i += blockDim.x) seen[i] = 0u;
  if (threadIdx.x == 0) bad = 0;
  __syncthreads();
  const int32_t* list = idx + static_cast<size_t>(b) * k_tot;
  for (int j = threadIdx.x; j < k_tot; j += blockDim.x) {
    const int i = __ldg(list + j);
    if (i < 0 || i >= N) {
      bad = 1;
      continue;
    }
    const uint32_t bit = 1u << (i & 31);
    if (atomicOr(&seen[i >> 5], bit) & bit) bad = 1;
  }
  __syncthreads();
  if (bad) {
    if (threadIdx.x == 0) record_status(status, CER_DEV_INDEX);
    return;
  }
  const int lane = threadIdx.x & 31;
  const int wpb = blockDim.x >> 5;
  for (int j = threadIdx.x >> 5; j < k_tot; j += wpb) {
    const int i = __ldg(list + j);
    uint4* row = h + (static_cast<size_t>(b) * N + i) * d16;
    const uint4* y = Y + (static_cast<size_t>(b) * k_tot + j) * d16;
    for (int c = lane; c < d16; c += 32) row[c] = add_row_vec(row[c], __ldg(y + c));
  }
}

static int row_grid(int M, int n_sm) {
  const int wpb = kRowThreads / 32;
  int blocks = (M + wpb - 1) / wpb;
  const int cap = n_sm * 4;  // 4 blocks x 16 warps per SM
  return blocks < cap ? blocks : cap;
}

// Shared memory the bulk gather may give one CTA's slots.
constexpr size_t kGatherSlotBytes = size_t(200) << 10;

cudaError_t launch_gather(const __nv_bfloat16* h, int B, int N, int d, const int32_t* idx, int k_tot,
                          __nv_bfloat16* X, int* status, int n_sm, cudaStream_t stream) {
  const int M = B * k_tot;
  if (M == 0 || d == 0) return cudaSuccess;
  const uint32_t row_bytes = static_cast<uint32_t>(d) * 2;
  const int max_slots = static_cast<int>(kGatherSlotBytes / row_bytes);
  // Bulk copies when the grid's slots take every row at once; with several
  // rows per slot each one waits a full round trip (global -> shared ->
  // global) and the vector-load kernel, with four loads in flight per lane
  // and no staging, measured faster (M = 14746 rows of 7 KB: 33 us against
  // 40 us).
  if (max_slots >= 1 && static_cast<long long>(M) <= static_cast<long long>(n_sm) * max_slots) {
    // as many slots per CTA as spread M over the SMs, within the budget
    int slots = (M + n_sm - 1) / n_sm;
    if (slots > max_slots) slots = max_slots;
    if (slots > 1024) slots = 1024;
    const int blocks = (M + slots - 1) / slots < n_sm ? (M + slots - 1) / slots : n_sm;
    const size_t smem = static_cast<size_t>(slots) * row_bytes + static_cast<size_t>(slots) * sizeof(uint64_t);
    cudaError_t e = ensure_max_smem(reinterpret_cast<const void*>(gather_rows_bulk_kernel),
                                    kGatherSlotBytes + 1024 * sizeof(uint64_t));
    if (e != cudaSuccess) return e;
    const int threads = (slots + 31) / 32 * 32;
    return launch_k(gather_rows_bulk_kernel, dim3(blocks), dim3(threads), smem, stream, 1,
                    reinterpret_cast<const char*>(h), N, row_bytes, idx, k_tot, M, slots, reinterpret_cast<char*>(X),
                    status);
  }
  return launch_k(gather_rows_kernel<false>, dim3(row_grid(M, n_sm)), dim3(kRowThreads), 0, stream, 1,
                  reinterpret_cast<const uint4*>(h), N, d / 8, idx, k_tot, M, reinterpret_cast<uint4*>(X), status,
                  static_cast<float2*>(nullptr), RopeFreqTable{});
}

cudaError_t launch_gather_rope(const __nv_bfloat16* h, int B, int N, int d, const int32_t* idx, int k_tot,
                               __nv_bfloat16* X, float2* cs, const RopeFreqTable& ft, int* status, int n_sm,
                               cudaStream_t stream) {
  const int M = B * k_tot;
  if (M == 0 || d == 0) return cudaSuccess;
  return launch_k(gather_rows_kernel<true>, dim3(row_grid(M, n_sm)), dim3(kRowThreads), 0, stream, 1,
                  reinterpret_cast<const uint4*>(h), N, d / 8, idx, k_tot, M, reinterpret_cast<uint4*>(X), status, cs,
                  ft);
}

cudaError_t launch_scatter_add(__nv_bfloat16* h, int B, int N, int d, const int32_t* idx, int k_tot,
                               const __nv_bfloat16* Y, int* status, int n_sm, cudaStream_t stream) {
  const int M = B * k_tot;
  if (M == 0 || d == 0) return cudaSuccess;
  return launch_k(scatter_add_kernel, dim3(row_grid(M, n_sm)), dim3(kRowThreads), 0, stream, 1,
                  reinterpret_cast<uint4*>(h), N, d / 8, idx, k_tot, M, reinterpret_cast<const uint4*>(Y), status);
}

cudaError_t launch_scatter_add_checked(__nv_bfloat16* h, int B, int N, int d, const int32_t* idx, int k_tot,
                                       const __nv_bfloat16* Y, int* status, cudaStream_t stream) {
  if (B == 0 || k_tot == 0 || d == 0) return cudaSuccess;
  const size_t smem = static_cast<size_t>((N + 31) / 32) * sizeof(uint32_t);
  return launch_k(scatter_add_checked_kernel, dim3(B), dim3(kRowThreads), smem, stream, 1, reinterpret_cast<uint4*>(h),
                  N, d / 8, idx, k_tot, reinterpret_cast<const uint4*>(Y), status);
}

}  // namespace cer
