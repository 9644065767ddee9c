// ucs_kernel.cu -- statistics of Unified Computation Scheduling (Sec. 3.4):
//   * drop-set Jaccard J and its random-adjusted form RDA (Eq. 10, Eq. 11),
//     the signals of diffusion-head cache reuse and denoising-step early exit;
//   * the layer-skipping redundancy gap g (Eq. 7).
#include <cuda_bf16.h>

#include "kernels.h"
#include "ptx.cuh"
#include "status.cuh"

namespace cer {

constexpr int kStatThreads = 256;

__device__ __forceinline__ int warp_sum_int(int v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// ---------------------------------------------------------------- Eq. 10 / 11

// One block per sequence.  D = routable tokens [r0, r1) not kept.  The counts
// are exact integers; J, J_rand and RDA are formed from them with explicit
// round-to-nearest fp64 operations in a fixed order, then rounded to fp32.
// Reading of J_rand: E|A&B| / E|A|B| for uniformly random drop sets of the
// same sizes a, b among the n routable tokens, E|A&B| = a b / n.  An empty
// union gives J = 1; J_rand = 1 gives RDA = 1.
constexpr int kDropThreads = 1024;

__global__ void __launch_bounds__(kDropThreads) drop_stats_kernel(const uint8_t* __restrict__ mask_t,
                                                                   const uint8_t* __restrict__ mask_ref, int N,
                                                                   int r0, int r1, float* jac, float* jrand,
                                                                   float* rda, int32_t* counts) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ int part[3][kDropThreads / 32];
  const int b = blockIdx.x;
  const uint8_t* mt = mask_t + static_cast<size_t>(b) * N;
  const uint8_t* mr = mask_ref + static_cast<size_t>(b) * N;
  int na = 0, nb = 0, ni = 0;
  for (int i = r0 + threadIdx.x; i < r1; i += blockDim.x) {
    const int da = mt[i] == 0, db = mr[i] == 0;
    na += da;
    nb += db;
    ni += da & db;
  }
  na = warp_sum_int(na);
  nb = warp_sum_int(nb);
  ni = warp_sum_int(ni);
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    part[0][warp] = na;
    part[1][warp] = nb;
    part[2][warp] = ni;
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  na = nb = ni = 0;
  for (int w = 0; w < kDropThreads / 32; ++w) {
    na += part[0][w];
    nb += part[1][w];
    ni += part[2][w];
  }
  const int uni = na + nb - ni;
  const double j = uni == 0 ? 1.0 : __ddiv_rn(static_cast<double>(ni), static_cast<double>(uni));
  const int n = r1 - r0;
  double jr = 1.0;
  if (na + nb != 0 && n != 0) {
    const double e = __ddiv_rn(__dmul_rn(static_cast<double>(na), static_cast<double>(nb)), static_cast<double>(n));
    jr = __ddiv_rn(e, __dsub_rn(static_cast<double>(na + nb), e));
  }
  const double rr = jr == 1.0 ? 1.0 : __ddiv_rn(__dsub_rn(j, jr), __dsub_rn(1.0, jr));
  jac[b] = static_cast<float>(j);
  if (jrand) jrand[b] = static_cast<float>(jr);
  if (rda) rda[b] = static_cast<float>(rr);
  if (counts) {
    counts[3 * b + 0] = na;
    counts[3 * b + 1] = nb;
    counts[3 * b + 2] = ni;
  }
}

// ---------------------------------------------------------------- Eq. 7

// One warp per token: cosine of the input and output rows (fp32 partial sums
// per lane, fixed xor-tree reduction).  A zero-norm pair gives 1 when the rows
// are bit-identical, else 0.  Seven blocks per SM (32 registers a thread,
// four K steps of loads in flight per lane): 56 warps, so B = 2 sequences of
// 4096 tokens (54 rows per SM) take one round of rows; at 40 registers six
// blocks fitted and a seventh ran as a second round (ncu: 31.4 us cold for
// 117 MB, 49 % of DRAM; the whole gap at that shape 48.5 us, against 45.0 us
// with seven).
__global__ void __launch_bounds__(kStatThreads, 7) row_cosine_kernel(const uint4* __restrict__ h_in,
                                                                   const uint4* __restrict__ h_out, int d8,
                                                                   long rows, float* __restrict__ cosv) {
  griddep_wait();
  griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const long wpb = blockDim.x >> 5;
  for (long r = blockIdx.x * wpb + (threadIdx.x >> 5); r < rows; r += static_cast<long>(gridDim.x) * wpb) {
    const uint4* a = h_in + r * d8;
    const uint4* o = h_out + r * d8;
    float dot = 0.f, na = 0.f, no = 0.f;
    unsigned diff = 0;
#pragma unroll 4
    for (int c = lane; c < d8; c += 32) {
      const uint4 va = __ldg(a + c), vo = __ldg(o + c);
      diff |= (va.x ^ vo.x) | (va.y ^ vo.y) | (va.z ^ vo.z) | (va.w ^ vo.w);
      const uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wo[4] = {vo.x, vo.y, vo.z, vo.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float2 fa = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&wa[k]));
        const float2 fo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&wo[k]));
        dot = fmaf(fa.x, fo.x, fmaf(fa.y, fo.y, dot));
        na = fmaf(fa.x, fa.x, fmaf(fa.y, fa.y, na));
        no = fmaf(fo.x, fo.x, fmaf(fo.y, fo.y, no));
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      dot += __shfl_xor_sync(0xffffffffu, dot, off);
      na += __shfl_xor_sync(0xffffffffu, na, off);
      no += __shfl_xor_sync(0xffffffffu, no, off);
      diff |= __shfl_xor_sync(0xffffffffu, diff, off);
    }
    if (lane == 0) {
      float c;
      if (na == 0.f || no == 0.f)
        c = diff ? 0.f : 1.f;
      else
        c = dot / (sqrtf(na) * sqrtf(no));
      cosv[r] = c;
    }
  }
}

// One block per sequence: g = mean_all(cos) - mean_R(cos), skip = g <= delta.
// fp32 sums in a fixed tree order (per-thread strided sums, xor-shuffle tree,
// warps in order): relative error about log2(N) * 2^-24.  FP64 arithmetic is
// very slow on this part, so it is kept out of this reduction.  Empty R gives
// g = 0.
__global__ void __launch_bounds__(kStatThreads) gap_reduce_kernel(const float* __restrict__ cosv,
                                                                   const uint8_t* __restrict__ mask, int N,
                                                                   float delta, float* gap, uint8_t* skip) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ float part_all[kStatThreads / 32], part_ret[kStatThreads / 32];
  __shared__ int part_n[kStatThreads / 32];
  const int b = blockIdx.x;
  const float* c = cosv + static_cast<size_t>(b) * N;
  const uint8_t* m = mask + static_cast<size_t>(b) * N;
  float s_all = 0.f, s_ret = 0.f;
  int n_ret = 0;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    const float v = c[i];
    s_all += v;
    if (m[i]) {
      s_ret += v;
      ++n_ret;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    s_all += __shfl_xor_sync(0xffffffffu, s_all, off);
    s_ret += __shfl_xor_sync(0xffffffffu, s_ret, off);
    n_ret += __shfl_xor_sync(0xffffffffu, n_ret, off);
  }
  const int warp = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    part_all[warp] = s_all;
    part_ret[warp] = s_ret;
    part_n[warp] = n_ret;
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  s_all = s_ret = 0.f;
  n_ret = 0;
  for (int w = 0; w < kStatThreads / 32; ++w) {
    s_all += part_all[w];
    s_ret += part_ret[w];
    n_ret += part_n[w];
  }
  const float g = (n_ret == 0 || N == 0) ? 0.f : s_all / static_cast<float>(N) - s_ret / static_cast<float>(n_ret);
  gap[b] = g;
  if (skip) skip[b] = g <= delta ? 1 : 0;
}

// ---------------------------------------------------------------- Eq. 8 / 9

// Per channel: s_c = mean over the retained rows of |z_c| times
// ||W_down[:, c]|| (the column norms are a static per-layer input); each block
// also sums its channels' saliency split at C_keep (kept channels first,
// the mask's pruned channels after), fixed order.
constexpr int kGateThreads = 256;

__global__ void __launch_bounds__(kGateThreads) saliency_kernel(const float* __restrict__ colsum, int n_parts,
                                                                 int M, int I, int C_keep,
                                                                 const float* __restrict__ norms, float* saliency,
                                                                 float* part_ws) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ double red[2][kGateThreads / 32];
  const int c = blockIdx.x * kGateThreads + threadIdx.x;
  double s = 0.0;
  if (c < I) {
    float acc = 0.f;
    for (int q = 0; q < n_parts; ++q) acc += colsum[static_cast<size_t>(q) * I + c];
    s = static_cast<double>(acc) / M * norms[c];
    if (saliency) saliency[c] = static_cast<float>(s);
  }
  double kept = (c < C_keep) ? s : 0.0, pruned = (c >= C_keep) ? s : 0.0;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    kept += __shfl_xor_sync(0xffffffffu, kept, off);
    pruned += __shfl_xor_sync(0xffffffffu, pruned, off);
  }
  if ((threadIdx.x & 31) == 0) {
    red[0][threadIdx.x >> 5] = kept;
    red[1][threadIdx.x >> 5] = pruned;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    kept = pruned = 0.0;
    for (int w = 0; w < kGateThreads / 32; ++w) {
      kept += red[0][w];
      pruned += red[1][w];
    }
    part_ws[2 * blockIdx.x] = static_cast<float>(kept);
    part_ws[2 * blockIdx.x + 1] = static_cast<float>(pruned);
  }
}

// One thread: leakage of Eq. 9 and the pruned-or-full decision.
__global__ void leakage_kernel(const float* part_ws, int n_blocks, float delta, float* leakage, uint8_t* use_pruned) {
  griddep_wait();
  griddep_launch_dependents();
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  double kept = 0.0, pruned = 0.0;
  for (int b = 0; b < n_blocks; ++b) {
    kept += part_ws[2 * b];
    pruned += part_ws[2 * b + 1];
  }
  const double total = kept + pruned;
  const double lam = total > 0.0 ? pruned / total : 0.0;
  if (leakage) *leakage = static_cast<float>(lam);
  *use_pruned = lam <= static_cast<double>(delta) ? 1 : 0;
}

// One warp per row: ||W[r, :]||_2 in fp32 (static per-layer input of Eq. 8).
__global__ void __launch_bounds__(kStatThreads) row_norm_kernel(const uint4* __restrict__ W, int d8, int rows,
                                                                 float* __restrict__ norms) {
  griddep_wait();
  griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int wpb = blockDim.x >> 5;
  for (int r = blockIdx.x * wpb + (threadIdx.x >> 5); r < rows; r += gridDim.x * wpb) {
    float s = 0.f;
    for (int c = lane; c < d8; c += 32) {
      const uint4 v = __ldg(W + static_cast<size_t>(r) * d8 + c);
      const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w4[k]));
        s = fmaf(f.x, f.x, fmaf(f.y, f.y, s));
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) norms[r] = sqrtf(s);
  }
}

// ---------------------------------------------------------------- launchers

cudaError_t launch_ffn_gate(const float* colsum, int n_parts, int M, int I, int C_keep, const float* norms,
                            float delta, float* saliency, float* part_ws, float* leakage, uint8_t* use_pruned,
                            cudaStream_t stream) {
  const int blocks = (I + kGateThreads - 1) / kGateThreads;
  cudaError_t e = launch_k(saliency_kernel, dim3(blocks), dim3(kGateThreads), 0, stream, 1, colsum, n_parts, M, I,
                           C_keep, norms, saliency, part_ws);
  if (e != cudaSuccess) return e;
  return launch_k(leakage_kernel, dim3(1), dim3(32), 0, stream, 1, static_cast<const float*>(part_ws), blocks, delta,
                  leakage, use_pruned);
}

cudaError_t launch_row_norms(const __nv_bfloat16* W, int rows, int d, float* norms, int n_sm, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  int blocks = (rows + 7) / 8;
  if (blocks > n_sm * 8) blocks = n_sm * 8;
  return launch_k(row_norm_kernel, dim3(blocks), dim3(kStatThreads), 0, stream, 1, reinterpret_cast<const uint4*>(W),
                  d / 8, rows, norms);
}

cudaError_t launch_drop_stats(const uint8_t* mask_t, const uint8_t* mask_ref, int B, int N, int r0, int r1,
                              float* jac, float* jrand, float* rda, int32_t* counts, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  return launch_k(drop_stats_kernel, dim3(B), dim3(kDropThreads), 0, stream, 1, mask_t, mask_ref, N, r0, r1, jac,
                  jrand, rda, counts);
}

cudaError_t launch_redundancy_gap(const __nv_bfloat16* h_in, const __nv_bfloat16* h_out, const uint8_t* mask,
                                  int B, int N, int d, float delta, float* gap, uint8_t* skip, float* cos_ws,
                                  int n_sm, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  const long rows = static_cast<long>(B) * N;
  if (rows > 0) {
    long blocks = (rows + 7) / 8;
    const long cap = static_cast<long>(n_sm) * 8;
    if (blocks > cap) blocks = cap;
    cudaError_t e = launch_k(row_cosine_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kStatThreads), 0, stream,
                             1, reinterpret_cast<const uint4*>(h_in), reinterpret_cast<const uint4*>(h_out), d / 8,
                             rows, cos_ws);
    if (e != cudaSuccess) return e;
  }
  return launch_k(gap_reduce_kernel, dim3(B), dim3(kStatThreads), 0, stream, 1, static_cast<const float*>(cos_ws),
                  mask, N, delta, gap, skip);
}

}  // namespace cer
