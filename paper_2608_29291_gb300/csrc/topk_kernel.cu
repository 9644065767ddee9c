// topk_kernel.cu -- S2: the per-sequence keep set R = TopK(sigmoid(l), K) of
// Eq. 6 (router_inference_outputs, Sec. 3.4), computed exactly on the fp32 logits (the sigmoid is
// monotonic, App. B.2).
//
// One 1024-thread CTA per sequence keeps the N order-preserving 32-bit keys in
// shared memory.  An MSB-first radix select (8-bit digits, shared histograms)
// finds the K-th largest routable key T and how many tokens equal to T must
// be taken; as soon as at most 32 routable keys share the digits found so
// far, one warp ranks those candidates exactly and the remaining passes are
// skipped (real-valued logits get there after one or two passes, heavy ties
// take all four).  Each warp then owns a contiguous run of tokens, read 32
// at a time (a token per lane, no bank conflicts): ballots rank every tie
// (lowest index first) and every kept token, and two scans over the warps'
// counts place them, so the kept list comes out in ascending token order with
// no sort.  When fed the scorer's partial sums it also reduces them (in chunk
// order) into the logits.
#include <cuda_runtime.h>

#include "kernels.h"
#include "ptx.cuh"
#include "status.cuh"

namespace cer {

constexpr int kTopkThreads = 1024;

// Monotone map from fp32 to uint32: a > b (as floats) iff key(a) > key(b);
// -0.0 is mapped like +0.0.
__device__ __forceinline__ uint32_t order_key(float v) {
  uint32_t u = __float_as_uint(v);
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive prefix sum over the block (all threads must call).
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* warp_tot) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    uint32_t t = lane < nw ? warp_tot[lane] : 0u;
    uint32_t ti = t;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t o = __shfl_up_sync(0xffffffffu, ti, off);
      if (lane >= off) ti += o;
    }
    if (lane < nw) warp_tot[lane] = ti - t;  // exclusive over warps
  }
  __syncthreads();
  const uint32_t r = warp_tot[warp] + incl - v;
  __syncthreads();
  return r;
}

// Histogram counts go to kSubHist copies (by warp) to spread the atomic
// contention of logits that share a few digit values; merged after each pass.
constexpr int kSubHist = 8;

// Tokens a thread reduces at once in the logits pass (their partial-sum loads
// are in flight together), and the keep-ballot store of the compaction.
constexpr int kLoadUnroll = 4;
constexpr int kMaxSteps = (kTopkMaxN + kTopkThreads - 1) / kTopkThreads;

// Logits from the scorer's partial sums, summed in chunk order, into the
// order keys: a thread takes U tokens at a time and reads their partial rows
// eight at a time, so up to 8U loads are in flight.
template <int U>
__device__ __forceinline__ void reduce_logits(const TopkArgs& a, size_t base, uint32_t* keys, int* s_nan) {
  const int N = a.N;
  for (int i0 = threadIdx.x; i0 < N; i0 += U * blockDim.x) {
    float v[U];
#pragma unroll
    for (int u = 0; u < U; ++u) v[u] = 0.f;
    for (int c0 = 0; c0 < a.n_chunks; c0 += 8) {
      float part[U][8];
      // Every load in bounds (token and chunk clamped), so all 8U go out
      // back to back; the clamped ones are not used.
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int i = min(i0 + u * static_cast<int>(blockDim.x), N - 1);
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const int cc = min(c0 + c, a.n_chunks - 1);
          part[u][c] = __ldg(a.src + static_cast<size_t>(cc) * a.chunk_stride + base + i);
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u)
#pragma unroll
        for (int c = 0; c < 8; ++c)
          if (c0 + c < a.n_chunks) v[u] = (c0 + c == 0) ? part[u][c] : v[u] + part[u][c];
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i0 + u * blockDim.x;
      if (i >= N) break;
      if (a.logits_out) a.logits_out[base + i] = v[u];
      if (a.probs_out) a.probs_out[base + i] = 1.0f / (1.0f + expf(-v[u]));
      if (i >= a.r0 && i < a.r1 && v[u] != v[u]) *s_nan = 1;
      keys[i] = order_key(v[u]);
    }
  }
}

__global__ void __launch_bounds__(kTopkThreads) topk_kernel(TopkArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ uint32_t keys[];
  __shared__ uint32_t hist[256];
  __shared__ uint32_t sub[kSubHist][256];
  __shared__ uint32_t warp_tot[32];
  __shared__ uint32_t s_prefix, s_remaining, s_count, s_ncand;
  __shared__ uint32_t s_cand[32];
  __shared__ int s_nan;
  __shared__ uint32_t s_ballot[kTopkThreads / 32][kMaxSteps];

  const int tid = threadIdx.x;
  const int b = blockIdx.x;
  const int N = a.N;
  const size_t base = static_cast<size_t>(b) * N;
  if (tid == 0) {
    s_nan = 0;
    s_ncand = 0;
  }
  __syncthreads();

  // 1. logits (reduced from partial sums in chunk order) -> keys
  if (N >= 2 * static_cast<int>(blockDim.x)) {
    reduce_logits<kLoadUnroll>(a, base, keys, &s_nan);
  } else {
    reduce_logits<1>(a, base, keys, &s_nan);
  }
  __syncthreads();

  const int Nr = a.r1 - a.r0;
  const int K = a.K;
  const bool keep_all = (K == Nr);
  const bool keep_none = (K == 0);
  uint32_t thr = 0, need_eq = 0;

  // 2. radix select of the K-th largest routable key
  if (!keep_all && !keep_none) {
    uint32_t prefix = 0, pmask = 0, remaining = static_cast<uint32_t>(K);
    for (int i = tid; i < kSubHist * 256; i += blockDim.x) (&sub[0][0])[i] = 0;
    __syncthreads();
    // Three barriers per pass: the merge also clears the sub-histograms for
    // the next pass, and s_prefix is rewritten only two barriers after every
    // thread has read it.
    for (int shift = 24; shift >= 0; shift -= 8) {
      uint32_t* my = sub[(tid >> 5) % kSubHist];
      for (int i = a.r0 + tid; i < a.r1; i += blockDim.x) {
        const uint32_t k = keys[i];
        if ((k & pmask) == prefix) atomicAdd(&my[(k >> shift) & 255u], 1u);
      }
      __syncthreads();
      for (int i = tid; i < 256; i += blockDim.x) {
        uint32_t c = 0;
#pragma unroll
        for (int q = 0; q < kSubHist; ++q) {
          c += sub[q][i];
          sub[q][i] = 0;
        }
        hist[i] = c;
      }
      __syncthreads();
      if (tid < 32) {
        const int lane = tid;
        uint32_t local[8];
        uint32_t tot = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          local[j] = hist[8 * lane + j];
          tot += local[j];
        }
        uint32_t incl = tot;  // sum over lanes >= lane
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const uint32_t o = __shfl_down_sync(0xffffffffu, incl, off);
          if (lane + off < 32) incl += o;
        }
        uint32_t cum = incl - tot;  // keys in higher digits than this lane's bins
#pragma unroll
        for (int j = 7; j >= 0; --j) {
          if (cum < remaining && cum + local[j] >= remaining) {
            s_prefix = prefix | (static_cast<uint32_t>(8 * lane + j) << shift);
            s_remaining = remaining - cum;
            s_count = local[j];
          }
          cum += local[j];
        }
      }
      __syncthreads();
      prefix = s_prefix;
      remaining = s_remaining;
      pmask |= 255u << shift;
      if (shift > 0 && s_count <= 32u) {
        // Few routable keys share the digits found so far (the usual case
        // for real-valued logits after one or two passes): gather them and
        // let one warp rank them exactly instead of running the remaining
        // passes.  The threshold is the candidate with fewer than
        // `remaining` larger candidates and at least `remaining` larger or
        // equal ones; need_eq is what is left of `remaining` above it.
        for (int i = a.r0 + tid; i < a.r1; i += blockDim.x) {
          const uint32_t k = keys[i];
          if ((k & pmask) == prefix) s_cand[atomicAdd(&s_ncand, 1u)] = k;
        }
        __syncthreads();
        if (tid < 32) {
          const uint32_t n = s_ncand;
          const uint32_t k = tid < static_cast<int>(n) ? s_cand[tid] : 0u;
          uint32_t gt = 0, ge = 0;
          for (uint32_t j = 0; j < n; ++j) {
            const uint32_t o = s_cand[j];
            gt += o > k ? 1u : 0u;
            ge += o >= k ? 1u : 0u;
          }
          if (tid < static_cast<int>(n) && gt < remaining && ge >= remaining) {
            s_prefix = k;                 // lanes holding equal keys write equal values
            s_remaining = remaining - gt;
          }
        }
        __syncthreads();
        prefix = s_prefix;
        remaining = s_remaining;
        break;
      }
    }
    thr = prefix;
    need_eq = remaining;
  }

  // 3. keep decisions in token order; ties to T ranked by index.  Warp w owns
  // tokens [w * steps * 32, (w + 1) * steps * 32), 32 per step.
  const int lane = tid & 31, warp = tid >> 5;
  const uint32_t lt = (1u << lane) - 1u;
  const int steps = (N + blockDim.x - 1) / blockDim.x;
  const int c0 = warp * steps * 32;
  const bool select = !keep_all && !keep_none;
  uint32_t eq_w = 0;
  if (select) {
    for (int st = 0; st < steps; ++st) {
      const int i = c0 + st * 32 + lane;
      const bool eq = i < N && i >= a.r0 && i < a.r1 && keys[i] == thr;
      eq_w += __popc(__ballot_sync(0xffffffffu, eq));
    }
  }
  uint32_t er = __shfl_sync(0xffffffffu, block_exclusive_scan(lane == 0 ? eq_w : 0u, warp_tot), 0);

  uint32_t keep_w = 0;
  for (int st = 0; st < steps; ++st) {
    const int i = c0 + st * 32 + lane;
    const bool valid = i < N;
    const bool routable = valid && i >= a.r0 && i < a.r1;
    const uint32_t k = valid ? keys[i] : 0u;
    const bool eq = select && routable && k == thr;
    const uint32_t eqb = __ballot_sync(0xffffffffu, eq);
    const uint32_t rank = er + __popc(eqb & lt);
    er += __popc(eqb);
    bool keep;
    if (!valid) keep = false;
    else if (!routable || keep_all) keep = true;
    else if (keep_none) keep = false;
    else keep = k > thr || (eq && rank < need_eq);
    const uint32_t kb = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) s_ballot[warp][st] = kb;
    keep_w += __popc(kb);
  }
  uint32_t pos = __shfl_sync(0xffffffffu, block_exclusive_scan(lane == 0 ? keep_w : 0u, warp_tot), 0);

  const int k_tot = K + N - Nr;
  int32_t* idx = a.idx + static_cast<size_t>(b) * k_tot;
  for (int st = 0; st < steps; ++st) {
    const int i = c0 + st * 32 + lane;
    const uint32_t kb = s_ballot[warp][st];   // written by this warp's lane 0 (block scan barriers since)
    const bool keep = (kb >> lane) & 1u;
    const uint32_t slot = pos + __popc(kb & lt);
    if (keep && slot < static_cast<uint32_t>(k_tot)) idx[slot] = i;
    if (a.mask && i < N) a.mask[base + i] = keep ? 1 : 0;
    pos += __popc(kb);
  }
  if (tid == 0 && s_nan) record_status(a.status, CER_DEV_NAN);
}

cudaError_t launch_topk(const TopkArgs& a, cudaStream_t stream) {
  if (a.B == 0 || a.N == 0) return cudaSuccess;
  const size_t smem = static_cast<size_t>(a.N) * sizeof(uint32_t);
  // The limit is raised once per device to the largest N ever accepted.
  cudaError_t e = ensure_max_smem(reinterpret_cast<const void*>(topk_kernel), kTopkMaxN * sizeof(uint32_t));
  if (e != cudaSuccess) return e;
  return launch_k(topk_kernel, dim3(a.B), dim3(kTopkThreads), smem, stream, 1, a);
}

}  // namespace cer
