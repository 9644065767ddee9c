// topk_kernel.cu -- S2: the per-sequence keep set R = TopK(sigmoid(l), K) of
// Eq. 6 (Sec. 3.4), computed exactly on the fp32 logits (the sigmoid is
// monotonic, App. B.2).
//
// A sequence is handled by a cluster of G <= 8 CTAs (G = 1 up to 4096
// tokens, else enough CTAs for about 4096 tokens each: measured on GB300, the
// cluster barriers and remote reads cost more than they save below that),
// CTA `rank` owning
// the tokens [rank * chunk, (rank + 1) * chunk).  Each CTA keeps the
// order-preserving 32-bit keys of its tokens in shared memory (reducing the
// scorer's partial sums, in chunk order, into the logits on the way).  An
// MSB-first radix select with 8-bit digits finds the K-th largest routable
// key T and how many tokens equal to T must be taken: every pass counts the
// CTA's keys into per-warp sub-histograms, publishes their sum, and after one
// cluster barrier every CTA adds up the G histograms through distributed
// shared memory and takes the same digit.  As soon as at most 32 routable
// keys share the digits found so far, each CTA publishes its candidates and
// one warp per CTA ranks all of them exactly (real-valued logits get there
// after one or two passes, heavy ties take all four).
//
// Compaction: each warp owns a contiguous run of its CTA's tokens.  The warps'
// counts of ties (key == T) and of tokens kept outright (key > T, or outside
// the routable range) are summed per CTA and published; after one more
// cluster barrier every CTA knows how many ties and kept tokens precede it,
// hence how many of its ties are taken (the lowest indices first) and where
// its kept tokens go, and writes its part of the ascending keep list with
// warp ballots -- no sort.
#include <cuda_runtime.h>

#include "kernels.h"
#include "ptx.cuh"
#include "status.cuh"

namespace cer {

constexpr int kTopkThreads = 512;
constexpr int kTopkWarps = kTopkThreads / 32;
constexpr int kTopkMaxCluster = 8;
// Tokens per CTA the cluster size aims at.
constexpr int kTopkChunkTarget = 4096;

// Monotone map from fp32 to uint32: a > b (as floats) iff key(a) > key(b);
// -0.0 is mapped like +0.0.
__device__ __forceinline__ uint32_t order_key(float v) {
  uint32_t u = __float_as_uint(v);
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Histogram counts go to kSubHist copies (by warp) to spread the atomic
// contention of logits that share a few digit values; merged after each pass.
constexpr int kSubHist = 8;

// Logits of tokens [lo, hi) from the scorer's partial sums, summed in chunk
// order, into the order keys; the routable keys are counted into pass 0's
// histogram (their top byte) on the way.  Vector form: a thread takes 4
// consecutive tokens, one float4 of each partial row, eight rows' loads in
// flight at once; it needs lo, the sequence base and the row stride to be
// multiples of 4 (checked by the caller).  The kernel runs once per step from
// a cold instruction cache, so its loops are kept short rather than unrolled.
__device__ __forceinline__ void key_out(const TopkArgs& a, size_t base, int lo, int i, float v, uint32_t* keys,
                                        uint32_t* hist0, bool count, int* s_nan) {
  if (a.logits_out) a.logits_out[base + i] = v;
  if (a.probs_out) a.probs_out[base + i] = 1.0f / (1.0f + expf(-v));
  const bool routable = i >= a.r0 && i < a.r1;
  if (routable && v != v) *s_nan = 1;
  const uint32_t k = order_key(v);
  keys[i - lo] = k;
  if (count && routable) atomicAdd(&hist0[k >> 24], 1u);
}

__device__ __forceinline__ float4 sum_partials4(const TopkArgs& a, const float4* src, size_t stride4, int q) {
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
  for (int c0 = 0; c0 < a.n_chunks; c0 += 8) {
    float4 part[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) part[c] = __ldg(src + static_cast<size_t>(min(c0 + c, a.n_chunks - 1)) * stride4 + q);
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      if (c0 + c >= a.n_chunks) break;
      if (c0 + c == 0) {
        v = part[c];
      } else {
        v.x += part[c].x;
        v.y += part[c].y;
        v.z += part[c].z;
        v.w += part[c].w;
      }
    }
  }
  return v;
}

__device__ __forceinline__ void reduce_logits_vec4(const TopkArgs& a, size_t base, int lo, int hi, uint32_t* keys,
                                                   uint32_t* hist0, bool count, int* s_nan) {
  const int q_hi = (hi + 3) / 4;
  const float4* src = reinterpret_cast<const float4*>(a.src + base);
  const size_t stride4 = a.chunk_stride / 4;
#pragma unroll 1
  for (int q = lo / 4 + threadIdx.x; q < q_hi; q += 2 * blockDim.x) {
    // two groups of 4 tokens: both groups' loads go out before either is summed
    const int q2 = min(q + static_cast<int>(blockDim.x), q_hi - 1);
    const float4 v0 = sum_partials4(a, src, stride4, q);
    const float4 v1 = sum_partials4(a, src, stride4, q2);
#pragma unroll
    for (int g = 0; g < 2; ++g) {
      const int qq = g == 0 ? q : q + blockDim.x;
      if (qq >= q_hi) break;
      const float4 v = g == 0 ? v0 : v1;
      const int i = 4 * qq;
      key_out(a, base, lo, i, v.x, keys, hist0, count, s_nan);
      if (i + 1 < hi) key_out(a, base, lo, i + 1, v.y, keys, hist0, count, s_nan);
      if (i + 2 < hi) key_out(a, base, lo, i + 2, v.z, keys, hist0, count, s_nan);
      if (i + 3 < hi) key_out(a, base, lo, i + 3, v.w, keys, hist0, count, s_nan);
    }
  }
}

// Scalar form for rows whose layout does not allow the vector loads.
__device__ __forceinline__ void reduce_logits_scalar(const TopkArgs& a, size_t base, int lo, int hi, uint32_t* keys,
                                                  uint32_t* hist0, bool count, int* s_nan) {
#pragma unroll 1
  for (int i = lo + threadIdx.x; i < hi; i += blockDim.x) {
    float v = __ldg(a.src + base + i);
#pragma unroll 1
    for (int c = 1; c < a.n_chunks; ++c) v += __ldg(a.src + static_cast<size_t>(c) * a.chunk_stride + base + i);
    key_out(a, base, lo, i, v, keys, hist0, count, s_nan);
  }
}

// Inclusive prefix sum over the lanes of a warp.
__device__ __forceinline__ uint32_t warp_inclusive_scan(uint32_t v, int lane) {
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t o = __shfl_up_sync(0xffffffffu, v, off);
    if (lane >= off) v += o;
  }
  return v;
}

__global__ void __launch_bounds__(kTopkThreads) topk_kernel(TopkArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ uint32_t keys[];           // keys of this CTA's tokens [lo, hi), at i - lo
  __shared__ uint32_t sub[kSubHist][256];
  __shared__ uint32_t hist[2][256];            // this CTA's histogram of a pass (by parity); read by the cluster
  __shared__ uint32_t s_cand[32];              // this CTA's candidate keys; read by the cluster
  __shared__ uint32_t s_ncand;
  __shared__ uint32_t s_cnt[2];                // this CTA's ties and outright keeps; read by the cluster
  __shared__ uint32_t s_prefix, s_remaining, s_count;
  __shared__ uint32_t w_eq[kTopkWarps], w_gt[kTopkWarps], w_eq_off[kTopkWarps], w_pos[kTopkWarps];
  __shared__ int s_nan;

  const int tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  const int G = static_cast<int>(cluster_nctarank());
  const int rank = static_cast<int>(cluster_ctarank());
  const int b = blockIdx.x / G;
  const int N = a.N;
  const int lo = rank * a.chunk;
  const int hi = min(N, lo + a.chunk);         // hi <= lo: this CTA holds no token
  const size_t base = static_cast<size_t>(b) * N;
  const int Nr = a.r1 - a.r0;
  const int K = a.K;
  const bool keep_all = (K == Nr);
  const bool keep_none = (K == 0);
  const bool select = !keep_all && !keep_none;
  const int rlo = max(lo, a.r0), rhi = min(hi, a.r1);   // this CTA's routable tokens
  uint32_t thr = 0, need_eq = 0;
  if (tid == 0) {
    s_nan = 0;
    s_ncand = 0;
  }
  for (int i = tid; i < kSubHist * 256; i += blockDim.x) (&sub[0][0])[i] = 0;
  __syncthreads();

  // 1. logits (reduced from partial sums in chunk order) -> keys, with pass
  // 0's histogram (top byte) of the routable keys
  uint32_t* my = sub[warp % kSubHist];
  if (a.vec4) {
    reduce_logits_vec4(a, base, lo, hi, keys, my, select, &s_nan);
  } else {
    reduce_logits_scalar(a, base, lo, hi, keys, my, select, &s_nan);
  }
  __syncthreads();

  // 2. radix select of the K-th largest routable key (every CTA of the
  // cluster takes the same branches: they all see the same histograms)
  if (select) {
    uint32_t prefix = 0, pmask = 0, remaining = static_cast<uint32_t>(K);
    int par = 0;
#pragma unroll 1
    for (int shift = 24; shift >= 0; shift -= 8, par ^= 1) {
      if (shift < 24) {   // pass 0 was counted with the keys
#pragma unroll 1
        for (int i = rlo + tid; i < rhi; i += blockDim.x) {
          const uint32_t k = keys[i - lo];
          if ((k & pmask) == prefix) atomicAdd(&my[(k >> shift) & 255u], 1u);
        }
        __syncthreads();
      }
      for (int i = tid; i < 256; i += blockDim.x) {
        uint32_t c = 0;
#pragma unroll
        for (int q = 0; q < kSubHist; ++q) {
          c += sub[q][i];
          sub[q][i] = 0;
        }
        hist[par][i] = c;
      }
      // Every CTA's histogram of this pass is complete.  The other buffer
      // (par ^ 1) is rewritten only in the next pass, after the next cluster
      // barrier, which no CTA passes before its reads of this pass are done.
      cluster_sync();
      if (warp == 0) {
        // The lane's 8 bins: its own CTA's counts, plus every other CTA's,
        // read through distributed shared memory with all loads of a CTA
        // issued before any is added (each one takes a round trip).
        uint32_t local[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) local[j] = hist[par][8 * lane + j];
        const uint32_t addr = smem_u32(&hist[par][8 * lane]);
        for (int r = 1; r < G; ++r) {
          const uint32_t remote = mapa_shared(addr, static_cast<uint32_t>((rank + r) % G));
          uint32_t v[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) v[j] = ld_dsmem_u32(remote + 4u * j);
#pragma unroll
          for (int j = 0; j < 8; ++j) local[j] += v[j];
        }
        uint32_t tot = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) tot += local[j];
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
        // At most 32 routable keys of the sequence share the digits found so
        // far: each CTA publishes its share of them, and one warp per CTA
        // ranks them all.  The threshold is the candidate with fewer than
        // `remaining` larger candidates and at least `remaining` larger or
        // equal ones; need_eq is what is left of `remaining` above it.
        for (int i = rlo + tid; i < rhi; i += blockDim.x) {
          const uint32_t k = keys[i - lo];
          if ((k & pmask) == prefix) s_cand[atomicAdd(&s_ncand, 1u)] = k;
        }
        cluster_sync();
        if (warp == 0) {
          // lane r < G reads CTA r's candidate count; a prefix over the lanes
          // gives each candidate's place; lane l then fetches candidate l.
          const uint32_t nr = lane < G ? ld_dsmem_u32(mapa_shared(smem_u32(&s_ncand), static_cast<uint32_t>(lane))) : 0u;
          const uint32_t before = warp_inclusive_scan(nr, lane) - nr;
          const uint32_t off = __shfl_sync(0xffffffffu, before + nr, G - 1);   // all candidates
          uint32_t k = 0;
          bool have = false;
          for (int r = 0; r < G; ++r) {
            const uint32_t br = __shfl_sync(0xffffffffu, before, r), n = __shfl_sync(0xffffffffu, nr, r);
            if (static_cast<uint32_t>(lane) >= br && static_cast<uint32_t>(lane) < br + n) {
              k = ld_dsmem_u32(mapa_shared(smem_u32(&s_cand[lane - br]), static_cast<uint32_t>(r)));
              have = true;
            }
          }
          uint32_t gt = 0, ge = 0;
          for (uint32_t j = 0; j < off; ++j) {
            const uint32_t o = __shfl_sync(0xffffffffu, k, static_cast<int>(j));
            gt += o > k ? 1u : 0u;
            ge += o >= k ? 1u : 0u;
          }
          if (have && gt < remaining && ge >= remaining) {
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

  // 3. keep decisions in token order.  Warp w owns tokens
  // [lo + w * steps * 32, lo + (w + 1) * steps * 32) of the CTA's range.
  const uint32_t lt = (1u << lane) - 1u;
  const int steps = (a.chunk + blockDim.x - 1) / blockDim.x;
  const int c0 = lo + warp * steps * 32;
  uint32_t eq_w = 0, gt_w = 0;
  for (int st = 0; st < steps; ++st) {
    const int i = c0 + st * 32 + lane;
    const bool valid = i < hi;
    const bool routable = valid && i >= a.r0 && i < a.r1;
    const uint32_t k = valid ? keys[i - lo] : 0u;
    const bool eq = select && routable && k == thr;
    const bool gt = valid && (!routable || keep_all || (select && k > thr));
    eq_w += __popc(__ballot_sync(0xffffffffu, eq));
    gt_w += __popc(__ballot_sync(0xffffffffu, gt));
  }
  if (lane == 0) {
    w_eq[warp] = eq_w;
    w_gt[warp] = gt_w;
  }
  __syncthreads();
  if (warp == 0) {
    const uint32_t e = lane < kTopkWarps ? w_eq[lane] : 0u, g = lane < kTopkWarps ? w_gt[lane] : 0u;
    const uint32_t ei = warp_inclusive_scan(e, lane), gi = warp_inclusive_scan(g, lane);
    if (lane == kTopkWarps - 1) {
      s_cnt[0] = ei;
      s_cnt[1] = gi;
    }
  }
  cluster_sync();   // every CTA's counts are published
  if (warp == 0) {
    // Ties and kept tokens before this CTA: CTA r takes
    // clamp(need_eq - (ties before r), 0, ties of r) of its ties.
    uint32_t er = 0, gr = 0;
    if (lane < G) {
      er = ld_dsmem_u32(mapa_shared(smem_u32(&s_cnt[0]), static_cast<uint32_t>(lane)));
      gr = ld_dsmem_u32(mapa_shared(smem_u32(&s_cnt[1]), static_cast<uint32_t>(lane)));
    }
    const uint32_t eb = warp_inclusive_scan(er, lane) - er;
    const uint32_t take = need_eq > eb ? min(need_eq - eb, er) : 0u;
    const uint32_t kr = gr + take;
    const uint32_t kb = warp_inclusive_scan(kr, lane) - kr;
    const uint32_t eq_before = __shfl_sync(0xffffffffu, eb, rank);
    const uint32_t keep_before = __shfl_sync(0xffffffffu, kb, rank);
    // the same within this CTA, over its warps
    const uint32_t e = lane < kTopkWarps ? w_eq[lane] : 0u, g = lane < kTopkWarps ? w_gt[lane] : 0u;
    const uint32_t ewb = eq_before + warp_inclusive_scan(e, lane) - e;
    const uint32_t wt = need_eq > ewb ? min(need_eq - ewb, e) : 0u;
    const uint32_t wk = g + wt;
    const uint32_t wkb = keep_before + warp_inclusive_scan(wk, lane) - wk;
    if (lane < kTopkWarps) {
      w_eq_off[lane] = ewb;
      w_pos[lane] = wkb;
    }
  }
  cluster_arrive();   // this CTA's reads of the others' shared memory are done
  __syncthreads();

  const int k_tot = K + N - Nr;
  int32_t* idx = a.idx + static_cast<size_t>(b) * k_tot;
  uint32_t er = w_eq_off[warp];
  uint32_t pos = w_pos[warp];
  for (int st = 0; st < steps; ++st) {
    const int i = c0 + st * 32 + lane;
    const bool valid = i < hi;
    const bool routable = valid && i >= a.r0 && i < a.r1;
    const uint32_t k = valid ? keys[i - lo] : 0u;
    const bool eq = select && routable && k == thr;
    const uint32_t eqb = __ballot_sync(0xffffffffu, eq);
    const uint32_t tie_rank = er + __popc(eqb & lt);
    er += __popc(eqb);
    const bool keep = valid && (!routable || keep_all || (select && (k > thr || (eq && tie_rank < need_eq))));
    const uint32_t kb = __ballot_sync(0xffffffffu, keep);
    const uint32_t slot = pos + __popc(kb & lt);
    if (keep && slot < static_cast<uint32_t>(k_tot)) idx[slot] = i;
    if (a.mask && valid) a.mask[base + i] = keep ? 1 : 0;
    pos += __popc(kb);
  }
  if (tid == 0 && s_nan) record_status(a.status, CER_DEV_NAN);
  cluster_wait();     // no CTA leaves while another may still read its shared memory
}

// Cluster size and tokens per CTA for sequences of N tokens.
static void topk_split(int N, int* G, int* chunk) {
  int g = N <= kTopkChunkTarget ? 1 : (N + kTopkChunkTarget - 1) / kTopkChunkTarget;
  g = g < 1 ? 1 : g > kTopkMaxCluster ? kTopkMaxCluster : g;
  int c = (N + g - 1) / g;
  c = (c + 31) / 32 * 32;
  *G = g;
  *chunk = c;
}

cudaError_t launch_topk(const TopkArgs& args, cudaStream_t stream) {
  if (args.B == 0 || args.N == 0) return cudaSuccess;
  TopkArgs a = args;
  int G = 1;
  topk_split(a.N, &G, &a.chunk);
  a.vec4 = (a.N % 4 == 0) && (a.chunk_stride % 4 == 0) && (reinterpret_cast<uintptr_t>(a.src) % 16 == 0);
  const size_t smem = static_cast<size_t>(a.chunk) * sizeof(uint32_t);
  // The limit is raised once per context to the largest chunk ever accepted.
  cudaError_t e = ensure_max_smem(reinterpret_cast<const void*>(topk_kernel), kTopkMaxN * sizeof(uint32_t));
  if (e != cudaSuccess) return e;
  return launch_k(topk_kernel, dim3(a.B * G), dim3(kTopkThreads), smem, stream, G, a);
}

}  // namespace cer
