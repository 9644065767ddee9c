// score_kernel.cu -- S1: routing logits of the core and expansion scorers
// (Sec. 3.2, Eq. 1) on tcgen05 tensor cores.
//
// The hidden layers of the core scorer and of the active expansion scorer are
// one GEMM, h [B*N, d] x [W1 ; W1e[m(t_b)]]^T, split into BN-wide hidden
// chunks.  A work tile is (sequence b, 128-token row tile, hidden chunk); its
// epilogue adds the per-sequence bias column (b1, or U emb(t_b) + b1e for the
// expansion), applies the exact-erf GELU in fp32 and folds the chunk into a
// per-token partial score w2 . GELU(.); each half of the chunk's columns
// (one per group of four epilogue warps) writes partial[2*chunk + half][b*N + n].
// The partial scores are summed in chunk order by the consumer (the reduce
// kernel below, or the top-K kernel in the fused block), so the logits do not
// depend on scheduling.
#include <cuda_bf16.h>

#include "kernels.h"
#include "umma_gemm.cuh"

namespace cer {

// ---------------------------------------------------------------- bias table

// One block per sequence.  bias_tab[b][j], w2_tab[b][j] for the concatenated
// hidden index j in [0, Hc + He): core columns take b1 and w2; expansion
// columns take U[m] emb(t_b) + b1e[m] and w2e[m] with m = m(t_b).
__global__ void time_bias_kernel(ScoreArgs a, float* bias_tab, float* w2_tab) {
  extern __shared__ float emb[];
  const int b = blockIdx.x;
  const int Ht = a.Hc + (a.gen ? a.He : 0);
  int m = 0;
  float t = 0.f;
  if (a.gen) {
    t = a.t[b];
    const double seg = floor(static_cast<double>(t) * a.S);
    m = seg < a.S - 1 ? static_cast<int>(seg) : a.S - 1;
    if (m < 0) m = 0;
    if (a.U != nullptr) {
      const int half = a.E / 2;
      for (int j = threadIdx.x; j < half; j += blockDim.x) {
        const double f = pow(10000.0, -static_cast<double>(j) / half);
        const double arg = 1000.0 * static_cast<double>(t) * f;
        emb[j] = static_cast<float>(cos(arg));
        emb[half + j] = static_cast<float>(sin(arg));
      }
    }
  }
  __syncthreads();
  for (int j = threadIdx.x; j < Ht; j += blockDim.x) {
    float bias, w2;
    if (j < a.Hc) {
      bias = a.b1 ? a.b1[j] : 0.f;
      w2 = a.w2[j];
    } else {
      const int jj = j - a.Hc;
      bias = a.b1e ? a.b1e[static_cast<size_t>(m) * a.He + jj] : 0.f;
      if (a.U != nullptr) {
        const __nv_bfloat16* u = a.U + (static_cast<size_t>(m) * a.He + jj) * a.E;
        float s = 0.f;
        for (int e = 0; e < a.E; ++e) s = fmaf(__bfloat162float(u[e]), emb[e], s);
        bias += s;
      }
      w2 = a.w2e[static_cast<size_t>(m) * a.He + jj];
    }
    bias_tab[static_cast<size_t>(b) * Ht + j] = bias;
    w2_tab[static_cast<size_t>(b) * Ht + j] = w2;
  }
}

// ---------------------------------------------------------------- scorer GEMM

__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

template <int BN_>
struct ScoreProblem {
  static constexpr int BN = BN_;
  static constexpr int STAGES = BN == 256 ? 4 : BN == 128 ? 6 : 8;
  static constexpr int B_MN_MAJOR = 0;
  static constexpr uint32_t kBStepBytes = 32;

  struct Params {
    CUtensorMap tm_h;    // h as [B*N, d], box 64 x 128
    CUtensorMap tm_w1;   // core W1 [Hc, d], box 64 x BN
    CUtensorMap tm_w1e;  // expansion W1e as [S*He, d], box 64 x BN
    const float* t;
    const float* bias_tab;
    const float* w2_tab;
    float* partial;
    int* status;
    int B, N, d, S, He, Ht;
    int n_rt, n_core, n_chunks;
  };
  struct ProdState {
    int b, rt, chunk, wrow;
  };

  __device__ static int num_tiles(const Params& p) { return p.B * p.n_rt * p.n_chunks; }
  __device__ static int num_kb(const Params& p) { return p.d / 64; }
  __device__ static void decode(const Params& p, int tile, int& b, int& rt, int& chunk) {
    chunk = tile % p.n_chunks;
    const int rest = tile / p.n_chunks;
    rt = rest % p.n_rt;
    b = rest / p.n_rt;
  }
  __device__ static void prod_tile(const Params& p, int tile, int lane, ProdState& st) {
    decode(p, tile, st.b, st.rt, st.chunk);
    if (st.chunk < p.n_core) {
      st.wrow = st.chunk * BN;
    } else {
      const double seg = floor(static_cast<double>(p.t[st.b]) * p.S);
      int m = seg < p.S - 1 ? static_cast<int>(seg) : p.S - 1;
      if (m < 0) m = 0;
      st.wrow = m * p.He + (st.chunk - p.n_core) * BN;
    }
  }
  __device__ static uint32_t stage_bytes(const Params&, int, int) { return kATileBytes + BN * 128; }
  __device__ static void prod_kb(const Params& p, const ProdState& st, int, int kb, int lane, uint8_t* a,
                                 uint8_t* b, uint64_t* bar) {
    if (lane == 0) {
      tma_load_2d(a, &p.tm_h, bar, kb * 64, st.b * p.N + st.rt * 128);
      if (st.chunk < p.n_core)
        tma_load_2d(b, &p.tm_w1, bar, kb * 64, st.wrow);
      else
        tma_load_2d(b, &p.tm_w1e, bar, kb * 64, st.wrow);
    }
  }
  __device__ static uint64_t bdesc(uint32_t saddr) { return sdesc_kmajor_sw128(saddr); }

  __device__ static void epilogue(const Params& p, int tile, int row, int half, uint32_t taddr) {
    int b, rt, chunk;
    decode(p, tile, b, rt, chunk);
    const float* bias = p.bias_tab + static_cast<size_t>(b) * p.Ht + chunk * BN;
    const float* w2 = p.w2_tab + static_cast<size_t>(b) * p.Ht + chunk * BN;
    float s = 0.f;
#pragma unroll 1
    for (int c = half * (BN / 64); c < (half + 1) * (BN / 64); ++c) {
      float v[32];
      tmem_ld_32x32(taddr + c * 32, v);
#pragma unroll
      for (int j = 0; j < 32; ++j) s = fmaf(__ldg(w2 + c * 32 + j), gelu_erf(v[j] + __ldg(bias + c * 32 + j)), s);
    }
    const int n = rt * 128 + row;
    if (n < p.N) p.partial[static_cast<size_t>(2 * chunk + half) * p.B * p.N + static_cast<size_t>(b) * p.N + n] = s;
  }
};

// ---------------------------------------------------------------- reduce

__global__ void score_reduce_kernel(const float* __restrict__ partial, int n_chunks, size_t total,
                                    float* __restrict__ logits, float* __restrict__ probs) {
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    float s = partial[i];
    for (int c = 1; c < n_chunks; ++c) s += partial[static_cast<size_t>(c) * total + i];
    logits[i] = s;
    if (probs) probs[i] = 1.0f / (1.0f + expf(-s));
  }
}

// ---------------------------------------------------------------- host side

int score_chunk_width(int Hc, int He, int gen) {
  for (int bn : {256, 128, 64}) {
    if (Hc % bn == 0 && (!gen || He % bn == 0)) return bn;
  }
  return 0;
}

int score_max_partials(int Hc, int He, int gen) {
  if (score_chunk_width(Hc, He, gen) == 0) return 0;
  return 2 * (Hc + (gen ? He : 0)) / 64;
}

// Chunk width for a launch: the widest that still gives every SM a tile,
// else the narrowest available (more, smaller tiles).
static int pick_chunk_width(const ScoreArgs& a, int n_sm) {
  const int Ht = a.Hc + (a.gen ? a.He : 0);
  const long rows = static_cast<long>(a.B) * ((a.N + 127) / 128);
  int best = 0;
  for (int bn : {256, 128, 64}) {
    if (a.Hc % bn != 0 || (a.gen && a.He % bn != 0)) continue;
    best = bn;
    if (rows * (Ht / bn) >= n_sm) return bn;
  }
  return best;
}

template <int BN>
static cudaError_t launch_score_gemm(const ScoreArgs& a, const float* bias_tab, const float* w2_tab,
                                     float* partial, int n_sm, cudaStream_t stream) {
  using P = ScoreProblem<BN>;
  typename P::Params p{};
  const int Ht = a.Hc + (a.gen ? a.He : 0);
  if (!encode_bf16_2d(&p.tm_h, a.h, static_cast<uint64_t>(a.B) * a.N, a.d, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_w1, a.W1, a.Hc, a.d, 64, BN)) return cudaErrorInvalidValue;
  if (a.gen) {
    if (!encode_bf16_2d(&p.tm_w1e, a.W1e, static_cast<uint64_t>(a.S) * a.He, a.d, 64, BN))
      return cudaErrorInvalidValue;
  } else {
    p.tm_w1e = p.tm_w1;
  }
  p.t = a.t;
  p.bias_tab = bias_tab;
  p.w2_tab = w2_tab;
  p.partial = partial;
  p.status = a.status;
  p.B = a.B;
  p.N = a.N;
  p.d = a.d;
  p.S = a.S;
  p.He = a.He;
  p.Ht = Ht;
  p.n_rt = (a.N + 127) / 128;
  p.n_core = a.Hc / BN;
  p.n_chunks = Ht / BN;
  const int tiles = a.B * p.n_rt * p.n_chunks;
  if (tiles == 0) return cudaSuccess;
  const size_t smem = gemm_smem_bytes<P>();
  cudaError_t e = ensure_max_smem(reinterpret_cast<const void*>(umma_gemm_kernel<P>), smem);
  if (e != cudaSuccess) return e;
  const int grid = tiles < n_sm ? tiles : n_sm;
  umma_gemm_kernel<P><<<grid, kGemmThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_score(const ScoreArgs& a, const ScoreWorkspace& ws, int n_sm, cudaStream_t stream,
                         int* n_partials) {
  const int emb_bytes = (a.gen && a.U) ? a.E * static_cast<int>(sizeof(float)) : 0;
  time_bias_kernel<<<a.B, 256, emb_bytes, stream>>>(a, ws.bias_tab, ws.w2_tab);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int bn = pick_chunk_width(a, n_sm);
  *n_partials = bn ? 2 * (a.Hc + (a.gen ? a.He : 0)) / bn : 0;
  switch (bn) {
    case 256: return launch_score_gemm<256>(a, ws.bias_tab, ws.w2_tab, ws.partial, n_sm, stream);
    case 128: return launch_score_gemm<128>(a, ws.bias_tab, ws.w2_tab, ws.partial, n_sm, stream);
    case 64: return launch_score_gemm<64>(a, ws.bias_tab, ws.w2_tab, ws.partial, n_sm, stream);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_score_reduce(const float* partial, int n_chunks, size_t total, float* logits, float* probs,
                                int n_sm, cudaStream_t stream) {
  if (total == 0) return cudaSuccess;
  size_t blocks = (total + 255) / 256;
  const size_t cap = static_cast<size_t>(n_sm) * 8;
  if (blocks > cap) blocks = cap;
  score_reduce_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(partial, n_chunks, total, logits, probs);
  return cudaGetLastError();
}

}  // namespace cer
