// score_kernel.cu -- S1: routing logits of the core and expansion scorers
// (Sec. 3.2, Eq. 4, core_expansion_formulation) on tcgen05 tensor cores.
//
// The hidden layers of the core scorer and of the active expansion scorer are
// one GEMM, h [B*N, d] x [W1 ; W1e[m(t_b)]]^T, split into BN-wide hidden
// chunks.  A work tile is (sequence b, 128-token row tile, hidden chunk); its
// epilogue adds the per-sequence bias column (b1, or U emb(t_b) + b1e for the
// expansion), applies the exact-erf GELU in fp32 and folds the chunk into a
// per-token partial score w2 . GELU(.), partial[chunk][b*N + n]: two groups of
// four epilogue warps each fold half the chunk's columns and the second group
// to finish a row adds the two halves.
// The partial scores are summed in chunk order by the consumer (the reduce
// kernel below, or the top-K kernel in the fused block), so the logits do not
// depend on scheduling.
#include <cuda_bf16.h>

#include <cmath>

#include "kernels.h"
#include "umma_gemm.cuh"

namespace cer {

// ---------------------------------------------------------------- bias table

// bias_tab[b][j], w2_tab[b][j] for the concatenated hidden index j in
// [0, Hc + He): core columns take b1 and w2; expansion columns take
// U[m] emb(t_b) + b1e[m] and w2e[m] with m = m(t_b).  Grid (B, nb), nb about
// the SM count over B: each block builds emb(t_b) in shared memory, then its
// 8 warps take the sequence's columns in turn, one column per warp at a time,
// reducing its U row across the lanes (coalesced reads).  About one block per
// SM leaves the registers of every SM to the scorer's CTAs, which start as
// soon as this kernel has: their copies and MMAs do not depend on it, only
// their epilogues read the tables.
//
// emb_j = cos / sin(1000 t f_j).  FP64 transcendentals are very slow on this
// part, so the argument is formed in turns -- x = (1000 t) * f_j / (2 pi), one
// fp64 product with the host-computed table -- reduced exactly in fp64
// (x - rint(x), |r| <= 1/2), and only then handed to the fp32 sincospif.  The
// result differs from the fp64 sinusoid by about 2e-7 before it is rounded
// to fp32.
constexpr int kBiasWarps = 8;

__device__ __forceinline__ void bias_column(const ScoreArgs& a, const float* emb, int m, int b, int j, int Ht,
                                            int lane, float* bias_tab, float* w2_tab) {
  float bias, w2;
  if (j < a.Hc) {
    bias = a.b1 ? a.b1[j] : 0.f;
    w2 = a.w2[j];
  } else {
    const int jj = j - a.Hc;
    float s = 0.f;
    if (a.U != nullptr) {
      const __nv_bfloat16* u = a.U + (static_cast<size_t>(m) * a.He + jj) * a.E;
      for (int e = lane; e < a.E; e += 32) s = fmaf(__bfloat162float(u[e]), emb[e], s);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    }
    bias = (a.b1e ? a.b1e[static_cast<size_t>(m) * a.He + jj] : 0.f) + s;
    w2 = a.w2e[static_cast<size_t>(m) * a.He + jj];
  }
  if (lane == 0) {
    bias_tab[static_cast<size_t>(b) * Ht + j] = bias;
    w2_tab[static_cast<size_t>(b) * Ht + j] = w2;
  }
}

__global__ void __launch_bounds__(32 * kBiasWarps) time_bias_kernel(ScoreArgs a,
                                                                    const __grid_constant__ EmbFreqTable ft,
                                                                    float* bias_tab, float* w2_tab) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ float emb[];
  const int b = blockIdx.x;
  const int Ht = a.Hc + (a.gen ? a.He : 0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int m = 0;
  if (a.gen) {
    const float t = a.t[b];
    const double seg = floor(static_cast<double>(t) * a.S);
    m = seg < a.S - 1 ? static_cast<int>(seg) : a.S - 1;
    if (m < 0) m = 0;
    if (a.U != nullptr) {
      const int half = a.E / 2;
      const double t1000 = 1000.0 * static_cast<double>(t);
      for (int j = threadIdx.x; j < half; j += blockDim.x) {
        const double x = t1000 * ft.g[j];                    // turns
        const float r = static_cast<float>(x - rint(x));     // exact reduction, |r| <= 1/2
        float sn, cs;
        sincospif(2.0f * r, &sn, &cs);
        emb[j] = cs;
        emb[half + j] = sn;
      }
    }
  }
  __syncthreads();
  const int step = gridDim.y * kBiasWarps;
  // two columns per round, their loads in flight together
  int j = blockIdx.y * kBiasWarps + warp;
  for (; j + step < Ht; j += 2 * step) {
    bias_column(a, emb, m, b, j, Ht, lane, bias_tab, w2_tab);
    bias_column(a, emb, m, b, j + step, Ht, lane, bias_tab, w2_tab);
  }
  if (j < Ht) bias_column(a, emb, m, b, j, Ht, lane, bias_tab, w2_tab);
}

// ---------------------------------------------------------------- scorer GEMM

// GELU(x) = x * Phi(x), Phi the standard normal CDF, with erf from the
// rational approximation of Abramowitz & Stegun, Handbook of Mathematical
// Functions, formula 7.1.26 (|error| <= 1.5e-7 for all z >= 0):
//   erf(z) = 1 - (a1 t + a2 t^2 + a3 t^3 + a4 t^4 + a5 t^5) exp(-z^2),
//   t = 1 / (1 + p z).
// With q = poly(t) exp(-z^2), z = |x|/sqrt(2): Phi(x) = 1 - q/2 for x >= 0
// and q/2 for x < 0.  Two MUFU operations and ~12 FMA-pipe instructions per
// element, against ~25 for erff; the scorer's epilogue evaluates one GELU
// per hidden unit and token, so this is its inner loop.  The approximation
// and the fast exponential/reciprocal add < 1e-6 |x| to GELU, far inside
// the score tolerance (checked against the fp64 oracle in the parity tests).
__device__ __forceinline__ float gelu_as(float x) {
  const float z = fabsf(x) * 0.70710678118654752f;
  const float t = __fdividef(1.0f, fmaf(0.3275911f, z, 1.0f));
  float poly = fmaf(1.061405429f, t, -1.453152027f);
  poly = fmaf(poly, t, 1.421413741f);
  poly = fmaf(poly, t, -0.284496736f);
  poly = fmaf(poly, t, 0.254829592f);
  poly *= t;
  const float q = poly * __expf(-z * z);
  const float phi = x >= 0.0f ? fmaf(-0.5f, q, 1.0f) : 0.5f * q;
  return x * phi;
}

// The two epilogue groups fold disjoint column halves of the same accumulator
// rows (warps w and w + 4 read the same TMEM lanes); whichever finishes a row
// second adds the halves, half 0's sum on the left (fp32 addition of two
// terms does not depend on their order either way).  Per accumulator buffer
// there is one sum slot per half and row and one arrival counter per row.
// A buffer's slots come round again two tiles later, after both groups have
// released that buffer; the counters only grow (an odd prior count marks the
// second arrival), so nothing waits and nothing is reset.  Returns whether
// this thread holds the row's chunk score in *out.
constexpr uint32_t kHalfSumBytes = 2 * 2 * 128 * 4;
constexpr uint32_t kHalfCountBytes = 2 * 128 * 4;
__device__ __forceinline__ bool combine_halves(const EpiCtx& ctx, int row, int half, float s, float* out) {
  volatile float* sum = reinterpret_cast<volatile float*>(ctx.smem) + ctx.acc * 256;   // [half][row]
  uint32_t* cnt = reinterpret_cast<uint32_t*>(ctx.smem + kHalfSumBytes) + ctx.acc * 128;
  sum[half * 128 + row] = s;
  __threadfence_block();
  const uint32_t prior = atomicAdd(&cnt[row], 1u);
  if ((prior & 1u) == 0u) return false;
  __threadfence_block();
  const float other = sum[(half ^ 1) * 128 + row];
  *out = half == 0 ? s + other : other + s;
  return true;
}

template <int BN_>
struct ScoreProblem {
  static constexpr int BN = BN_;
  static constexpr int MMA_PAIR = 0;
  static constexpr int CLUSTER = 1;
  static constexpr int KSUB = BN == 256 ? 1 : 2;   // K blocks per ring slot
  static constexpr int STAGES = BN == 128 ? 3 : 4;
  static constexpr int B_MN_MAJOR = 0;
  static constexpr int EPI_WARPS = 8;
  static constexpr uint32_t kBStepBytes = 32;
  static constexpr uint32_t kEpiSmemBytes = kHalfSumBytes + kHalfCountBytes;
  static constexpr uint32_t kEpiZeroBytes = kEpiSmemBytes;

  struct Params {
    CUtensorMap tm_h;    // h as [B*N, d], box 64 x 128
    CUtensorMap tm_w1;   // core W1 [Hc, d], box 64 x BN
    CUtensorMap tm_w1e;  // expansion W1e as [S*He, d], box 64 x BN
    const float* t;
    const float* bias_tab;   // [B][Ht], or NULL: columns take b1 (or 0) and w2 directly
    const float* w2_tab;
    const float* b1;
    const float* w2;
    float* partial;
    int* status;
    int B, N, d, S, He, Ht;
    int n_rt, n_core, n_chunks;
    int acts_first;      // the previous kernel (the bias-table kernel) writes no h
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
  __device__ static void prod_tile(const Params& p, int tile, int, ProdState& st) {
    decode(p, tile, st.b, st.rt, st.chunk);
    if (st.chunk < p.n_core) {
      st.wrow = st.chunk * BN;
    } else {
      int m = 0;
      if (p.S > 1) {
        const double seg = floor(static_cast<double>(p.t[st.b]) * p.S);
        m = seg < p.S - 1 ? static_cast<int>(seg) : p.S - 1;
        if (m < 0) m = 0;
      }
      st.wrow = m * p.He + (st.chunk - p.n_core) * BN;
    }
  }
  // With several expansion segments the weight rows depend on t, which a
  // previous kernel may write; with one, the weights may go out first.
  __device__ static bool weights_first(const Params& p) { return p.S <= 1; }
  __device__ static bool acts_first(const Params& p) { return p.acts_first != 0; }
  __device__ static uint32_t stage_bytes(const Params&, int, int, int part) {
    return ((part & kPartAct) ? kATileBytes : 0u) + ((part & kPartWeights) ? BN * 128u : 0u);
  }
  __device__ static void prod_kb(const Params& p, const ProdState& st, int, int kb, int lane, uint8_t* a,
                                 uint8_t* b, uint64_t* bar, int part) {
    if (lane == 0) {
      const int x = kb * 64;   // K blocks past d load as zeros
      if (part & kPartAct) tma_load_2d(a, &p.tm_h, bar, x, st.b * p.N + st.rt * 128);
      if (part & kPartWeights) tma_load_2d(b, st.chunk < p.n_core ? &p.tm_w1 : &p.tm_w1e, bar, x, st.wrow);
    }
  }
  __device__ static uint64_t bdesc(uint32_t saddr) { return sdesc_kmajor_sw128(saddr); }
  __device__ static void prefetch(const Params& p) {
    tma_prefetch_desc(&p.tm_h);
    tma_prefetch_desc(&p.tm_w1);
    tma_prefetch_desc(&p.tm_w1e);
  }

  __device__ static void epilogue_done(const Params&, int, int) {}
  __device__ static bool epilogue(const Params& p, int tile, int row, int half, uint32_t taddr, EpiCtx& ctx) {
    int b, rt, chunk;
    decode(p, tile, b, rt, chunk);
    const float* bias = p.bias_tab ? p.bias_tab + static_cast<size_t>(b) * p.Ht + chunk * BN
                                   : (p.b1 ? p.b1 + chunk * BN : nullptr);
    const float* w2 = p.w2_tab ? p.w2_tab + static_cast<size_t>(b) * p.Ht + chunk * BN : p.w2 + chunk * BN;
    float s = 0.f;
#pragma unroll 1
    for (int c = half * (BN / 64); c < (half + 1) * (BN / 64); ++c) {
      float v[32];
      tmem_ld_32x32(taddr + c * 32, v);
      const float4* b4 = bias ? reinterpret_cast<const float4*>(bias + c * 32) : nullptr;
      const float4* w4 = reinterpret_cast<const float4*>(w2 + c * 32);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float4 bb = b4 ? __ldg(b4 + q) : make_float4(0.f, 0.f, 0.f, 0.f), ww = __ldg(w4 + q);
        s = fmaf(ww.x, gelu_as(v[4 * q + 0] + bb.x), s);
        s = fmaf(ww.y, gelu_as(v[4 * q + 1] + bb.y), s);
        s = fmaf(ww.z, gelu_as(v[4 * q + 2] + bb.z), s);
        s = fmaf(ww.w, gelu_as(v[4 * q + 3] + bb.w), s);
      }
    }
    const int n = rt * 128 + row;
    float score;
    if (combine_halves(ctx, row, half, s, &score) && n < p.N)
      p.partial[static_cast<size_t>(chunk) * p.B * p.N + static_cast<size_t>(b) * p.N + n] = score;
    return true;
  }
};

// The same scorer as pair MMAs (tcgen05 cta_group::2) for wide hidden layers,
// where the scorer is bound by the tensor pipe (Hc + He >= 512): a work tile
// is 256 consecutive rows of h viewed as [B*N, d] (tiles may straddle
// sequences) times one 256-wide hidden chunk.  Each CTA of the pair loads its
// 128 rows and 128 of the chunk's weight rows, so an SM takes in 32 KB per
// 64-wide K block for a 128 x 256 x 64 product instead of the 48 KB of a
// one-CTA 128 x 256 tile.  Each CTA's tensor memory receives all 256
// columns of its 128 rows; its epilogue is ScoreProblem's, with the bias and
// w2 tables looked up per row (b = row / N).  One expansion segment only
// (the weight chunk must be the same for both CTAs of a pair).
struct ScorePairProblem {
  static constexpr int BN = 256;
  static constexpr int MMA_PAIR = 1;
  static constexpr int CLUSTER = 2;
  static constexpr int KSUB = 2;
  static constexpr int STAGES = 3;
  static constexpr int B_MN_MAJOR = 0;
  static constexpr int EPI_WARPS = 8;
  static constexpr uint32_t kBStepBytes = 32;
  static constexpr uint32_t kEpiSmemBytes = kHalfSumBytes + kHalfCountBytes;
  static constexpr uint32_t kEpiZeroBytes = kEpiSmemBytes;
  static constexpr uint32_t kBoxBytes = 128 * 128;   // 128 weight rows x 64 bf16

  struct Params {
    CUtensorMap tm_h;    // h as [B*N, d], box 64 x 128
    CUtensorMap tm_w1;   // core W1 [Hc, d], box 64 x 128
    CUtensorMap tm_w1e;  // expansion W1e [He, d], box 64 x 128
    const float* bias_tab;   // [B][Ht], or NULL: columns take b1 (or 0) and w2 directly
    const float* w2_tab;
    const float* b1;
    const float* w2;
    float* partial;
    int* status;
    int rows, N, d, Ht;      // rows = B * N
    int n_rp, n_core, n_chunks;
    int acts_first;          // the previous kernel (the bias-table kernel) writes no h
  };
  struct ProdState {
    int m0, wrow, core;
  };

  // Cluster tile t: row pair t / n_chunks (rows 256 (t / n_chunks) + 128 rank ..), chunk t % n_chunks.
  // The chunks of a row pair are consecutive tiles, so they run side by side
  // and read the pair's rows of h from L2 while they are there (chunk-major
  // order measured 56.5 against 54.2 us at long_7b).
  __device__ static int num_tiles(const Params& p) { return p.n_rp * p.n_chunks; }
  __device__ static int num_kb(const Params& p) { return p.d / 64; }
  __device__ static bool weights_first(const Params&) { return true; }
  __device__ static bool acts_first(const Params& p) { return p.acts_first != 0; }
  __device__ static uint32_t stage_bytes(const Params&, int, int, int part) {
    return 2 * (((part & kPartAct) ? kATileBytes : 0u) + ((part & kPartWeights) ? kBoxBytes : 0u));
  }
  __device__ static void prod_tile(const Params& p, int tile, int rank, ProdState& st) {
    const int chunk = tile % p.n_chunks;
    st.m0 = (2 * (tile / p.n_chunks) + rank) * 128;   // rows past B*N load as zeros
    st.core = chunk < p.n_core;
    st.wrow = (st.core ? chunk : chunk - p.n_core) * BN + rank * 128;
  }
  __device__ static void prod_kb(const Params& p, const ProdState& st, int, int kb, int lane, uint8_t* a,
                                 uint8_t* b, uint32_t leader_bar, int part) {
    if (lane == 0) {
      const int x = kb * 64;
      if (part & kPartAct) tma_load_2d_pair(a, &p.tm_h, leader_bar, x, st.m0);
      if (part & kPartWeights) tma_load_2d_pair(b, st.core ? &p.tm_w1 : &p.tm_w1e, leader_bar, x, st.wrow);
    }
  }
  __device__ static uint64_t bdesc(uint32_t saddr) { return sdesc_kmajor_sw128(saddr); }
  __device__ static void prefetch(const Params& p) {
    tma_prefetch_desc(&p.tm_h);
    tma_prefetch_desc(&p.tm_w1);
    tma_prefetch_desc(&p.tm_w1e);
  }

  __device__ static void epilogue_done(const Params&, int, int) {}
  __device__ static bool epilogue(const Params& p, int tile, int row, int half, uint32_t taddr, EpiCtx& ctx) {
    const int chunk = tile % p.n_chunks;
    const int grow = (2 * (tile / p.n_chunks) + ctx.rank) * 128 + row;
    // Rows past B*N (the ragged last tile) still take part in every tensor
    // memory load -- tcgen05.ld is warp-collective (.sync.aligned) -- and
    // only skip the store; their bias and w2 come from the last sequence.
    const bool valid = grow < p.rows;
    const int b = (valid ? grow : p.rows - 1) / p.N;
    const float* bias = p.bias_tab ? p.bias_tab + static_cast<size_t>(b) * p.Ht + chunk * BN
                                   : (p.b1 ? p.b1 + chunk * BN : nullptr);
    const float* w2 = p.w2_tab ? p.w2_tab + static_cast<size_t>(b) * p.Ht + chunk * BN : p.w2 + chunk * BN;
    float s = 0.f;
#pragma unroll 1
    for (int c = half * 4; c < half * 4 + 4; ++c) {
      float v[32];
      tmem_ld_32x32(taddr + c * 32, v);
      const float4* b4 = bias ? reinterpret_cast<const float4*>(bias + c * 32) : nullptr;
      const float4* w4 = reinterpret_cast<const float4*>(w2 + c * 32);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float4 bb = b4 ? __ldg(b4 + q) : make_float4(0.f, 0.f, 0.f, 0.f), ww = __ldg(w4 + q);
        s = fmaf(ww.x, gelu_as(v[4 * q + 0] + bb.x), s);
        s = fmaf(ww.y, gelu_as(v[4 * q + 1] + bb.y), s);
        s = fmaf(ww.z, gelu_as(v[4 * q + 2] + bb.z), s);
        s = fmaf(ww.w, gelu_as(v[4 * q + 3] + bb.w), s);
      }
    }
    float score;
    if (combine_halves(ctx, row, half, s, &score) && valid) p.partial[static_cast<size_t>(chunk) * p.rows + grow] = score;
    return true;
  }
};

// ---------------------------------------------------------------- reduce

__global__ void score_reduce_kernel(const float* __restrict__ partial, int n_chunks, size_t total,
                                    float* __restrict__ logits, float* __restrict__ probs) {
  griddep_wait();
  griddep_launch_dependents();
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
  return (Hc + (gen ? He : 0)) / 64;
}

// Chunk width for a launch: the widest whose tiles fill at least ~90% of a
// wave, else the narrowest available (more, smaller tiles).  Generation at
// B = 8, N = 1088 (144 tiles of 256 hidden units on 152 SMs) measured 2 us
// faster as one 256-wide wave than as two waves of 128-wide tiles.
static int pick_chunk_width(const ScoreArgs& a, int n_sm) {
  const int Ht = a.Hc + (a.gen ? a.He : 0);
  const long rows = static_cast<long>(a.B) * ((a.N + 127) / 128);
  int best = 0;
  for (int bn : {256, 128, 64}) {
    if (a.Hc % bn != 0 || (a.gen && a.He % bn != 0)) continue;
    best = bn;
    if (10 * rows * (Ht / bn) >= 9 * static_cast<long>(n_sm)) return bn;   // at least ~90% of a wave
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
  p.b1 = a.b1;
  p.w2 = a.w2;
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
  p.acts_first = bias_tab != nullptr;   // generation: right behind the bias-table kernel
  return launch_gemm<P>(p, a.B * p.n_rt * p.n_chunks, a.d / 64, nullptr, n_sm, stream);
}

// Whether the pair-MMA scorer takes this launch: wide hidden layers (the
// tensor-bound case), whole 256-wide chunks, one expansion segment.
static bool use_pair_scorer(const ScoreArgs& a) {
  const int Ht = a.Hc + (a.gen ? a.He : 0);
  return Ht >= 512 && a.Hc % 256 == 0 && (!a.gen || (a.He % 256 == 0 && a.S == 1));
}

static cudaError_t launch_score_pair(const ScoreArgs& a, const float* bias_tab, const float* w2_tab, float* partial,
                                     const StreamKArea* sk, int n_sm, cudaStream_t stream) {
  using P = ScorePairProblem;
  P::Params p{};
  const int Ht = a.Hc + (a.gen ? a.He : 0);
  const uint64_t rows = static_cast<uint64_t>(a.B) * a.N;
  if (!encode_bf16_2d(&p.tm_h, a.h, rows, a.d, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_w1, a.W1, a.Hc, a.d, 64, 128)) return cudaErrorInvalidValue;
  if (a.gen) {
    if (!encode_bf16_2d(&p.tm_w1e, a.W1e, a.He, a.d, 64, 128)) return cudaErrorInvalidValue;
  } else {
    p.tm_w1e = p.tm_w1;
  }
  p.bias_tab = bias_tab;
  p.w2_tab = w2_tab;
  p.b1 = a.b1;
  p.w2 = a.w2;
  p.partial = partial;
  p.status = a.status;
  p.rows = static_cast<int>(rows);
  p.N = a.N;
  p.d = a.d;
  p.Ht = Ht;
  p.n_rp = static_cast<int>((rows + 255) / 256);
  p.n_core = a.Hc / 256;
  p.n_chunks = Ht / 256;
  p.acts_first = bias_tab != nullptr;   // generation: right behind the bias-table kernel
  return launch_gemm<P>(p, p.n_rp * p.n_chunks, a.d / 64, sk, n_sm, stream);
}

// Understanding reads b1 and w2 directly (bias/w2 tables NULL); generation
// first builds the per-sequence tables.
static cudaError_t launch_score_chunks(const ScoreArgs& a, const float* bias_tab, const float* w2_tab,
                                       float* partial, const StreamKArea* sk, int n_sm, cudaStream_t stream,
                                       int* n_partials) {
  if (use_pair_scorer(a)) {
    *n_partials = (a.Hc + (a.gen ? a.He : 0)) / 256;
    return launch_score_pair(a, bias_tab, w2_tab, partial, sk, n_sm, stream);
  }
  const int bn = pick_chunk_width(a, n_sm);
  *n_partials = bn ? (a.Hc + (a.gen ? a.He : 0)) / bn : 0;
  switch (bn) {
    case 256: return launch_score_gemm<256>(a, bias_tab, w2_tab, partial, n_sm, stream);
    case 128: return launch_score_gemm<128>(a, bias_tab, w2_tab, partial, n_sm, stream);
    case 64: return launch_score_gemm<64>(a, bias_tab, w2_tab, partial, n_sm, stream);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_score(const ScoreArgs& a, const ScoreWorkspace& ws, const StreamKArea* sk, int n_sm,
                         cudaStream_t stream, int* n_partials) {
  if (!a.gen) return launch_score_chunks(a, nullptr, nullptr, ws.partial, sk, n_sm, stream, n_partials);
  const int emb_bytes = a.U ? a.E * static_cast<int>(sizeof(float)) : 0;
  const int Ht = a.Hc + a.He;
  EmbFreqTable ft;
  const int half = (a.gen && a.U) ? a.E / 2 : 0;
  for (int j = 0; j < half; ++j) ft.g[j] = std::pow(10000.0, -static_cast<double>(j) / half) / (2.0 * M_PI);
  for (int j = half; j < 512; ++j) ft.g[j] = 0.0;
  int nb = (n_sm + a.B - 1) / a.B;
  const int max_nb = (Ht + kBiasWarps - 1) / kBiasWarps;
  if (nb > max_nb) nb = max_nb;
  if (nb < 1) nb = 1;
  const dim3 bias_grid(a.B, nb);
  cudaError_t e = launch_k(time_bias_kernel, bias_grid, dim3(32 * kBiasWarps), emb_bytes, stream, 1, a, ft,
                           ws.bias_tab, ws.w2_tab);
  if (e != cudaSuccess) return e;
  return launch_score_chunks(a, ws.bias_tab, ws.w2_tab, ws.partial, sk, n_sm, stream, n_partials);
}

cudaError_t launch_score_reduce(const float* partial, int n_chunks, size_t total, float* logits, float* probs,
                                int n_sm, cudaStream_t stream) {
  if (total == 0) return cudaSuccess;
  size_t blocks = (total + 255) / 256;
  const size_t cap = static_cast<size_t>(n_sm) * 8;
  if (blocks > cap) blocks = cap;
  return launch_k(score_reduce_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, stream, 1, partial,
                  n_chunks, total, logits, probs);
}

}  // namespace cer
