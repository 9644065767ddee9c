// ffn_kernel.cu -- S4 (+S5 fused): the channel-pruned SwiGLU FFN on the
// packed rows (Sec. 3.4 compaction and FFN pruning; SwiGLU of the Qwen2.5
// backbone, App. A.5), as two tcgen05 GEMMs over dense operands.
//
// The kept rows X [M, d] and the kept-channel weight slices Wg, Wu, WdT
// [C, d] arrive packed (row gathers run as separate HBM-bound copies: TMA
// 4-row gathers inside the GEMM producer measured 2.4x slower), so every
// operand tile is one TMA box.
//
// gate/up:  act[m, c] = SiLU(Wg[c] . x_m) * (Wu[c] . x_m)
//   One 128x256 MMA tile holds gate (columns 0..127) and up (128..255) for
//   the same 128 channels, so the SwiGLU runs in the epilogue and act is
//   written once, as bf16: each half of the epilogue warps stages its
//   128 x 64 act box in shared memory (128-byte swizzle, conflict-free) and
//   one thread writes it with a TMA store, overlapping the next tile.
// down:     y[m, n] = sum_c act[m, c] * WdT[c, n]
//   B is MN-major: 64 channel rows x BN output columns (BN = 128, 192 or 256,
//   picked per launch so the tiles fill the SMs), one 64-column TMA box per
//   64 columns per K block.  Epilogue: Y = bf16(y), or, fused, the unpack
//   out[b, idx[m], n] = bf16(h[b, idx[m], n] + y) -- the kept rows are
//   distinct, so no atomics; dropped rows are never touched.
#include <cuda_bf16.h>

#include "kernels.h"
#include "umma_gemm.cuh"

namespace cer {

// SiLU(g) * u with the fast exponential and division: the result is rounded
// to bf16 (8 significant bits), far coarser than their error.  The exponent
// argument is clamped so 1 + e^-g stays finite (SiLU(g) ~ 0 there anyway).
__device__ __forceinline__ float silu_mul(float g, float u) {
  return __fdividef(g * u, 1.0f + __expf(fminf(-g, 80.0f)));
}

// ---------------------------------------------------------------- gate/up

// Two CTAs of a cluster take adjacent 128-row tiles of the same 128 channels
// as one M=256 x N=256 pair MMA: rank 0 holds the gate rows of the weight
// tile, rank 1 the up rows, and each CTA receives only its own 32 KB per K
// block (the one-CTA form with the weight tile multicast to both received
// 48 KB and measured 3-6% slower); the ring has room for six slots.
template <int EPI_WARPS_>
struct GateUpProblemT {
  static constexpr int BN = 256;
  static constexpr int MMA_PAIR = 1;
  static constexpr int KSUB = 2;
  static constexpr int STAGES = 3;
  static constexpr int B_MN_MAJOR = 0;
  static constexpr int EPI_WARPS = EPI_WARPS_;
  static constexpr int kGroups = EPI_WARPS / 4;
  // A group's SwiGLU reads the gate columns of its channels and the up
  // columns 128 further on; with two groups each would read columns of the
  // other group's half, which a stream-K owner fixes up only for its own
  // half (and eight warps measured 3% slower anyway).
  static_assert(EPI_WARPS == 4, "one epilogue group reads both accumulator halves");
  static constexpr int CLUSTER = 2;
  static constexpr uint32_t kBStepBytes = 32;
  static constexpr uint32_t kBoxBytes = 128 * 128;          // 128 rows x 64 bf16
  static constexpr uint32_t kEpiSmemBytes = 2 * kBoxBytes;  // the act tile as two TMA boxes
  static constexpr uint32_t kEpiZeroBytes = 0;

  struct Params {
    CUtensorMap tm_x;    // X [M, d], box 64 x 128
    CUtensorMap tm_wg;   // Wg [C, d], box 64 x 128
    CUtensorMap tm_wu;   // Wu [C, d], box 64 x 128
    CUtensorMap tm_act;  // act [M, C], box 64 x 128 (store)
    float* colsum;       // optional [2 * n_mt][C]: sum of |act| over each half of a row tile
    int* status;
    int M, d, C, n_mt, n_mtp, n_ct;
  };
  struct ProdState {
    int m0, c0, rank;
  };

  // Cluster tile t covers row tiles 2*(t % n_mtp) + {0, 1} and channel tile t / n_mtp.
  __device__ static int num_tiles(const Params& p) { return p.n_mtp * p.n_ct; }
  __device__ static int num_kb(const Params& p) { return p.d / 64; }
  __device__ static uint32_t stage_bytes(const Params&, int, int, int part) {
    return 2 * (((part & kPartAct) ? kATileBytes : 0u) + ((part & kPartWeights) ? kBoxBytes : 0u));
  }
  __device__ static void prod_tile(const Params& p, int tile, int rank, ProdState& st) {
    st.c0 = (tile / p.n_mtp) * 128;
    st.m0 = (2 * (tile % p.n_mtp) + rank) * 128;   // rows past M load as zeros
    st.rank = rank;
  }
  // Pair MMA: N columns 0..127 (gate) come from rank 0's B slot, 128..255 (up)
  // from rank 1's; every copy counts on the even CTA's barrier.  `part`
  // selects the activation copy, the weight copy or both (kPart*).
  __device__ static bool weights_first(const Params&) { return true; }
  __device__ static bool acts_first(const Params&) { return false; }   // X comes from the row gather
  __device__ static void prod_kb(const Params& p, const ProdState& st, int, int kb, int lane, uint8_t* a,
                                 uint8_t* b, uint32_t leader_bar, int part) {
    if (lane == 0) {
      const int x = kb * 64;   // K blocks past d load as zeros
      if (part & kPartAct) tma_load_2d_pair(a, &p.tm_x, leader_bar, x, st.m0);
      if (part & kPartWeights) tma_load_2d_pair(b, st.rank == 0 ? &p.tm_wg : &p.tm_wu, leader_bar, x, st.c0);
    }
  }
  __device__ static uint64_t bdesc(uint32_t saddr) { return sdesc_kmajor_sw128(saddr); }
  __device__ static void prefetch(const Params& p) {
    tma_prefetch_desc(&p.tm_x);
    tma_prefetch_desc(&p.tm_wg);
    tma_prefetch_desc(&p.tm_wu);
    tma_prefetch_desc(&p.tm_act);
  }

  // Group `grp` (four warps, 128 threads, one accumulator row each) produces
  // the 64-channel boxes grp*2/kGroups .. of the tile's 128 channels.
  __device__ static bool epilogue(const Params& p, int tile, int row, int grp, uint32_t taddr, EpiCtx& ctx) {
    const int ct = tile / p.n_mtp;
    const int mt = 2 * (tile % p.n_mtp) + ctx.rank;
    const bool leader = (row == 0);
#pragma unroll 1
    for (int bi = 0; bi < 2 / kGroups; ++bi) {
      const int bx = grp * (2 / kGroups) + bi;     // box: channels [64*bx, 64*bx + 64)
      uint8_t* box = ctx.smem + bx * kBoxBytes;
      if (leader) bulk_wait_group_read0();         // the previous store has read the boxes
      if (!ctx.sync()) return false;
      uint8_t* my_row = box + row * 128;
#pragma unroll 1
      for (int c = 0; c < 2; ++c) {
        float g[32], u[32];
        const int col = 64 * bx + 32 * c;
        tmem_ld2_32x32(taddr + col, taddr + 128 + col, g, u);
        uint32_t pk[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) pk[j] = pack_bf16x2(silu_mul(g[2 * j], u[2 * j]), silu_mul(g[2 * j + 1], u[2 * j + 1]));
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const int chunk16 = (4 * c + v) ^ (row & 7);   // 128-byte swizzle of the TMA box
          *reinterpret_cast<uint4*>(my_row + chunk16 * 16) = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
        }
      }
      fence_proxy_async_smem();
      if (!ctx.sync()) return false;
      const int x = ct * 128 + 64 * bx;
      if (leader && x < p.C && mt < p.n_mt) {
        tma_store_2d(&p.tm_act, box, x, mt * 128);
        bulk_commit_group();
      }
      if (p.colsum != nullptr && mt < p.n_mt) {
        // Column sums of |act| for the UCS saliency (Eq. 8): thread `row`
        // sums channel row % 64 of the box over rows [64 * (row / 64), +64),
        // reading the staged (swizzled) box; rows past M hold zeros.
        const int j = row & 63, rh = row >> 6;
        float acc = 0.f;
#pragma unroll 8
        for (int r = 64 * rh; r < 64 * rh + 64; ++r) {
          const int off = r * 128 + ((((j >> 3) ^ (r & 7))) << 4) + ((j & 7) << 1);
          acc += fabsf(__bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(box + off)));
        }
        const int ch = x + j;
        if (ch < p.C) p.colsum[static_cast<size_t>(2 * mt + rh) * p.C + ch] = acc;
      }
    }
    return true;
  }
  __device__ static void epilogue_done(const Params&, int row, int) {
    if (row == 0) bulk_wait_group0();
  }
};

using GateUpProblem = GateUpProblemT<4>;

// ---------------------------------------------------------------- down

// PAIR_ = 0: one CTA per 128 x BN tile.
// PAIR_ = 1: two CTAs of a cluster take adjacent 128-row tiles as one M=256 x
// N=BN pair MMA; each holds its act rows and BN/2 of the B columns, so it
// streams 16 KB of act and BN*64 bytes of WdT per K block for a 128 x BN
// output tile.
template <int BN_, int PAIR_>
struct DownProblem {
  static constexpr int BN = BN_;
  static constexpr int MMA_PAIR = PAIR_;
  static constexpr int CLUSTER = PAIR_ ? 2 : 1;
  static constexpr int CTA_N = PAIR_ ? BN / 2 : BN;   // B columns in one CTA's ring slot
  static constexpr int ATOMS = CTA_N / 64;
  // Two K blocks per slot where three slots fit.
  static constexpr int KSUB = (PAIR_ || BN == 128) ? 2 : 1;
  static constexpr int STAGES = KSUB == 2 ? 3 : BN == 256 ? 4 : 5;
  static constexpr int B_MN_MAJOR = 1;
  static constexpr int EPI_WARPS = 8;
  static constexpr uint32_t kBStepBytes = 2048;     // 16 K-rows = two 1024 B row groups
  static constexpr uint32_t kAtomBytes = 64 * 128;  // 64 K-rows x 64 columns
  static constexpr uint32_t kEpiSmemBytes = 0;
  static constexpr uint32_t kEpiZeroBytes = 0;
  static_assert(CTA_N % 64 == 0, "whole 64-column B atoms per CTA");

  struct Params {
    CUtensorMap tm_act;  // act [M, C], box 64 x 128
    CUtensorMap tm_wdt;  // WdT [C, d] as [d/64][C][64], box 64 x 64 x ATOMS: one K block's atoms
    const int32_t* idx;          // scatter mode: keep list [B][k_tot]
    const __nv_bfloat16* hin;    // scatter mode: residual input
    __nv_bfloat16* out;          // Y [M, d] or the residual output
    const uint8_t* use_small_k;  // optional device flag: contract only the first C_small channels
    const float2* rope_cs;       // optional rotary (cos, sin) per row (plain mode, BN == 256)
    int* status;
    int scatter;
    int rope_heads;
    int M, d, C, C_small, N, k_tot, n_mt, n_mtp, n_nt;   // n_mtp: row-tile pairs
  };
  struct ProdState {
    int m0, atom0;
  };

  // Tile t: N tile t / R and row tile t % R (pair: rows 2 (t % R) + rank),
  // R = row tiles (pairs).
  __device__ static int rows_per_n(const Params& p) { return PAIR_ ? p.n_mtp : p.n_mt; }
  __device__ static int num_tiles(const Params& p) { return rows_per_n(p) * p.n_nt; }
  __device__ static int row_tile(const Params& p, int tile, int rank) {
    const int r = tile % rows_per_n(p);
    return PAIR_ ? 2 * r + rank : r;
  }
  __device__ static int num_kb(const Params& p) {
    return (p.use_small_k != nullptr && *p.use_small_k) ? p.C_small / 64 : p.C / 64;
  }
  // Whole boxes always: atoms past d and K blocks past C load as zeros, so
  // every slot's byte count is fixed (and, for a pair, known to the even CTA).
  __device__ static uint32_t stage_bytes(const Params&, int, int, int part) {
    return (PAIR_ ? 2 : 1) * (((part & kPartAct) ? kATileBytes : 0u) + ((part & kPartWeights) ? ATOMS * kAtomBytes : 0u));
  }
  __device__ static void prod_tile(const Params& p, int tile, int rank, ProdState& st) {
    const int nt = tile / rows_per_n(p);
    st.m0 = row_tile(p, tile, rank) * 128;   // rows past M load as zeros
    st.atom0 = (nt * BN + (PAIR_ ? rank * CTA_N : 0)) / 64;
  }
  // The K extent may come from a device flag the previous kernel writes (the
  // UCS gate); only without it may the weights go out before that kernel ends.
  __device__ static bool weights_first(const Params& p) { return p.use_small_k == nullptr; }
  __device__ static bool acts_first(const Params&) { return false; }   // act comes from the gate/up GEMM
  __device__ static void prod_kb(const Params& p, const ProdState& st, int, int kb, int lane, uint8_t* a,
                                 uint8_t* b, uint64_t* bar, int part) {
    if (lane == 0) {
      if (part & kPartAct) tma_load_2d(a, &p.tm_act, bar, kb * 64, st.m0);
      if (part & kPartWeights) tma_load_3d(b, &p.tm_wdt, bar, 0, kb * 64, st.atom0);
    }
  }
  __device__ static void prod_kb(const Params& p, const ProdState& st, int, int kb, int lane, uint8_t* a,
                                 uint8_t* b, uint32_t leader_bar, int part) {
    if (lane == 0) {
      if (part & kPartAct) tma_load_2d_pair(a, &p.tm_act, leader_bar, kb * 64, st.m0);
      if (part & kPartWeights) tma_load_3d_pair(b, &p.tm_wdt, leader_bar, 0, kb * 64, st.atom0);
    }
  }
  __device__ static uint64_t bdesc(uint32_t saddr) { return sdesc_mnmajor_sw128(saddr, kAtomBytes, 1024); }
  __device__ static void prefetch(const Params& p) {
    tma_prefetch_desc(&p.tm_act);
    tma_prefetch_desc(&p.tm_wdt);
  }

  __device__ static void epilogue_done(const Params&, int, int) {}
  __device__ static bool epilogue(const Params& p, int tile, int row, int half, uint32_t taddr, EpiCtx& ctx) {
    const int nt = tile / rows_per_n(p);
    const int m = row_tile(p, tile, ctx.rank) * 128 + row;
    bool valid = m < p.M;
    size_t dst_row = 0;
    if (valid) {
      if (p.scatter) {
        const int tok = __ldg(p.idx + m);
        if (tok < 0 || tok >= p.N) {
          record_status(p.status, CER_DEV_INDEX);
          valid = false;
        }
        dst_row = static_cast<size_t>(m / p.k_tot) * p.N + tok;
      } else {
        dst_row = static_cast<size_t>(m);
      }
    }
    constexpr int kChunksPerHalf = BN / 64;
    if constexpr (BN == 256) {
      // Rotary embedding: with BN = 256 an epilogue half is one whole head
      // (128 columns), so pair (j, j + 64) is chunk q and chunk q + 2 of the
      // half.  Rotated from the fp32 accumulator, rounded once.
      const int col0 = nt * BN + half * 128;
      if (p.rope_cs != nullptr && !p.scatter && col0 < p.rope_heads * kHeadDim) {
        const float4* cs4 = reinterpret_cast<const float4*>(p.rope_cs + static_cast<size_t>(valid ? m : 0) * 64);
#pragma unroll 1
        for (int q = 0; q < 2; ++q) {
          float a[32], bv[32];
          tmem_ld_32x32(taddr + (4 * half + q) * 32, a);
          tmem_ld_32x32(taddr + (4 * half + q + 2) * 32, bv);
          if (valid) {
            uint32_t lo[16], hi[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              const float4 t = __ldg(cs4 + 16 * q + e);   // cos, sin of j = 32q + 2e and j + 1
              lo[e] = pack_bf16x2(fmaf(a[2 * e], t.x, -bv[2 * e] * t.y), fmaf(a[2 * e + 1], t.z, -bv[2 * e + 1] * t.w));
              hi[e] = pack_bf16x2(fmaf(bv[2 * e], t.x, a[2 * e] * t.y), fmaf(bv[2 * e + 1], t.z, a[2 * e + 1] * t.w));
            }
            uint4* dlo = reinterpret_cast<uint4*>(p.out + dst_row * p.d + col0 + 32 * q);
            uint4* dhi = reinterpret_cast<uint4*>(p.out + dst_row * p.d + col0 + 64 + 32 * q);
#pragma unroll
            for (int w = 0; w < 4; ++w) {
              dlo[w] = make_uint4(lo[4 * w], lo[4 * w + 1], lo[4 * w + 2], lo[4 * w + 3]);
              dhi[w] = make_uint4(hi[4 * w], hi[4 * w + 1], hi[4 * w + 2], hi[4 * w + 3]);
            }
          }
        }
        return true;
      }
    }
#pragma unroll 1
    for (int c = kChunksPerHalf * half; c < kChunksPerHalf * (half + 1); ++c) {
      float v[32];
      tmem_ld_32x32(taddr + c * 32, v);
      const int n0 = nt * BN + c * 32;
      if (valid && n0 < p.d) {
        uint32_t pk[16];
        if (p.scatter) {
          const uint4* src = reinterpret_cast<const uint4*>(p.hin + dst_row * p.d + n0);
          uint4 hv[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) hv[q] = src[q];
          const uint32_t* hw = reinterpret_cast<const uint32_t*>(hv);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            __nv_bfloat162 hb = *reinterpret_cast<const __nv_bfloat162*>(&hw[j]);
            const float2 hf = __bfloat1622float2(hb);
            pk[j] = pack_bf16x2(hf.x + v[2 * j], hf.y + v[2 * j + 1]);
          }
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) pk[j] = pack_bf16x2(v[2 * j], v[2 * j + 1]);
        }
        uint4* dst = reinterpret_cast<uint4*>(p.out + dst_row * p.d + n0);
#pragma unroll
        for (int q = 0; q < 4; ++q) dst[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
      }
    }
    return true;
  }
};

// ---------------------------------------------------------------- launchers

cudaError_t launch_ffn_gateup(const FfnArgs& a, int n_sm, cudaStream_t stream) {
  GateUpProblem::Params p{};
  if (!encode_bf16_2d(&p.tm_x, a.X, a.M, a.d, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_wg, a.Wg, a.C, a.d, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_wu, a.Wu, a.C, a.d, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_act, a.act, a.M, a.C, 64, 128)) return cudaErrorInvalidValue;
  p.colsum = a.colsum;
  p.status = a.status;
  p.M = a.M;
  p.d = a.d;
  p.C = a.C;
  p.n_mt = (a.M + 127) / 128;
  p.n_mtp = (p.n_mt + 1) / 2;
  p.n_ct = (a.C + 127) / 128;
  return launch_gemm<GateUpProblem>(p, p.n_mtp * p.n_ct, a.d / 64, &a.sk, n_sm, stream);
}

template <int BN, int PAIR>
static cudaError_t launch_down(const FfnArgs& a, int n_sm, cudaStream_t stream) {
  using P = DownProblem<BN, PAIR>;
  typename P::Params p{};
  if (!encode_bf16_2d(&p.tm_act, a.act, a.M, a.C, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_col_blocks(&p.tm_wdt, a.WdT, a.C, a.d, 64, P::ATOMS)) return cudaErrorInvalidValue;
  p.idx = a.idx;
  p.hin = a.h;
  p.out = a.scatter ? a.out : a.Y;
  p.use_small_k = a.use_small_k;
  p.rope_cs = a.rope_cs;
  p.rope_heads = a.rope_heads;
  p.status = a.status;
  p.scatter = a.scatter;
  p.M = a.M;
  p.d = a.d;
  p.C = a.C;
  p.C_small = a.C_small;
  p.N = a.N;
  p.k_tot = a.k_tot;
  p.n_mt = (a.M + 127) / 128;
  p.n_mtp = (p.n_mt + 1) / 2;
  p.n_nt = (a.d + BN - 1) / BN;
  const int nkb = (a.use_small_k != nullptr ? a.C_small : a.C) / 64;
  return launch_gemm<P>(p, (PAIR ? p.n_mtp : p.n_mt) * p.n_nt, nkb, &a.sk, n_sm, stream);
}

// Tile shape of the down GEMM.  With at least two row tiles: 256-row pair
// tiles 256 columns wide (the act and WdT streams per flop are what bound
// this contraction; the one-CTA 128 x 192 tile measured about 1.3x slower
// even where it fills every SM).  Otherwise one CTA per 128 x BN tile, BN the
// width with the least per-SM work (waves x width), the wider on a tie.
int down_tile_width(int M, int d, int n_sm) {
  const long n_mt = (M + 127) / 128;
  if (n_mt >= 2) return 0;
  int best = 256;
  long best_cost = -1;
  for (int bn : {256, 192, 128}) {
    const long tiles = n_mt * ((d + bn - 1) / bn);
    const long cost = ((tiles + n_sm - 1) / n_sm) * bn;
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

cudaError_t launch_ffn_down(const FfnArgs& a, int n_sm, cudaStream_t stream) {
  const int width = down_tile_width(a.M, a.d, n_sm);
  if (a.rope_cs != nullptr) {
    // the fused rotary embedding wants whole heads in each epilogue half
    return width == 0 ? launch_down<256, 1>(a, n_sm, stream) : launch_down<256, 0>(a, n_sm, stream);
  }
  switch (width) {
    case 0: return launch_down<256, 1>(a, n_sm, stream);
    case 192: return launch_down<192, 0>(a, n_sm, stream);
    case 128: return launch_down<128, 0>(a, n_sm, stream);
    default: return launch_down<256, 0>(a, n_sm, stream);
  }
}

}  // namespace cer
