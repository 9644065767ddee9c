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
//   written once, as bf16.
// down:     y[m, n] = sum_c act[m, c] * WdT[c, n]
//   B is MN-major: 64 channel rows x 256 output columns, four 64-column TMA
//   boxes per K block.  Epilogue: Y = bf16(y), or, fused, the unpack
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

struct GateUpProblem {
  static constexpr int BN = 256;
  static constexpr int STAGES = 4;
  static constexpr int B_MN_MAJOR = 0;
  static constexpr uint32_t kBStepBytes = 32;

  struct Params {
    CUtensorMap tm_x;   // X [M, d], box 64 x 128
    CUtensorMap tm_wg;  // Wg [C, d], box 64 x 128
    CUtensorMap tm_wu;  // Wu [C, d], box 64 x 128
    __nv_bfloat16* act;
    int* status;
    int M, d, C, n_mt, n_ct;
  };
  struct ProdState {
    int m0, c0;
  };

  __device__ static int num_tiles(const Params& p) { return p.n_mt * p.n_ct; }
  __device__ static int num_kb(const Params& p) { return p.d / 64; }
  __device__ static uint32_t stage_bytes(const Params&, int, int) { return kATileBytes + BN * 128; }
  __device__ static void prod_tile(const Params& p, int tile, int, ProdState& st) {
    st.c0 = (tile / p.n_mt) * 128;
    st.m0 = (tile % p.n_mt) * 128;
  }
  __device__ static void prod_kb(const Params& p, const ProdState& st, int, int kb, int lane, uint8_t* a,
                                 uint8_t* b, uint64_t* bar) {
    if (lane == 0) {
      const int x = kb * 64;
      tma_load_2d(a, &p.tm_x, bar, x, st.m0);
      tma_load_2d(b, &p.tm_wg, bar, x, st.c0);
      tma_load_2d(b + 128 * 128, &p.tm_wu, bar, x, st.c0);
    }
  }
  __device__ static uint64_t bdesc(uint32_t saddr) { return sdesc_kmajor_sw128(saddr); }

  __device__ static void epilogue(const Params& p, int tile, int row, int half, uint32_t taddr) {
    const int ct = tile / p.n_mt;
    const int m = (tile % p.n_mt) * 128 + row;
    const bool valid = m < p.M;
#pragma unroll 1
    for (int c = 2 * half; c < 2 * half + 2; ++c) {
      float g[32], u[32];
      tmem_ld2_32x32(taddr + c * 32, taddr + 128 + c * 32, g, u);
      const int ch0 = ct * 128 + c * 32;
      if (valid && ch0 < p.C) {
        uint32_t pk[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) pk[j] = pack_bf16x2(silu_mul(g[2 * j], u[2 * j]), silu_mul(g[2 * j + 1], u[2 * j + 1]));
        uint4* dst = reinterpret_cast<uint4*>(p.act + static_cast<size_t>(m) * p.C + ch0);
#pragma unroll
        for (int v = 0; v < 4; ++v) dst[v] = make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
      }
    }
  }
};

// ---------------------------------------------------------------- down

struct DownProblem {
  static constexpr int BN = 256;
  static constexpr int STAGES = 4;
  static constexpr int B_MN_MAJOR = 1;
  static constexpr uint32_t kBStepBytes = 2048;     // 16 K-rows = two 1024 B row groups
  static constexpr uint32_t kAtomBytes = 64 * 128;  // 64 K-rows x 64 columns

  struct Params {
    CUtensorMap tm_act;  // act [M, C], box 64 x 128
    CUtensorMap tm_wdt;  // WdT [C, d], box 64 x 64
    const int32_t* idx;          // scatter mode: keep list [B][k_tot]
    const __nv_bfloat16* hin;    // scatter mode: residual input
    __nv_bfloat16* out;          // Y [M, d] or the residual output
    int* status;
    int scatter;
    int M, d, C, N, k_tot, n_mt, n_nt;
  };
  struct ProdState {
    int m0, n0, n_atoms;
  };

  __device__ static int num_tiles(const Params& p) { return p.n_mt * p.n_nt; }
  __device__ static int num_kb(const Params& p) { return p.C / 64; }
  __device__ static int atoms(const Params& p, int nt) {
    const int left = (p.d - nt * 256) / 64;
    return left < 4 ? left : 4;
  }
  __device__ static uint32_t stage_bytes(const Params& p, int tile, int) {
    return kATileBytes + atoms(p, tile / p.n_mt) * kAtomBytes;
  }
  __device__ static void prod_tile(const Params& p, int tile, int, ProdState& st) {
    const int nt = tile / p.n_mt;
    st.n0 = nt * 256;
    st.m0 = (tile % p.n_mt) * 128;
    st.n_atoms = atoms(p, nt);
  }
  __device__ static void prod_kb(const Params& p, const ProdState& st, int, int kb, int lane, uint8_t* a,
                                 uint8_t* b, uint64_t* bar) {
    if (lane == 0) {
      tma_load_2d(a, &p.tm_act, bar, kb * 64, st.m0);
      for (int at = 0; at < st.n_atoms; ++at) tma_load_2d(b + at * kAtomBytes, &p.tm_wdt, bar, st.n0 + at * 64, kb * 64);
    }
  }
  __device__ static uint64_t bdesc(uint32_t saddr) { return sdesc_mnmajor_sw128(saddr, kAtomBytes, 1024); }

  __device__ static void epilogue(const Params& p, int tile, int row, int half, uint32_t taddr) {
    const int nt = tile / p.n_mt;
    const int m = (tile % p.n_mt) * 128 + row;
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
#pragma unroll 1
    for (int c = 4 * half; c < 4 * half + 4; ++c) {
      float v[32];
      tmem_ld_32x32(taddr + c * 32, v);
      const int n0 = nt * 256 + c * 32;
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
  }
};

// ---------------------------------------------------------------- launchers

template <class P>
static cudaError_t launch_gemm(const typename P::Params& p, int tiles, int n_sm, cudaStream_t stream) {
  if (tiles == 0) return cudaSuccess;
  const size_t smem = gemm_smem_bytes<P>();
  cudaError_t e = ensure_max_smem(reinterpret_cast<const void*>(umma_gemm_kernel<P>), smem);
  if (e != cudaSuccess) return e;
  const int grid = tiles < n_sm ? tiles : n_sm;
  umma_gemm_kernel<P><<<grid, kGemmThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_ffn_gateup(const FfnArgs& a, int n_sm, cudaStream_t stream) {
  GateUpProblem::Params p{};
  if (!encode_bf16_2d(&p.tm_x, a.X, a.M, a.d, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_wg, a.Wg, a.C, a.d, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_wu, a.Wu, a.C, a.d, 64, 128)) return cudaErrorInvalidValue;
  p.act = a.act;
  p.status = a.status;
  p.M = a.M;
  p.d = a.d;
  p.C = a.C;
  p.n_mt = (a.M + 127) / 128;
  p.n_ct = (a.C + 127) / 128;
  return launch_gemm<GateUpProblem>(p, p.n_mt * p.n_ct, n_sm, stream);
}

cudaError_t launch_ffn_down(const FfnArgs& a, int n_sm, cudaStream_t stream) {
  DownProblem::Params p{};
  if (!encode_bf16_2d(&p.tm_act, a.act, a.M, a.C, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_wdt, a.WdT, a.C, a.d, 64, 64)) return cudaErrorInvalidValue;
  p.idx = a.idx;
  p.hin = a.h;
  p.out = a.scatter ? a.out : a.Y;
  p.status = a.status;
  p.scatter = a.scatter;
  p.M = a.M;
  p.d = a.d;
  p.C = a.C;
  p.N = a.N;
  p.k_tot = a.k_tot;
  p.n_mt = (a.M + 127) / 128;
  p.n_nt = (a.d + 255) / 256;
  return launch_gemm<DownProblem>(p, p.n_mt * p.n_nt, n_sm, stream);
}

}  // namespace cer
