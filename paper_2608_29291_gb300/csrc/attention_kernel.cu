// attention_kernel.cu -- attention on the packed sequence (Sec. 3.4: the
// retained tokens are packed into a shorter sequence for attention and FFN;
// for understanding the packed keys and values are the compressed KV cache),
// with the rotary position embedding of the Qwen2.5 backbone (App. A.5).
//
// Packed rows are laid out as one bf16 matrix qkv [B * L, (Hq + 2 Hkv) * 128]:
// per row Hq query heads, Hkv key heads, Hkv value heads of 128 values.  A
// packed token keeps its original position (its index in the full sequence)
// for the rotary embedding, and the keep list is ascending, so masking by
// original position is the causal mask on the packed order.
//
// rope_kernel: one warp per packed row rotates its query and key heads in
// place (rotate-half pairing (j, j + 64)).
//
// packed_attention_kernel: persistent, one CTA per SM, one work item per
// (query tile of 128 packed tokens, sequence, query head), the tiles with the
// most key blocks first.  192 threads:
//   warp 0     TMA: the Q tile once per item (two 64-column boxes, K-major)
//              and, per key block of 128 tokens, K (K-major, a three-slot
//              ring freed as soon as S is computed) and V (four 64 x 64
//              MN-major atoms, a two-slot ring), each K one block ahead of
//              its V;
//   warp 1     allocates TMEM (two S buffers of 128 columns, O of 128) and
//              issues tcgen05.mma: S_j = Q K_j^T into S[j % 2] -- issued one
//              block ahead, so it overlaps the softmax of block j - 1 -- and
//              O += P_j V_j once the softmax has written P_j;
//   warps 2-5  softmax, one query row per thread (its TMEM lane), the whole
//              S row in one 128-column TMEM load: masked row maximum in the
//              log2 domain, kept until a block's exceeds it by more than 8,
//              so O is rescaled in TMEM rarely; P_j = exp2(s - m) written as
//              bf16 into a 128-byte-swizzled tile (the A operand of P V), the
//              running sum kept in fp32; at the end O / l goes out as bf16.
// Every wait is bounded like the GEMM skeleton's (umma_gemm.cuh).
#include <cuda_bf16.h>

#include "kernels.h"
#include "umma_gemm.cuh"

namespace cer {

// ------------------------------------------------------------------ rotary embedding

constexpr int kRopeThreads = 256;   // 8 warps, one packed row per warp at a time

// One warp per row: lane l rotates pairs j = 8 (l % 8) .. + 7 of heads
// l / 8, l / 8 + 4, ... with 16-byte loads of both halves.  The angle
// a = pos * theta_j is formed in turns, x = pos * g_j with g_j = theta_j /
// (2 pi) from the host's fp64 table, reduced exactly in fp64 (x - rint(x))
// and handed to fp32 sincospif: accurate to ~2e-7 for any position, where an
// fp32 product pos * theta_j would lose the angle.
__global__ void __launch_bounds__(kRopeThreads)
    rope_kernel(__nv_bfloat16* qkv, long long rows, int Hq, int Hkv, const int32_t* __restrict__ pos,
                const __grid_constant__ RopeFreqTable ft, int* status) {
  griddep_wait();
  griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int j0 = 8 * (lane & 7);
  const int width = (Hq + 2 * Hkv) * kHeadDim;
  const int heads = Hq + Hkv;
  const long long warps = static_cast<long long>(gridDim.x) * (kRopeThreads / 32);
  for (long long row = blockIdx.x * (kRopeThreads / 32) + (threadIdx.x >> 5); row < rows; row += warps) {
    const int p = __ldg(pos + row);
    __nv_bfloat16* r = qkv + row * width;
    // Heads lane/8, lane/8 + 4, ... in batches of four: a batch's loads are
    // issued before the angles (and the previous batch's stores) are needed.
    for (int h0 = lane >> 3; h0 < heads; h0 += 16) {
      uint4 lo[4], hi[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int h = h0 + 4 * i;
        if (h < heads) {
          lo[i] = *reinterpret_cast<const uint4*>(r + h * kHeadDim + j0);
          hi[i] = *reinterpret_cast<const uint4*>(r + h * kHeadDim + 64 + j0);
        }
      }
      if (p < 0) break;
      float c[8], s[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const double x = static_cast<double>(p) * ft.g[j0 + e];
        sincospif(2.0f * static_cast<float>(x - rint(x)), &s[e], &c[e]);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int h = h0 + 4 * i;
        if (h >= heads) break;
        uint32_t* lw = reinterpret_cast<uint32_t*>(&lo[i]);
        uint32_t* hw = reinterpret_cast<uint32_t*>(&hi[i]);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 a = __bfloat1622float2(*reinterpret_cast<__nv_bfloat162*>(&lw[e]));
          const float2 b = __bfloat1622float2(*reinterpret_cast<__nv_bfloat162*>(&hw[e]));
          const int k = 2 * e;
          lw[e] = pack_bf16x2(fmaf(a.x, c[k], -b.x * s[k]), fmaf(a.y, c[k + 1], -b.y * s[k + 1]));
          hw[e] = pack_bf16x2(fmaf(b.x, c[k], a.x * s[k]), fmaf(b.y, c[k + 1], a.y * s[k + 1]));
        }
        *reinterpret_cast<uint4*>(r + h * kHeadDim + j0) = lo[i];
        *reinterpret_cast<uint4*>(r + h * kHeadDim + 64 + j0) = hi[i];
      }
    }
    if (p < 0 && lane == 0) record_status(status, CER_DEV_INDEX);
  }
}

cudaError_t launch_rope(__nv_bfloat16* qkv, long long rows, int Hq, int Hkv, const int32_t* pos,
                        const RopeFreqTable& ft, int* status, int n_sm, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  const long long per_block = kRopeThreads / 32;
  long long blocks = (rows + per_block - 1) / per_block;
  const long long cap = static_cast<long long>(n_sm) * 8;
  if (blocks > cap) blocks = cap;
  return launch_k(rope_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kRopeThreads), 0, stream, 1, qkv, rows, Hq,
                  Hkv, pos, ft, status);
}

// ------------------------------------------------------------------ attention

struct AttnParams {
  CUtensorMap tm_qk;   // qkv, box 64 x 128 (Q and K tiles)
  CUtensorMap tm_v;    // qkv, box 64 x 64 (V atoms)
  __nv_bfloat16* out;  // [B * L, Hq * 128]
  int* status;
  int B, L, Hq, Hkv, causal, n_qt, n_items;
  float scale_log2;    // log2(e) / sqrt(128)
};

constexpr int kAttnThreads = 192;
constexpr uint32_t kBox = 128 * 128;              // 128 rows x 64 bf16
constexpr uint32_t kQBytes = 2 * kBox;            // Q tile: 128 tokens x 128
constexpr uint32_t kKBytes = 2 * kBox;            // K tile: 128 keys x 128 (two K-major boxes)
constexpr uint32_t kVBytes = 2 * kBox;            // V tile: four 64 x 64 MN-major atoms
constexpr uint32_t kPBytes = 2 * kBox;            // P tile: 128 queries x 128 keys, bf16
constexpr int kKSlots = 3;                        // K is freed as soon as S is computed: one block more in flight
constexpr int kVSlots = 2;
constexpr size_t kAttnSmem = 1024 + kQBytes + kKSlots * kKBytes + kVSlots * kVBytes + kPBytes + 256;
constexpr uint32_t kIdescS = idesc_bf16(128, 128, 0);    // Q (K-major) x K (K-major)
constexpr uint32_t kIdescPV = idesc_bf16(128, 128, 1);   // P (K-major) x V (MN-major)

struct AttnItem {
  int b, h, kh, qt, n_kv;
};

__device__ __forceinline__ AttnItem attn_item(const AttnParams& p, int item) {
  AttnItem it;
  const int per_tile = p.B * p.Hq;
  it.qt = p.n_qt - 1 - item / per_tile;   // the tiles with the most key blocks first
  const int rest = item % per_tile;
  it.b = rest / p.Hq;
  it.h = rest % p.Hq;
  it.kh = it.h / (p.Hq / p.Hkv);
  it.n_kv = p.causal ? it.qt + 1 : p.n_qt;
  return it;
}

// 2^x with the hardware's approximate exponential (relative error ~2^-22,
// far below the bf16 rounding the weights then receive); 2^-inf = 0.
__device__ __forceinline__ float exp2_fast(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__global__ void __launch_bounds__(kAttnThreads, 1) packed_attention_kernel(const __grid_constant__ AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* q_tile = smem;
  uint8_t* k_ring = q_tile + kQBytes;
  uint8_t* v_ring = k_ring + kKSlots * kKBytes;   // slot s: atom (key half kh, dim half na) at kh*16K + na*8K
  uint8_t* p_tile = v_ring + kVSlots * kVBytes;
  uint64_t* q_full = reinterpret_cast<uint64_t*>(p_tile + kPBytes);
  uint64_t* q_empty = q_full + 1;
  uint64_t* k_full = q_empty + 1;          // [kKSlots]
  uint64_t* k_empty = k_full + kKSlots;    // [kKSlots]
  uint64_t* v_full = k_empty + kKSlots;    // [kVSlots]
  uint64_t* v_empty = v_full + kVSlots;    // [kVSlots]
  uint64_t* s_full = v_empty + kVSlots;    // [2]
  uint64_t* s_free = s_full + 2;           // [2]
  uint64_t* p_full = s_free + 2;
  uint64_t* o_done = p_full + 1;
  uint64_t* o_free = o_done + 1;
  uint64_t* drain = o_free + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 32) {
    tma_prefetch_desc(&p.tm_qk);
    tma_prefetch_desc(&p.tm_v);
  }
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int s = 0; s < kKSlots; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < kVSlots; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&s_full[s], 1);
      mbar_init(&s_free[s], 4);   // one arrival per softmax warp
    }
    mbar_init(p_full, 4);
    mbar_init(o_done, 1);
    mbar_init(o_free, 4);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  griddep_wait();   // qkv written by the previous kernel is visible
  griddep_launch_dependents();

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    // Key block j's K goes out one block ahead of its V: K_j, then V_{j-1}
    // (carried across items), so the keys for S_{j+1} are in flight while
    // P_j V_j waits.
    uint32_t gk = 0, gv = 0, items = 0;
    bool ok = true;
    bool pend = false;
    int pend_row = 0, pend_col = 0;
    auto load_v = [&](int row, int col) -> bool {
      const uint32_t s = gv % kVSlots;
      if (!warp_wait(&v_empty[s], ((gv / kVSlots) & 1) ^ 1, abort_flag, p.status)) return false;
      if (lane == 0) {
        uint8_t* slot = v_ring + s * kVBytes;
        mbar_arrive_expect_tx(&v_full[s], kVBytes);
        for (int kh = 0; kh < 2; ++kh)
          for (int na = 0; na < 2; ++na)
            tma_load_2d(slot + kh * 16384 + na * 8192, &p.tm_v, &v_full[s], col + na * 64, row + kh * 64);
      }
      __syncwarp();
      ++gv;
      return true;
    };
    for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x, ++items) {
      const AttnItem it = attn_item(p, item);
      const int row0 = it.b * p.L;
      if (!warp_wait(q_empty, (items & 1) ^ 1, abort_flag, p.status)) {
        ok = false;
        break;
      }
      if (lane == 0) {
        mbar_arrive_expect_tx(q_full, kQBytes);
        tma_load_2d(q_tile, &p.tm_qk, q_full, it.h * kHeadDim, row0 + it.qt * 128);
        tma_load_2d(q_tile + kBox, &p.tm_qk, q_full, it.h * kHeadDim + 64, row0 + it.qt * 128);
      }
      __syncwarp();
      const int kcol = (p.Hq + it.kh) * kHeadDim;
      const int vcol = (p.Hq + p.Hkv + it.kh) * kHeadDim;
      for (int j = 0; j < it.n_kv; ++j) {
        const uint32_t s = gk % kKSlots;
        if (!warp_wait(&k_empty[s], ((gk / kKSlots) & 1) ^ 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          uint8_t* slot = k_ring + s * kKBytes;
          mbar_arrive_expect_tx(&k_full[s], kKBytes);
          tma_load_2d(slot, &p.tm_qk, &k_full[s], kcol, row0 + j * 128);
          tma_load_2d(slot + kBox, &p.tm_qk, &k_full[s], kcol + 64, row0 + j * 128);
        }
        __syncwarp();
        ++gk;
        if (pend && !load_v(pend_row, pend_col)) {
          ok = false;
          break;
        }
        pend = true;
        pend_row = row0 + j * 128;
        pend_col = vcol;
      }
    }
    if (ok && pend) ok = load_v(pend_row, pend_col);
    if (!ok && lane == 0) unwind_pause(1000000ull);
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    uint32_t gk = 0, gv = 0;   // K / V blocks consumed
    uint32_t cs = 0;           // S tiles issued (buffer cs % 2)
    uint32_t cp = 0;           // P tiles consumed
    uint32_t items = 0;
    bool ok = true;
    bool issued_any = false;
    const uint32_t q_base = smem_u32(q_tile), p_base = smem_u32(p_tile);
    const uint32_t o_tm = tmem_base + 256;
    for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x, ++items) {
      const AttnItem it = attn_item(p, item);
      if (!warp_wait(q_full, items & 1, abort_flag, p.status)) {
        ok = false;
        break;
      }
      tc_fence_after();
      for (int j = -1; j < it.n_kv && ok; ++j) {
        // S_{j+1} = Q K_{j+1}^T, one block ahead of P_j V_j.
        if (j + 1 < it.n_kv) {
          const uint32_t ks = gk % kKSlots;
          const uint32_t buf = cs & 1;
          if (!warp_wait(&k_full[ks], (gk / kKSlots) & 1, abort_flag, p.status) ||
              !warp_wait(&s_free[buf], ((cs >> 1) & 1) ^ 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          if (lane == 0) {
            const uint32_t k_base = smem_u32(k_ring + ks * kKBytes);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const uint32_t off = (k >> 2) * kBox + (k & 3) * 32;
              umma_bf16(tmem_base + buf * 128, sdesc_kmajor_sw128(q_base + off), sdesc_kmajor_sw128(k_base + off),
                        kIdescS, k > 0 ? 1u : 0u);
            }
            umma_commit(&s_full[buf]);
            umma_commit(&k_empty[ks]);
            if (j + 2 == it.n_kv) umma_commit(q_empty);   // the item's last S: the Q tile may be reloaded
            issued_any = true;
          }
          __syncwarp();
          ++gk;
          ++cs;
        }
        if (j < 0) continue;
        // O += P_j V_j once the softmax has written P_j (and, for the item's
        // first block, has read out the previous item's O).
        if (!warp_wait(p_full, cp & 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        ++cp;
        const uint32_t vs = gv % kVSlots;
        if ((j == 0 && !warp_wait(o_free, (items & 1) ^ 1, abort_flag, p.status)) ||
            !warp_wait(&v_full[vs], (gv / kVSlots) & 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (lane == 0) {
          const uint32_t v_base = smem_u32(v_ring + vs * kVBytes);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint64_t adesc = sdesc_kmajor_sw128(p_base + (k >> 2) * kBox + (k & 3) * 32);
            const uint64_t bdesc = sdesc_mnmajor_sw128(v_base + (k >> 2) * 16384 + (k & 3) * 2048, 8192, 1024);
            umma_bf16(o_tm, adesc, bdesc, kIdescPV, (j > 0 || k > 0) ? 1u : 0u);
          }
          umma_commit(&v_empty[vs]);
          umma_commit(o_done);
        }
        __syncwarp();
        ++gv;
      }
    }
    if (!ok && lane == 0 && issued_any) {
      umma_commit(drain);
      drain_wait(drain, 0);
    }
  } else {
    // ---------------------------------------------------------------- softmax
    const int qd = warp & 3;            // TMEM lane quadrant
    const int r = qd * 32 + lane;       // query row of the tile
    const uint32_t lane_off = static_cast<uint32_t>(qd * 32) << 16;
    const uint32_t o_tm = tmem_base + lane_off + 256;
    const float sc = p.scale_log2;
    uint32_t cs = 0, co = 0, items = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x, ++items) {
      const AttnItem it = attn_item(p, item);
      const int qi = it.qt * 128 + r;
      // Keys past the sequence, and (causal) past the query, are masked.
      const int lim = p.causal ? (qi + 1 < p.L ? qi + 1 : p.L) : p.L;
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < it.n_kv; ++j, ++cs) {
        const uint32_t buf = cs & 1;
        if (!warp_wait(&s_full[buf], (cs >> 1) & 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int n_ok = lim - j * 128;   // admissible keys of this block: [0, n_ok)
        uint32_t sv[128];
        tmem_ld_32x32_x128(tmem_base + lane_off + buf * 128, sv);   // the whole S row
        float mx8[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx8[e] = -INFINITY;
        if (n_ok >= 128) {
#pragma unroll
          for (int e = 0; e < 128; ++e) mx8[e & 7] = fmaxf(mx8[e & 7], __uint_as_float(sv[e]));
        } else {
#pragma unroll
          for (int e = 0; e < 128; ++e)
            if (e < n_ok) mx8[e & 7] = fmaxf(mx8[e & 7], __uint_as_float(sv[e]));
        }
        const float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                               fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
        // The running maximum moves only when the block's exceeds it by more
        // than 8 (log2 units): with a stale maximum the weights stay below
        // 2^8, far inside bf16 and fp32, and O is rescaled rarely.  The
        // result is unchanged: O and l share the same shift.
        const float mb = mx * sc;
        const float m_new = (mb > m + 8.0f) ? mb : m;   // the first block always takes its maximum
        const float alpha = exp2_fast(m - m_new);       // 0 for the first block, else 1 or < 2^-8
        if (j > 0) {
          // P_{j-1} V_{j-1} is complete: the P tile is free and O may be rescaled.
          if (!warp_wait(o_done, co & 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          ++co;
          tc_fence_after();
          if (__any_sync(0xffffffffu, alpha != 1.0f)) {
#pragma unroll 1
            for (int c = 0; c < 4; ++c) {
              float ov[32];
              tmem_ld_32x32(o_tm + c * 32, ov);
#pragma unroll
              for (int e = 0; e < 32; ++e) ov[e] *= alpha;
              tmem_st_32x32(o_tm + c * 32, ov);
            }
          }
        }
        // P = exp2(s * scale - m) as bf16 into the swizzled A tile of P V.
        const float neg = -m_new;
        float rs4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int c = 0; c < 16; ++c) {   // 16-byte chunks of 8 keys
          uint32_t pk[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int k0 = 8 * c + 2 * e;
            float p0 = exp2_fast(fmaf(__uint_as_float(sv[k0]), sc, neg));
            float p1 = exp2_fast(fmaf(__uint_as_float(sv[k0 + 1]), sc, neg));
            if (n_ok < 128) {
              p0 = k0 < n_ok ? p0 : 0.f;
              p1 = k0 + 1 < n_ok ? p1 : 0.f;
            }
            rs4[e] += p0 + p1;
            pk[e] = pack_bf16x2(p0, p1);
          }
          const int chunk = (c & 7) ^ (r & 7);   // 128-byte swizzle within each 64-key box
          *reinterpret_cast<uint4*>(p_tile + (c >> 3) * kBox + r * 128 + chunk * 16) =
              make_uint4(pk[0], pk[1], pk[2], pk[3]);
        }
        tc_fence_before();
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&s_free[buf]);
          mbar_arrive(p_full);
        }
        l = l * alpha + ((rs4[0] + rs4[1]) + (rs4[2] + rs4[3]));
        m = m_new;
      }
      if (!ok) break;
      if (!warp_wait(o_done, co & 1, abort_flag, p.status)) {
        ok = false;
        break;
      }
      ++co;
      tc_fence_after();
      const float inv = 1.0f / l;
      uint32_t ov[128];
      tmem_ld_32x32_x128(o_tm, ov);
      if (qi < p.L) {
        uint4* d4 = reinterpret_cast<uint4*>(p.out + (static_cast<size_t>(it.b) * p.L + qi) *
                                                         (static_cast<size_t>(p.Hq) * kHeadDim) +
                                             static_cast<size_t>(it.h) * kHeadDim);
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          uint32_t pk[4];
#pragma unroll
          for (int e = 0; e < 4; ++e)
            pk[e] = pack_bf16x2(__uint_as_float(ov[8 * q + 2 * e]) * inv, __uint_as_float(ov[8 * q + 2 * e + 1]) * inv);
          d4[q] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(o_free);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

cudaError_t launch_packed_attention(const __nv_bfloat16* qkv, int B, int L, int Hq, int Hkv, int causal,
                                    __nv_bfloat16* out, int* status, int n_sm, cudaStream_t stream) {
  if (B == 0 || L == 0) return cudaSuccess;
  AttnParams p{};
  const uint64_t rows = static_cast<uint64_t>(B) * L;
  const uint64_t width = static_cast<uint64_t>(Hq + 2 * Hkv) * kHeadDim;
  if (!encode_bf16_2d(&p.tm_qk, qkv, rows, width, 64, 128)) return cudaErrorInvalidValue;
  if (!encode_bf16_2d(&p.tm_v, qkv, rows, width, 64, 64)) return cudaErrorInvalidValue;
  p.out = out;
  p.status = status;
  p.B = B;
  p.L = L;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.causal = causal;
  p.n_qt = (L + 127) / 128;
  p.n_items = B * Hq * p.n_qt;
  p.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));
  cudaError_t e = ensure_max_smem(reinterpret_cast<const void*>(packed_attention_kernel), kAttnSmem);
  if (e != cudaSuccess) return e;
  const int grid = p.n_items < n_sm ? p.n_items : n_sm;
  return launch_k(packed_attention_kernel, dim3(grid), dim3(kAttnThreads), kAttnSmem, stream, 1, p);
}

}  // namespace cer
