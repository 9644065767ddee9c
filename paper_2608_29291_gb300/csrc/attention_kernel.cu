// attention_kernel.cu -- attention on the packed sequence (Sec. 3.4, token
// compaction: only the kept tokens of R take part in attention, as in the
// FFN, and in understanding mode their keys and values are the reduced KV
// cache), with the rotary position embedding of the Qwen2.5 backbone
// (App. A.5).
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
// most key blocks first.  352 threads:
//   warp 0     TMA: the Q tile once per item and K blocks of 128 keys
//              (K-major, a three-slot ring), streaming ahead of V;
//   warp 10    TMA: V blocks (two MN-major 64 x 128 boxes, a two-slot ring);
//   warp 1     allocates TMEM (three S buffers of 128 columns, O of 128) and
//              issues tcgen05.mma: S_j = Q K_j^T two blocks ahead of the
//              softmax, and O += P_j V_j with P_j read from tensor memory;
//   warps 2-9  softmax, two warps per TMEM lane quadrant splitting the key
//              columns: masked row maximum in the log2 domain (exchanged
//              between the two halves through shared memory), kept until a
//              block's exceeds it by more than 8, so O is rescaled rarely;
//              P_j = exp2(s - m) packed to bf16 over the S buffer it came
//              from, the running sum kept in fp32; at the end O / l goes
//              out as bf16.
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
// fp32 product pos * theta_j would lose the angle.  (A two-part fp32 form of
// the reduction measured slower than these eight fp64 products per row.)
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
    // The angles depend on the row and the lane's pairs only: they are formed
    // once, after the first batch's loads (fp64 is slow on this part).
    float c[8], s[8];
    bool have_angles = false;
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
      if (!have_angles) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const double x = static_cast<double>(p) * ft.g[j0 + e];
          sincospif(2.0f * static_cast<float>(x - rint(x)), &s[e], &c[e]);
        }
        have_angles = true;
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
  CUtensorMap tm_qkv;  // qkv, box 64 columns x 128 rows (Q, K and V tiles)
  __nv_bfloat16* out;  // [B * L, Hq * 128]
  int* status;
  int B, L, Hq, Hkv, causal, group, n_qt, n_items;
  float scale_log2;    // log2(e) / sqrt(128)
};

constexpr int kAttnThreads = 352;                 // Q/K producer, MMA, eight softmax warps, V producer
constexpr uint32_t kBox = 128 * 128;              // 128 rows x 64 bf16
constexpr uint32_t kQBytes = 2 * kBox;            // Q tile: 128 tokens x 128 (two K-major boxes)
constexpr uint32_t kKBytes = 2 * kBox;            // K block: 128 keys x 128 (two K-major boxes)
constexpr uint32_t kVBytes = 2 * kBox;            // V block: two MN-major boxes (dims 0-63, 64-127) of 128 keys
constexpr int kKSlots = 3;
constexpr int kVSlots = 2;
constexpr int kSBufs = 3;                         // S buffers in tensor memory
constexpr uint32_t kXchBytes = 2 * 2 * 128 * 4;   // row-maximum exchange: [parity][half][row]
constexpr size_t kAttnSmem = 1024 + kQBytes + kKSlots * kKBytes + kVSlots * kVBytes + kXchBytes + 512;
constexpr uint32_t kIdescS = idesc_bf16(128, 128, 0);    // Q (K-major) x K (K-major)
constexpr uint32_t kIdescPV = idesc_bf16(128, 128, 1);   // P (tensor memory) x V (MN-major)

// A work item: one 128-query tile of one sequence and query head.
struct AttnItem {
  int b, h, kh, qt, n_kv;
};

// Tiles with the most key blocks first; a key/value head's query heads on
// neighbouring items, so their K and V blocks are read from L2.
__device__ __forceinline__ AttnItem attn_item(const AttnParams& p, int item) {
  AttnItem it;
  const int per_tile = p.B * p.Hq;
  it.qt = p.n_qt - 1 - item / per_tile;
  const int rest = item % per_tile;
  it.b = rest / p.Hq;
  it.h = rest % p.Hq;
  it.kh = it.h / p.group;
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

// 32 lanes x 64 columns of fp32 in one load, the wait in the same asm statement.
__device__ __forceinline__ void tmem_ld_32x32_x64(uint32_t taddr, uint32_t (&r)[64]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, "
      "%36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, "
      "%57, %58, %59, %60, %61, %62, %63}, [%64];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
        "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
        "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(taddr)
      : "memory");
}

// Tensor memory, 512 columns: three S buffers at [0,128), [128,256),
// [256,384) and O at [384,512).  Key blocks, counted over all of a CTA's
// items (gb), rotate through the S buffers; P(gb) (bf16, two keys per
// column) overwrites the first 64 columns of S(gb)'s buffer once the softmax
// has read S(gb), and is the A operand of O += P(gb) V.  S(gb + 3) reuses the
// buffer after that product has completed -- by then long done, as S(gb + 3)
// is issued after P(gb + 1) V.  So the MMA warp issues P(j) V and S(j + 2)
// back to back as soon as P(j) is written, and S(j + 1) and S(j + 2) are
// computed while the softmax works on block j.
//
// Softmax: warps 2-9, two per TMEM lane quadrant: warp half hf takes key
// columns [64 hf, 64 hf + 64) of its 32 query rows.  The two halves exchange
// their row maxima through shared memory once per block (an mbarrier of two
// arrivals per quadrant, bounded like every wait) and their row sums once
// per item.
__global__ void __launch_bounds__(kAttnThreads, 1) packed_attention_kernel(const __grid_constant__ AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* q_tile = smem;
  uint8_t* k_ring = q_tile + kQBytes;
  uint8_t* v_ring = k_ring + kKSlots * kKBytes;   // slot s: dims 64 na .. 64 na + 63 of 128 keys at na*16K
  float* xch_val = reinterpret_cast<float*>(v_ring + kVSlots * kVBytes);   // [parity][half][row]
  uint64_t* q_full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(xch_val) + kXchBytes);
  uint64_t* q_empty = q_full + 1;
  uint64_t* k_full = q_empty + 1;          // [kKSlots]
  uint64_t* k_empty = k_full + kKSlots;    // [kKSlots]
  uint64_t* v_full = k_empty + kKSlots;    // [kVSlots]
  uint64_t* v_empty = v_full + kVSlots;    // [kVSlots]
  uint64_t* s_full = v_empty + kVSlots;    // [kSBufs]
  uint64_t* p_full = s_full + kSBufs;      // [kSBufs]
  uint64_t* pv_done = p_full + kSBufs;     // [kSBufs]: P(gb) V complete
  uint64_t* o_done = pv_done + kSBufs;     // an item's last P V product
  uint64_t* o_free = o_done + 1;
  uint64_t* xch = o_free + 1;              // [4]: per lane quadrant
  uint64_t* drain = xch + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 32) tma_prefetch_desc(&p.tm_qkv);
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
    for (int i = 0; i < kSBufs; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 8);   // one arrival per softmax warp
      mbar_init(&pv_done[i], 1);
    }
    mbar_init(o_done, 1);
    mbar_init(o_free, 8);
    for (int i = 0; i < 4; ++i) mbar_init(&xch[i], 2);
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
    // ---------------------------------------------------------------- Q and K producer
    // One thread issues everything here (TMA copies, mbarrier operations,
    // tcgen05.mma and commits are per thread): warp-wide waits would only
    // add a broadcast and a reconvergence to every step.
    if (lane == 0) {
      // K streams ahead, limited only by its own ring: S(j) needs just K_j.
      uint32_t gk = 0, items = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x, ++items) {
        const AttnItem it = attn_item(p, item);
        const int row0 = it.b * p.L;
        if (!mbar_wait(q_empty, (items & 1) ^ 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          const int qrow = row0 + it.qt * 128;
          mbar_arrive_expect_tx(q_full, kQBytes);
          tma_load_2d(q_tile, &p.tm_qkv, q_full, it.h * kHeadDim, qrow);
          tma_load_2d(q_tile + kBox, &p.tm_qkv, q_full, it.h * kHeadDim + 64, qrow);
        }
        const int kcol = (p.Hq + it.kh) * kHeadDim;
        for (int j = 0; j < it.n_kv && ok; ++j) {
          const uint32_t ks = gk % kKSlots;
          if (!mbar_wait(&k_empty[ks], ((gk / kKSlots) & 1) ^ 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          if (lane == 0) {
            uint8_t* slot = k_ring + ks * kKBytes;
            mbar_arrive_expect_tx(&k_full[ks], kKBytes);
            tma_load_2d(slot, &p.tm_qkv, &k_full[ks], kcol, row0 + j * 128);
            tma_load_2d(slot + kBox, &p.tm_qkv, &k_full[ks], kcol + 64, row0 + j * 128);
          }
          ++gk;
        }
      }
      if (!ok && lane == 0) unwind_pause(1000000ull);
    }
    __syncwarp();
  } else if (warp == 10) {
    // ---------------------------------------------------------------- V producer
    if (lane == 0) {
      uint32_t gv = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x) {
        const AttnItem it = attn_item(p, item);
        const int row0 = it.b * p.L;
        const int vcol = (p.Hq + p.Hkv + it.kh) * kHeadDim;
        for (int j = 0; j < it.n_kv && ok; ++j) {
          const uint32_t vs = gv % kVSlots;
          if (!mbar_wait(&v_empty[vs], ((gv / kVSlots) & 1) ^ 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          if (lane == 0) {
            uint8_t* slot = v_ring + vs * kVBytes;
            mbar_arrive_expect_tx(&v_full[vs], kVBytes);
            tma_load_2d(slot, &p.tm_qkv, &v_full[vs], vcol, row0 + j * 128);
            tma_load_2d(slot + kBox, &p.tm_qkv, &v_full[vs], vcol + 64, row0 + j * 128);
          }
          ++gv;
        }
      }
      if (!ok && lane == 0) unwind_pause(1000000ull);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      // Per item: S(0), S(1); then per key block j: S(j + 2), P(j) V_j.
      uint32_t gk = 0, gv = 0, items = 0, g = 0, o_taken = 0;
      bool ok = true;
      bool issued_any = false;
      // S(gb) = Q K^T from K slot ks, once P(gb - 3) V (the buffer's previous
      // reader) has completed.  That wait cannot meet a barrier two phases
      // ahead: P(gb) V needs S(gb).
      auto issue_s = [&](uint32_t ks, uint32_t gb) -> bool {
        const uint32_t buf = gb % kSBufs;
        if (gb >= kSBufs &&
            !mbar_wait(&pv_done[buf], ((gb - kSBufs) / kSBufs) & 1, abort_flag, p.status))
          return false;
        tc_fence_after();
        if (lane == 0) {
          const uint32_t q_base = smem_u32(q_tile);
          const uint32_t k_base = smem_u32(k_ring + ks * kKBytes);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t off = (k >> 2) * kBox + (k & 3) * 32;
            umma_bf16(tmem_base + buf * 128, sdesc_kmajor_sw128(q_base + off), sdesc_kmajor_sw128(k_base + off),
                      kIdescS, k > 0 ? 1u : 0u);
          }
          umma_commit(&s_full[buf]);
          issued_any = true;
        }
        return true;
      };
      // O (+)= P(gb) V from V slot vs; first: the item's first block (also waits
      // until the previous item's O has been read out); last: its last block.
      auto issue_pv = [&](uint32_t vs, uint32_t gb, bool first, bool last) -> bool {
        const uint32_t buf = gb % kSBufs;
        if (!mbar_wait(&p_full[buf], (gb / kSBufs) & 1, abort_flag, p.status)) return false;
        if (first) {
          if (!mbar_wait(o_free, (o_taken & 1) ^ 1, abort_flag, p.status)) return false;
          ++o_taken;
        }
        tc_fence_after();
        if (lane == 0) {
          const uint32_t v_base = smem_u32(v_ring + vs * kVBytes);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint64_t bdesc = sdesc_mnmajor_sw128(v_base + k * 2048, kBox, 1024);
            umma_bf16_tmem_a(tmem_base + 384, tmem_base + buf * 128 + k * 8, bdesc, kIdescPV,
                             (!first || k > 0) ? 1u : 0u);
          }
          umma_commit(&pv_done[buf]);
          if (last) umma_commit(o_done);
          issued_any = true;
        }
        return true;
      };
      for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x, ++items) {
        const AttnItem it = attn_item(p, item);
        const int n = it.n_kv;
        if (!mbar_wait(q_full, items & 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        for (int j = 0; j < 2 && j < n; ++j) {
          const uint32_t ks = gk % kKSlots;
          if (!mbar_wait(&k_full[ks], (gk / kKSlots) & 1, abort_flag, p.status) || !issue_s(ks, g + j)) {
            ok = false;
            break;
          }
          if (lane == 0) {
            umma_commit(&k_empty[ks]);
            if (j + 1 == n) umma_commit(q_empty);
          }
          ++gk;
        }
        for (int j = 0; j < n && ok; ++j) {
          // S(j + 2) first: it needs only K and P(j - 1) V, so it runs while
          // the softmax still works on block j.
          if (j + 2 < n) {
            const uint32_t ks = gk % kKSlots;
            if (!mbar_wait(&k_full[ks], (gk / kKSlots) & 1, abort_flag, p.status) || !issue_s(ks, g + j + 2)) {
              ok = false;
              break;
            }
            if (lane == 0) {
              umma_commit(&k_empty[ks]);
              if (j + 3 == n) umma_commit(q_empty);
            }
            ++gk;
          }
          const uint32_t vs = gv % kVSlots;
          if (!mbar_wait(&v_full[vs], (gv / kVSlots) & 1, abort_flag, p.status) ||
              !issue_pv(vs, g + j, j == 0, j + 1 == n)) {
            ok = false;
            break;
          }
          if (lane == 0) umma_commit(&v_empty[vs]);
          ++gv;
        }
        g += n;
      }
      if (!ok && lane == 0 && issued_any) {
        umma_commit(drain);
        drain_wait(drain, 0);
      }
    }
    __syncwarp();
  } else if (warp < 10) {
    // ---------------------------------------------------------------- softmax
    const int qd = warp & 3;            // TMEM lane quadrant
    const int hf = (warp - 2) >> 2;     // key-column half
    const int r = qd * 32 + lane;       // query row of the tile
    const uint32_t row_tm = tmem_base + (static_cast<uint32_t>(qd * 32) << 16);
    const uint32_t o_tm = row_tm + 384 + hf * 64;
    const float sc = p.scale_log2;
    uint32_t g = 0, done = 0, xp = 0;   // key blocks, items, exchanges so far
    bool ok = true;
    // Swap a value with the other half's warp of this quadrant.
    auto exchange = [&](float v, float& other) -> bool {
      float* slot = xch_val + (xp & 1) * 256;
      slot[hf * 128 + r] = v;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&xch[qd]);
      if (!warp_wait(&xch[qd], xp & 1, abort_flag, p.status)) return false;
      tc_fence_after();
      other = slot[(hf ^ 1) * 128 + r];
      ++xp;
      return true;
    };
    for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x) {
      const AttnItem it = attn_item(p, item);
      const int qi = it.qt * 128 + r;
      // Keys past the sequence, and (causal) past the query, are masked.
      const int lim = p.causal ? (qi + 1 < p.L ? qi + 1 : p.L) : p.L;
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < it.n_kv; ++j) {
        const uint32_t gb = g + j, buf = gb % kSBufs;
        if (!warp_wait(&s_full[buf], (gb / kSBufs) & 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int n_ok = lim - j * 128 - hf * 64;   // admissible keys of this half: [0, n_ok)
        uint32_t sv[64];
        tmem_ld_32x32_x64(row_tm + buf * 128 + hf * 64, sv);
        float mx8[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mx8[e] = -INFINITY;
        if (n_ok >= 64) {
#pragma unroll
          for (int e = 0; e < 64; ++e) mx8[e & 7] = fmaxf(mx8[e & 7], __uint_as_float(sv[e]));
        } else {
#pragma unroll
          for (int e = 0; e < 64; ++e)
            if (e < n_ok) mx8[e & 7] = fmaxf(mx8[e & 7], __uint_as_float(sv[e]));
        }
        float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                         fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
        // Both halves have read their S columns before either writes P over them.
        float mx_other;
        if (!exchange(mx, mx_other)) {
          ok = false;
          break;
        }
        mx = fmaxf(mx, mx_other);
        // The running maximum moves only when the block's exceeds it by more
        // than 8 (log2 units): with a stale maximum the weights stay below
        // 2^8, far inside bf16 and fp32, and O is rescaled rarely.  The
        // result is unchanged: O and l share the same shift.  A block with no
        // admissible key (mx = -inf) leaves it where it is.
        const float mb = mx * sc;
        const float m_new = (mb > m + 8.0f) ? mb : m;   // the first block always takes its maximum
        const float alpha = exp2_fast(m - m_new);       // 0 for the first block, else 1 or < 2^-8
        // P = exp2(s * scale - m), packed to bf16 pairs: this half's keys
        // 64hf + 32hh + (0..31) go to buffer columns 32hf + 16hh + (0..15).
        const float neg = -m_new;
        float rs4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int k0 = hh * 32 + 2 * e;
            float p0 = exp2_fast(fmaf(__uint_as_float(sv[k0]), sc, neg));
            float p1 = exp2_fast(fmaf(__uint_as_float(sv[k0 + 1]), sc, neg));
            if (n_ok < 64) {
              p0 = k0 < n_ok ? p0 : 0.f;
              p1 = k0 + 1 < n_ok ? p1 : 0.f;
            }
            rs4[e & 3] += p0 + p1;
            pk[e] = pack_bf16x2(p0, p1);
          }
          tmem_st_32x32_x16_nowait(row_tm + buf * 128 + hf * 32 + hh * 16, pk);
        }
        // Rescale this half's O columns when the maximum moved, once P(gb - 1)
        // V has completed (it cannot be two phases ahead: P(gb + 2) V needs
        // this warp's P(gb + 2)).
        if (j > 0 && __any_sync(0xffffffffu, alpha != 1.0f)) {
          const uint32_t pb = gb - 1;
          if (!warp_wait(&pv_done[pb % kSBufs], (pb / kSBufs) & 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < 2; ++c) {
            float ov[32];
            tmem_ld_32x32(o_tm + c * 32, ov);
#pragma unroll
            for (int e = 0; e < 32; ++e) ov[e] *= alpha;
            tmem_st_32x32(o_tm + c * 32, ov);
          }
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[buf]);
        l = l * alpha + ((rs4[0] + rs4[1]) + (rs4[2] + rs4[3]));
        m = m_new;
      }
      if (!ok) break;
      g += it.n_kv;
      float l_other;
      if (!exchange(l, l_other) || !warp_wait(o_done, done & 1, abort_flag, p.status)) {
        ok = false;
        break;
      }
      ++done;
      tc_fence_after();
      const float inv = 1.0f / (hf == 0 ? l + l_other : l_other + l);
#pragma unroll 1
      for (int c = 0; c < 2; ++c) {
        float ov[32];
        tmem_ld_32x32(o_tm + c * 32, ov);
        if (qi < p.L) {
          uint4* d4 = reinterpret_cast<uint4*>(p.out + (static_cast<size_t>(it.b) * p.L + qi) *
                                                           (static_cast<size_t>(p.Hq) * kHeadDim) +
                                               static_cast<size_t>(it.h) * kHeadDim + hf * 64 + c * 32);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint32_t w4[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) w4[e] = pack_bf16x2(ov[8 * q + 2 * e] * inv, ov[8 * q + 2 * e + 1] * inv);
            d4[q] = make_uint4(w4[0], w4[1], w4[2], w4[3]);
          }
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
  if (!encode_bf16_2d(&p.tm_qkv, qkv, rows, width, 64, 128)) return cudaErrorInvalidValue;
  p.out = out;
  p.status = status;
  p.B = B;
  p.L = L;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.causal = causal;
  p.group = Hq / Hkv;
  p.n_qt = (L + 127) / 128;
  p.n_items = B * Hq * p.n_qt;
  p.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));
  cudaError_t e = ensure_max_smem(reinterpret_cast<const void*>(packed_attention_kernel), kAttnSmem);
  if (e != cudaSuccess) return e;
  const int grid = p.n_items < n_sm ? p.n_items : n_sm;
  return launch_k(packed_attention_kernel, dim3(grid), dim3(kAttnThreads), kAttnSmem, stream, 1, p);
}

}  // namespace cer
