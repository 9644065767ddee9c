// umma_gemm.cuh -- persistent, warp-specialised tcgen05 GEMM skeleton for
// sm_103a, shared by the scorer and the two FFN contractions.
//
// One CTA per SM (64 + 32*EPI_WARPS threads, up to ~225 KB shared memory,
// 2*BN TMEM columns):
//   warp 0     producer: TMA box loads of the A tile (128 rows x 64 bf16)
//              and the B tile (BN rows x 64 bf16, or 64 K-rows x BN for an
//              MN-major B) into a STAGES-deep ring;
//   warp 1     allocates TMEM, one elected lane issues tcgen05.mma
//              (M=128, N=BN, K=16) four times per 64-wide K block and
//              commits the ring slot back to the producer;
//   warps 2..  epilogue, EPI_WARPS = 4 or 8: read the fp32 accumulator out of
//              TMEM (lane = tile row; with 8 warps, warps 2-5 take the first
//              half of the columns and warps 6-9 the second) and apply the
//              problem's fused epilogue.
// The accumulator is double-buffered in TMEM so the epilogue of tile i
// overlaps the MMAs of tile i+1.  Tiles are visited with a stride of the
// number of clusters.  With CLUSTER == 2 the two CTAs of a cluster work on
// one cluster tile (two adjacent 128-row tiles sharing a B tile): each loads
// half of B and multicasts it to both, each MMA commit frees the ring slot
// in both CTAs, and cluster barriers bracket start-up and teardown so no CTA
// exits while its peer may still write into its shared memory.
//
// With MMA_PAIR == 1 (CLUSTER == 2) the cluster runs one M=256 x N=BN pair MMA
// per K step instead (tcgen05 cta_group::2): each CTA loads its 128 A rows
// and its half of the B tile into its own ring, all of the pair's copies are
// counted on the even CTA's ring barrier, the even CTA's warp 1 issues the
// MMAs and its commits free the ring slot and publish the accumulator in both
// CTAs, and each epilogue warp frees its accumulator buffer with one arrival
// on the even CTA's barrier.  Each SM then streams 128 x 64 of A plus
// BN/2 x 64 of B per K step instead of the whole B tile.
//
// Every wait is bounded (ptx.cuh); on a timeout the CTA unwinds, waits
// briefly for its own copies and MMAs, frees TMEM and exits.
//
// A problem class P supplies:
//   BN, STAGES, B_MN_MAJOR, EPI_WARPS, CLUSTER, MMA_PAIR, kBStepBytes,
//   Params (with `int* status`), num_tiles(p) (cluster tiles),
//   num_kb(p), prod_tile(p, tile, rank, state),
//   prod_kb(p, state, tile, kb, lane, a_smem, b_smem, bar) (with MMA_PAIR,
//   `bar` is the cluster address of the even CTA's ring barrier),
//   stage_bytes(p, tile, kb) (with MMA_PAIR, the bytes of both CTAs),
//   bdesc(saddr),
//   kEpiSmemBytes (shared memory reserved for the epilogue, may be 0),
//   epilogue(p, tile, row, half, taddr, ctx) -> false to abort (ctx.rank is
//   the CTA's rank in its cluster): columns
//   [half*BN/H, (half+1)*BN/H) of accumulator row `row` (H = EPI_WARPS/4
//   groups of four warps), taddr addressing
//   column 0 of that row's lanes, ctx the reserved shared memory and a
//   bounded barrier over the 128 threads of the half;
//   epilogue_done(p, row, half): once, after the last tile.
#pragma once

#include "ptx.cuh"

namespace cer {

template <class P>
constexpr int gemm_threads() {
  return 64 + 32 * P::EPI_WARPS;
}
constexpr uint32_t kATileBytes = 128 * 128;  // 128 rows x 64 bf16

template <int BN>
struct TmemCols {
  static constexpr uint32_t need = 2 * BN;
  static constexpr uint32_t value = need <= 32 ? 32 : need <= 64 ? 64 : need <= 128 ? 128 : need <= 256 ? 256 : 512;
};

// Bytes of one ring slot's B tile in one CTA (half of it with a pair MMA).
template <class P>
__host__ __device__ constexpr uint32_t b_stage_bytes() {
  return static_cast<uint32_t>(P::MMA_PAIR ? P::BN / 2 : P::BN) * 128u;
}

template <class P>
constexpr size_t gemm_smem_bytes() {
  return 1024 + static_cast<size_t>(P::STAGES) * (kATileBytes + b_stage_bytes<P>()) + P::kEpiSmemBytes + 256;
}

// Sleep about `ns` nanoseconds (bounded; used only while unwinding).
__device__ __forceinline__ void unwind_pause(uint64_t ns) {
  const uint64_t t0 = globaltimer_ns();
  while (globaltimer_ns() - t0 < ns) __nanosleep(1000);
}

// A short, abort-independent wait used only while unwinding.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > 100000000ull) return;
  }
}

// Lane 0 waits, the whole warp takes its verdict: keeps every branch after a
// wait warp-uniform, which the .sync.aligned tcgen05 instructions require.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* status) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort_flag, status) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

// What an epilogue half (4 warps, 128 threads) shares: the reserved shared
// memory and a barrier over its threads whose wait is bounded like every
// other wait (an mbarrier of count 128; each thread tracks the phase).
struct EpiCtx {
  uint8_t* smem;
  int rank;
  uint64_t* half_bar;
  uint32_t phase;
  volatile int* abort_flag;
  int* status;
  __device__ __forceinline__ bool sync() {
    mbar_arrive(half_bar);
    const bool ok = mbar_wait(half_bar, phase, abort_flag, status);
    phase ^= 1;
    return ok;
  }
};

template <class P>
__global__ void __launch_bounds__(gemm_threads<P>(), 1) umma_gemm_kernel(const __grid_constant__ typename P::Params p) {
  static_assert(P::EPI_WARPS == 4 || P::EPI_WARPS == 8, "epilogue is one or two groups of four warps");
  static_assert(P::CLUSTER == 1 || P::CLUSTER == 2, "clusters of one or two CTAs");
  constexpr bool PAIR = P::MMA_PAIR != 0;
  static_assert(!PAIR || P::CLUSTER == 2, "a pair MMA runs on a 2-CTA cluster");
  constexpr uint16_t kPairMask = 0x3;
  constexpr int BN = P::BN;
  constexpr int STAGES = P::STAGES;
  constexpr uint32_t B_BYTES = b_stage_bytes<P>();
  constexpr uint32_t TMEM_COLS = TmemCols<BN>::value;
  constexpr uint32_t IDESC = idesc_bf16(PAIR ? 256 : 128, BN, P::B_MN_MAJOR);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* a_ring = smem;
  uint8_t* b_ring = smem + STAGES * kATileBytes;
  uint8_t* epi_smem = b_ring + STAGES * B_BYTES;  // 1024-byte aligned
  uint64_t* full = reinterpret_cast<uint64_t*>(epi_smem + P::kEpiSmemBytes);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* half_bar = drain + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(half_bar + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int rank = P::CLUSTER > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  const int cluster_id = blockIdx.x / P::CLUSTER;
  const int n_clusters = gridDim.x / P::CLUSTER;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      // One MMA commit from each CTA of the cluster (from the even CTA alone with a pair MMA).
      mbar_init(&empty[s], PAIR ? 1 : P::CLUSTER);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      // Every epilogue thread (with a pair MMA: every epilogue warp of both CTAs).
      mbar_init(&tempty[a], PAIR ? 2 * P::EPI_WARPS : 32 * P::EPI_WARPS);
    }
    mbar_init(drain, 1);
    mbar_init(&half_bar[0], 128);
    mbar_init(&half_bar[1], 128);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    if (PAIR) {
      tmem_alloc_pair(tmem_slot, TMEM_COLS);   // together with warp 1 of the peer CTA
      tmem_relinquish_pair();
    } else {
      tmem_alloc(tmem_slot, TMEM_COLS);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  if (P::CLUSTER > 1) {
    cluster_sync();      // the peer's barriers exist before any multicast reaches them
  } else {
    __syncthreads();
  }
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  griddep_wait();                 // inputs written by the previous kernel are visible
  griddep_launch_dependents();

  const int ntiles = P::num_tiles(p);
  const int nkb = P::num_kb(p);

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    typename P::ProdState st;
    int stage = 0;
    uint32_t phase = 0;
    long issued = 0;
    bool ok = true;
    // With a pair MMA the even CTA's ring barriers count both CTAs' copies.
    const uint32_t leader_full = PAIR ? mapa_shared(smem_u32(full), 0) : 0u;
    for (int tile = cluster_id; tile < ntiles && ok; tile += n_clusters) {
      P::prod_tile(p, tile, rank, st);
      for (int kb = 0; kb < nkb; ++kb) {
        if (!warp_wait(&empty[stage], phase ^ 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        if (!PAIR || rank == 0) {
          const uint32_t bytes = P::stage_bytes(p, tile, kb);
          if (lane == 0) mbar_arrive_expect_tx(&full[stage], bytes);
        }
        __syncwarp();
        if constexpr (PAIR) {
          P::prod_kb(p, st, tile, kb, lane, a_ring + stage * kATileBytes, b_ring + stage * B_BYTES,
                     leader_full + static_cast<uint32_t>(stage) * 8u);
        } else {
          P::prod_kb(p, st, tile, kb, lane, a_ring + stage * kATileBytes, b_ring + stage * B_BYTES, &full[stage]);
        }
        ++issued;
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
    }
    if (!ok && lane == 0) {
      // Let the copies already issued land before the CTA's memory goes away
      // (the odd CTA of a pair cannot see the barrier its copies count on).
      if (PAIR && rank != 0) {
        unwind_pause(1000000ull);
      } else {
        for (long n = issued - 1; n >= 0 && n >= issued - STAGES; --n)
          drain_wait(&full[n % STAGES], static_cast<uint32_t>((n / STAGES) & 1));
      }
    }
  } else if (warp == 1 && (!PAIR || rank == 0)) {
    // ---------------------------------------------------------------- MMA issuer
    int stage = 0;
    uint32_t phase = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    bool issued_any = false;
    for (int tile = cluster_id; tile < ntiles && ok; tile += n_clusters) {
      if (!warp_wait(&tempty[acc], acc_phase ^ 1, abort_flag, p.status)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
      for (int kb = 0; kb < nkb; ++kb) {
        if (!warp_wait(&full[stage], phase, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (lane == 0) {
          const uint32_t a_base = smem_u32(a_ring + stage * kATileBytes);
          const uint32_t b_base = smem_u32(b_ring + stage * B_BYTES);
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint64_t adesc = sdesc_kmajor_sw128(a_base + k * 32);
            const uint64_t bdesc = P::bdesc(b_base + k * P::kBStepBytes);
            if (PAIR)
              umma_bf16_pair(d_tmem, adesc, bdesc, IDESC, (kb | k) != 0 ? 1u : 0u);
            else
              umma_bf16(d_tmem, adesc, bdesc, IDESC, (kb | k) != 0 ? 1u : 0u);
          }
          if (PAIR)
            umma_commit_pair_multicast(&empty[stage], kPairMask);
          else if (P::CLUSTER > 1)
            umma_commit_multicast(&empty[stage], kPairMask);   // frees the slot in both CTAs
          else
            umma_commit(&empty[stage]);
          issued_any = true;
        }
        __syncwarp();
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (!ok) break;
      if (lane == 0) {
        if (PAIR)
          umma_commit_pair_multicast(&tfull[acc], kPairMask);   // both CTAs' epilogues
        else
          umma_commit(&tfull[acc]);
      }
      __syncwarp();
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1;
      }
    }
    if (!ok && lane == 0 && issued_any) {
      if (PAIR)
        umma_commit_pair(drain);
      else
        umma_commit(drain);
      drain_wait(drain, 0);
    }
  } else if (warp >= 2) {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;            // TMEM lane quadrant this warp may access
    const int row = q * 32 + lane;     // accumulator row = TMEM lane
    const int half = (warp - 2) >> 2;  // which half of the accumulator columns
    EpiCtx ctx{epi_smem, rank, &half_bar[half], 0u, abort_flag, p.status};
    const uint32_t leader_tempty = PAIR ? mapa_shared(smem_u32(tempty), 0) : 0u;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = cluster_id; tile < ntiles; tile += n_clusters) {
      if (!warp_wait(&tfull[acc], acc_phase, abort_flag, p.status)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      const bool ok = P::epilogue(p, tile, row, half, taddr, ctx);
      tc_fence_before();
      if (PAIR) {
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(leader_tempty + static_cast<uint32_t>(acc) * 8u);
      } else {
        mbar_arrive(&tempty[acc]);
      }
      if (!ok) break;
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1;
      }
    }
    P::epilogue_done(p, row, half);
  }

  tc_fence_before();
  if (P::CLUSTER > 1) {
    cluster_sync();      // the peer no longer multicasts into this CTA
  } else {
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    if (PAIR)
      tmem_dealloc_pair(tmem_base, TMEM_COLS);   // together with warp 1 of the peer CTA
    else
      tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

}  // namespace cer
