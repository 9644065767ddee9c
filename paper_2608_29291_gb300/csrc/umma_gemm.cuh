// umma_gemm.cuh -- persistent, warp-specialised tcgen05 GEMM skeleton for
// sm_103a, shared by the scorer and the two FFN contractions.
//
// One CTA per SM (96 + 32*EPI_WARPS threads, up to ~225 KB shared memory,
// 2*BN TMEM columns):
//   warp 0     activation producer: TMA loads of the A tile (128 rows x 64
//              bf16 per K block) into a STAGES-deep ring;
//   warp 2     weight producer: TMA loads of the B tile (BN rows x 64 bf16,
//              or 64 K-rows x BN for an MN-major B) into the same ring; a
//              ring slot holds KSUB consecutive 64-wide K blocks, each with
//              its own "full" barrier and one "empty" barrier for the slot;
//   warp 1     allocates TMEM, one elected lane issues tcgen05.mma
//              (M=128, N=BN, K=16) four times per 64-wide K block and
//              commits the ring slot back to both producers;
//   warps 3..  epilogue, EPI_WARPS = 4 or 8: read the fp32 accumulator out of
//              TMEM (lane = tile row; with 8 warps, warps 3-6 take the first
//              half of the columns and warps 7-10 the second) and apply the
//              problem's fused epilogue.
// The accumulator is double-buffered in TMEM so the epilogue of one tile
// overlaps the MMAs of the next.
//
// With MMA_PAIR == 1 (CLUSTER == 2) the two CTAs of a cluster run one
// M=256 x N=BN pair MMA per K step (tcgen05 cta_group::2): each CTA loads its
// 128 A rows and its half of the B tile into its own ring, all of the pair's
// copies are counted on the even CTA's ring barrier, the even CTA's warp 1
// issues the MMAs and its commits free the ring slot and publish the
// accumulator in both CTAs, and each epilogue warp frees its accumulator
// buffer with one arrival on the even CTA's barrier.  Each SM then streams
// 128 x 64 of A plus BN/2 x 64 of B per K step.  Cluster barriers bracket
// start-up and teardown so no CTA exits while its peer may still use it.
//
// Work split.  A cluster is a "slot"; the grid holds as many slots as can be
// resident at once.  Tiles [0, dp_tiles) go round-robin to the slots whole.
// The K blocks of the remaining tiles (stream-K) are cut into one contiguous
// run per slot, so every slot gets the same number of K blocks however the
// tile count divides.  A run splits into segments at tile boundaries:
//   - a segment that starts at K block 0 belongs to the tile's owner, which
//     runs the problem's epilogue once the tile is complete;
//   - a segment that starts later (only a run's first segment can) is a
//     contribution: its fp32 accumulator goes to the slot's region of the
//     partial buffer and the slot publishes a flag.
// The owner of a split tile waits (bounded) for the flags of the following
// slots whose runs start inside the tile, adds their partials into its TMEM
// accumulator, clears the flags and calls the epilogue as for a whole tile.
// Contributions are made at the start of a run and consumed at the end of
// another, so the owner rarely waits; every slot of the grid is resident.
// The owner's segment ends its run, so by the time its accumulator is full
// the ring is idle: each partial comes in with one bulk copy per epilogue
// half.  Partials are stored per (slot, CTA, half) as 128 rows of the half's
// columns with the 16-byte chunks of row r permuted by r % 8, so that the
// owner's threads, one row each, read shared memory without bank conflicts.
//
// When every slot is busy these contractions are bound by L2 bandwidth (the
// K-block rate per slot drops as slots are added), so splitting only pays
// where a last wave would leave most slots idle; see stream_k_plan.
//
// Slots, barriers and threads, as measured on GB300 (globaltimer traces of
// the FFN GEMMs):
//   - every slot costs the MMA thread a wait, a fence and a commit; with one
//     64-wide K block per slot that overhead made the 256 x 256 pair tile
//     ~10% slower than with two (KSUB = 2);
//   - a ring of three 64 KB slots gives a freed slot ~1 us to refill before
//     the MMAs need it, about one copy latency; with a single barrier per
//     slot the MMA thread waited for data a fifth of its time.  A "full"
//     barrier per K block lets the MMAs start on the first half of a slot
//     while the second half still streams in;
//   - each slot costs a producer thread an empty-slot wait, an expect_tx and
//     one TMA instruction per box, a few hundred cycles whatever the box
//     size; one thread per operand keeps that below the MMA time.
// When the weights come from no earlier kernel the weight producer never
// waits for it (programmatic dependent launch): its copies start at once.
//
// Every wait is bounded (ptx.cuh); on a timeout the CTA unwinds, waits
// briefly for its own copies and MMAs, frees TMEM and exits.
//
// A problem class P supplies:
//   BN, STAGES, B_MN_MAJOR, EPI_WARPS, CLUSTER, MMA_PAIR, kBStepBytes,
//   KSUB (64-wide K blocks per ring slot, 1 or 2),
//   Params (with `int* status`), num_tiles(p) (cluster tiles),
//   num_kb(p) (64-wide K blocks; K blocks of the last slot past the end are
//   still copied -- zeros or unused data -- but their MMAs are skipped),
//   prod_tile(p, tile, rank, state),
//   prod_kb(p, state, tile, kb, lane, a_smem, b_smem, bar, part): the copies
//   of 64-wide K block kb (with MMA_PAIR, `bar` is the cluster address of
//   the even CTA's barrier; `part` selects the activation copy, the weight
//   copy or both),
//   weights_first(p): true when num_tiles, num_kb, prod_tile and the weight
//   copies read nothing a previous kernel may write, so the weight producer
//   need not wait for that kernel to finish,
//   acts_first(p): the same for the activation copies,
//   stage_bytes(p, tile, kb, part) (the bytes of the selected copies of one
//   K block; with MMA_PAIR, of both CTAs),
//   bdesc(saddr), prefetch(p) (prefetches the tensor maps' descriptors),
//   kEpiSmemBytes (shared memory reserved for the epilogue, may be 0),
//   kEpiZeroBytes (how much of it, from its start, is zeroed before any
//   thread starts its role),
//   epilogue(p, tile, row, half, taddr, ctx) -> false to abort (ctx.rank is
//   the CTA's rank in its cluster): columns
//   [half*BN/H, (half+1)*BN/H) of accumulator row `row` (H = EPI_WARPS/4
//   groups of four warps), taddr addressing
//   column 0 of that row's lanes, ctx the reserved shared memory, a
//   bounded barrier over the 128 threads of the half and the accumulator
//   buffer (0 or 1) the tile is in -- that buffer's next tile is delivered
//   only after every epilogue thread has returned from this one;
//   epilogue_done(p, row, half): once, after the last tile.
#pragma once

#include <atomic>

namespace cer {
// Parts of a K block's copies (prod_kb, stage_bytes): each producer thread
// issues one of them.
constexpr int kPartAct = 1;       // the A operand, produced by the previous kernel
constexpr int kPartWeights = 2;   // the B operand, static weights
}

#include "kernels.h"
#include "ptx.cuh"

namespace cer {

template <class P>
constexpr int gemm_threads() {
  return 96 + 32 * P::EPI_WARPS;
}
constexpr int kFirstEpiWarp = 3;
constexpr uint32_t kATileBytes = 128 * 128;  // 128 rows x 64 bf16

template <int BN>
struct TmemCols {
  static constexpr uint32_t need = 2 * BN;
  static constexpr uint32_t value = need <= 32 ? 32 : need <= 64 ? 64 : need <= 128 ? 128 : need <= 256 ? 256 : 512;
};

// Bytes of one 64-wide K block of the B tile in one CTA (half of it with a
// pair MMA).
template <class P>
__host__ __device__ constexpr uint32_t b_stage_bytes() {
  return static_cast<uint32_t>(P::MMA_PAIR ? P::BN / 2 : P::BN) * 128u;
}

// One ring slot (KSUB K blocks) of each operand in one CTA.
template <class P>
__host__ __device__ constexpr uint32_t a_slot_bytes() {
  return static_cast<uint32_t>(P::KSUB) * kATileBytes;
}
template <class P>
__host__ __device__ constexpr uint32_t b_slot_bytes() {
  return static_cast<uint32_t>(P::KSUB) * b_stage_bytes<P>();
}

template <class P>
constexpr size_t gemm_smem_bytes() {
  return 1024 + static_cast<size_t>(P::STAGES) * (a_slot_bytes<P>() + b_slot_bytes<P>()) + P::kEpiSmemBytes + 256;
}

// Stream-K split of a launch (see above).  partial == nullptr: every tile
// whole, round-robin over the slots.
struct StreamK {
  float* partial;               // [slots][CLUSTER][128][BN] fp32, one contribution per slot
  unsigned long long* flags;    // [slots][CLUSTER][EPI_WARPS / 4]; 0 or a launch token
  unsigned long long token;     // non-zero value a contributor publishes
  int dp_tiles;                 // tiles handed out whole
};

// First stream-K unit (K block) of slot s of S over U units.
__host__ __device__ __forceinline__ long long sk_first_unit(long long U, int s, int S) {
  return U * s / S;
}

// Host side: how a launch splits its tiles.  With every slot busy these
// contractions are bound by L2 bandwidth (the K-block rate per slot drops as
// slots are added), so a split that keeps them all busy only adds partial
// traffic.  Two cases pay:
//   - a last wave that would leave most slots idle: when the tiles fill at
//     least one wave, the last wave is at most half full and the contraction
//     has at least 64 K blocks, the last full wave and the remainder are split,
//     every run covering at least one tile (at most two contributors a tile);
//   - fewer tiles than half the slots (a small M): every tile is split over up
//     to four slots when each run keeps at least 8 K blocks, so the operands
//     stream into four times as many SMs; runs are then shorter than a tile
//     and a tile has up to four contributors.
// (Splitting the scorer's short contractions was measured slower: the
// owners' GELU epilogues then run on a quarter of the SMs.)
struct SplitPlan {
  int slots;      // clusters to launch
  int dp_tiles;   // tiles handed out whole (== tiles: no split)
};

constexpr int kMaxSplit = 4;

//   - balance_waves (the tensor-bound pair scorer, whose tiles are few and
//     long): whenever the tiles fill at least one wave but not a whole number
//     of them, the last full wave and the remainder are split, so every slot
//     takes the same number of K blocks.
inline SplitPlan stream_k_plan(int tiles, int nkb, int slots, bool balance_waves = false) {
  const SplitPlan whole{tiles < slots ? tiles : slots, tiles};
  if (slots <= 1 || tiles <= 0) return whole;
  const int q = tiles / slots;
  const int r = tiles % slots;
  if (balance_waves && q > 0 && r > 0) return SplitPlan{slots, (q - 1) * slots};
  if (q == 0) {
    if (2 * tiles > slots) return whole;
    const int s = tiles * kMaxSplit < slots ? tiles * kMaxSplit : slots;
    if (static_cast<long long>(tiles) * nkb < 8LL * s) return whole;
    return SplitPlan{s, 0};
  }
  if (nkb < 64 || r == 0 || 2 * r > slots) return whole;
  return SplitPlan{slots, (q - 1) * slots};
}

// The segments a slot works through, in order: its whole tiles, then its
// stream-K run cut at tile boundaries.  Producer, MMA issuer and epilogue
// each walk their own copy.
struct SegCursor {
  int n_slots, nkb, dp_tiles, next_dp;
  long long u, u_end;

  __device__ SegCursor(int slot, int n_slots_, int ntiles, int nkb_, int dp_tiles_)
      : n_slots(n_slots_), nkb(nkb_), dp_tiles(dp_tiles_), next_dp(slot) {
    const long long U = static_cast<long long>(ntiles - dp_tiles_) * nkb_;
    u = sk_first_unit(U, slot, n_slots_);
    u_end = sk_first_unit(U, slot + 1, n_slots_);
  }
  __device__ bool next(int& tile, int& kb0, int& kb1) {
    if (next_dp < dp_tiles) {
      tile = next_dp;
      kb0 = 0;
      kb1 = nkb;
      next_dp += n_slots;
      return true;
    }
    if (u < u_end) {
      const long long t = u / nkb;
      tile = dp_tiles + static_cast<int>(t);
      kb0 = static_cast<int>(u - t * nkb);
      const long long end = u_end - t * nkb;
      kb1 = end < nkb ? static_cast<int>(end) : nkb;
      u += kb1 - kb0;
      return true;
    }
    return false;
  }
};

// A short, abort-independent wait used only while unwinding.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > 100000000ull) return;
  }
}

// Sleep about `ns` nanoseconds (bounded; used only while unwinding).
__device__ __forceinline__ void unwind_pause(uint64_t ns) {
  const uint64_t t0 = globaltimer_ns();
  while (globaltimer_ns() - t0 < ns) __nanosleep(1000);
}

// Every lane waits on the same barrier; one vote gives the warp a single
// verdict, so every branch after a wait stays warp-uniform, which the
// .sync.aligned tcgen05 instructions require.  (Lane 0 waiting alone and
// broadcasting its result costs a divergence and a reconvergence per wait.)
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* status) {
  const bool ok = mbar_wait(bar, parity, abort_flag, status);
  return __all_sync(0xffffffffu, ok);
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
  int acc = 0;   // the tile's TMEM accumulator buffer
  __device__ __forceinline__ bool sync() {
    mbar_arrive(half_bar);
    const bool ok = mbar_wait(half_bar, phase, abort_flag, status);
    phase ^= 1;
    return ok;
  }
};

template <class P>
__global__ void __launch_bounds__(gemm_threads<P>(), 1)
    umma_gemm_kernel(const __grid_constant__ typename P::Params p, const __grid_constant__ StreamK sk) {
  static_assert(P::EPI_WARPS == 4 || P::EPI_WARPS == 8, "epilogue is one or two groups of four warps");
  constexpr bool PAIR = P::MMA_PAIR != 0;
  static_assert(P::CLUSTER == (PAIR ? 2 : 1), "a pair MMA runs on a 2-CTA cluster, anything else on one CTA");
  constexpr uint16_t kPairMask = 0x3;
  constexpr int BN = P::BN;
  constexpr int STAGES = P::STAGES;
  constexpr int HALVES = P::EPI_WARPS / 4;
  constexpr int HALF_COLS = BN / HALVES;
  constexpr int KSUB = P::KSUB;
  static_assert(KSUB == 1 || KSUB == 2, "one or two K blocks per ring slot");
  constexpr uint32_t A_BYTES = a_slot_bytes<P>();
  constexpr uint32_t B_BYTES = b_slot_bytes<P>();
  constexpr uint32_t TMEM_COLS = TmemCols<BN>::value;
  constexpr uint32_t IDESC = idesc_bf16(PAIR ? 256 : 128, BN, P::B_MN_MAJOR);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* a_ring = smem;
  uint8_t* b_ring = smem + STAGES * A_BYTES;
  uint8_t* epi_smem = b_ring + STAGES * B_BYTES;  // 1024-byte aligned
  uint64_t* full = reinterpret_cast<uint64_t*>(epi_smem + P::kEpiSmemBytes);   // [STAGES][KSUB]
  uint64_t* empty = full + STAGES * KSUB;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* half_bar = drain + 1;
  uint64_t* sk_bar = half_bar + 2;   // the owner's partial copies, one per epilogue half
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sk_bar + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int rank = PAIR ? static_cast<int>(cluster_ctarank()) : 0;
  const int slot = blockIdx.x / P::CLUSTER;
  const int n_slots = gridDim.x / P::CLUSTER;

  if (threadIdx.x == 32) P::prefetch(p);   // tensor-map descriptors, ahead of the first copy
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES * KSUB; ++s)
      mbar_init(&full[s], 2);    // the two producers' expect_tx (the even CTA's, with a pair MMA)
    for (int s = 0; s < STAGES; ++s)
      mbar_init(&empty[s], 1);   // one MMA commit (the even CTA's, with a pair MMA)
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      // Every epilogue thread (with a pair MMA: every epilogue warp of both CTAs).
      mbar_init(&tempty[a], PAIR ? 2 * P::EPI_WARPS : 32 * P::EPI_WARPS);
    }
    mbar_init(drain, 1);
    mbar_init(&half_bar[0], 128);
    mbar_init(&half_bar[1], 128);
    mbar_init(&sk_bar[0], 1);
    mbar_init(&sk_bar[1], 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  static_assert(P::kEpiZeroBytes <= P::kEpiSmemBytes && P::kEpiZeroBytes % 4 == 0, "zeroed epilogue smem");
  if constexpr (P::kEpiZeroBytes > 0) {
    for (uint32_t i = threadIdx.x; i < P::kEpiZeroBytes / 4; i += blockDim.x)
      reinterpret_cast<uint32_t*>(epi_smem)[i] = 0u;
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
  if (PAIR) {
    cluster_sync();      // the peer's barriers exist before any copy or commit reaches them
  } else {
    __syncthreads();
  }
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // Inputs written by the previous kernel are visible after this wait
  // (programmatic dependent launch starts this kernel while the previous one
  // is still finishing).  The weight producer skips it when the weights and
  // the tile walk depend on nothing that kernel writes.  It then does not
  // signal the dependents either: the first signal of any thread releases
  // the CTA, and every CTA signalling only after its own wait keeps the rule
  // that when a kernel starts, the kernels two or more launches back have
  // completed -- which is what makes weights written there safe to read
  // without the wait.
  // The activation producer (and, when neither operand waits, the MMA
  // issuer, which reads no global memory) likewise skip it when the previous
  // kernel writes nothing the activation copies read (acts_first: the
  // scorer behind the generation bias-table kernel); the epilogue always
  // waits.
  const bool weights_first = P::weights_first(p);
  const bool acts_first = P::acts_first(p);
  const bool skip_wait = (warp == 2 && weights_first) || (warp == 0 && acts_first) ||
                         (warp == 1 && weights_first && acts_first);
  if (!skip_wait) {
    griddep_wait();
    griddep_launch_dependents();
  }

  const int ntiles = P::num_tiles(p);
  const int nk64 = P::num_kb(p);                 // 64-wide K blocks
  const int nkb = (nk64 + KSUB - 1) / KSUB;      // ring slots per tile
  const int dp_tiles = sk.partial != nullptr && sk.dp_tiles < ntiles ? sk.dp_tiles : ntiles;

  if (warp == 0 || warp == 2) {
    // ---------------------------------------------------------------- producers
    // One thread each: TMA copies and mbarrier operations are per thread, and
    // a warp-wide wait (test, broadcast, reconverge) would double the cost of
    // issuing a slot.  Warp 0 copies the activations, warp 2 the weights;
    // both walk the same slots and each adds its own bytes to a slot's count.
    if (lane == 0) {
      const int part = warp == 0 ? kPartAct : kPartWeights;
      typename P::ProdState st;
      SegCursor cur(slot, n_slots, ntiles, nkb, dp_tiles);
      int stage = 0;
      uint32_t phase = 0;
      long issued = 0;
      bool ok = true;
      // With a pair MMA the even CTA's ring barriers count both CTAs' copies.
      const uint32_t leader_full = PAIR ? mapa_shared(smem_u32(full), 0) : 0u;
      int tile, kb0, kb1;
      while (ok && cur.next(tile, kb0, kb1)) {
        P::prod_tile(p, tile, rank, st);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.status)) {   // a fresh slot passes at once
            ok = false;
            break;
          }
#pragma unroll
          for (int j = 0; j < KSUB; ++j) {
            const int k64 = kb * KSUB + j;
            const int fb = stage * KSUB + j;
            uint8_t* a_dst = a_ring + stage * A_BYTES + j * kATileBytes;
            uint8_t* b_dst = b_ring + stage * B_BYTES + j * b_stage_bytes<P>();
            if (!PAIR || rank == 0) mbar_arrive_expect_tx(&full[fb], P::stage_bytes(p, tile, k64, part));
            if constexpr (PAIR) {
              P::prod_kb(p, st, tile, k64, 0, a_dst, b_dst, leader_full + static_cast<uint32_t>(fb) * 8u, part);
            } else {
              P::prod_kb(p, st, tile, k64, 0, a_dst, b_dst, &full[fb], part);
            }
          }
          ++issued;
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok) {
        // Let the copies already issued land before the CTA's memory goes away
        // (the odd CTA of a pair cannot see the barrier its copies count on).
        if (PAIR && rank != 0) {
          unwind_pause(1000000ull);
        } else {
          for (long n = issued - 1; n >= 0 && n >= issued - STAGES; --n)
            for (int j = 0; j < KSUB; ++j)
              drain_wait(&full[(n % STAGES) * KSUB + j], static_cast<uint32_t>((n / STAGES) & 1));
        }
      }
    }
    __syncwarp();
  } else if (warp == 1 && (!PAIR || rank == 0)) {
    // ---------------------------------------------------------------- MMA issuer
    // One thread, like the producer (tcgen05.mma and tcgen05.commit are
    // issued by a single thread).
    if (lane == 0) {
      SegCursor cur(slot, n_slots, ntiles, nkb, dp_tiles);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      bool issued_any = false;
      int tile, kb0, kb1;
      while (ok && cur.next(tile, kb0, kb1)) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
        for (int kb = kb0; kb < kb1; ++kb) {
          const uint32_t a_base = smem_u32(a_ring + stage * A_BYTES);
          const uint32_t b_base = smem_u32(b_ring + stage * B_BYTES);
          const int nsub = nk64 - kb * KSUB < KSUB ? nk64 - kb * KSUB : KSUB;   // K blocks in this slot
#pragma unroll
          for (int j = 0; j < KSUB; ++j) {
            // Every K block of the slot was copied (the barrier phases stay in
            // step); only those inside the contraction are multiplied.
            if (!mbar_wait(&full[stage * KSUB + j], phase, abort_flag, p.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            if (j < nsub) {
              issued_any = true;
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const uint64_t adesc = sdesc_kmajor_sw128(a_base + j * kATileBytes + k * 32);
                const uint64_t bdesc = P::bdesc(b_base + j * b_stage_bytes<P>() + k * P::kBStepBytes);
                const uint32_t accumulate = ((kb - kb0) | j | k) != 0 ? 1u : 0u;
                if (PAIR)
                  umma_bf16_pair(d_tmem, adesc, bdesc, IDESC, accumulate);
                else
                  umma_bf16(d_tmem, adesc, bdesc, IDESC, accumulate);
              }
            }
          }
          if (!ok) break;
          if (PAIR)
            umma_commit_pair_multicast(&empty[stage], kPairMask);   // frees the slot in both CTAs
          else
            umma_commit(&empty[stage]);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        if (PAIR)
          umma_commit_pair_multicast(&tfull[acc], kPairMask);   // both CTAs' epilogues
        else
          umma_commit(&tfull[acc]);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1;
        }
      }
      if (!ok && issued_any) {
        if (PAIR)
          umma_commit_pair(drain);
        else
          umma_commit(drain);
        drain_wait(drain, 0);
      }
    }
    __syncwarp();
  } else if (warp >= kFirstEpiWarp) {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;                        // TMEM lane quadrant this warp may access
    const int row = q * 32 + lane;                 // accumulator row = TMEM lane
    const int half = (warp - kFirstEpiWarp) >> 2;  // which half of the accumulator columns
    EpiCtx ctx{epi_smem, rank, &half_bar[half], 0u, abort_flag, p.status};
    const uint32_t leader_tempty = PAIR ? mapa_shared(smem_u32(tempty), 0) : 0u;
    const long long sk_units = static_cast<long long>(ntiles - dp_tiles) * nkb;
    uint32_t sk_phase = 0;
    SegCursor cur(slot, n_slots, ntiles, nkb, dp_tiles);
    int acc = 0;
    uint32_t acc_phase = 0;
    int tile, kb0, kb1;
    while (cur.next(tile, kb0, kb1)) {
      if (!warp_wait(&tfull[acc], acc_phase, abort_flag, p.status)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      bool ok = true;
      if (kb0 > 0) {
        // A contribution: this half's columns of the row go to the slot's
        // partial region (chunks permuted by row), then the half publishes
        // its flag.
        float4* dst = reinterpret_cast<float4*>(sk.partial) +
                      (static_cast<size_t>((slot * P::CLUSTER + rank) * HALVES + half) * 128 + row) * (HALF_COLS / 4);
#pragma unroll 1
        for (int c = 0; c < HALF_COLS; c += 32) {
          float v[32];
          tmem_ld_32x32(taddr + half * HALF_COLS + c, v);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            __stcg(dst + ((c / 4 + j) ^ (row & 7)), make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]));
        }
        __threadfence();
        ok = ctx.sync();
        if (ok && row == 0) st_release_u64(&sk.flags[(slot * P::CLUSTER + rank) * HALVES + half], sk.token);
      } else {
        if (kb1 < nkb) {
          // The owner of a split tile: the runs of the following slots that
          // start inside this tile hold the rest of its K blocks.  Each
          // partial is copied into the (idle) ring, then added into TMEM.
          const long long tile_end = static_cast<long long>(tile - dp_tiles + 1) * nkb;
          constexpr uint32_t kHalfBytes = 128u * HALF_COLS * 4u;
          static_assert(HALVES * kHalfBytes <= STAGES * (A_BYTES + B_BYTES), "partials fit in the ring");
          static_assert(kHalfBytes % 16384 == 0, "copied in 16 KB pieces");
          const float4* stage = reinterpret_cast<const float4*>(a_ring + half * kHalfBytes) + row * (HALF_COLS / 4);
          for (int s2 = slot + 1; ok && s2 < n_slots && sk_first_unit(sk_units, s2, n_slots) < tile_end; ++s2) {
            unsigned long long* flag = &sk.flags[(s2 * P::CLUSTER + rank) * HALVES + half];
            if (row == 0) {
              ok = flag_wait(flag, sk.token, abort_flag, p.status);
              if (ok) {
                fence_proxy_async_global();
                const char* src = reinterpret_cast<const char*>(sk.partial) +
                                  static_cast<size_t>((s2 * P::CLUSTER + rank) * HALVES + half) * kHalfBytes;
                mbar_arrive_expect_tx(&sk_bar[half], kHalfBytes);
                for (uint32_t off = 0; off < kHalfBytes; off += 16384)
                  bulk_load(a_ring + half * kHalfBytes + off, src + off, 16384, &sk_bar[half]);
              }
            }
            ok = ctx.sync() && !*abort_flag;
            if (ok) ok = mbar_wait(&sk_bar[half], sk_phase, abort_flag, p.status);
            sk_phase ^= 1;
            if (!ok) break;
#pragma unroll 1
            for (int c = 0; c < HALF_COLS; c += 32) {
              float v[32];
              tmem_ld_32x32(taddr + half * HALF_COLS + c, v);
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                const float4 w = stage[(c / 4 + j) ^ (row & 7)];
                v[4 * j] += w.x;
                v[4 * j + 1] += w.y;
                v[4 * j + 2] += w.z;
                v[4 * j + 3] += w.w;
              }
              tmem_st_32x32(taddr + half * HALF_COLS + c, v);
            }
            ok = ctx.sync();   // the stage is read before the next copy overwrites it
            if (ok && row == 0) st_relaxed_u64(flag, 0ull);
          }
        }
        ctx.acc = acc;
        if (ok) ok = P::epilogue(p, tile, row, half, taddr, ctx);
      }
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
  if (PAIR) {
    cluster_sync();      // the peer no longer copies into, commits to or arrives on this CTA
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

// ---------------------------------------------------------------- host side

// A launch's stream-K token: never 0, and hashed (SplitMix64 finaliser) so
// that whatever a fresh workspace holds is not taken for a published flag.
inline unsigned long long next_stream_k_token() {
  static std::atomic<unsigned long long> counter{0};
  unsigned long long z = counter.fetch_add(1) + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  z ^= z >> 31;
  return z | 1ull;
}

// Launches umma_gemm_kernel<P> over `tiles` cluster tiles of `nkb` 64-wide
// K blocks (the fewest the kernel may take, for a contraction length decided
// on the device).  The persistent grid holds at most as many slots (clusters) as can
// be resident at once; with a stream-K region the tiles may be split.
template <class P>
cudaError_t launch_gemm(const typename P::Params& p, int tiles, int nkb, const StreamKArea* area, int n_sm,
                        cudaStream_t stream, bool balance_waves = false) {
  if (tiles == 0) return cudaSuccess;
  const size_t smem = gemm_smem_bytes<P>();
  cudaError_t e = ensure_max_smem(reinterpret_cast<const void*>(umma_gemm_kernel<P>), smem);
  if (e != cudaSuccess) return e;
  int slots = n_sm;
  if (P::CLUSTER > 1) {
    // Clusters must fit inside GPC boundaries: ask how many can be resident.
    static int resident[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    int& max_clusters = resident[dev & 63];
    if (max_clusters == 0) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(n_sm / P::CLUSTER * P::CLUSTER, 1, 1);
      cfg.blockDim = dim3(gemm_threads<P>(), 1, 1);
      cfg.dynamicSmemBytes = smem;
      cfg.stream = stream;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = P::CLUSTER;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      e = cudaOccupancyMaxActiveClusters(&n, umma_gemm_kernel<P>, &cfg);
      if (e != cudaSuccess) return e;
      max_clusters = n > 0 ? n : 1;
    }
    slots = max_clusters;
  }
  StreamK sk{};
  SplitPlan plan{tiles < slots ? tiles : slots, tiles};
  if (area != nullptr && area->partial != nullptr && area->flags != nullptr) {
    const SplitPlan split = stream_k_plan(tiles, nkb, slots, balance_waves);
    const size_t partial = static_cast<size_t>(split.slots) * P::CLUSTER * 128 * P::BN * sizeof(float);
    const size_t flags = static_cast<size_t>(split.slots) * P::CLUSTER * (P::EPI_WARPS / 4) * sizeof(unsigned long long);
    if (split.dp_tiles < tiles && partial <= kStreamKPartialBytes && flags <= kStreamKFlagBytes) {
      plan = split;
      sk.partial = area->partial;
      sk.flags = area->flags;
      sk.token = next_stream_k_token();
      sk.dp_tiles = split.dp_tiles;
    }
  }
  return launch_k(umma_gemm_kernel<P>, dim3(plan.slots * P::CLUSTER), dim3(gemm_threads<P>()), smem, stream,
                  P::CLUSTER, p, sk);
}

}  // namespace cer
