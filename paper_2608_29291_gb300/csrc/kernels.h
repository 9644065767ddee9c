// kernels.h -- internal launch interface between the C ABI (cer_api.cu) and
// the kernel translation units.  Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstddef>
#include <cstdint>

#include "../../include/cer_api.h"

namespace cer {

// Encode a 2-D bf16 tensor map (rows x cols, row pitch cols*2 bytes) with a
// box of box_cols x box_rows elements, 128-byte swizzle, zero fill.
bool encode_bf16_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_cols,
                    uint32_t box_rows);

// Encode a row-major bf16 matrix (rows x cols, cols a multiple of 64) as the
// 3-D tensor [cols / 64][rows][64] with a box of 64 x box_rows x box_blocks:
// one copy brings box_blocks consecutive 64-column blocks of box_rows rows,
// each block a 128-byte-swizzled [box_rows][64] tile, the blocks one after
// another in shared memory.  The innermost coordinate is always 0.
bool encode_bf16_col_blocks(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
                            uint32_t box_blocks);

// Launch `kernel` with programmatic dependent launch allowed (and a cluster
// dimension when cluster_x > 1): it may start while the previous kernel on
// the stream finishes; its griddep_wait() orders it after that kernel.
// Every kernel of this library prefers the largest shared-memory carveout,
// so the SMs keep one configuration and a kernel with large shared memory
// (the GEMMs) can be resident beside a small one that runs before it (an SM
// whose carveout must change has to drain first).  Set once per context.
cudaError_t prefer_max_shared(const void* func);

template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                            int cluster_x, Args&&... args) {
  cudaError_t e = prefer_max_shared(reinterpret_cast<const void*>(kernel));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  int n = 0;
  attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Record a printf-style message for cer_get_error() and return `status`.
cer_status internal_fail(cer_status status, const char* fmt, ...);

// CER_OK if the current device is an sm_103 GPU this library can run on;
// otherwise the status and message every entry point gives for it.
cer_status require_supported_device();

// Identity of the current CUDA context (cuCtxGetId), 0 if none is current.
// Device addresses of module symbols and per-function attributes belong to a
// context: a cache of them is valid only while this value is unchanged (a
// cudaDeviceReset, for one, makes a new primary context).
unsigned long long current_context_id();

// The bounded-wait self-test kernel: kind 0 waits for *flag == token, kind 1
// for an mbarrier phase (completed only when arrive != 0), at most limit_ns.
cudaError_t launch_bounded_wait_selftest(int kind, const unsigned long long* flag, unsigned long long token,
                                         int arrive, unsigned long long limit_ns, int* status, cudaStream_t stream);

// Raise a kernel's dynamic shared-memory limit to `bytes` (its largest
// launch) once per device.
cudaError_t ensure_max_smem(const void* func, size_t bytes);

// Bytes of the GEMMs' stream-K partial buffer and of its flags (a launch uses
// at most this much; see umma_gemm.cuh).
constexpr size_t kStreamKPartialBytes = size_t(24) << 20;
constexpr size_t kStreamKFlagBytes = 8192;

// A stream-K region of a workspace (both NULL: tiles are never split).  The
// kernels that use it run one after another on a stream and leave every flag
// cleared, so one region serves the scorer and both FFN GEMMs of a block.
struct StreamKArea {
  float* partial;               // kStreamKPartialBytes
  unsigned long long* flags;    // kStreamKFlagBytes
};

// ------------------------------------------------------------------ S1 score
struct ScoreArgs {
  const __nv_bfloat16* h;
  int B, N, d;
  const __nv_bfloat16* W1;
  const float* b1;
  const float* w2;
  int Hc;
  const __nv_bfloat16* W1e;
  const float* b1e;
  const float* w2e;
  const __nv_bfloat16* U;
  int He, E, S;
  const float* t;
  int gen;
  int* status;
};

// Frequencies of the sinusoidal progress embedding divided by 2*pi, in fp64:
// g[j] = 10000^(-j/(E/2)) / (2*pi), j < E/2 <= 512 (computed on the host).
struct EmbFreqTable {
  double g[512];
};

struct ScoreWorkspace {
  float* bias_tab;  // [B][Hc + He]
  float* w2_tab;    // [B][Hc + He]
  float* partial;   // [n_partials][B*N], n_partials = (Hc + He) / chunk width <= (Hc + He) / 64
};

// Largest hidden-chunk width the scorer may use for these widths (0: none).
int score_chunk_width(int Hc, int He, int gen);
// Upper bound of the partial-score rows the scorer writes.
int score_max_partials(int Hc, int He, int gen);
// Launches the bias-table and scorer kernels; *n_partials receives the number
// of partial-score rows written (to be summed in order by the consumer).
// With a stream-K area (sk non-NULL, as inside the fused block) the pair-MMA
// scorer may split tiles by K block like the FFN GEMMs.
cudaError_t launch_score(const ScoreArgs& a, const ScoreWorkspace& ws, const StreamKArea* sk, int n_sm,
                         cudaStream_t stream, int* n_partials);
cudaError_t launch_score_reduce(const float* partial, int n_chunks, size_t total, float* logits, float* probs,
                                int n_sm, cudaStream_t stream);

// ------------------------------------------------------------------ S2 select
struct TopkArgs {
  const float* src;      // logits [B*N] (n_chunks == 1) or scorer partial sums [n_chunks][B*N]
  int n_chunks;
  size_t chunk_stride;
  int B, N, r0, r1, K;
  float* logits_out;     // nullable
  float* probs_out;      // nullable
  int32_t* idx;          // [B][k_tot]
  uint8_t* mask;         // nullable
  int* status;
  int chunk;             // tokens per CTA of a sequence's cluster (set by launch_topk)
  int vec4;              // the partial rows may be read as float4 (set by launch_topk)
};
constexpr int kTopkMaxN = 49152;
cudaError_t launch_topk(const TopkArgs& a, cudaStream_t stream);

// ------------------------------------------------------------------ S3 / S5 rows
cudaError_t launch_gather(const __nv_bfloat16* h, int B, int N, int d, const int32_t* idx, int k_tot,
                          __nv_bfloat16* X, int* status, int n_sm, cudaStream_t stream);
cudaError_t launch_scatter_add(__nv_bfloat16* h, int B, int N, int d, const int32_t* idx, int k_tot,
                               const __nv_bfloat16* Y, int* status, int n_sm, cudaStream_t stream);
// The validating scatter-add: a sequence whose index list holds an entry out
// of [0, N) or a repeated entry records CER_ERR_INDEX and is left unwritten.
// N <= kScatterCheckedMaxN (its bitmap lives in shared memory).
constexpr int kScatterCheckedMaxN = 393216;
cudaError_t launch_scatter_add_checked(__nv_bfloat16* h, int B, int N, int d, const int32_t* idx, int k_tot,
                                       const __nv_bfloat16* Y, int* status, cudaStream_t stream);

// ------------------------------------------------------------------ S4 FFN
struct FfnArgs {
  const __nv_bfloat16* X;     // packed kept rows [M, d]
  int M, d, C;
  const __nv_bfloat16* Wg;    // kept-channel slices [C, d]
  const __nv_bfloat16* Wu;
  const __nv_bfloat16* WdT;
  __nv_bfloat16* act;         // workspace [M, C]
  // Output: Y [M, d] (scatter == 0) or out[b, idx] = bf16(h + y) (scatter == 1).
  __nv_bfloat16* Y;
  const __nv_bfloat16* h;
  __nv_bfloat16* out;
  const int32_t* idx;
  int N, k_tot;
  int scatter;
  // UCS FFN gate (Sec. 3.4, Eq. 8/9): gate/up also writes column sums of
  // |act| (colsum [2 * ceil(M/128)][C], optional); the down GEMM contracts
  // only the first C_small channels when *use_small_k is set (optional).
  float* colsum;
  const uint8_t* use_small_k;
  int C_small;
  StreamKArea sk;   // optional
  // Rotary embedding fused into a plain-output down GEMM (the attention
  // sublayer's QKV projection): with rope_cs != NULL, output columns of heads
  // [0, rope_heads) (128 columns each) are rotated, pair (j, j + 64) by the
  // angle of row m whose (cos, sin) is rope_cs[m * 64 + j].
  const float2* rope_cs;
  int rope_heads;
  int* status;
};
cudaError_t launch_ffn_gateup(const FfnArgs& a, int n_sm, cudaStream_t stream);
cudaError_t launch_ffn_down(const FfnArgs& a, int n_sm, cudaStream_t stream);

// ------------------------------------------------------------------ UCS FFN gate
// saliency s_c = (sum_parts colsum[part][c] / M) * norm_c; leakage =
// sum_{c >= C_keep} s_c / sum_c s_c; *use_pruned = leakage <= delta.
// part_ws holds 2 * ceil(I / 256) floats.
cudaError_t launch_ffn_gate(const float* colsum, int n_parts, int M, int I, int C_keep, const float* norms,
                            float delta, float* saliency, float* part_ws, float* leakage, uint8_t* use_pruned,
                            cudaStream_t stream);
cudaError_t launch_row_norms(const __nv_bfloat16* W, int rows, int d, float* norms, int n_sm, cudaStream_t stream);

// ------------------------------------------------------------------ UCS statistics
cudaError_t launch_drop_stats(const uint8_t* mask_t, const uint8_t* mask_ref, int B, int N, int r0, int r1,
                              float* jac, float* jrand, float* rda, int32_t* counts, cudaStream_t stream);
cudaError_t launch_redundancy_gap(const __nv_bfloat16* h_in, const __nv_bfloat16* h_out, const uint8_t* mask,
                                  int B, int N, int d, float delta, float* gap, uint8_t* skip, float* cos_ws,
                                  int n_sm, cudaStream_t stream);

// ------------------------------------------------------------------ attention on the packed sequence
// qkv: bf16 [B * L, (Hq + 2 Hkv) * 128]; each row holds the token's Hq query
// heads, then Hkv key heads, then Hkv value heads (head size 128).
constexpr int kHeadDim = 128;

// Frequencies of the rotary embedding divided by 2*pi, in fp64:
// g[j] = base^(-2j/128) / (2*pi), j < 64 (computed on the host).
struct RopeFreqTable {
  double g[kHeadDim / 2];
};

// Rotates the query and key heads of every packed row in place at the row's
// original position pos[row] (the keep list, [B * L]).
cudaError_t launch_rope(__nv_bfloat16* qkv, long long rows, int Hq, int Hkv, const int32_t* pos,
                        const RopeFreqTable& ft, int* status, int n_sm, cudaStream_t stream);
// The row gather (S3) that also writes, for every packed row m, the rotary
// (cos, sin) of its position idx[m] for the 64 frequencies: cs [M][64], the
// same arithmetic as the rotary-embedding kernel.
cudaError_t launch_gather_rope(const __nv_bfloat16* h, int B, int N, int d, const int32_t* idx, int k_tot,
                               __nv_bfloat16* X, float2* cs, const RopeFreqTable& ft, int* status, int n_sm,
                               cudaStream_t stream);

// out [B * L, Hq * 128] = softmax(Q K^T / sqrt(128)) V per sequence and query
// head over the packed tokens (causal: key index <= query index).
cudaError_t launch_packed_attention(const __nv_bfloat16* qkv, int B, int L, int Hq, int Hkv, int causal,
                                    __nv_bfloat16* out, int* status, int n_sm, cudaStream_t stream);

}  // namespace cer
