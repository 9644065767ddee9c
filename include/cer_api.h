/*
 * cer_api.h -- C ABI of the GB300 (sm_103a) token-routed compacted block of
 * CE-Router (core-expansion routing): score every token, keep the top-K per
 * sequence, pack the kept rows, run a channel-pruned SwiGLU FFN on them and add
 * the result back into the residual stream; dropped tokens bypass unchanged.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * Memory.   Every tensor argument is DEVICE memory owned by the caller, dense
 *           row-major, on the device current when the call is made.  bf16
 *           tensors are passed as `const void*` (2-byte IEEE bfloat16), fp32 as
 *           float*, indices as int32_t*, masks as uint8_t*.  The library never
 *           allocates device memory: entry points that need scratch take a
 *           caller-supplied `workspace` of at least the size reported by the
 *           matching *_workspace_size() function (256-byte aligned).
 * Alignment. Every tensor pointer must be 16-byte aligned (CER_ERR_ALIGN).
 *           A pointer to a tensor with no elements may be NULL.
 * Streams.  Work is enqueued asynchronously on `stream` (0 = legacy default
 *           stream); a call returns before the GPU finishes.
 * Errors.   Argument checks run on the host before any launch: on failure
 *           nothing is enqueued, the status is returned and a message is
 *           available from cer_get_error() (per host thread).  Errors found
 *           by a kernel (a NaN routable logit, a bounded wait that gave up,
 *           an out-of-range index) are recorded in a per-device status word
 *           that cer_sync_status() reads and clears.  Nothing throws across
 *           the ABI.
 * Device.   The library holds sm_103a code only; a call on another device
 *           returns CER_ERR_DEVICE.
 *
 * Notation: B sequences of N tokens with hidden size d; routable range
 * [r0, r1) with N_r = r1 - r0 tokens (tokens outside it are always kept);
 * K routable tokens kept per sequence; k_tot = K + N - N_r kept per sequence;
 * M = B * k_tot packed rows; I full FFN intermediate width; C kept channels.
 */
#ifndef CER_API_H
#define CER_API_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum cer_status {
  CER_OK = 0,
  CER_ERR_NULL = 1,      /* a required pointer is NULL                                  */
  CER_ERR_SHAPE = 2,     /* a size is out of range or not a supported multiple          */
  CER_ERR_ALIGN = 3,     /* a tensor pointer is not 16-byte aligned                     */
  CER_ERR_RANGE = 4,     /* a count or index is out of range (K > N_r, r0 > r1, ...)    */
  CER_ERR_NAN = 5,       /* device: a routable logit was NaN                            */
  CER_ERR_DEVICE = 6,    /* not an sm_103 device, or a CUDA runtime error               */
  CER_ERR_TIMEOUT = 7,   /* device: a bounded wait inside a kernel gave up              */
  CER_ERR_LAUNCH = 8,    /* a kernel launch failed                                      */
  CER_ERR_WORKSPACE = 9, /* workspace NULL or smaller than *_workspace_size() reports   */
  CER_ERR_INDEX = 10     /* device: an index list entry was out of range                */
} cer_status;

typedef enum cer_task { CER_TASK_UND = 0, CER_TASK_GEN = 1 } cer_task;

/*
 * One token-wise scorer MLP with a scalar output (Sec. 3.2: the core scorer
 * c_l, or the M generation expansion scorers e_{l,m}, one per denoising
 * segment).  Score of a token h:  w2[m] . GELU(W1[m] h + b1[m] + U[m] emb(t)),
 * GELU with the exact Gaussian CDF; emb(t) the E-dim sinusoid
 * [cos(1000 t f_j), sin(1000 t f_j)], f_j = 10000^(-j/(E/2)), j < E/2.
 * Segment m(t) = min(n_segments-1, floor(t * n_segments)) (equal-width
 * progress segments).  The core has n_segments == 1 and no U.
 */
typedef struct cer_scorer {
  const void*  W1;        /* bf16 [n_segments][hidden][d]                                  */
  const float* b1;        /* fp32 [n_segments][hidden], or NULL for no bias                */
  const float* w2;        /* fp32 [n_segments][hidden]                                     */
  const void*  U;         /* bf16 [n_segments][hidden][emb_dim], or NULL (no time input)   */
  int hidden;             /* hidden width, a multiple of 64, <= 4096                       */
  int emb_dim;            /* even, <= 1024; ignored when U is NULL                         */
  int n_segments;         /* >= 1, <= 64                                                   */
} cer_scorer;

/* ------------------------------------------------------------------ S1 score
 * Routing logits of Eq. 4 (Sec. 3.2, core_expansion_formulation): l^U = c(h) for understanding,
 * l^G = c(h) + e_{m(t)}(h) for generation.
 *   h        bf16 [B, N, d]; d a multiple of 64, <= 16384
 *   core     the core scorer (n_segments must be 1, U must be NULL)
 *   exp      the expansion scorers; read only when task == CER_TASK_GEN
 *            (may be NULL for CER_TASK_UND); its hidden width may differ
 *   t        fp32 [B] denoising progress per sequence (read for CER_TASK_GEN)
 *   logits   fp32 [B, N] output
 *   probs    fp32 [B, N] output p = sigmoid(l) of Eq. 6, or NULL
 * Workspace: cer_score_workspace_size(B, N, core->hidden, exp hidden, task).
 * The GEMM runs on tcgen05 tensor cores (bf16 operands, fp32 accumulation);
 * bias, GELU and the w2 dot product are applied in fp32.                     */
cer_status cer_score(const void* h, int B, int N, int d,
                     const cer_scorer* core, const cer_scorer* exp,
                     const float* t, int task,
                     float* logits, float* probs,
                     void* workspace, size_t workspace_bytes, cudaStream_t stream);
size_t cer_score_workspace_size(int B, int N, int core_hidden, int exp_hidden, int task);

/* ------------------------------------------------------------------ S1 without allocation
 * cer_score_static: cer_score for callers that cannot allocate device memory
 * (a plug-in or custom-operator host that gives its operators no workspace
 * and forbids allocation after load, or a real-time loop whose memory budget
 * is fixed at start-up).  The paper has no counterpart: this is a deployment
 * convenience of this library.  Same arguments and results as cer_score, but
 * no workspace: the scratch lives in one static device array of 4 MiB
 * (4194304 bytes), present on every GPU that loads the library until the
 * process exits.  Sizes whose cer_score_workspace_size() exceeds 4 MiB are
 * rejected with CER_ERR_WORKSPACE before any work is enqueued.  The call
 * allocates nothing.  Its first call on a device looks up the array's device
 * address (with that device current), and so does the first call in a new
 * context of that device (after cudaDeviceReset, say); make that first call
 * before any stream capture.  All calls share the array: calls whose GPU work can
 * overlap (other streams, other host threads) race on it; calls on one
 * stream are safe.                                                          */
cer_status cer_score_static(const void* h, int B, int N, int d,
                            const cer_scorer* core, const cer_scorer* exp,
                            const float* t, int task,
                            float* logits, float* probs, cudaStream_t stream);

/* ------------------------------------------------------------------ S2 select
 * Keep set R of Eq. 6 (Sec. 3.4, router_inference_outputs) per sequence: the K tokens of [r0, r1) with
 * the largest logit (ranking logits equals ranking sigmoid(l), App. B.2), ties
 * to the lower token index, -0.0 equal to +0.0, -inf allowed; plus every
 * token outside [r0, r1).  Exact: integer radix select on order-preserving
 * keys of the fp32 bits.
 *   logits   fp32 [B, N]
 *   idx      int32 [B, k_tot] output, kept token indices in ascending order
 *   mask     uint8 [B, N] output (1 = kept), or NULL
 * A NaN logit inside [r0, r1) sets CER_ERR_NAN in the device status word (the
 * outputs are then unspecified).  N <= 49152.                                 */
cer_status cer_select_topk(const float* logits, int B, int N, int r0, int r1, int K,
                           int32_t* idx, uint8_t* mask, cudaStream_t stream);

/* ------------------------------------------------------------------ S3 gather
 * Token compaction (Sec. 3.4): X[b*k_tot + j, :] = h[b, idx[b, j], :].
 *   h bf16 [B, N, d] (d a multiple of 8), idx int32 [B, k_tot], X bf16 [B*k_tot, d].
 * An index outside [0, N) sets CER_ERR_INDEX and its row is left unwritten.   */
cer_status cer_gather(const void* h, int B, int N, int d, const int32_t* idx, int k_tot,
                      void* X, cudaStream_t stream);

/* ------------------------------------------------------------------ S4 FFN
 * Channel-pruned SwiGLU FFN on the packed rows (Sec. 3.4 FFN pruning; Qwen2.5
 * backbone of App. A.5):
 *   Y[m, :] = sum_{c in Cs} WdT[c, :] * SiLU(Wg[c] . X[m]) * (Wu[c] . X[m])
 *   X     bf16 [M, d], d a multiple of 64
 *   Wg,Wu bf16 [I, d]   gate and up projections, one row per channel
 *   WdT   bf16 [I, d]   down projection stored channel-major (row c is
 *                       W_down[:, c]), so that pruning is a row selection
 *   chan  int32 [C] kept channel indices in [0, I), or NULL: then the weight
 *         arrays hold exactly the C channels to use (C == I), e.g. the full
 *         FFN or slices made once by cer_pack_ffn_weights; C a multiple of 64
 *   Y     bf16 [M, d] output
 * Two tcgen05 GEMMs (bf16 operands, fp32 accumulation in TMEM) over dense
 * TMA tiles; with chan != NULL the kept weight rows are first copied into the
 * workspace (3*C*d*2 bytes moved twice per call).  The SwiGLU activation
 * passes through the workspace as bf16 [M, C]; for M > 0 the workspace also
 * holds 24 MiB + 8 KiB in which the two GEMMs split output tiles by
 * contraction block across SM pairs and add the fp32 partial sums.
 * Workspace: cer_routed_ffn_workspace_size(M, d, C, chan != NULL).         */
cer_status cer_routed_ffn(const void* X, int M, int d,
                          const void* Wg, const void* Wu, const void* WdT, int I,
                          const int32_t* chan, int C, void* Y,
                          void* workspace, size_t workspace_bytes, cudaStream_t stream);
size_t cer_routed_ffn_workspace_size(int M, int d, int C, int with_chan);

/* ------------------------------------------------------------------ weight slices
 * The static channel-pruning mask of Sec. 3.4 (FFN pruning; App. A.4: the
 * candidate mask is fixed per layer) applied once: copies the kept rows of
 * Wg, Wu and WdT (all bf16 [I, d], d a multiple of 8) into Wg_out, Wu_out,
 * WdT_out (bf16 [C, d]) in the order of chan (int32 [C], entries in [0, I)).
 * Passing the outputs with chan == NULL and I == C to cer_routed_ffn or
 * cer_routed_block runs the pruned FFN without per-call copies.           */
cer_status cer_pack_ffn_weights(const void* Wg, const void* Wu, const void* WdT, int I, int d,
                                const int32_t* chan, int C,
                                void* Wg_out, void* Wu_out, void* WdT_out, cudaStream_t stream);

/* ------------------------------------------------------------------ S5 scatter
 * Unpack (Sec. 3.4): h[b, idx[b, j], :] = bf16(h + Y[b*k_tot + j, :]) in place,
 * fp32 sum rounded to nearest even; rows not in idx are not touched.
 *   h bf16 [B, N, d] (d a multiple of 8), idx int32 [B, k_tot] without
 *   duplicates within a sequence, Y bf16 [B*k_tot, d].                        */
cer_status cer_scatter_add(void* h, int B, int N, int d, const int32_t* idx, int k_tot,
                           const void* Y, cudaStream_t stream);

/* cer_scatter_add_checked: the same unpack for index lists that may break
 * cer_scatter_add's precondition (no paper counterpart: a validation mode).
 * Each sequence's list is first checked on the device: an entry outside
 * [0, N) or an entry repeated within the sequence (two updates of one row
 * would race) sets CER_ERR_INDEX in the device status word, and then none of
 * that sequence's rows is written; valid sequences are updated exactly as by
 * cer_scatter_add.  One CTA per sequence, so slower than cer_scatter_add for
 * few sequences.  N <= 393216.                                              */
cer_status cer_scatter_add_checked(void* h, int B, int N, int d, const int32_t* idx, int k_tot,
                                   const void* Y, cudaStream_t stream);

/* ------------------------------------------------------------------ fused block
 * The whole routed block S1..S5 on one stream:
 *   scorer GEMM -> top-K (also reduces the scorer's partial sums) ->
 *   row gather of the kept tokens (and, with chan != NULL, of the kept
 *   weight rows) -> gate/up GEMM with the SwiGLU epilogue -> down GEMM whose
 *   epilogue adds into the kept rows of the output.
 *   h, out   bf16 [B, N, d]; out == h (or NULL) updates h in place and moves
 *            no bytes for dropped rows; otherwise out must not overlap h and
 *            dropped rows are copied (bypass)
 *   core, exp, t, task   as for cer_score
 *   r0, r1, K            as for cer_select_topk
 *   Wg, Wu, WdT, I, chan, C   as for cer_routed_ffn
 *   logits   fp32 [B, N] output, or NULL
 *   idx      int32 [B, k_tot] output, or NULL
 *   mask     uint8 [B, N] output, or NULL
 *   stage_events  NULL, or n_stage_events == 6 caller-created CUDA events
 *            recorded on `stream` at the start, after the scorer, after the
 *            top-K, after the row gather, after the gate/up GEMM and after
 *            the down GEMM (for per-stage timing).
 * Workspace: cer_routed_block_workspace_size(..., chan != NULL).           */
cer_status cer_routed_block(void* h, void* out, int B, int N, int d,
                            const cer_scorer* core, const cer_scorer* exp,
                            const float* t, int task, int r0, int r1, int K,
                            const void* Wg, const void* Wu, const void* WdT, int I,
                            const int32_t* chan, int C,
                            float* logits, int32_t* idx, uint8_t* mask,
                            void* workspace, size_t workspace_bytes,
                            cudaEvent_t* stage_events, int n_stage_events,
                            cudaStream_t stream);
size_t cer_routed_block_workspace_size(int B, int N, int d, int core_hidden, int exp_hidden,
                                       int task, int r0, int r1, int K, int C, int with_chan);

/* ------------------------------------------------------------------ UCS FFN gate
 * FFN pruning of Unified Computation Scheduling (Sec. 3.4 (2), Eq. 8 and
 * Eq. 9; App. A.4: delta_FFN = 0.150).  The static mask proposes a pruned
 * channel set P; per call, the saliency of every channel on the retained rows,
 *   s_c = mean_i |z_{i,c}| * ||W_down[:, c]||_2,
 * gives the leakage lambda = sum_{c in P} s_c / sum_c s_c, and the pruned FFN
 * runs only if lambda <= delta (else the full FFN).  The saliency needs the
 * activation of every channel, so the gate/up GEMM runs over all I channels;
 * the decision sets how many channels the down GEMM contracts -- on the
 * device, without a host round trip.  One decision per call, over every
 * retained row of the batch (one sequence per call gives the per-sample rule).
 *
 * Weights: Wg, Wu, WdT bf16 [I, d] holding all channels with the C_keep
 * kept channels first and the mask's pruned channels after (pack once with
 * cer_pack_ffn_weights and that permutation as chan); norms fp32 [I] the
 * W_down column norms in the same order (cer_ffn_channel_norms, once).
 * I and C_keep multiples of 64.  Outputs: saliency fp32 [I] or NULL, leakage
 * fp32 [1] or NULL, use_pruned uint8 [1] (1 = pruned FFN ran) or NULL.     */
cer_status cer_ffn_channel_norms(const void* WdT, int I, int d, float* norms, cudaStream_t stream);

cer_status cer_routed_ffn_gated(const void* X, int M, int d,
                                const void* Wg, const void* Wu, const void* WdT, int I, int C_keep,
                                const float* norms, float delta, void* Y,
                                float* saliency, float* leakage, uint8_t* use_pruned,
                                void* workspace, size_t workspace_bytes, cudaStream_t stream);
size_t cer_routed_ffn_gated_workspace_size(int M, int d, int I);

/* The fused block with the gate (arguments as for cer_routed_block and the
 * gated FFN above; stage event 4 follows the gate/up GEMM and the gate).   */
cer_status cer_routed_block_gated(void* h, void* out, int B, int N, int d,
                                  const cer_scorer* core, const cer_scorer* exp,
                                  const float* t, int task, int r0, int r1, int K,
                                  const void* Wg, const void* Wu, const void* WdT, int I, int C_keep,
                                  const float* norms, float delta,
                                  float* saliency, float* leakage, uint8_t* use_pruned,
                                  float* logits, int32_t* idx, uint8_t* mask,
                                  void* workspace, size_t workspace_bytes,
                                  cudaEvent_t* stage_events, int n_stage_events, cudaStream_t stream);
size_t cer_routed_block_gated_workspace_size(int B, int N, int d, int core_hidden, int exp_hidden,
                                             int task, int r0, int r1, int K, int I);

/* ------------------------------------------------------------------ UCS statistics
 * Signals of Unified Computation Scheduling (Sec. 3.4), computed from the
 * router's decisions.
 *
 * cer_drop_set_stats: drop-set similarity of two routing decisions per
 * sequence (Eq. 10 and Eq. 11; diffusion-head cache reuse compares t with the
 * last refresh, early exit compares adjacent steps).  D is the routable tokens
 * [r0, r1) a keep mask does not keep.
 *   mask_t, mask_ref  uint8 [B, N] keep masks (1 = kept), e.g. from
 *                     cer_select_topk or cer_routed_block
 *   jaccard  fp32 [B]  J = |D_t & D_ref| / |D_t | D_ref| (1 if both empty)
 *   j_rand   fp32 [B]  expected J of random drop sets of the same sizes among
 *                      the n = r1 - r0 routable tokens, taken as
 *                      E|A&B| / E|A|B| with E|A&B| = |A||B|/n; or NULL
 *   rda      fp32 [B]  (J - J_rand) / (1 - J_rand) (1 if J_rand = 1); or NULL
 *   counts   int32 [B, 3]  |D_t|, |D_ref|, |D_t & D_ref|; or NULL
 * The counts are exact; the ratios are formed in fp64 from them.            */
cer_status cer_drop_set_stats(const uint8_t* mask_t, const uint8_t* mask_ref, int B, int N, int r0, int r1,
                              float* jaccard, float* j_rand, float* rda, int32_t* counts,
                              cudaStream_t stream);

/* cer_redundancy_gap: layer-skipping statistic of Eq. 7 per sequence,
 * g = mean over all tokens of cos(h_in_i, h_out_i) minus the mean over the
 * retained tokens R (mask 1); skip[b] = (g <= delta), delta_LS = 0.0040 in
 * App. A.4.
 *   h_in, h_out  bf16 [B, N, d] (d a multiple of 8), the block's input and output
 *   mask         uint8 [B, N]
 *   gap          fp32 [B] output; skip uint8 [B] output or NULL
 * Cosines accumulate in fp32 per token (a zero-norm pair counts 1 if equal,
 * else 0); the means are fp32 fixed-order tree sums.  Empty R gives g = 0.
 * Workspace: cer_redundancy_gap_workspace_size(B, N).                      */
cer_status cer_redundancy_gap(const void* h_in, const void* h_out, const uint8_t* mask, int B, int N, int d,
                              float delta, float* gap, uint8_t* skip,
                              void* workspace, size_t workspace_bytes, cudaStream_t stream);
size_t cer_redundancy_gap_workspace_size(int B, int N);

/* ------------------------------------------------------------------ attention on the packed sequence
 * Sec. 3.4 (task-adaptive token compaction): attention, like the FFN, runs
 * only over the kept tokens of R, gathered into a compact sequence; in
 * understanding mode the keys and values of that compact sequence are the
 * reduced key-value cache later decoding steps read.  Backbone (App. A.5):
 * Qwen2.5, head size 128, grouped key/value heads, rotary embedding.
 *
 * Packed rows: qkv bf16 [B * L, (Hq + 2 Hkv) * 128] (device, 16-byte
 * aligned): per row the token's Hq query heads, then Hkv key heads, then Hkv
 * value heads, 128 values each; L = the packed length of every sequence (the
 * k_tot of cer_select_topk).  Requires Hq >= 1, Hkv >= 1, Hq % Hkv == 0.
 *
 * cer_rope_packed: rotary position embedding of the query and key heads, in
 * place, each packed row at its original position (a packed token keeps its
 * index in the full sequence).
 *   pos   int32 [B * L] device: the rows' original positions, e.g. the keep
 *         list of cer_select_topk; a negative position is reported as
 *         CER_ERR_INDEX by cer_sync_status and that row is left unrotated
 *   base  rotary base (1e6 for Qwen2.5): for j < 64 the pair (j, j + 64) of a
 *         head is rotated by pos * base^(-2j/128) (rotate-half pairing)
 * Angles are formed in fp64 turns and reduced exactly before an fp32 sine
 * and cosine; rotated values are rounded to bf16.
 *
 * cer_packed_attention: softmax attention over each packed sequence,
 *   out[b, i, h] = sum_j softmax_j(q_{b,i,h} . k_{b,j,g} / sqrt(128)) v_{b,j,g},
 *   g = h / (Hq / Hkv), over the packed tokens j of sequence b (j <= i when
 *   causal: the keep list is ascending, so this is the causal mask by
 *   original position).
 *   qkv   as above (rotated); not modified
 *   out   bf16 [B * L, Hq * 128] device
 * Q K^T accumulates in fp32 on the tensor cores; the softmax weights are
 * rounded to bf16 for their product with V (fp32 accumulation); out is the
 * normalised fp32 result rounded to bf16.                                    */
cer_status cer_rope_packed(void* qkv, int B, int L, int Hq, int Hkv, const int32_t* pos, double base,
                           cudaStream_t stream);
cer_status cer_packed_attention(const void* qkv, int B, int L, int Hq, int Hkv, int causal, void* out,
                                cudaStream_t stream);

/* cer_routed_attention: the attention sublayer on the packed sequence,
 *   X = h[b, idx[b, :]] (packed, [B * L, d]),
 *   qkv = X WqkvT, rotated at the original positions idx (as cer_rope_packed),
 *   A = cer_packed_attention(qkv),
 *   out[b, idx[b, j]] = bf16(h[b, idx[b, j]] + (A WoT)[b * L + j]); other rows
 *   bypass (bit-identical; copied when out != h).
 *   h      bf16 [B, N, d] device; out NULL or == h: in place
 *   idx    int32 [B, L] device: ascending keep list per sequence (e.g. from
 *          cer_select_topk); out-of-range entries are reported as
 *          CER_ERR_INDEX by cer_sync_status and their rows skipped
 *   WqkvT  bf16 [d, (Hq + 2 Hkv) * 128] device: the QKV projection stored
 *          input-major (column j of W_qkv's transpose per output feature)
 *   WoT    bf16 [Hq * 128, d] device: the output projection, input-major
 *   qkv    NULL, or bf16 [B * L, (Hq + 2 Hkv) * 128] device: receives the
 *          rotated packed rows; their key and value heads are the compressed
 *          KV cache of the sublayer
 * Requires d a multiple of 64 in [64, 16384] and the head conditions above.
 * The projections accumulate in fp32 on the tensor cores (tcgen05 pair
 * MMA) and round to bf16, like the FFN; the rotary embedding is applied to
 * the QKV projection's fp32 accumulator before that rounding (one rounding
 * instead of cer_rope_packed's two), with the same angles.
 * Workspace: cer_routed_attention_workspace_size(B, L, d, Hq, Hkv): the
 * packed rows, qkv, the attention output, the rows' rotary (cos, sin) and
 * the stream-K area.                                                       */
cer_status cer_routed_attention(void* h, void* out, int B, int N, int d, const int32_t* idx, int L,
                                const void* WqkvT, const void* WoT, int Hq, int Hkv, int causal, double base,
                                void* qkv, void* workspace, size_t workspace_bytes, cudaStream_t stream);
size_t cer_routed_attention_workspace_size(int B, int L, int d, int Hq, int Hkv);

/* ------------------------------------------------------------------ bounded-wait self-test
 * cer_selftest_bounded_wait: a check of this library's failure detection (no
 * paper counterpart).  Every wait inside its kernels (on an mbarrier phase or
 * on a flag another CTA publishes) gives up after a limit, records
 * CER_ERR_TIMEOUT in the device status word and unwinds.  This entry point
 * launches one single-thread kernel that waits the same way, with a limit of
 * limit_us microseconds (1 .. 100000), for
 *   kind 0: the device word *flag (8-byte aligned device memory) to equal
 *           token, polled with acquire loads;
 *   kind 1: an mbarrier phase in the kernel's shared memory, completed only
 *           if arrive != 0 (the thread then arrives on it before waiting);
 *           flag is not read.
 * When the wait runs out, the kernel records CER_ERR_TIMEOUT and returns with
 * nothing in flight, so the context stays usable: cer_sync_status then
 * returns CER_ERR_TIMEOUT and clears it.                                    */
cer_status cer_selftest_bounded_wait(int kind, const unsigned long long* flag, unsigned long long token,
                                     int arrive, int limit_us, cudaStream_t stream);

/* ------------------------------------------------------------------ status
 * cer_sync_status: synchronise `stream`, then return and clear the current
 * device's status word (the first kernel-detected error since the last call),
 * or CER_ERR_DEVICE if the synchronisation itself failed.
 * cer_get_error: message of the last failing call on this host thread.
 * cer_status_string: name of a status code.  cer_version: ABI version.     */
cer_status  cer_sync_status(cudaStream_t stream);
const char* cer_get_error(void);
const char* cer_status_string(cer_status s);
int         cer_version(void);

#ifdef __cplusplus
}
#endif
#endif /* CER_API_H */
