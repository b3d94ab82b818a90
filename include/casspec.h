/*
 * casspec.h -- C ABI of the CAS-Spec token-tree decode step for NVIDIA GB300 (sm_103a).
 *
 * CAS-Spec (arXiv 2510.26843) drafts with "virtual" draft models derived from the target model
 * itself by dynamically switchable inference acceleration (DSIA, Sec. 4.1, Def. 4.1) and verifies
 * token trees with tree attention (Sec. 4.2).  Every draft and verify pass is the same operation:
 * one forward of a Llama-style decoder over n tree nodes (1 <= n <= 64) against a prefix KV cache,
 * optionally with some layers switched off (layer-sparsity DSIA) or with W8A8 GEMMs
 * (activation-quantisation DSIA, App. C).  After the target's pass, the longest root-to-node path
 * that greedy decoding would have produced is accepted (lossless, Sec. 5.1) and its K/V entries are
 * moved into the committed cache.  This library implements exactly that hot path.
 *
 * Conventions shared by every entry point
 *  - Pointers marked "dev" are device pointers on the current CUDA device; "host" are host
 *    pointers.  The library allocates no device memory: model weights, the KV cache and all
 *    scratch live in caller-provided buffers sized by the *_bytes() queries.  It keeps only small
 *    host handles and never retains tokens / parent_idx / output pointers after a call returns.
 *  - Work is enqueued asynchronously on the model's stream (casspec_set_stream; default: the legacy
 *    default stream).  Only casspec_kv_length and casspec_get_status synchronise it.
 *  - Return value: CASSPEC_OK or a negative casspec_status.  Argument errors are reported
 *    synchronously and enqueue nothing.  Errors detected on the device (invalid parent_idx, an
 *    inconsistent accepted path, an expired bounded wait) are written to a device status word (the
 *    first error wins) and read with casspec_get_status; nothing traps.
 *  - bf16 tensors are passed as uint16_t bit patterns; matrices are row-major.  A weight W of a
 *    linear layer is [out][in] and the layer computes y = x * W^T.
 */
#ifndef CASSPEC_H
#define CASSPEC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Entry points are the library's only exported symbols. */
#define CASSPEC_API __attribute__((visibility("default")))

#define CASSPEC_MAX_TREE 64 /* tree slots per round; also the largest n of one call */
#define CASSPEC_SKIP_ATTN 0x2u /* skip-mask flag: the layer's attention block is skipped */
#define CASSPEC_SKIP_FFN 0x4u  /* skip-mask flag: the layer's FFN block is skipped */

typedef enum casspec_status {
  CASSPEC_OK = 0,
  CASSPEC_E_INVAL = -1,    /* NULL pointer, bad enum value, inconsistent configuration */
  CASSPEC_E_SHAPE = -2,    /* a size outside the supported range */
  CASSPEC_E_CAPACITY = -3, /* tree or KV capacity exceeded, or a caller buffer too small */
  CASSPEC_E_CUDA = -4,     /* a CUDA runtime call failed (including a failed launch) */
  CASSPEC_E_TREE = -5,     /* device: parent_idx invalid, or accepted path inconsistent */
  CASSPEC_E_TIMEOUT = -6,  /* device: a bounded wait inside a kernel expired */
  CASSPEC_E_STATE = -7     /* call-order rule violated (e.g. a layer's tree K/V missing) */
} casspec_status;

/* Model shape.  Requirements: d_model = n_heads * head_dim; head_dim in {64, 128};
 * d_model % 128 == 0, d_model <= 16384; ffn % 16 == 0, ffn <= 65536; vocab % 8 == 0,
 * vocab <= 131072; 1 <= n_layers <= 256.  casspec_create_model further returns CASSPEC_E_SHAPE
 * when the projection chain cannot hold the model on this GPU: a CTA's slice of any projection
 * (rows / number of SMs, in 16-row groups; gate and up count twice) must stay within 224 rows, and a
 * projection's input width within 256 blocks of 64 columns (d_model, ffn <= 16384).  On 152 SMs that
 * is 3 * d_model, 2 * ffn and vocab <= 34048 (up to rounding to 16-row groups). */
typedef struct casspec_model_config {
  int32_t n_layers;
  int32_t d_model;
  int32_t n_heads;
  int32_t head_dim;
  int32_t ffn;       /* SwiGLU hidden size F */
  int32_t vocab;
  float rope_base;   /* rotary base (10000 for Llama-2) */
  float rms_eps;     /* RMSNorm epsilon (1e-5 for Llama-2) */
  int32_t with_int8; /* nonzero: reserve int8 weights + scales so quant_mode 1 can run */
} casspec_model_config;

typedef struct casspec_model casspec_model; /* opaque host handle */
typedef struct casspec_kv casspec_kv;       /* opaque host handle */

/* Weight tensors (casspec_tensor).  Shapes for d = d_model, F = ffn, V = vocab:
 *   EMBED [V][d] bf16, LM_HEAD [V][d] bf16, FINAL_NORM [d] fp32       (layer ignored)
 *   ATTN_NORM [d] fp32, FFN_NORM [d] fp32 (RMSNorm gains)
 *   WQKV [3d][d] bf16 (rows: Wq, then Wk, then Wv), WO [d][d], WG [F][d], WU [F][d], WD [d][F] bf16
 * The int8 copies (written by casspec_quantize_weights) are WQKV_Q .. WD_Q int8 with the same
 * shapes and WQKV_S .. WD_S fp32 per-output-row scales.  The int4 copies (W4A4, same call) are
 * WQKV_Q4 .. WD_Q4 with rows of K / 2 bytes (column 2j in the low nibble of byte j, two's
 * complement codes in [-7, 7]) and WQKV_S4 .. WD_S4 fp32 scales (amax / 7); WQKV_F8 .. WD_F8 hold
 * the same codes as one FP8 e4m3 byte each (the tensor-core W4A4 path).
 * Step state (read-only views of the model's scratch, valid until the next step on the model; layer
 * ignored; for tests and for callers that want the hidden state):
 *   RESIDUAL [64][d] fp32: the residual stream after the step's last active layer (before the final
 *     RMSNorm), rows 0 .. n-1 valid;
 *   ACT_Q [64][K] int8 and ACT_S [64] fp32: codes and per-token scales of the latest quantised
 *     projection input of a W8A8 or W4A4 step (the down projection's input, K = ffn, when the last
 *     active layer ran its FFN block). */
enum casspec_tensor_id {
  CASSPEC_T_EMBED = 0,
  CASSPEC_T_LM_HEAD = 1,
  CASSPEC_T_FINAL_NORM = 2,
  CASSPEC_T_ATTN_NORM = 3,
  CASSPEC_T_FFN_NORM = 4,
  CASSPEC_T_WQKV = 5,
  CASSPEC_T_WO = 6,
  CASSPEC_T_WG = 7,
  CASSPEC_T_WU = 8,
  CASSPEC_T_WD = 9,
  CASSPEC_T_WQKV_Q = 10,
  CASSPEC_T_WO_Q = 11,
  CASSPEC_T_WG_Q = 12,
  CASSPEC_T_WU_Q = 13,
  CASSPEC_T_WD_Q = 14,
  CASSPEC_T_WQKV_S = 15,
  CASSPEC_T_WO_S = 16,
  CASSPEC_T_WG_S = 17,
  CASSPEC_T_WU_S = 18,
  CASSPEC_T_WD_S = 19,
  CASSPEC_T_RESIDUAL = 20,
  CASSPEC_T_ACT_Q = 21,
  CASSPEC_T_ACT_S = 22,
  CASSPEC_T_WQKV_Q4 = 23,
  CASSPEC_T_WO_Q4 = 24,
  CASSPEC_T_WG_Q4 = 25,
  CASSPEC_T_WU_Q4 = 26,
  CASSPEC_T_WD_Q4 = 27,
  CASSPEC_T_WQKV_S4 = 28,
  CASSPEC_T_WO_S4 = 29,
  CASSPEC_T_WG_S4 = 30,
  CASSPEC_T_WU_S4 = 31,
  CASSPEC_T_WD_S4 = 32,
  CASSPEC_T_WQKV_F8 = 33,
  CASSPEC_T_WO_F8 = 34,
  CASSPEC_T_WG_F8 = 35,
  CASSPEC_T_WU_F8 = 36,
  CASSPEC_T_WD_F8 = 37
};

/* Option bits for casspec_set_options. */
#define CASSPEC_OPT_PDL 1u    /* programmatic dependent launch between the step's kernels (default on) */
#define CASSPEC_OPT_GRAPHS 2u /* replay a captured CUDA graph per (call shape, pointers) (default off) */
/* Test hook for the failure path (default off): while set, a bf16 tree step with two or more
 * projections in one chain launch makes that launch's second phase wait for an arrival that never
 * comes; the bounded wait expires (2 s), the step reports CASSPEC_E_TIMEOUT through
 * casspec_get_status, and the model stays usable once the bit is cleared.  Such steps run
 * eagerly (never captured into a graph). */
#define CASSPEC_OPT_TEST_STALL 4u
#define CASSPEC_OPT_W4_TC 8u /* quant_mode 2 on the tensor cores with e4m3 codes (default on); off: 4-bit
                                codes through the integer mma.sync path */
#define CASSPEC_OPT_W8_TC 16u /* quant_mode 1 on the tensor cores (default on): int8 codes widened to fp16
                                 in shared memory, exact int32 sums (App. C's W8A8); off: the integer
                                 mma.sync path.  Both give the same logits bit for bit. */

/* ---------------------------------------------------------------------------------------------
 * Model
 * ------------------------------------------------------------------------------------------- */

/* Bytes of device memory a model with `cfg` needs (weights, optional int8 copies, step scratch,
 * tensor-map-aligned).  Returns 0 if cfg is invalid. */
CASSPEC_API size_t casspec_model_bytes(const casspec_model_config* cfg);

/* Create a model in caller memory `dev_mem` (dev, >= casspec_model_bytes(cfg), 256-byte aligned).
 * Weights are not initialised: write them through casspec_tensor.  The caller keeps ownership of
 * dev_mem and must keep it alive until casspec_destroy_model.  Errors: E_INVAL, E_CAPACITY, E_CUDA. */
CASSPEC_API int casspec_create_model(const casspec_model_config* cfg, void* dev_mem, size_t bytes, casspec_model** out);

/* Release the host handle (and any captured graphs).  Does not free dev_mem. */
CASSPEC_API void casspec_destroy_model(casspec_model* m);

/* Stream on which all of the model's work is enqueued (a cudaStream_t; NULL = legacy default). */
CASSPEC_API int casspec_set_stream(casspec_model* m, void* cuda_stream);

/* Set option bits (CASSPEC_OPT_*); returns the previous bits in *old_flags if non-NULL. */
CASSPEC_API int casspec_set_options(casspec_model* m, unsigned flags, unsigned* old_flags);

/* Activation sparsity (App. C: the TEAL draft of the DSIA family), a model setting for every step.
 * With 0 < s < 1, before each of Wqkv, Wo, Wgate/Wup and Wdown every token's floor(s * K) inputs of
 * smallest magnitude (after RMSNorm) become 0; among equal magnitudes the lower index is kept.  A
 * bf16 step selects on the split activation's value (hi + lo); a quantised step (App. C's mixed
 * drafts, e.g. W4A4 with sparsity) selects on the bf16 activation it then quantises.  The
 * projections themselves stay dense, so a sparse step moves the same weight bytes as a dense one
 * (this is the draft's arithmetic, not its speed).  s = 0, the default, is the dense step.  Changing
 * s drops captured graphs.  Errors: CASSPEC_E_INVAL (null model, s outside [0, 1)). */
CASSPEC_API int casspec_set_act_sparsity(casspec_model* m, float s);

/* The sparsity rule of casspec_set_act_sparsity on a split activation x_split (dev, [128][ld] bf16:
 * hi plane rows 0..63, lo plane rows 64..127, value = hi + lo in fp32): rows 0..n-1, columns
 * 0..K-1, zeroed in both planes, in place, enqueued on `cuda_stream` (for tests and callers that
 * apply the rule themselves).  Errors: CASSPEC_E_INVAL (null pointer, s outside [0, 1)),
 * CASSPEC_E_SHAPE (n outside 1..64, K outside 1..16384, ld < K), CASSPEC_E_CUDA. */
CASSPEC_API int casspec_sparsify_rows(uint16_t* x_split, int ld, int n, int K, float s, void* cuda_stream);

/* Device address and size of weight tensor `tensor` (casspec_tensor_id) of `layer` (ignored for
 * the layer-independent tensors).  The caller writes weights there (e.g. cudaMemcpyAsync).
 * After writing the tensor maps stay valid: they are built once from these addresses.
 * Errors: E_INVAL (bad id / layer, int8 tensor of a model created without with_int8). */
CASSPEC_API int casspec_tensor(casspec_model* m, int tensor, int layer, void** dev_ptr, size_t* bytes);

/* Per-output-channel symmetric int8 copies of WQKV, WO, WG, WU, WD for every layer (App. C
 * activation-quantisation DSIA, W8A8 reading): for each row, a = max|w|, q = rint(w * (127/a))
 * with ties to even (fp32, IEEE division and multiply), clamped to +-127, scale = a / 127; a = 0
 * gives q = 0, scale 0.  Enqueued on the model stream.  Errors: E_INVAL (no int8 storage). */
CASSPEC_API int casspec_quantize_weights(casspec_model* m);

/* ---------------------------------------------------------------------------------------------
 * KV cache: one cache shared by the target and all its self-drafts (Sec. 2 and 4.1: self-
 * speculation keeps no separate draft cache).  Layout per layer: K then V, each
 * [n_heads][max_ctx][head_dim] bf16.  Slots [0, P) hold the committed prefix, slots
 * [P, P + T) hold the current token tree (T <= 64).
 * ------------------------------------------------------------------------------------------- */

/* Bytes for a cache of `max_ctx` slots (max_ctx is rounded up to a multiple of 64). */
CASSPEC_API size_t casspec_kv_bytes(const casspec_model_config* cfg, int max_ctx);

/* Create a cache for model m in caller memory `dev_mem` (dev, 256-byte aligned).  The memory is
 * zeroed on the model stream; P = T = 0.  Errors: E_INVAL, E_CAPACITY, E_CUDA. */
CASSPEC_API int casspec_kv_create(casspec_model* m, int max_ctx, void* dev_mem, size_t bytes, casspec_kv** out);
CASSPEC_API void casspec_kv_destroy(casspec_kv* kv);

/* K and V of `layer` (dev, [n_heads][ld_slots][head_dim] bf16) so a caller can install a prefix. */
CASSPEC_API int casspec_kv_layer(casspec_kv* kv, int layer, void** k_dev, void** v_dev, int* ld_slots);

/* Declare slots [0, P) committed in every layer and clear the tree (T = 0).  Enqueued. */
CASSPEC_API int casspec_kv_set_prefix(casspec_kv* kv, int P);

/* Discard the current tree (T = 0) without committing anything, e.g. before a verify pass that
 * re-runs the whole draft tree.  Host-side bookkeeping only. */
CASSPEC_API int casspec_kv_reset_tree(casspec_kv* kv);

/* Synchronise the model stream and return the committed length P and the tree length T. */
CASSPEC_API int casspec_kv_length(casspec_kv* kv, int* P_out, int* T_out);

/* ---------------------------------------------------------------------------------------------
 * The tree step (Sec. 4.2: tree attention for parallel drafting and parallel verification).
 * ------------------------------------------------------------------------------------------- */

/* One decoder forward over n new tree nodes appended at tree slots T .. T+n-1.
 *   tokens      dev int32 [n]   token id of each node (0 <= id < vocab; clamped if not)
 *   parent_idx  dev int32 [n]   tree slot of each node's parent, in [-1, T + i); -1 makes the node
 *                               a child of the last committed token (depth 0, position P).  A node
 *                               at depth t sits at position P + t and attends to the whole prefix
 *                               plus exactly its ancestors and itself.
 *   n           1 .. 64, T + n <= 64, P + T + n <= max_ctx
 *   skip_mask   host uint8 [n_layers] or NULL (all layers on); 0 switches layer l off: the layer
 *               is the identity on the residual stream and writes no K/V (layer-sparsity DSIA,
 *               Sec. 4.1).  A non-zero byte keeps the layer on except for the sub-blocks whose
 *               flag it carries (Sec. 4.1 also names attention / FFN sub-blocks as the unit):
 *               CASSPEC_SKIP_ATTN drops the attention block (no residual update, no K/V
 *               written), CASSPEC_SKIP_FFN the FFN block; both flags equal 0.  Other bits are
 *               ignored.
 *               Rule: every layer whose attention runs must hold K/V for all T existing tree
 *               slots (nested masks, as in a layer-sparsity cascade); otherwise E_STATE.
 *   quant_mode  0: bf16 weights, fp32 accumulation.  1: W8A8 GEMMs for WQKV, WO, WG/WU, WD with
 *               per-token dynamic int8 activations (activation-quantisation DSIA); attention, K/V
 *               and the LM head stay bf16.  2: the same with 4-bit weights and activations (W4A4,
 *               codes in [-7, 7]).  Modes 1 and 2 need casspec_quantize_weights first.
 *   logits_out  dev fp32 [n][vocab] or NULL.
 * The row argmax of the logits (ties to the lowest id) and the top-2 margin of every node are
 * always computed and kept in the model (casspec_argmax).  Invalid parent_idx values are reported
 * through the status word (E_TREE); the step still runs, treating such a node as a depth-0 node.
 * Errors (synchronous): E_INVAL, E_SHAPE, E_CAPACITY, E_STATE, E_CUDA. */
CASSPEC_API int casspec_tree_step(casspec_model* m, casspec_kv* kv, const int32_t* tokens, const int32_t* parent_idx,
                      int n, const uint8_t* skip_mask, int quant_mode, float* logits_out);

/* Device pointers to the argmax (int32 [64]) and top-2 margin (fp32 [64]) of the latest tree
 * step's nodes.  Valid until the next tree step on this model. */
CASSPEC_API int casspec_argmax(casspec_model* m, const int32_t** argmax_dev, const float** margin_dev);

/* Greedy lossless acceptance (Sec. 5.1) over a whole verified tree of n nodes.
 *   logits        dev fp32 [n][vocab] of the target's pass, or NULL to use the model's fused
 *                 argmax of its latest tree step (which must then have covered these n nodes).
 *   tokens, parent_idx  dev int32 [n]; node 0 must be the only root (parent -1) and
 *                 parent_idx[c] < c for c > 0 (else E_TREE on the status word, accepted L = 0).
 *   accepted_out  dev int32 [n + 2]: [0] = L (>= 1), [1 .. L] = node indices of the accepted path
 *                 root first, [L + 1] = bonus token (the target's argmax at the last accepted node).
 * A node matches when its parent matches and its token equals the parent's argmax (node 0 always
 * matches); the accepted node is the deepest match, the lowest index among equally deep ones. */
CASSPEC_API int casspec_accept_greedy(casspec_model* m, const float* logits, const int32_t* tokens, const int32_t* parent_idx,
                          int n, int32_t* accepted_out);

/* Move the K/V of the accepted path (accepted_out as written by casspec_accept_greedy, dev) from
 * tree slots to committed slots P .. P+L-1 in every layer, then P += L and T = 0.  All layers must
 * hold the tree's K/V (the verify pass ran with every layer on), else E_STATE.  A path that is
 * inconsistent with the current tree (L < 1, L > T, an index >= T, a first node other than the
 * root, slot 0, or a node whose parent is not the node before it) sets E_TREE on the status word
 * and leaves the cache unchanged. */
CASSPEC_API int casspec_kv_compact(casspec_kv* kv, const int32_t* accepted_out);

/* ---------------------------------------------------------------------------------------------
 * Tracing: per-kernel device time measured with CUDA events on the launch stream.
 * ------------------------------------------------------------------------------------------- */
enum casspec_kernel_kind {
  CASSPEC_K_QKV = 0,    /* QKV projection + rotary + K/V write */
  CASSPEC_K_ATTN = 1,   /* tree attention */
  CASSPEC_K_WO = 2,     /* output projection + residual */
  CASSPEC_K_GATEUP = 3, /* gate/up projection + SwiGLU */
  CASSPEC_K_DOWN = 4,   /* down projection + residual */
  CASSPEC_K_LMHEAD = 5, /* LM head + argmax partials */
  CASSPEC_K_OTHER = 6,  /* tree prep, embedding, RMSNorm, quantisation, argmax merge */
  CASSPEC_K_COUNT = 7
};

/* enable != 0: clear the records and bracket every kernel the model launches eagerly from now on
 * with a CUDA event pair (graph replays are not instrumented); enable == 0: stop recording. */
CASSPEC_API int casspec_profile(casspec_model* m, int enable);

/* Synchronise the model stream; total device time in ms and number of recorded launches of
 * kernel kind `kind` (casspec_kernel_kind) since profiling was enabled. */
CASSPEC_API int casspec_profile_read(casspec_model* m, int kind, double* total_ms, int* launches);

/* Number of kernels the model has enqueued so far: eager launches plus the kernels contained in
 * every replayed CUDA graph. */
CASSPEC_API int casspec_launch_count(casspec_model* m, uint64_t* count);

/* Synchronise the model stream; return and clear the device status word. */
CASSPEC_API int casspec_get_status(casspec_model* m, int* status_out);

CASSPEC_API const char* casspec_status_string(int status);

/* ---------------------------------------------------------------------------------------------
 * Stateless kernels of the step, exposed for composition and for per-kernel checks.  All run on
 * `cuda_stream`; scratch is caller-provided.
 * ------------------------------------------------------------------------------------------- */

/* Scratch bytes needed by casspec_linear_bf16 for an [N][K] weight and n tokens. */
CASSPEC_API size_t casspec_linear_workspace_bytes(int N, int K, int n);

/* Y[i][o] = sum_k X[i][k] * W[o][k] (fp32 accumulation on the tensor cores) for i < n, o < N.
 *   W dev bf16 [N][K], X dev bf16 [n][K] (row stride K), Y dev fp32 [n][ldy], ldy >= N.
 *   1 <= n <= 64, K % 8 == 0, N >= 1; W and X 16-byte aligned.
 *   N <= 130,944 (1023 tiles of 128 rows).
 *   workspace dev, >= casspec_linear_workspace_bytes(N, K, n) bytes; its first 4 KB must be zero
 *   before the first call and are left zero by every call that completes.  A call whose bounded
 *   device wait expired leaves CASSPEC_E_TIMEOUT in the int32 at byte offset 4092 of the workspace
 *   (its status word; Y is then incomplete) and the 4 KB must be zeroed again before the next call. */
CASSPEC_API int casspec_linear_bf16(const uint16_t* W, int N, int K, const uint16_t* X, int n, float* Y, int ldy,
                        void* workspace, size_t workspace_bytes, void* cuda_stream);

/* casspec_linear_bf16 without a caller workspace: the same projection (Y = X W^T, fp32 accumulation
 * on the tensor cores, same arguments and layout as casspec_linear_bf16), with its stream-K scratch
 * in a static device array of the library (8 MB + 4 KB per device).  The paper has no counterpart:
 * this is plumbing for callers that cannot allocate device memory at the call site.
 *   Allocates nothing.  The first call on a device looks up the scratch address (with that device
 *   current); make that first call before capturing any stream.  Every call clears the scratch's
 *   counter block on `cuda_stream` before its kernel, so nothing needs to be zeroed by the caller.
 *   The scratch is shared by all calls on a device: calls that overlap in time (other streams or
 *   threads) race on it and must be serialised by the caller.
 *   Returns CASSPEC_E_CAPACITY when ceil(N / 128) + min(ceil(N/128) * ceil(K/64), SM count) > 256
 *   (N up to 13,312 on a 152-SM GB300); other errors as casspec_linear_bf16.
 *   A bounded device wait of the kernel that expires leaves CASSPEC_E_TIMEOUT in the scratch's
 *   status word (Y is then incomplete); casspec_linear_bf16_static_status reads it. */
CASSPEC_API int casspec_linear_bf16_static(const uint16_t* W, int N, int K, const uint16_t* X, int n, float* Y, int ldy,
                               void* cuda_stream);
/* Status word of the latest casspec_linear_bf16_static call on the current device (0 or
 * CASSPEC_E_TIMEOUT): waits for cuda_stream, then copies the word to *status_out (no allocation).
 * Each call clears the word when it starts. */
CASSPEC_API int casspec_linear_bf16_static_status(void* cuda_stream, int* status_out);

/* RMSNorm of n rows (Llama pre-norm): y = x / sqrt(mean(x^2) + eps) * g, fp32 arithmetic.
 *   x dev fp32 [n][d]; g dev fp32 [d]; y_bf16 dev bf16 [n][d] (may be NULL if q is given).
 *   If q_out (dev int8 [n][d]) and s_out (dev fp32 [n]) are non-NULL, each bf16 output row is also
 *   quantised with the per-row int8 rule of casspec_quantize_weights (that rule, applied per token,
 *   is the activation quantisation of the W8A8 draft). */
CASSPEC_API int casspec_rmsnorm(const float* x, const float* g, int n, int d, float eps, uint16_t* y_bf16, int8_t* q_out,
                    float* s_out, void* cuda_stream);

/* Per-row int8 quantisation of bf16 rows x [n][d] -> q [n][d], s [n] (same rule). */
CASSPEC_API int casspec_quantize_rows(const uint16_t* x, int n, int d, int8_t* q_out, float* s_out, void* cuda_stream);
/* The same with codes in [-7, 7] (the W4A4 draft's activations, App. C): inv = 7 / amax, scale amax / 7,
 * q4_out (dev [n][d / 2] bytes) two codes per byte, column 2j in the low nibble of byte j.  d % 8 == 0. */
CASSPEC_API int casspec_quantize_rows4(const uint16_t* x, int n, int d, uint8_t* q4_out, float* s_out,
                                       void* cuda_stream);

/* ---------------------------------------------------------------------------------------------
 * Dynamic Tree Cascade scheduling (DyTC): host code, no GPU work; thread-compatible (one scheduler
 * per thread).  It decides which draft configuration drafts how many tokens below which node of the
 * draft tree; the caller runs those drafts with casspec_tree_step and verifies the tree.
 * ------------------------------------------------------------------------------------------- */

/* Expected walltime improvement factors under i.i.d. Bernoulli acceptance (Sec. 3):
 *   casspec_ewif_sd: T_SD = (1 - a^(k+1)) / ((1 - a)(c k + 1)), draft acceptance a, cost coefficient c
 *     (draft step time / target step time), draft length k;
 *   casspec_ewif_hc: horizontal cascade, d1 drafts k1 tokens then d2 drafts k2:
 *     [(1 - a1^(k1+1)) / (1 - a1) + a1^k1 a2 (1 - a2^k2) / (1 - a2)] / (1 + k1 c1 + k2 c2);
 *   casspec_ewif_vc: vertical cascade, n rounds of d2 drafting k tokens for d1:
 *     (1 - a phi(a)^n) / ((1 - a)(1 + n c1 + n k c2)), phi(x) = 1 + (x - 1)(1 - (a12 x)^(k+1)) / (1 - a12 x),
 *     a = acceptance of d1 by the target, a12 = acceptance of d2 by d1; phi^n is the n-th power.
 * Return NaN for out-of-range arguments (acceptance outside [0, 1], negative lengths; a = 1 for the
 * cascade forms). */
CASSPEC_API double casspec_ewif_sd(double alpha, double c, int k);
CASSPEC_API double casspec_ewif_hc(double a1, double c1, int k1, double a2, double c2, int k2);
CASSPEC_API double casspec_ewif_vc(double alpha, double alpha12, double c1, double c2, int n, int k);

/* The step objective of Eq. 5 (Sec. 4.2): T_s = (E_acc + a^k a_dn) / (c k + c_dn), with
 * E_acc = a (1 - a^k) / (1 - a) (= k at a = 1) and (a_dn, c_dn) the bottom draft's acceptance and cost
 * (its "least future speedup").  NaN where Algorithm 2 skips the pair (c k + c_dn ~ 0) or k < 1. */
CASSPEC_API double casspec_dytc_objective(double alpha, double c, int k, double alpha_dn, double c_dn);

/* The latency model behind the cost coefficients (Sec. 4.2: hardware-aware latency prediction by
 * Bayesian linear regression): latency = w0 + w1 x with x the bytes a step moves (its roofline is
 * linear in them), prior w ~ N(mu0, diag(sd0^2)) (mu0, sd0 host [2]), Gaussian noise of standard
 * deviation noise_sd, fitted to m measured steps (x, y host [m]; m = 0 returns the prior).  Writes the
 * posterior mean to w_out [2] and, if non-NULL, the posterior covariance to cov_out [2][2].  A draft's
 * cost coefficient is then (w0 + w1 x_draft) / (w0 + w1 x_target).  Errors: E_INVAL. */
CASSPEC_API int casspec_latency_fit(const double* x, const double* y, int m, const double* mu0, const double* sd0,
                                    double noise_sd, double* w_out, double* cov_out);

/* Algorithmic bytes of one tree step (the regressor of the latency model): for every layer whose
 * attention block runs (skip_mask as for casspec_tree_step, NULL = all on) its Wqkv and Wo, the prefix
 * K/V of P slots read and the n new K/V written; for every FFN block that runs its Wg, Wu and Wd; the
 * LM head read and the n rows of fp32 logits written.  Weights count 2 bytes in bf16 (quant_mode 0),
 * 1 byte plus 4 per output row in W8A8 (quant_mode 1), half a byte plus 4 per row in W4A4 (quant_mode
 * 2, the 4-bit codes).  Host only.  Returns -1 on bad arguments. */
CASSPEC_API double casspec_step_bytes(const casspec_model_config* cfg, const uint8_t* skip_mask, int quant_mode, int n,
                                      int P);

#define CASSPEC_DYTC_MAX_CFG 16
#define CASSPEC_TOPK_MAX 8 /* largest K of casspec_topk and of the DyTC tree */
typedef struct casspec_dytc casspec_dytc;
typedef struct {
  int n_cfg;        /* candidate draft configurations, 1..CASSPEC_DYTC_MAX_CFG */
  double alpha_dn;  /* bottom draft: acceptance rate ... */
  double c_dn;      /* ... and cost coefficient (0 = free: the stop rule never fires) */
  int k_max;        /* longest draft per expansion (Algorithm 1's k_max), 1..CASSPEC_MAX_TREE */
  double t_min;     /* stop when alpha_dn / c_dn * P_acc(leaf) < t_min (Sec. 4.2) */
  int m_max;        /* largest tree, root included, 1..CASSPEC_MAX_TREE */
  double lambda;    /* EMA weight of the previous estimate (the paper uses 0.7) */
  int window;       /* outcomes per configuration in the recent mean (the paper uses H = 20) */
  int topk;         /* Algorithm 1's K: candidates per drafted position, 1..CASSPEC_TOPK_MAX (1: a chain) */
  double p_tree;    /* Algorithm 1's P_tree: top-P mass of the kept candidates, (0, 1] */
} casspec_dytc_params;

/* Create a scheduler over n_cfg candidate configurations with initial acceptance estimates
 * alpha_init[n_cfg] (host, in [0, 1]; e.g. from a calibration run, App. D) and cost coefficients
 * cost[n_cfg] (host, >= 0).  Errors: E_INVAL for out-of-range parameters, E_CAPACITY. */
CASSPEC_API int casspec_dytc_create(const casspec_dytc_params* p, const double* alpha_init, const double* cost,
                                    casspec_dytc** out);
CASSPEC_API void casspec_dytc_destroy(casspec_dytc* s);
/* The parameters a scheduler was created with. */
CASSPEC_API int casspec_dytc_get_params(const casspec_dytc* s, casspec_dytc_params* out);
/* Replace a configuration's cost coefficient (e.g. from measured step times). */
CASSPEC_API int casspec_dytc_set_cost(casspec_dytc* s, int cfg, double cost);
/* The latency model fed by measured steps (Sec. 4.2, hardware-aware latency prediction).  Steps of
 * different arithmetic (bf16, W8A8, W4A4) do not share one bytes-to-time line -- the quantised
 * projections are limited by their integer or conversion work, not only by the bytes they stream --
 * so each class (CASSPEC_DYTC_MAX_CLASS of them; use the step's quant_mode) has its own regression:
 *   casspec_dytc_observe records one measured step of class cls (bytes it moved, microseconds; the
 *   scheduler keeps the most recent 512 per class);
 *   casspec_dytc_fit_costs fits casspec_latency_fit to each class's recorded steps (prior mu0, sd0,
 *   noise_sd; a class without steps keeps the prior) and sets every configuration's cost coefficient
 *   to its predicted latency over the target's, c = max(w0 + w1 cfg_bytes[i], 0) / (v0 + v1 target_bytes),
 *   with w the fit of the configuration's class cfg_class[i] and v that of class 0, the target's
 *   (cfg_class, cfg_bytes host [n_cfg]; bytes e.g. from casspec_step_bytes).  w_out (host
 *   [CASSPEC_DYTC_MAX_CLASS][2], may be NULL) receives every class's fitted w.  Errors: E_INVAL (bad
 *   arguments, a class out of range, a non-positive predicted target latency). */
#define CASSPEC_DYTC_MAX_CLASS 4
CASSPEC_API int casspec_dytc_observe(casspec_dytc* s, int cls, double bytes, double us);
CASSPEC_API int casspec_dytc_fit_costs(casspec_dytc* s, const int* cfg_class, const double* cfg_bytes,
                                       double target_bytes, const double* mu0, const double* sd0, double noise_sd,
                                       double* w_out);
/* Current acceptance estimate and cost coefficient of a configuration. */
CASSPEC_API int casspec_dytc_alpha(const casspec_dytc* s, int cfg, double* alpha_out);
CASSPEC_API int casspec_dytc_cost(const casspec_dytc* s, int cfg, double* cost_out);
/* Algorithm 2 (App. D) with the current estimates: the configuration and draft length k in
 * [1, k_max] maximising Eq. 5, first maximum on ties; *cfg_out = -1 and *k_out = 0 when no pair has
 * a positive objective.  *obj_out (may be NULL) receives the maximum. */
CASSPEC_API int casspec_dytc_best_config(const casspec_dytc* s, int* cfg_out, int* k_out, double* obj_out);
/* Acceptance bookkeeping (Sec. 4.2): record whether the first token that configuration cfg drafted
 * in this round was accepted (the last `window` outcomes are kept); at the end of a round,
 * casspec_dytc_end_step sets alpha <- lambda alpha + (1 - lambda) mean(outcomes) for every
 * configuration recorded since the previous end of round; the others keep their estimate (App. D). */
CASSPEC_API int casspec_dytc_record(casspec_dytc* s, int cfg, int accepted);
CASSPEC_API int casspec_dytc_end_step(casspec_dytc* s);
/* Algorithm 1 (Sec. 4.2), driven by the caller (one drafted token per position here; K candidates per
 * position with casspec_dytc_tree_begin / casspec_dytc_tree_add below):
 *   casspec_dytc_tree_reset: the tree holds the root (node 0: the last committed token), P_acc = 1;
 *   casspec_dytc_tree_plan: returns 1 with the active leaf of highest P_acc (lowest index on ties),
 *     the configuration and k of Algorithm 2; returns 0 (stop) when the tree holds m_max nodes, no
 *     leaf is active, alpha_dn / c_dn * P_acc(leaf) < t_min, or no configuration has a positive
 *     objective (that leaf is then deactivated);
 *   casspec_dytc_tree_extend: appends the k tokens drafted by cfg below `leaf` as a chain, each with
 *     P_acc = P_acc(parent) * alpha(cfg); the leaf and each new node that gets a child stop being
 *     active leaves.  Stops at m_max nodes; returns the number of nodes appended (or an error);
 *   casspec_dytc_tree_get: the tree in node order, arrays of m_max entries (any may be NULL):
 *     parent (-1 for the root), token (-1 for the root), cfg (-1 for the root), P_acc. */
CASSPEC_API int casspec_dytc_tree_reset(casspec_dytc* s);
CASSPEC_API int casspec_dytc_tree_plan(casspec_dytc* s, int* leaf_out, int* cfg_out, int* k_out);
CASSPEC_API int casspec_dytc_tree_extend(casspec_dytc* s, int leaf, int cfg, int k, const int32_t* tokens);
CASSPEC_API int casspec_dytc_tree_get(const casspec_dytc* s, int* n_out, int32_t* parent_out, int32_t* token_out,
                                      int32_t* cfg_out, double* p_acc_out);
/* Algorithm 1 with K candidates per drafted position and sibling-parallel drafting (Sec. 4.2):
 *   casspec_dytc_tree_begin: the branches of an expansion of `leaf` (planned by casspec_dytc_tree_plan):
 *     the leaf and, when `siblings` is non-zero and the leaf is not the root, every active sibling of
 *     the leaf (same parent) in node order; branches_out (host int32 [CASSPEC_MAX_TREE]), *nb_out their
 *     number.  A neural draft passes siblings = 1 and extends every branch in the same draft steps; a
 *     retrieval draft passes 0.
 *   casspec_dytc_tree_add: one drafted position below `node` (a branch's current node): tokens and
 *     probabilities (host [kc], rank order, kc in 1..CASSPEC_TOPK_MAX; e.g. casspec_topk of the draft's
 *     logits row of `node`) are normalised over the kc; candidates are kept in rank order, the first
 *     always and each further one while the normalised mass kept before it is below p_tree; each
 *     becomes a child of `node` with P_acc = P_acc(node) * alpha(cfg) * its normalised probability;
 *     `node` stops being an active leaf.  Returns the index of the top-1 child (the branch's next
 *     node), 0 when the tree already holds m_max nodes (nothing added), or an error.  Stops adding at
 *     m_max nodes.  With kc = 1 it appends one node with P_acc(node) * alpha(cfg), like tree_extend. */
CASSPEC_API int casspec_dytc_tree_begin(casspec_dytc* s, int leaf, int siblings, int32_t* branches_out, int* nb_out);
CASSPEC_API int casspec_dytc_tree_add(casspec_dytc* s, int node, int cfg, const int32_t* tokens, const float* probs,
                                      int kc);

/* Prompt-lookup bottom draft (PLD: the default bottom draft M_dn, Sec. 4.1; its match length is its
 * confidence, Sec. 4.2).  Over the history tokens (dev int32 [L], L >= 0), find the longest n in
 * [n_min, n_max] (1 <= n_min <= n_max <= 64) such that the last n tokens occurred earlier, ending at a
 * position p < L - 1; among those occurrences take the latest; draft the tokens x[p+1 .. p+k] (cut at
 * the history's end, k <= CASSPEC_MAX_TREE).  out (dev int32 [2 + k]) receives {n (0: no match),
 * drafted count, tokens...}.  One kernel on cuda_stream; the library's models are not involved.
 * Errors: E_INVAL (arguments), E_CUDA (launch). */
CASSPEC_API int casspec_pld_draft(const int32_t* tokens, int L, int n_min, int n_max, int k, int32_t* out,
                                  void* cuda_stream);

/* K-best candidates per row (Sec. 4.2, Algorithm 1: the top-K tokens of each drafted position; their
 * normalised probabilities rank the sibling candidates).  logits dev fp32 [n][V] (e.g. a tree step's
 * logits_out); for each row, idx_out (dev int32 [n][K]) receives the K largest logits' token ids in
 * descending order (lower id first on ties; -1 past V) and prob_out (dev fp32 [n][K]) their softmax
 * probabilities over the whole row.  1 <= K <= 8.  One kernel on cuda_stream.  Errors: E_INVAL, E_CUDA. */
CASSPEC_API int casspec_topk(const float* logits, int n, int V, int K, int32_t* idx_out, float* prob_out,
                             void* cuda_stream);

/* One holistic round of the vertical cascade VC(d_i, d_n) (Sec. 4.2; its draft length depends on how
 * many low-level tokens are accepted): d_n proposed proposals[j] (host) below a leaf, and d_i's greedy
 * choices are argmax[0] at the leaf and argmax[r] after the r-th proposal (host [j + 1]).  out (host
 * [j + 1]) receives the proposals d_i accepts, in order up to the first mismatch, then d_i's own next
 * token.  Returns their count (1 .. j + 1) or E_INVAL. */
CASSPEC_API int casspec_vc_accept(const int32_t* proposals, int j, const int32_t* argmax, int32_t* out);

/* A draft configuration (Sec. 4.1), one of:
 *   - a DSIA draft of the model: layer mask and GEMM mode as for casspec_tree_step (skip_mask host
 *     uint8 [n_layers], NULL = all layers on; quant_mode 0 bf16, 1 W8A8), pld_n_max = 0;
 *   - the prompt-lookup bottom draft: pld_n_max > 0, vc = 0 (casspec_pld_draft with n in
 *     [1, pld_n_max] over the committed history and the path to the leaf);
 *   - the vertical cascade VC(model draft, prompt lookup): pld_n_max > 0, vc != 0; the prompt lookup
 *     proposes up to k tokens below the leaf and the model draft checks them in one tree step
 *     (casspec_vc_accept).  Its acceptance estimate is that of the model draft's tokens (App. D). */
typedef struct {
  const uint8_t* skip_mask;
  int quant_mode;
  int pld_n_max;
  int vc;
} casspec_draft_cfg;

/* One round of DyTC speculative decoding (Sec. 4.2: Algorithm 1, then verification by the target).
 * Configuration i of scheduler s runs as cfgs[i].  root_token is the last generated token, not yet
 * in the cache (the previous round's bonus token); kv must hold a committed prefix with no tree (T = 0).
 *   K = 1 (the scheduler's topk): each expansion (leaf, cfg, k) that Algorithm 1 plans runs the chosen
 *   draft over root .. leaf as one chain and then once per further drafted token (greedy argmax), and
 *   appends the k tokens.
 *   K > 1 with a neural draft: the draft runs over root .. leaf plus the leaf's active siblings (the
 *   branches, casspec_dytc_tree_begin) in one tree step, then once per further position over the
 *   branches' top-1 children; at each position casspec_topk of each branch's logits row gives the
 *   candidates that casspec_dytc_tree_add keeps.  dev_logits (device fp32 [CASSPEC_MAX_TREE][vocab])
 *   receives the draft's logits; it may be NULL when K = 1.
 *   The target then verifies the whole tree (casspec_tree_step, all layers, bf16), the longest matching
 *   path is accepted (casspec_accept_greedy) and compacted into the cache (casspec_kv_compact).  For
 *   every branch of an expansion whose node was accepted, whether its top-1 child was accepted is
 *   recorded (the first drafted token's outcome), and the estimates are updated (casspec_dytc_end_step).
 *   A prompt-lookup configuration drafts from history (dev int32, the committed tokens, the last
 *   being root_token; hist_len entries, room for CASSPEC_MAX_TREE more, which the round overwrites);
 *   finding no earlier occurrence counts as a rejected first token and ends the drafting.  A vertical
 *   cascade configuration runs its model draft once over root .. leaf plus the lookup's proposals
 *   (none when nothing matches) and appends the tokens casspec_vc_accept gives.  history may be NULL
 *   when no configuration uses the prompt lookup.
 *   dev_work: device int32 [CASSPEC_DYTC_WORK] (caller-owned scratch).  out_tokens (host int32
 *   [CASSPEC_MAX_TREE]) receives the tokens this round commits after the root, the last being the
 *   bonus token (the next root); *n_out their count (>= 1); *n_drafted_out (may be NULL) the drafted
 *   nodes.  Synchronises the model's stream several times (it reads drafted tokens back).
 *   Errors: E_INVAL, E_STATE (kv holds a tree), E_TREE (device-reported), errors of the calls above. */
CASSPEC_API int casspec_dytc_round(casspec_dytc* s, casspec_model* m, casspec_kv* kv, const casspec_draft_cfg* cfgs,
                                   int32_t root_token, int32_t* history, int hist_len, int32_t* dev_work,
                                   float* dev_logits, int32_t* out_tokens, int* n_out, int* n_drafted_out);
#define CASSPEC_DYTC_WORK (24 * CASSPEC_MAX_TREE) /* int32 entries of casspec_dytc_round's dev_work */

#ifdef __cplusplus
}
#endif

#endif /* CASSPEC_H */
