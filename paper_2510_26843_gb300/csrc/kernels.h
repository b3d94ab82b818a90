// Internal interface between the host runtime (api.cu) and the kernel translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace casspec {

// Epilogue applied to a finished 128-row x n tile of a projection (output rows = channels).
enum Epi : int {
  EPI_STORE = 0,   // y[i][o] = v                              (stateless linear)
  EPI_RESID = 1,   // y[i][o] += v                             (Wo, Wd: residual add in fp32)
  EPI_QKV = 2,     // rotary on q,k at tree positions; q -> q_out, k,v -> cache slots P+T+i
  EPI_GLU = 3,     // tile = 64 gate rows + 64 up rows: u_out = split(silu(g) * up)
  EPI_LMHEAD = 4,  // logits[i][o] = v (optional) + per-tile (max, argmax, 2nd max) per token
};

struct EpiParams {
  int n;        // valid tokens (columns)
  int N;        // output channels of the projection (for EPI_GLU: F)
  float* y;     // EPI_STORE / EPI_RESID: [n][ldy] fp32
  int ldy;
  // EPI_QKV
  uint16_t* q_out;      // [64][d] bf16
  uint16_t* kc;         // this layer's K cache [H][ctx][hd]
  uint16_t* vc;         // this layer's V cache
  int ctx, d, hd, T;
  const int* dP;        // device committed length P
  const int* pos;       // [n] position of each new node (P + depth)
  const float2* rope;   // [ctx][hd/2] (cos, sin) of p * base^(-2j/hd) for every position p
  float* ss_out;        // EPI_RESID (optional): [tiles][64] sum over the tile's columns of updated y^2
  uint16_t* xa_out;     // EPI_RESID (optional): split(y * g_next) as [128][ldy] bf16 (see below)
  const float* g_next;  // RMSNorm gains of the projection that reads xa_out
  // EPI_GLU
  uint16_t* u_out;      // split(silu(g) * up) as [128][N] bf16
  // A "split" activation matrix holds fp32 values v as two bf16 planes, hi = bf16(v) in rows
  // 0..63 and lo = bf16(v - hi) in rows 64..127 (16 significant bits in all): the B operand of the
  // chained tensor-core projections, which multiply both planes with the same weights.
  // EPI_LMHEAD
  float* logits;        // [n][V] fp32 or null
  float* am_v1;         // [tiles][64] partial max
  int* am_i1;           // [tiles][64] partial argmax (vocab id)
  float* am_v2;         // [tiles][64] partial second max
};

struct GemmArgs {
  int tiles;     // 128-row output tiles
  int kblocks;   // ceil(K / 64)
  int w_blocked; // weights stored tile-blocked: box (t, k) is rows [(t * kblocks + k) * R, +R) of a 64-wide map
  float* partials;     // stream-K partial tiles, (tiles + grid) slots of 64 x 128 fp32
  unsigned* counters;  // [tiles], zero between launches
  int* status;
  EpiParams ep;
};

// int8 (W8A8) projection arguments
struct GemmI8Args {
  const int8_t* W;   // [N][K] int8, or with w4 [N][K / 2] bytes of two 4-bit codes (column 2j low nibble)
  const float* sw;   // [N]
  const int8_t* W2;  // EPI_GLU: up weights (gate in W)
  const float* sw2;
  const int8_t* X;   // [64][K] quantised activations
  const float* sx;   // [64]
  int N, K, ksplit;  // ksplit CTAs share one 128-row tile along K
  int tiles;
  int w4;            // weights are packed 4-bit codes (W4A4: activations are codes in [-7, 7] too)
  int* partials;     // [tiles][ksplit][64][128] int32
  unsigned* counters;
  int* status;
  EpiParams ep;
};

// exact W4A4 projection on the tensor cores (e4m3 codes in [-7, 7], fp32 accumulation is exact)
struct GemmF8Args {
  int tiles;     // 128-row output tiles (EPI_GLU: 64 gate + 64 up rows per tile)
  int kblocks;   // ceil(K / 128)
  int N;         // output channels (EPI_GLU: F)
  const float* sw;   // [N] weight scales (EPI_GLU: gate)
  const float* sw2;  // EPI_GLU: up weight scales
  const float* sx;   // [64] activation scales
  const uint8_t* wpk;  // the weight codes packed as 16 KB tile images (launch_pack_tiles8), or null:
                       // then read through the tensor maps
  float* partials;     // stream-K partial tiles, (tiles + grid) slots of 64 x 128 fp32
  unsigned* counters;  // [tiles], zero between launches
  int* status;
  EpiParams ep;
};

constexpr int kAttnMaxSplits = 8;  // the splits of a head form one thread-block cluster (portable size)
struct AttnArgs {
  const uint16_t* q;    // [64][d] bf16 (rotated)
  uint16_t* o;          // split attention output [128][d] bf16
  const unsigned long long* anc;  // [n] ancestor masks over tree slots
  const int* dP;
  int T, n, ctx, d, n_heads;
  int layer;            // K/V rows of this layer in the cache tensor map: ((layer * 2 + kv) * H + h) * ctx + slot
  int splits;           // CTAs per head (split-KV, one cluster), <= kAttnMaxSplits; n_heads * splits <= 2 * SMs
  float scale_log2;     // log2(e) / sqrt(hd)
  int* status;
};

// ---- the persistent projection chain (chain.cu) ----
// A projection of N output rows is split among the G CTAs of a launch by 16-row groups: CTA c owns
// groups [g0, g0 + ng) of the balanced split below (the first N/16 % G CTAs take one group more).
constexpr int kRowGroup = 16;
struct RowSlice {
  int g0, ng;
};
__host__ __device__ inline RowSlice row_slice(int c, int NG, int G) {
  const int base = NG / G, extra = NG % G;
  return RowSlice{c * base + (c < extra ? c : extra), base + (c < extra ? 1 : 0)};
}
// CTA that owns group g under row_slice
__host__ __device__ inline int row_slice_owner(int g, int NG, int G) {
  const int base = NG / G, extra = NG % G;
  return g < extra * (base + 1) ? g / (base + 1) : extra + (g - extra * (base + 1)) / (base > 0 ? base : 1);
}

// The part of a phase one CTA runs: rows [16 g0, 16 (g0 + ng)) of the output and the k-blocks
// klo + (rot + j) % len, j = 0 .. len-1, of the input (S = 1: all of K; S = 2: CTA pair c / 2 shares
// the rows, rank c % 2 takes one half of K).
struct PhasePart {
  int g0, ng, rank, klo, len, rot, slice;  // slice: index of the row slice (per-slice partials)
};
__host__ __device__ inline PhasePart phase_part(int c, int G, int NG, int kb, int S, int rot_groups) {
  PhasePart q;
  if (S == 2) {
    const int Gc = G / 2, cl = c / 2;
    const RowSlice s = row_slice(cl, NG, Gc);
    q.g0 = s.g0;
    q.ng = s.ng;
    q.rank = c & 1;
    q.klo = q.rank ? kb / 2 : 0;
    q.len = q.rank ? kb - kb / 2 : kb / 2;
    q.rot = q.len > 0 ? (cl * q.len) / Gc : 0;
    q.slice = cl;
  } else {
    const RowSlice s = row_slice(c, NG, G);
    q.g0 = s.g0;
    q.ng = s.ng;
    q.rank = 0;
    q.klo = 0;
    q.len = kb;
    q.rot = rot_groups > 0 ? (row_slice(c, rot_groups, G).g0 * kRowGroup / 64) % kb : 0;
    q.slice = c;
  }
  return q;
}

// How the rows of a projection's weights are packed (pack_rows_kernel).
enum PackKind : int {
  PACK_PLAIN = 0,  // rows in order
  PACK_GLU = 1,    // gate and up rows of the same channels in one slice (gate first)
  PACK_QKV = 2,    // [Wq; Wk; Wv] with each 16-row group holding 8 rotary pairs of one head
};

// One phase: Y = RMSNorm?(X) W^T with X the split activation of tensor map ChainMaps::x; when `ss` is
// set X holds x * g (gains applied by its producer) and each token's result is multiplied by
// rsqrt(sum(ss partials) / K + eps), which equals projecting RMSNorm(x) * g.
constexpr int kMaxPhases = 4;
constexpr int kReadyPerPhase = 256;  // readiness counters per phase (64-column blocks of its output)
struct ChainPhase {
  int epi;            // EPI_RESID, EPI_GLU, EPI_QKV or EPI_LMHEAD
  int N;              // output rows (EPI_GLU: F channels; the packed slice holds gate then up rows)
  int K, kb;          // input width and its 64-column blocks
  const uint8_t* wp;  // packed weights (pack_rows_kernel with this launch's G)
  int rot_groups;     // 16-row groups of the split that produced the input (the CTA's first k-block is
                      // the one holding its own slice of that split); must match the packing
  int in_phase;       // phase of this launch that produces the input, -1: an earlier kernel
  int in_N;           // output rows of that phase (the readiness targets)
  int publish;        // a later phase of this launch reads this phase's output
  int in_S;           // split factor of that phase (its rows are counted in once per split)
  int S;              // 1: the CTA's rows over all of K; 2 (EPI_RESID in a launch of CTA pairs): the
                      // pair's rows, each CTA one half of K, the halves summed through shared memory
  const float* ss;    // partial sums of squares [ss_parts][64] of the normalised input (null: none)
  int ss_parts;
  float eps;
  EpiParams ep;       // outputs; ss_out and the argmax partials are [slices][64], indexed by slice
};
struct ChainArgs {
  int nphases;
  int bn;              // token rows loaded per plane: n rounded up to 16
  ChainPhase ph[kMaxPhases];
  unsigned* ready;     // [kMaxPhases][kReadyPerPhase], zero between launches
  unsigned* done;      // [kMaxPhases + 1] CTAs finished per phase + exit counter, zero between launches
  int* status;
  int stall_phase;     // test hook: this phase's first readiness wait needs one row more than ever come (-1: off)
  int pairs;           // 1: launched as clusters of two CTAs (phases with S = 2 allowed)
};
struct ChainMaps {
  CUtensorMap x[kMaxPhases];  // split activations [128][K] bf16: 64 x bn boxes (bn = 64: 64 x 128, both planes)
};

// ---- launchers (return cudaSuccess or the launch error) ----
bool encode_tmap_bf16(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t rows, uint64_t row_stride_bytes,
                      uint32_t box_inner, uint32_t box_rows);
int gemm_bf16_grid(int tiles, int kblocks, int num_sms);
size_t gemm_partials_floats(int tiles, int grid);
cudaError_t launch_gemm_bf16(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int BN, int epi,
                             const GemmArgs& args, int grid, cudaStream_t stream, bool pdl);

bool encode_tmap_u8(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t rows, uint64_t row_stride_bytes,
                    uint32_t box_inner, uint32_t box_rows);
cudaError_t launch_gemm_f8(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int BN, int epi,
                           const GemmF8Args& args, int grid, cudaStream_t stream, bool pdl);
// W8A8 on the tensor cores: int8 weight and activation codes (the 128-byte-swizzled byte tiles of
// gemm_f8) widened to fp16 in shared memory; exact int32 sums, the same values as gemm_i8.
// Weight codes ([N][K] bytes, K a multiple of 16; EPI_GLU: gate and up) as contiguous 16 KB images of
// 128 x 128-code tiles with the 128-byte swizzle, in the order gemm_f8 / gemm_s8tc stream them.
size_t pack_tiles8_bytes(int N, int K, int glu);
cudaError_t launch_pack_tiles8(const uint8_t* src, const uint8_t* src2, int N, int K, int glu, uint8_t* dst,
                               cudaStream_t stream);
cudaError_t launch_gemm_s8tc(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int BN,
                             int epi, const GemmF8Args& args, int grid, cudaStream_t stream, bool pdl);

int gemm_i8_ksplit(int tiles, int K, int num_sms);
cudaError_t launch_gemm_i8(const GemmI8Args& args, int BN, int epi, cudaStream_t stream, bool pdl);

int attn_splits(int n_heads, int num_sms);
cudaError_t launch_tree_attention(const CUtensorMap& tmKV, const AttnArgs& a, int hd, cudaStream_t stream, bool pdl);

cudaError_t launch_tree_prep(const int* parent, int n, int T, const int* dP, int* tdepth, unsigned long long* tanc,
                             int* pos, unsigned long long* anc_new, int* status, cudaStream_t s, bool pdl);
cudaError_t launch_embed(const uint16_t* E, const int* tokens, int n, int d, int vocab, const float* g, float* x,
                         float* ss, uint16_t* xa, cudaStream_t s, bool pdl);
int chain_grid(int num_sms);
size_t chain_smem_bytes();
int chain_slice_rows(int N, int G, bool glu);
cudaError_t launch_chain(const ChainMaps& maps, const ChainArgs& args, int grid, cudaStream_t stream, bool pdl);
constexpr int kChainMaxSliceRows = 224;  // output rows (GLU: 2 x channels) of a CTA's slice: one k-block per weight stage
constexpr int kPairMaxRows = 80;  // rows of an S = 2 slice that the pair's exchange buffer holds
size_t pack_rows_bytes(int N, int K, int kind);
cudaError_t launch_pack_rows(const uint16_t* W, const uint16_t* W2, int N, int rows, int K, int G, int S, int kind,
                             int d, int hd, int rot_groups, uint8_t* out, cudaStream_t s);
int chain_pairs_fit(int grid);  // 1 if a launch of grid / 2 CTA pairs fits the GPU at once
// Quantised outputs: fmt 0 int8 codes, 1 (quant_rows only) two 4-bit codes per byte, 2 e4m3 bytes of
// codes in [-7, 7].
cudaError_t launch_rmsnorm(const float* x, const float* g, int n, int d, float eps, uint16_t* y, int8_t* q, float* sq,
                           cudaStream_t s, bool pdl, int qmax = 127, int fmt = 0);
// Activation sparsity of a split activation [128][ld] (hi rows 0..63, lo rows 64..127): in each of
// the n token rows the floor(s K) smallest-magnitude entries of hi + lo become 0 (ties: lower index kept).
// planes = 1: the magnitudes of the hi plane alone, and only the hi plane is written.
cudaError_t launch_sparsify(uint16_t* x, int ld, int n, int K, float s, cudaStream_t st, bool pdl, int planes = 2);
cudaError_t launch_quant_rows(const uint16_t* x, int n, int d, int ldx, int8_t* q, int ldq, float* sq, cudaStream_t s,
                              bool pdl, int qmax = 127, int fmt = 0);
cudaError_t launch_argmax_reduce(const float* v1, const int* i1, const float* v2, int tiles, int n, int* am,
                                 float* margin, cudaStream_t s, bool pdl);
cudaError_t launch_row_argmax(const float* logits, int n, int V, int* am, cudaStream_t s);
cudaError_t launch_accept(const int* am, const int* tokens, const int* parent, int n, int* acc, int* status,
                          cudaStream_t s);
cudaError_t launch_kv_compact(uint16_t* kv, int n_layers, int n_heads, int ctx, int hd, const int* acc,
                              const unsigned long long* tanc, int T, int* dP, unsigned* counter, int* status,
                              cudaStream_t s);
cudaError_t launch_set_int(int* p, int v, cudaStream_t s);

}  // namespace casspec
