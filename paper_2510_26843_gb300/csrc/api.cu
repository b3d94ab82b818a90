// Host runtime of the C ABI (include/casspec.h): model and KV-cache descriptors in caller memory,
// argument validation, the launch sequence of one tree step, and optional CUDA-graph replay.
#include <cmath>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <tuple>
#include <vector>

#include "kernels.h"
#include "../../include/casspec.h"

using namespace casspec;

namespace {

constexpr int kSmsBound = 256;  // scratch is sized for up to this many SMs
constexpr int kMaxTree = CASSPEC_MAX_TREE;

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

struct LayerPtrs {
  float *attn_norm, *ffn_norm;
  uint16_t *wqkv, *wo, *wg, *wu, *wd;
  int8_t *qkv_q, *wo_q, *wg_q, *wu_q, *wd_q;
  float *qkv_s, *wo_s, *wg_s, *wu_s, *wd_s;
  int8_t *qkv_q4, *wo_q4, *wg_q4, *wu_q4, *wd_q4;  // W4A4: two 4-bit codes per byte
  float *qkv_s4, *wo_s4, *wg_s4, *wu_s4, *wd_s4;
  uint8_t *qkv_f8, *wo_f8, *wg_f8, *wu_f8, *wd_f8;  // W4A4: the same codes as e4m3 bytes (tensor-core path)
  // the tensor-core paths' weight codes as contiguous 16 KB tile images (launch_pack_tiles8): W8A8 int8
  // codes (..._qp) and W4A4 e4m3 codes (..._fp); gate and up share one stream
  uint8_t *qkv_qp, *wo_qp, *wgu_qp, *wd_qp, *qkv_fp, *wo_fp, *wgu_fp, *wd_fp;
  CUtensorMap tm_qkv8, tm_o8, tm_g8, tm_u8, tm_d8;
  CUtensorMap tm_qkvq, tm_oq, tm_gq, tm_uq, tm_dq;  // W8A8 int8 codes as byte tiles (tensor-core path)
  CUtensorMap tm_qkv, tm_o, tm_g, tm_u, tm_d;
  uint8_t *wqkv_p, *wo_p, *wgu_p, *wd_p;  // the projections packed per CTA for the chain (pack_rows_kernel)
};

// Byte layout of a model's device memory (weights, int8 copies, step scratch).
struct Layout {
  size_t total = 0;
  size_t embed, lm_head, final_norm;
  std::vector<size_t> attn_norm, ffn_norm, wqkv, wo, wg, wu, wd;
  std::vector<size_t> qkv_q, wo_q, wg_q, wu_q, wd_q, qkv_s, wo_s, wg_s, wu_s, wd_s;
  std::vector<size_t> wqkv_p, wo_p, wgu_p, wd_p;
  size_t lm_p;
  std::vector<size_t> qkv_q4, wo_q4, wg_q4, wu_q4, wd_q4, qkv_s4, wo_s4, wg_s4, wu_s4, wd_s4;
  std::vector<size_t> qkv_f8, wo_f8, wg_f8, wu_f8, wd_f8;
  std::vector<size_t> qkv_qp, wo_qp, wgu_qp, wd_qp, qkv_fp, wo_fp, wgu_fp, wd_fp;
  size_t x, q, o, u, xa, xq, xs, ssp, pos, anc, am_v1, am_i1, am_v2, am, margin, am2;
  size_t gemm_part, gemm_cnt, chain_ready, chain_done, i8_part, i8_cnt, status;
  size_t scratch_begin;
  int max_tiles, lm_tiles;
};

bool config_ok(const casspec_model_config* c) {
  if (c == nullptr) return false;
  if (c->n_layers < 1 || c->n_layers > 256) return false;
  if (c->head_dim != 64 && c->head_dim != 128) return false;
  if (c->n_heads < 1 || c->d_model != c->n_heads * c->head_dim) return false;
  if (c->d_model % 128 != 0 || c->d_model > 16384) return false;
  if (c->ffn < 16 || c->ffn % 16 != 0 || c->ffn > 65536) return false;
  if (c->vocab < 16 || c->vocab % 8 != 0 || c->vocab > 131072) return false;
  if (!(c->rope_base > 0.f) || !(c->rms_eps >= 0.f)) return false;
  return true;
}

int cdiv(long long a, long long b) { return (int)((a + b - 1) / b); }
int roundup16(int n) { return (n + 15) / 16 * 16; }

Layout make_layout(const casspec_model_config& c) {
  Layout L;
  const size_t d = c.d_model, F = c.ffn, V = c.vocab, NL = c.n_layers;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    off = align_up(off, 256);
    size_t r = off;
    off += bytes;
    return r;
  };
  L.embed = take(V * d * 2);
  L.lm_head = take(V * d * 2);
  L.final_norm = take(d * 4);
  for (size_t l = 0; l < NL; ++l) {
    L.attn_norm.push_back(take(d * 4));
    L.ffn_norm.push_back(take(d * 4));
    L.wqkv.push_back(take(3 * d * d * 2));
    L.wo.push_back(take(d * d * 2));
    L.wg.push_back(take(F * d * 2));
    L.wu.push_back(take(F * d * 2));
    L.wd.push_back(take(d * F * 2));
  }
  // the bf16 projections once more, packed per CTA in the order the projection chain streams them
  // (the row-major tensors stay for filling, export, quantisation and the stand-alone GEMM)
  for (size_t l = 0; l < NL; ++l) {
    L.wqkv_p.push_back(take(pack_rows_bytes((int)(3 * d), (int)d, PACK_QKV)));
    L.wo_p.push_back(take(pack_rows_bytes((int)d, (int)d, PACK_PLAIN)));
    L.wgu_p.push_back(take(pack_rows_bytes((int)F, (int)d, PACK_GLU)));
    L.wd_p.push_back(take(pack_rows_bytes((int)d, (int)F, PACK_PLAIN)));
  }
  L.lm_p = take(pack_rows_bytes(roundup16((int)V), (int)d, PACK_PLAIN));
  if (c.with_int8) {
    for (size_t l = 0; l < NL; ++l) {
      L.qkv_q.push_back(take(3 * d * d));
      L.wo_q.push_back(take(d * d));
      L.wg_q.push_back(take(F * d));
      L.wu_q.push_back(take(F * d));
      L.wd_q.push_back(take(d * F));
      L.qkv_s.push_back(take(3 * d * 4));
      L.wo_s.push_back(take(d * 4));
      L.wg_s.push_back(take(F * 4));
      L.wu_s.push_back(take(F * 4));
      L.wd_s.push_back(take(d * 4));
      L.qkv_q4.push_back(take(3 * d * d / 2));
      L.wo_q4.push_back(take(d * d / 2));
      L.wg_q4.push_back(take(F * d / 2));
      L.wu_q4.push_back(take(F * d / 2));
      L.wd_q4.push_back(take(d * F / 2));
      L.qkv_s4.push_back(take(3 * d * 4));
      L.wo_s4.push_back(take(d * 4));
      L.wg_s4.push_back(take(F * 4));
      L.wu_s4.push_back(take(F * 4));
      L.wd_s4.push_back(take(d * 4));
      L.qkv_f8.push_back(take(3 * d * d));
      L.wo_f8.push_back(take(d * d));
      L.wg_f8.push_back(take(F * d));
      L.wu_f8.push_back(take(F * d));
      L.wd_f8.push_back(take(d * F));
      for (int f = 0; f < 2; ++f) {
        (f ? L.qkv_fp : L.qkv_qp).push_back(take(pack_tiles8_bytes((int)(3 * d), (int)d, 0)));
        (f ? L.wo_fp : L.wo_qp).push_back(take(pack_tiles8_bytes((int)d, (int)d, 0)));
        (f ? L.wgu_fp : L.wgu_qp).push_back(take(pack_tiles8_bytes((int)F, (int)d, 1)));
        (f ? L.wd_fp : L.wd_qp).push_back(take(pack_tiles8_bytes((int)d, (int)F, 0)));
      }
    }
  }
  L.scratch_begin = align_up(off, 256);
  const size_t T = kMaxTree;
  L.lm_tiles = cdiv(V, 128);
  L.max_tiles = std::max(std::max(cdiv(3 * d, 128), cdiv(F, 64)), L.lm_tiles);
  L.x = take(T * d * 4);
  L.q = take(T * d * 2);
  L.o = take(2 * T * d * 2);  // split activations: hi plane rows 0..63, lo plane rows 64..127
  L.u = take(2 * T * F * 2);
  L.xa = take(2 * T * d * 2);
  L.xq = take(T * std::max(d, F));
  L.xs = take(T * 4);
  L.ssp = take((size_t)std::max<size_t>(d / 128, kSmsBound) * T * 4);  // per-slice partial sums of squares
  L.pos = take(T * 4);
  L.anc = take(T * 8);
  L.am_v1 = take((size_t)kSmsBound * T * 4);  // per-slice LM-head (max, argmax, second max)
  L.am_i1 = take((size_t)kSmsBound * T * 4);
  L.am_v2 = take((size_t)kSmsBound * T * 4);
  L.am = take(T * 4);
  L.margin = take(T * 4);
  L.am2 = take(T * 4);
  L.gemm_part = take(gemm_partials_floats(L.max_tiles, kSmsBound) * 4);
  L.gemm_cnt = take((size_t)L.max_tiles * 4);
  L.chain_ready = take((size_t)kMaxPhases * kReadyPerPhase * 4);
  L.chain_done = take(256);
  {  // int32 partial tiles of the W8A8 projections: tiles x ksplit slots of 64 x 128
    const size_t kq = (size_t)(cdiv(d, 128) + 3) / 4, kf = (size_t)(cdiv(F, 128) + 3) / 4;
    const size_t slots = std::max(std::max((size_t)cdiv(3 * d, 128) * kq, (size_t)cdiv(F, 64) * kq),
                                  (size_t)cdiv(d, 128) * kf);
    L.i8_part = take(slots * 64 * 128 * 4);
  }
  L.i8_cnt = take((size_t)L.max_tiles * 4);
  L.status = take(256);
  L.total = align_up(off, 256);
  return L;
}

int num_sms_of_current_device() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return sms;
}

}  // namespace

struct GraphKey {
  const void* kv;
  const void* tokens;
  const void* parent;
  const void* logits;
  int n, T, mode;
  std::vector<uint8_t> mask;
  bool operator<(const GraphKey& o) const {
    return std::tie(kv, tokens, parent, logits, n, T, mode, mask) <
           std::tie(o.kv, o.tokens, o.parent, o.logits, o.n, o.T, o.mode, o.mask);
  }
};

struct casspec_model {
  casspec_model_config cfg;
  Layout lay;
  uint8_t* base = nullptr;
  cudaStream_t stream = nullptr;
  cudaStream_t cap_stream = nullptr;
  unsigned flags = CASSPEC_OPT_PDL | CASSPEC_OPT_W4_TC | CASSPEC_OPT_W8_TC;
  int num_sms = 0;
  uint16_t *embed, *lm_head;
  float* final_norm;
  std::vector<LayerPtrs> layers;
  CUtensorMap tm_lm;
  float *x, *ssp;
  uint16_t *q, *o, *u, *xa;       // o, u, xa: split activations [128][K] bf16 (hi, lo planes)
  // their 64 x BN boxes, BN = 16, 32, 48, 64, and [4]: 64 x 128 boxes (both planes of all 64 tokens
  // in one load, used when n > 48)
  CUtensorMap tm_o[5], tm_u[5], tm_xa[5];
  CUtensorMap tm_xq8_d[4], tm_xq8_f[4];    // activation codes (int8 or e4m3 bytes), rows of d or F, 128 x BN boxes
  int8_t* xq;
  float* xs;
  unsigned *chain_ready, *chain_done;
  uint8_t* lm_p = nullptr;   // the LM head packed for the chain
  int resid_split = 1;       // 2: the chain runs as CTA pairs and the residual projections split K in two
  float act_sparsity = 0.f;  // App. C activation sparsity of the bf16 steps (0: dense)
  bool pack_dirty = true;    // the row-major weights may have changed since the last packing
  bool pack8_dirty = true;   // the row-major W8A8 / W4A4 codes may have changed since their packing
  int* pos;
  unsigned long long* anc;
  float *am_v1, *am_v2, *margin;
  int *am_i1, *am, *am2;
  float* gemm_part;
  unsigned* gemm_cnt;
  int* i8_part;
  unsigned* i8_cnt;
  int* status;
  std::map<GraphKey, std::pair<cudaGraphExec_t, int>> graphs;  // exec + kernels it contains
  std::mutex mu;
  bool prof_on = false;
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> prof_ev[CASSPEC_K_COUNT];
  int prof_used[CASSPEC_K_COUNT] = {};
  uint64_t launches = 0;
};

struct casspec_kv {
  casspec_model* m;
  uint16_t* base;
  int ctx;
  int* dP;
  int* tdepth;
  unsigned long long* tanc;
  unsigned* compact_cnt;
  float2* rope;  // [ctx][hd/2] rotary (cos, sin) per position
  CUtensorMap tm_kv;  // the whole cache as [layers * 2 * heads * ctx][hd] bf16, 64 x 64 boxes
  int T = 0;
  long long P_upper = 0;
  std::vector<int> layer_valid;  // tree slots [0, layer_valid[l]) hold K/V of layer l
};

namespace {

size_t kv_region_bytes(const casspec_model_config& c, int ctx) {
  return (size_t)c.n_layers * 2 * c.n_heads * ctx * c.head_dim * 2;
}
int kv_ctx(int max_ctx) { return (max_ctx + 63) / 64 * 64; }
size_t kv_meta_bytes(const casspec_model_config& c, int ctx) {
  return 1024 + (size_t)ctx * (c.head_dim / 2) * 8;
}

uint16_t* kv_layer_k(casspec_kv* kv, int l) {
  const auto& c = kv->m->cfg;
  return kv->base + (size_t)l * 2 * c.n_heads * kv->ctx * c.head_dim;
}
uint16_t* kv_layer_v(casspec_kv* kv, int l) {
  const auto& c = kv->m->cfg;
  return kv_layer_k(kv, l) + (size_t)c.n_heads * kv->ctx * c.head_dim;
}

#define CK(call)                              \
  do {                                        \
    cudaError_t e_ = (call);                  \
    if (e_ != cudaSuccess) return CASSPEC_E_CUDA; \
  } while (0)

// Event pair bracketing one launch of `kind` while profiling (eager launches only).
cudaEvent_t prof_begin(casspec_model* m, int kind, cudaStream_t s) {
  auto& v = m->prof_ev[kind];
  int& used = m->prof_used[kind];
  if (used == (int)v.size()) {
    cudaEvent_t a, b;
    if (cudaEventCreate(&a) != cudaSuccess) return nullptr;
    if (cudaEventCreate(&b) != cudaSuccess) {
      cudaEventDestroy(a);
      return nullptr;
    }
    v.emplace_back(a, b);
  }
  cudaEventRecord(v[used].first, s);
  return v[used].second;
}

// Launch `call` (a cudaError_t expression) as one kernel of kind `kind`: count it, and bracket it
// with events when profiling an eager step.
#define LAUNCH(kind, call)                                                   \
  do {                                                                       \
    cudaEvent_t stop_ = prof ? prof_begin(m, (kind), s) : nullptr;            \
    const cudaError_t e_ = (call);                                           \
    if (e_ != cudaSuccess) return CASSPEC_E_CUDA;                            \
    if (stop_ != nullptr) {                                                  \
      cudaEventRecord(stop_, s);                                             \
      m->prof_used[(kind)]++;                                                \
    }                                                                        \
    ++count;                                                                 \
  } while (0)

// Refresh the chain's packed weight copies from the row-major tensors (on the model's stream).
int pack_weights(casspec_model* m, int& count) {
  const auto& c = m->cfg;
  const int d = c.d_model, F = c.ffn, V = c.vocab, hd = c.head_dim;
  const int G = chain_grid(m->num_sms);
  for (int l = 0; l < c.n_layers; ++l) {
    LayerPtrs& p = m->layers[l];
    const int Sr = m->resid_split;  // the residual projections' split (CTA pairs: 2)
    CK(launch_pack_rows(p.wqkv, nullptr, 3 * d, 3 * d, d, G, 1, PACK_QKV, d, hd, d / kRowGroup, p.wqkv_p, m->stream));
    CK(launch_pack_rows(p.wo, nullptr, d, d, d, G, Sr, PACK_PLAIN, d, hd, d / kRowGroup, p.wo_p, m->stream));
    CK(launch_pack_rows(p.wg, p.wu, F, F, d, G, 1, PACK_GLU, d, hd, d / kRowGroup, p.wgu_p, m->stream));
    CK(launch_pack_rows(p.wd, nullptr, d, d, F, G, Sr, PACK_PLAIN, d, hd, F / kRowGroup, p.wd_p, m->stream));
    count += 4;
  }
  CK(launch_pack_rows(m->lm_head, nullptr, roundup16(V), V, d, G, 1, PACK_PLAIN, d, hd, d / kRowGroup, m->lm_p,
                      m->stream));
  ++count;
  m->pack_dirty = false;
  return CASSPEC_OK;
}

// Refresh the tensor-core projections' tile images of the W8A8 int8 and W4A4 e4m3 codes.
int pack_codes(casspec_model* m, int& count) {
  const auto& c = m->cfg;
  const int d = c.d_model, F = c.ffn;
  for (int l = 0; l < c.n_layers; ++l) {
    LayerPtrs& p = m->layers[l];
    const uint8_t* q8[5] = {reinterpret_cast<uint8_t*>(p.qkv_q), reinterpret_cast<uint8_t*>(p.wo_q),
                            reinterpret_cast<uint8_t*>(p.wg_q), reinterpret_cast<uint8_t*>(p.wu_q),
                            reinterpret_cast<uint8_t*>(p.wd_q)};
    const uint8_t* f8[5] = {p.qkv_f8, p.wo_f8, p.wg_f8, p.wu_f8, p.wd_f8};
    for (int f = 0; f < 2; ++f) {
      const uint8_t* const* w = f ? f8 : q8;
      CK(launch_pack_tiles8(w[0], nullptr, 3 * d, d, 0, f ? p.qkv_fp : p.qkv_qp, m->stream));
      CK(launch_pack_tiles8(w[1], nullptr, d, d, 0, f ? p.wo_fp : p.wo_qp, m->stream));
      CK(launch_pack_tiles8(w[2], w[3], F, d, 1, f ? p.wgu_fp : p.wgu_qp, m->stream));
      CK(launch_pack_tiles8(w[4], nullptr, d, F, 0, f ? p.wd_fp : p.wd_qp, m->stream));
      count += 4;
    }
  }
  m->pack8_dirty = false;
  return CASSPEC_OK;
}

// Sub-blocks of a layer that a step runs (from a skip-mask byte).
constexpr uint8_t kBlockAttn = 1, kBlockFfn = 2;
uint8_t layer_blocks(uint8_t code) {
  if (code == 0) return 0;
  return (uint8_t)(((code & CASSPEC_SKIP_ATTN) ? 0 : kBlockAttn) | ((code & CASSPEC_SKIP_FFN) ? 0 : kBlockFfn));
}
// One projection or attention of a step (`l`: its layer, -1 for the LM head).
enum { IT_QKV, IT_ATTN, IT_WO, IT_GU, IT_DOWN, IT_LM };
struct StepItem {
  int kind, l;
};

// Enqueue one tree step on stream s (argument checks already done).  `count` receives the number
// of kernels enqueued; profiling events are recorded only when `prof` is set.
//   bf16 mode: tree prep -> embedding (+ row sums of squares) -> chain launches of consecutive
//   projections, each attention ending one (with every block on: chain[QKV of the first layer],
//   then per layer attention and chain[Wo, Wgate/Wup, Wdown, next layer's QKV or the LM head]) ->
//   argmax merge.  RMSNorm is folded into the chain phases that consume it.
//   int8 mode: per-projection W8A8 kernels with RMSNorm / quantisation kernels, then chain[LM head].
int enqueue_step(casspec_model* m, casspec_kv* kv, const int32_t* tokens, const int32_t* parent, int n,
                 const std::vector<uint8_t>& on, int mode, float* logits, cudaStream_t s, bool prof, int& count) {
  const auto& c = m->cfg;
  const int d = c.d_model, F = c.ffn, V = c.vocab, hd = c.head_dim, H = c.n_heads;
  const bool pdl = (m->flags & CASSPEC_OPT_PDL) != 0;
  const int BN = roundup16(n);
  const int T = kv->T;
  std::vector<int> act;
  for (int l = 0; l < c.n_layers; ++l)
    if (on[l]) act.push_back(l);
  // The step as a list of projections and attentions: per active layer QKV, attention and Wo when
  // its attention block is on, gate/up and down when its FFN block is on; the LM head last.
  // Every residual projection (Wo, down) is followed by a projection that reads x.
  std::vector<StepItem> items;
  for (int l : act) {
    if (on[l] & kBlockAttn) {
      items.push_back({IT_QKV, l});
      items.push_back({IT_ATTN, l});
      items.push_back({IT_WO, l});
    }
    if (on[l] & kBlockFfn) {
      items.push_back({IT_GU, l});
      items.push_back({IT_DOWN, l});
    }
  }
  items.push_back({IT_LM, -1});
  // gains of the RMSNorm that a projection reading x applies
  auto reader_gain = [&](const StepItem& it) -> const float* {
    return it.kind == IT_QKV ? m->layers[it.l].attn_norm : it.kind == IT_GU ? m->layers[it.l].ffn_norm : m->final_norm;
  };

  LAUNCH(CASSPEC_K_OTHER, launch_tree_prep(parent, n, T, kv->dP, kv->tdepth, kv->tanc, m->pos, m->anc, m->status, s,
                                           pdl));
  // the first projection that reads x normalises it with these gains (null: an int8 layer does)
  const float* g_first = (mode == 0 || act.empty()) ? reader_gain(items[0]) : nullptr;
  LAUNCH(CASSPEC_K_OTHER, launch_embed(m->embed, tokens, n, d, V, g_first, m->x, m->ssp, m->xa, s, pdl));
  const int bi = BN / 16 - 1;  // tensor maps of the split activations for this BN
  const int cx = BN == 64 ? 4 : bi;  // the chain loads both planes in one box at BN = 64

  EpiParams base = {};
  base.n = n;
  base.ctx = kv->ctx;
  base.d = d;
  base.hd = hd;
  base.T = T;
  base.dP = kv->dP;
  base.pos = m->pos;
  base.rope = kv->rope;

  // ---- phases of the projection chain ----
  const int G = chain_grid(m->num_sms);
  const int Sr = m->resid_split;
  const int resid_parts = std::min(d / kRowGroup, G / Sr);  // partial sums of squares a residual phase leaves
  auto ph_qkv = [&](int l, int ss_parts, ChainPhase& p, CUtensorMap& x) {
    p = ChainPhase{};
    p.epi = EPI_QKV;
    p.N = 3 * d;
    p.K = d;
    p.kb = cdiv(d, 64);
    p.wp = m->layers[l].wqkv_p;
    p.rot_groups = d / kRowGroup;
    p.ss = m->ssp;
    p.ss_parts = ss_parts;
    p.eps = c.rms_eps;
    p.ep = base;
    p.ep.N = 3 * d;
    p.ep.q_out = m->q;
    p.ep.kc = kv_layer_k(kv, l);
    p.ep.vc = kv_layer_v(kv, l);
    x = m->tm_xa[cx];
  };
  // residual projection; g_next: gains of the RMSNorm that the next projection applies to x
  auto ph_resid = [&](int K, const uint8_t* wp, int rot_groups, const float* g_next, ChainPhase& p) {
    p = ChainPhase{};
    p.epi = EPI_RESID;
    p.S = Sr;
    p.N = d;
    p.K = K;
    p.kb = cdiv(K, 64);
    p.wp = wp;
    p.rot_groups = rot_groups;
    p.ep = base;
    p.ep.N = d;
    p.ep.y = m->x;
    p.ep.ldy = d;
    p.ep.ss_out = m->ssp;
    p.ep.xa_out = m->xa;
    p.ep.g_next = g_next;
  };
  auto ph_gu = [&](int l, int ss_parts, ChainPhase& p) {
    p = ChainPhase{};
    p.epi = EPI_GLU;
    p.N = F;
    p.K = d;
    p.kb = cdiv(d, 64);
    p.wp = m->layers[l].wgu_p;
    p.rot_groups = d / kRowGroup;
    p.ss = m->ssp;
    p.ss_parts = ss_parts;
    p.eps = c.rms_eps;
    p.ep = base;
    p.ep.N = F;
    p.ep.u_out = m->u;
  };
  auto ph_lm = [&](int ss_parts, ChainPhase& p, CUtensorMap& x) {
    p = ChainPhase{};
    p.epi = EPI_LMHEAD;
    p.N = roundup16(V);
    p.K = d;
    p.kb = cdiv(d, 64);
    p.wp = m->lm_p;
    p.rot_groups = d / kRowGroup;
    p.ss = m->ssp;
    p.ss_parts = ss_parts;
    p.eps = c.rms_eps;
    p.ep = base;
    p.ep.N = V;
    p.ep.logits = logits;
    p.ep.am_v1 = m->am_v1;
    p.ep.am_i1 = m->am_i1;
    p.ep.am_v2 = m->am_v2;
    x = m->tm_xa[cx];
  };
  bool stall_pending = (m->flags & CASSPEC_OPT_TEST_STALL) != 0;
  auto chain = [&](ChainArgs& ca, ChainMaps& cm, int kind) -> int {
    ca.bn = BN;
    ca.ready = m->chain_ready;
    ca.done = m->chain_done;
    ca.status = m->status;
    ca.stall_phase = -1;
    ca.pairs = Sr == 2 ? 1 : 0;
    if (stall_pending && ca.nphases >= 2) {  // test hook: the first multi-phase launch of the step
      ca.stall_phase = 1;
      stall_pending = false;
    }
    for (int p = 0; p < ca.nphases; ++p) {  // consecutive phases feed each other
      if (ca.ph[p].S == 0) ca.ph[p].S = 1;
      ca.ph[p].in_phase = p - 1;
      ca.ph[p].in_N = p > 0 ? ca.ph[p - 1].N : 0;
      ca.ph[p].in_S = p > 0 ? ca.ph[p - 1].S : 1;
      ca.ph[p].publish = p + 1 < ca.nphases ? 1 : 0;
    }
    LAUNCH(kind, launch_chain(cm, ca, G, s, pdl));
    return CASSPEC_OK;
  };
  auto attention = [&](int l) -> int {
    AttnArgs at = {};
    at.q = m->q;
    at.o = m->o;
    at.anc = m->anc;
    at.dP = kv->dP;
    at.T = T;
    at.n = n;
    at.ctx = kv->ctx;
    at.d = d;
    at.n_heads = H;
    at.layer = l;
    at.splits = attn_splits(H, m->num_sms);
    at.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)hd));
    at.status = m->status;
    LAUNCH(CASSPEC_K_ATTN, launch_tree_attention(kv->tm_kv, at, hd, s, pdl));
    return CASSPEC_OK;
  };

  if (mode == 0) {
    // Consecutive projections share one chain launch (up to kMaxPhases phases); every attention
    // ends the current chain.  With all blocks on this gives [QKV], then [Wo, gate/up, down,
    // next QKV or LM head] after each attention.
    ChainArgs ca = {};
    ChainMaps cm = {};
    int nph = 0, nchains = 0;
    auto flush = [&]() -> int {
      if (nph == 0) return CASSPEC_OK;
      ca.nphases = nph;
      const int kind = (nph == 1 && ca.ph[0].epi == EPI_LMHEAD) ? CASSPEC_K_LMHEAD
                       : (nchains == 0 && ca.ph[0].epi == EPI_QKV) ? CASSPEC_K_QKV
                                                                   : CASSPEC_K_GATEUP;
      const int rc = chain(ca, cm, kind);
      ca = ChainArgs{};
      cm = ChainMaps{};
      nph = 0;
      ++nchains;
      return rc;
    };
    int rc;
    for (size_t i = 0; i < items.size(); ++i) {
      const StepItem& it = items[i];
      if (it.kind == IT_ATTN) {
        if ((rc = flush()) != CASSPEC_OK || (rc = attention(it.l)) != CASSPEC_OK) return rc;
        continue;
      }
      if (nph == kMaxPhases && (rc = flush()) != CASSPEC_OK) return rc;
      // Activation sparsity (App. C): the projection's input loses its smallest-magnitude entries
      // before the projection, so the projection starts its own launch after the sparsity kernel.
      const float sp = m->act_sparsity;
      if (sp > 0.f && it.kind != IT_LM) {
        if ((rc = flush()) != CASSPEC_OK) return rc;
        uint16_t* in = it.kind == IT_WO ? m->o : it.kind == IT_DOWN ? m->u : m->xa;
        const int K = it.kind == IT_DOWN ? F : d;
        LAUNCH(CASSPEC_K_OTHER, launch_sparsify(in, K, n, K, sp, s, pdl));
      }
      const int ss_parts = i == 0 ? 1 : resid_parts;  // the embedding leaves one partial, a residual phase one per slice
      ChainPhase& p = ca.ph[nph];
      switch (it.kind) {
        case IT_QKV:
          ph_qkv(it.l, ss_parts, p, cm.x[nph]);
          break;
        case IT_WO:
          ph_resid(d, m->layers[it.l].wo_p, d / kRowGroup, reader_gain(items[i + 1]), p);
          cm.x[nph] = m->tm_o[cx];
          break;
        case IT_GU:
          ph_gu(it.l, ss_parts, p);
          cm.x[nph] = m->tm_xa[cx];
          break;
        case IT_DOWN:
          ph_resid(F, m->layers[it.l].wd_p, F / kRowGroup, reader_gain(items[i + 1]), p);
          cm.x[nph] = m->tm_u[cx];
          break;
        default:
          ph_lm(ss_parts, p, cm.x[nph]);
          break;
      }
      ++nph;
    }
    if ((rc = flush()) != CASSPEC_OK) return rc;
  } else {
    // mode 1: W8A8 (codes in [-127, 127]); mode 2: W4A4 (codes in [-7, 7], weights two per byte)
    const bool w4 = mode == 2;
    const int qmax = w4 ? 7 : 127;
    // W4A4 on the tensor cores: e4m3 codes, exact fp32 accumulation (casspec gemm_f8); otherwise the
    // 4-bit codes go through the s8 MMA of gemm_i8
    const bool tc4 = w4 && (m->flags & CASSPEC_OPT_W4_TC) != 0;
    // W8A8 on the tensor cores: int8 codes widened to bf16 in shared memory (casspec gemm_s8tc), the
    // same exact int32 sums as gemm_i8
    const bool tc8 = !w4 && (m->flags & CASSPEC_OPT_W8_TC) != 0;
    const bool tc = tc4 || tc8;
    const int afmt = tc4 ? 2 : 0;  // activation codes as e4m3 bytes for the tensor-core path
    auto gemmf8 = [&](const CUtensorMap& tw, const CUtensorMap& tw2, const uint8_t* wpk, const CUtensorMap& tx,
                      const float* sw, const float* sw2, int N, int K, int tiles, int epi,
                      const EpiParams& e) -> cudaError_t {
      GemmF8Args g = {};
      g.wpk = wpk;
      g.tiles = tiles;
      g.kblocks = cdiv(K, 128);
      g.N = N;
      g.sw = sw;
      g.sw2 = sw2;
      g.sx = m->xs;
      g.partials = m->gemm_part;
      g.counters = m->gemm_cnt;
      g.status = m->status;
      g.ep = e;
      const int grid = gemm_bf16_grid(tiles, g.kblocks, m->num_sms);
      return tc8 ? launch_gemm_s8tc(tw, tw2, tx, BN, epi, g, grid, s, pdl)
                 : launch_gemm_f8(tw, tw2, tx, BN, epi, g, grid, s, pdl);
    };
    auto gemm8 = [&](const int8_t* W, const float* sw, const int8_t* W2, const float* sw2, int N, int K, int tiles,
                     int epi, const EpiParams& e) -> cudaError_t {
      GemmI8Args g8 = {};
      g8.W = W;
      g8.sw = sw;
      g8.W2 = W2;
      g8.sw2 = sw2;
      g8.X = m->xq;
      g8.sx = m->xs;
      g8.N = N;
      g8.K = K;
      g8.tiles = tiles;
      g8.ksplit = gemm_i8_ksplit(tiles, K, m->num_sms);
      g8.w4 = w4 ? 1 : 0;
      g8.partials = m->i8_part;
      g8.counters = m->i8_cnt;
      g8.status = m->status;
      g8.ep = e;
      return launch_gemm_i8(g8, BN, epi, s, pdl);
    };
    EpiParams er = base;  // residual projections
    er.N = d;
    er.y = m->x;
    er.ldy = d;
    for (size_t i = 0; i < items.size(); ++i) {
      const StepItem& it = items[i];
      int rc;
      if (it.kind == IT_LM) {  // the LM head stays bf16: the chain, after the W8A8 layers' residual tiles
        ChainArgs ca = {};
        ChainMaps cm = {};
        ca.nphases = 1;
        ph_lm(i == 0 ? 1 : d / 128, ca.ph[0], cm.x[0]);
        if ((rc = chain(ca, cm, CASSPEC_K_LMHEAD)) != CASSPEC_OK) return rc;
        continue;
      }
      if (it.kind == IT_ATTN) {
        if ((rc = attention(it.l)) != CASSPEC_OK) return rc;
        continue;
      }
      LayerPtrs& Lp = m->layers[it.l];
      const int8_t *q_qkv = w4 ? Lp.qkv_q4 : Lp.qkv_q, *q_wo = w4 ? Lp.wo_q4 : Lp.wo_q;
      const int8_t *q_wg = w4 ? Lp.wg_q4 : Lp.wg_q, *q_wu = w4 ? Lp.wu_q4 : Lp.wu_q, *q_wd = w4 ? Lp.wd_q4 : Lp.wd_q;
      const float *s_qkv = w4 ? Lp.qkv_s4 : Lp.qkv_s, *s_wo = w4 ? Lp.wo_s4 : Lp.wo_s;
      const float *s_wg = w4 ? Lp.wg_s4 : Lp.wg_s, *s_wu = w4 ? Lp.wu_s4 : Lp.wu_s, *s_wd = w4 ? Lp.wd_s4 : Lp.wd_s;
      EpiParams ed = er;
      if ((it.kind == IT_WO || it.kind == IT_DOWN) && items[i + 1].kind == IT_LM) {
        ed.ss_out = m->ssp;  // the last residual projection leaves the LM head's RMSNorm inputs
        ed.xa_out = m->xa;
        ed.g_next = m->final_norm;
      }
      // the tensor-core path's weight maps and tile images of this layer (W8A8 int8 / W4A4 e4m3 codes)
      const CUtensorMap &t_qkv = tc8 ? Lp.tm_qkvq : Lp.tm_qkv8, &t_wo = tc8 ? Lp.tm_oq : Lp.tm_o8;
      const CUtensorMap &t_wg = tc8 ? Lp.tm_gq : Lp.tm_g8, &t_wu = tc8 ? Lp.tm_uq : Lp.tm_u8;
      const CUtensorMap& t_wd = tc8 ? Lp.tm_dq : Lp.tm_d8;
      const uint8_t *p_qkv = tc8 ? Lp.qkv_qp : Lp.qkv_fp, *p_wo = tc8 ? Lp.wo_qp : Lp.wo_fp;
      const uint8_t *p_wgu = tc8 ? Lp.wgu_qp : Lp.wgu_fp, *p_wd = tc8 ? Lp.wd_qp : Lp.wd_fp;
      // the projection's quantised input: with activation sparsity (App. C's mixed draft) the bf16
      // activation first loses its smallest-magnitude entries (selected on that bf16 value), then
      // the same row quantiser runs on it
      const float sp = m->act_sparsity;
      auto norm_quant = [&](const float* gain) -> int {
        if (sp > 0.f) {
          LAUNCH(CASSPEC_K_OTHER, launch_rmsnorm(m->x, gain, n, d, c.rms_eps, m->xa, nullptr, nullptr, s, pdl, qmax, afmt));
          LAUNCH(CASSPEC_K_OTHER, launch_sparsify(m->xa, d, n, d, sp, s, pdl, 1));
          LAUNCH(CASSPEC_K_OTHER, launch_quant_rows(m->xa, n, d, d, m->xq, d, m->xs, s, pdl, qmax, afmt));
        } else {
          LAUNCH(CASSPEC_K_OTHER, launch_rmsnorm(m->x, gain, n, d, c.rms_eps, nullptr, m->xq, m->xs, s, pdl, qmax, afmt));
        }
        return CASSPEC_OK;
      };
      auto quant = [&](uint16_t* in, int K) -> int {
        if (sp > 0.f) LAUNCH(CASSPEC_K_OTHER, launch_sparsify(in, K, n, K, sp, s, pdl, 1));
        LAUNCH(CASSPEC_K_OTHER, launch_quant_rows(in, n, K, K, m->xq, K, m->xs, s, pdl, qmax, afmt));
        return CASSPEC_OK;
      };
      if (it.kind == IT_QKV) {
        if ((rc = norm_quant(Lp.attn_norm)) != CASSPEC_OK) return rc;
        EpiParams e = base;
        e.N = 3 * d;
        e.q_out = m->q;
        e.kc = kv_layer_k(kv, it.l);
        e.vc = kv_layer_v(kv, it.l);
        if (tc)
          LAUNCH(CASSPEC_K_QKV,
                 gemmf8(t_qkv, t_qkv, p_qkv, m->tm_xq8_d[bi], s_qkv, nullptr, 3 * d, d, 3 * d / 128, EPI_QKV, e));
        else
          LAUNCH(CASSPEC_K_QKV, gemm8(q_qkv, s_qkv, nullptr, nullptr, 3 * d, d, 3 * d / 128, EPI_QKV, e));
      } else if (it.kind == IT_WO) {
        // W8A8 activations are the bf16 values: the hi plane of the split output
        if ((rc = quant(m->o, d)) != CASSPEC_OK) return rc;
        if (tc)
          LAUNCH(CASSPEC_K_WO, gemmf8(t_wo, t_wo, p_wo, m->tm_xq8_d[bi], s_wo, nullptr, d, d, d / 128, EPI_RESID, ed));
        else
          LAUNCH(CASSPEC_K_WO, gemm8(q_wo, s_wo, nullptr, nullptr, d, d, d / 128, EPI_RESID, ed));
      } else if (it.kind == IT_GU) {
        if ((rc = norm_quant(Lp.ffn_norm)) != CASSPEC_OK) return rc;
        EpiParams eg = base;
        eg.N = F;
        eg.u_out = m->u;
        if (tc)
          LAUNCH(CASSPEC_K_GATEUP,
                 gemmf8(t_wg, t_wu, p_wgu, m->tm_xq8_d[bi], s_wg, s_wu, F, d, cdiv(F, 64), EPI_GLU, eg));
        else
          LAUNCH(CASSPEC_K_GATEUP, gemm8(q_wg, s_wg, q_wu, s_wu, F, d, cdiv(F, 64), EPI_GLU, eg));
      } else {
        if ((rc = quant(m->u, F)) != CASSPEC_OK) return rc;
        if (tc)
          LAUNCH(CASSPEC_K_DOWN, gemmf8(t_wd, t_wd, p_wd, m->tm_xq8_f[bi], s_wd, nullptr, d, F, d / 128, EPI_RESID, ed));
        else
          LAUNCH(CASSPEC_K_DOWN, gemm8(q_wd, s_wd, nullptr, nullptr, d, F, d / 128, EPI_RESID, ed));
      }
    }
  }
  LAUNCH(CASSPEC_K_OTHER, launch_argmax_reduce(m->am_v1, m->am_i1, m->am_v2, std::min(roundup16(V) / kRowGroup, G), n,
                                               m->am, m->margin, s, pdl));
  return CASSPEC_OK;
}

bool build_tensor_maps(casspec_model* m) {
  const auto& c = m->cfg;
  const uint64_t d = c.d_model, F = c.ffn, V = c.vocab;
  bool ok = true;
  for (int l = 0; l < c.n_layers; ++l) {
    LayerPtrs& Lp = m->layers[l];
    ok = ok && encode_tmap_bf16(&Lp.tm_qkv, Lp.wqkv, d, 3 * d, d * 2, 64, 128);
    ok = ok && encode_tmap_bf16(&Lp.tm_o, Lp.wo, d, d, d * 2, 64, 128);
    ok = ok && encode_tmap_bf16(&Lp.tm_g, Lp.wg, d, F, d * 2, 64, 64);
    ok = ok && encode_tmap_bf16(&Lp.tm_u, Lp.wu, d, F, d * 2, 64, 64);
    ok = ok && encode_tmap_bf16(&Lp.tm_d, Lp.wd, F, d, F * 2, 64, 128);
  }
  ok = ok && encode_tmap_bf16(&m->tm_lm, m->lm_head, d, V, d * 2, 64, 128);
  if (c.with_int8) {
    for (int l = 0; l < c.n_layers; ++l) {
      LayerPtrs& Lp = m->layers[l];
      ok = ok && encode_tmap_u8(&Lp.tm_qkv8, Lp.qkv_f8, d, 3 * d, d, 128, 128);
      ok = ok && encode_tmap_u8(&Lp.tm_o8, Lp.wo_f8, d, d, d, 128, 128);
      ok = ok && encode_tmap_u8(&Lp.tm_g8, Lp.wg_f8, d, F, d, 128, 64);
      ok = ok && encode_tmap_u8(&Lp.tm_u8, Lp.wu_f8, d, F, d, 128, 64);
      ok = ok && encode_tmap_u8(&Lp.tm_d8, Lp.wd_f8, F, d, F, 128, 128);
      ok = ok && encode_tmap_u8(&Lp.tm_qkvq, Lp.qkv_q, d, 3 * d, d, 128, 128);
      ok = ok && encode_tmap_u8(&Lp.tm_oq, Lp.wo_q, d, d, d, 128, 128);
      ok = ok && encode_tmap_u8(&Lp.tm_gq, Lp.wg_q, d, F, d, 128, 64);
      ok = ok && encode_tmap_u8(&Lp.tm_uq, Lp.wu_q, d, F, d, 128, 64);
      ok = ok && encode_tmap_u8(&Lp.tm_dq, Lp.wd_q, F, d, F, 128, 128);
    }
    for (int b = 0; b < 4; ++b) {
      const uint32_t BN = 16u * (uint32_t)(b + 1);
      ok = ok && encode_tmap_u8(&m->tm_xq8_d[b], m->xq, d, kMaxTree, d, 128, BN);
      ok = ok && encode_tmap_u8(&m->tm_xq8_f[b], m->xq, F, kMaxTree, F, 128, BN);
    }
  }
  for (int b = 0; b < 4; ++b) {
    const uint32_t BN = 16u * (uint32_t)(b + 1);
    ok = ok && encode_tmap_bf16(&m->tm_o[b], m->o, d, 2 * kMaxTree, d * 2, 64, BN);
    ok = ok && encode_tmap_bf16(&m->tm_u[b], m->u, F, 2 * kMaxTree, F * 2, 64, BN);
    ok = ok && encode_tmap_bf16(&m->tm_xa[b], m->xa, d, 2 * kMaxTree, d * 2, 64, BN);
  }
  {
    const uint32_t rows = 2 * kMaxTree;
    ok = ok && encode_tmap_bf16(&m->tm_o[4], m->o, d, rows, d * 2, 64, rows);
    ok = ok && encode_tmap_bf16(&m->tm_u[4], m->u, F, rows, F * 2, 64, rows);
    ok = ok && encode_tmap_bf16(&m->tm_xa[4], m->xa, d, rows, d * 2, 64, rows);
  }
  return ok;
}

}  // namespace

// =============================================================================================
// C ABI
// =============================================================================================
extern "C" {

size_t casspec_model_bytes(const casspec_model_config* cfg) {
  if (!config_ok(cfg)) return 0;
  return make_layout(*cfg).total;
}

int casspec_create_model(const casspec_model_config* cfg, void* dev_mem, size_t bytes, casspec_model** out) {
  if (out == nullptr || dev_mem == nullptr || !config_ok(cfg)) return CASSPEC_E_INVAL;
  if ((reinterpret_cast<uintptr_t>(dev_mem) & 255) != 0) return CASSPEC_E_INVAL;
  Layout L = make_layout(*cfg);
  if (bytes < L.total) return CASSPEC_E_CAPACITY;
  const int sms = num_sms_of_current_device();
  if (sms <= 0 || sms > kSmsBound) return CASSPEC_E_CUDA;
  {  // the projection chain's per-CTA slices must fit one MMA (and a residual slice the epilogue)
    const int G = chain_grid(sms), d = cfg->d_model, F = cfg->ffn;
    if (chain_slice_rows(3 * d, G, false) > kChainMaxSliceRows || chain_slice_rows(F, G, true) > kChainMaxSliceRows ||
        chain_slice_rows(roundup16(cfg->vocab), G, false) > kChainMaxSliceRows ||
        cdiv(F, 64) > kReadyPerPhase || cdiv(d, 64) > kReadyPerPhase)
      return CASSPEC_E_SHAPE;
  }
  // The residual projections (d output rows) split K over CTA pairs when pairs of CTAs fit the GPU
  // at once and a pair's rows fit its exchange buffer; otherwise each CTA runs all of K for its rows.
  int resid_split = 1;
  {
    const int G = chain_grid(sms), d = cfg->d_model;
    if (chain_slice_rows(d, G / 2, false) <= kPairMaxRows && cdiv(d, 64) >= 2 && cdiv(cfg->ffn, 64) >= 2 &&
        chain_pairs_fit(G))
      resid_split = 2;
    else if (chain_slice_rows(d, G, false) > 64)
      return CASSPEC_E_SHAPE;
  }
  casspec_model* m = new (std::nothrow) casspec_model();
  if (m == nullptr) return CASSPEC_E_CAPACITY;
  m->cfg = *cfg;
  m->resid_split = resid_split;
  m->lay = L;
  m->num_sms = sms;
  uint8_t* b = static_cast<uint8_t*>(dev_mem);
  m->base = b;
  m->embed = reinterpret_cast<uint16_t*>(b + L.embed);
  m->lm_head = reinterpret_cast<uint16_t*>(b + L.lm_head);
  m->final_norm = reinterpret_cast<float*>(b + L.final_norm);
  m->layers.resize(cfg->n_layers);
  for (int l = 0; l < cfg->n_layers; ++l) {
    LayerPtrs& p = m->layers[l];
    std::memset(&p, 0, sizeof(p));
    p.attn_norm = reinterpret_cast<float*>(b + L.attn_norm[l]);
    p.ffn_norm = reinterpret_cast<float*>(b + L.ffn_norm[l]);
    p.wqkv = reinterpret_cast<uint16_t*>(b + L.wqkv[l]);
    p.wo = reinterpret_cast<uint16_t*>(b + L.wo[l]);
    p.wg = reinterpret_cast<uint16_t*>(b + L.wg[l]);
    p.wu = reinterpret_cast<uint16_t*>(b + L.wu[l]);
    p.wd = reinterpret_cast<uint16_t*>(b + L.wd[l]);
    p.wqkv_p = b + L.wqkv_p[l];
    p.wo_p = b + L.wo_p[l];
    p.wgu_p = b + L.wgu_p[l];
    p.wd_p = b + L.wd_p[l];
    if (cfg->with_int8) {
      p.qkv_q = reinterpret_cast<int8_t*>(b + L.qkv_q[l]);
      p.wo_q = reinterpret_cast<int8_t*>(b + L.wo_q[l]);
      p.wg_q = reinterpret_cast<int8_t*>(b + L.wg_q[l]);
      p.wu_q = reinterpret_cast<int8_t*>(b + L.wu_q[l]);
      p.wd_q = reinterpret_cast<int8_t*>(b + L.wd_q[l]);
      p.qkv_s = reinterpret_cast<float*>(b + L.qkv_s[l]);
      p.wo_s = reinterpret_cast<float*>(b + L.wo_s[l]);
      p.wg_s = reinterpret_cast<float*>(b + L.wg_s[l]);
      p.wu_s = reinterpret_cast<float*>(b + L.wu_s[l]);
      p.wd_s = reinterpret_cast<float*>(b + L.wd_s[l]);
      p.qkv_q4 = reinterpret_cast<int8_t*>(b + L.qkv_q4[l]);
      p.wo_q4 = reinterpret_cast<int8_t*>(b + L.wo_q4[l]);
      p.wg_q4 = reinterpret_cast<int8_t*>(b + L.wg_q4[l]);
      p.wu_q4 = reinterpret_cast<int8_t*>(b + L.wu_q4[l]);
      p.wd_q4 = reinterpret_cast<int8_t*>(b + L.wd_q4[l]);
      p.qkv_s4 = reinterpret_cast<float*>(b + L.qkv_s4[l]);
      p.wo_s4 = reinterpret_cast<float*>(b + L.wo_s4[l]);
      p.wg_s4 = reinterpret_cast<float*>(b + L.wg_s4[l]);
      p.wu_s4 = reinterpret_cast<float*>(b + L.wu_s4[l]);
      p.wd_s4 = reinterpret_cast<float*>(b + L.wd_s4[l]);
      p.qkv_f8 = b + L.qkv_f8[l];
      p.wo_f8 = b + L.wo_f8[l];
      p.wg_f8 = b + L.wg_f8[l];
      p.wu_f8 = b + L.wu_f8[l];
      p.wd_f8 = b + L.wd_f8[l];
      p.qkv_qp = b + L.qkv_qp[l];
      p.wo_qp = b + L.wo_qp[l];
      p.wgu_qp = b + L.wgu_qp[l];
      p.wd_qp = b + L.wd_qp[l];
      p.qkv_fp = b + L.qkv_fp[l];
      p.wo_fp = b + L.wo_fp[l];
      p.wgu_fp = b + L.wgu_fp[l];
      p.wd_fp = b + L.wd_fp[l];
    }
  }
  m->x = reinterpret_cast<float*>(b + L.x);
  m->q = reinterpret_cast<uint16_t*>(b + L.q);
  m->o = reinterpret_cast<uint16_t*>(b + L.o);
  m->u = reinterpret_cast<uint16_t*>(b + L.u);
  m->xa = reinterpret_cast<uint16_t*>(b + L.xa);
  m->ssp = reinterpret_cast<float*>(b + L.ssp);
  m->chain_ready = reinterpret_cast<unsigned*>(b + L.chain_ready);
  m->chain_done = reinterpret_cast<unsigned*>(b + L.chain_done);
  m->lm_p = b + L.lm_p;
  m->xq = reinterpret_cast<int8_t*>(b + L.xq);
  m->xs = reinterpret_cast<float*>(b + L.xs);
  m->pos = reinterpret_cast<int*>(b + L.pos);
  m->anc = reinterpret_cast<unsigned long long*>(b + L.anc);
  m->am_v1 = reinterpret_cast<float*>(b + L.am_v1);
  m->am_i1 = reinterpret_cast<int*>(b + L.am_i1);
  m->am_v2 = reinterpret_cast<float*>(b + L.am_v2);
  m->am = reinterpret_cast<int*>(b + L.am);
  m->margin = reinterpret_cast<float*>(b + L.margin);
  m->am2 = reinterpret_cast<int*>(b + L.am2);
  m->gemm_part = reinterpret_cast<float*>(b + L.gemm_part);
  m->gemm_cnt = reinterpret_cast<unsigned*>(b + L.gemm_cnt);
  m->i8_part = reinterpret_cast<int*>(b + L.i8_part);
  m->i8_cnt = reinterpret_cast<unsigned*>(b + L.i8_cnt);
  m->status = reinterpret_cast<int*>(b + L.status);

  if (cudaMemset(b + L.scratch_begin, 0, L.total - L.scratch_begin) != cudaSuccess ||
      cudaStreamCreateWithFlags(&m->cap_stream, cudaStreamNonBlocking) != cudaSuccess) {
    delete m;
    return CASSPEC_E_CUDA;
  }
  // RMSNorm gains default to 1.0
  std::vector<float> ones(cfg->d_model, 1.0f);
  bool ok = cudaMemcpy(m->final_norm, ones.data(), ones.size() * 4, cudaMemcpyHostToDevice) == cudaSuccess;
  for (int l = 0; ok && l < cfg->n_layers; ++l) {
    ok = cudaMemcpy(m->layers[l].attn_norm, ones.data(), ones.size() * 4, cudaMemcpyHostToDevice) == cudaSuccess &&
         cudaMemcpy(m->layers[l].ffn_norm, ones.data(), ones.size() * 4, cudaMemcpyHostToDevice) == cudaSuccess;
  }
  if (!ok || !build_tensor_maps(m)) {
    cudaStreamDestroy(m->cap_stream);
    delete m;
    return CASSPEC_E_CUDA;
  }
  *out = m;
  return CASSPEC_OK;
}

void casspec_destroy_model(casspec_model* m) {
  if (m == nullptr) return;
  for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second.first);
  for (auto& v : m->prof_ev)
    for (auto& e : v) {
      cudaEventDestroy(e.first);
      cudaEventDestroy(e.second);
    }
  if (m->cap_stream) cudaStreamDestroy(m->cap_stream);
  delete m;
}

int casspec_set_stream(casspec_model* m, void* stream) {
  if (m == nullptr) return CASSPEC_E_INVAL;
  m->stream = static_cast<cudaStream_t>(stream);
  return CASSPEC_OK;
}

int casspec_set_act_sparsity(casspec_model* m, float s) {
  if (m == nullptr || !(s >= 0.f && s < 1.f)) return CASSPEC_E_INVAL;
  if (s != m->act_sparsity) {  // the step's launches differ: captured steps are rebuilt
    for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second.first);
    m->graphs.clear();
  }
  m->act_sparsity = s;
  return CASSPEC_OK;
}

int casspec_sparsify_rows(uint16_t* x_split, int ld, int n, int K, float s, void* stream) {
  if (x_split == nullptr || !(s >= 0.f && s < 1.f)) return CASSPEC_E_INVAL;
  if (n < 1 || n > kMaxTree || K < 1 || K > 16384 || ld < K) return CASSPEC_E_SHAPE;
  CK(launch_sparsify(x_split, ld, n, K, s, static_cast<cudaStream_t>(stream), false));
  return CASSPEC_OK;
}

int casspec_set_options(casspec_model* m, unsigned flags, unsigned* old_flags) {
  if (m == nullptr ||
      (flags & ~(CASSPEC_OPT_PDL | CASSPEC_OPT_GRAPHS | CASSPEC_OPT_TEST_STALL | CASSPEC_OPT_W4_TC |
                 CASSPEC_OPT_W8_TC)) != 0)
    return CASSPEC_E_INVAL;
  if (old_flags) *old_flags = m->flags;
  if (flags != m->flags) {
    for (auto& kv : m->graphs) cudaGraphExecDestroy(kv.second.first);
    m->graphs.clear();
  }
  m->flags = flags;
  return CASSPEC_OK;
}

int casspec_tensor(casspec_model* m, int tensor, int layer, void** dev_ptr, size_t* bytes) {
  if (m == nullptr || dev_ptr == nullptr) return CASSPEC_E_INVAL;
  if (tensor <= CASSPEC_T_WD) m->pack_dirty = true;  // the caller may write through the pointer
  if ((tensor >= CASSPEC_T_WQKV_Q && tensor <= CASSPEC_T_WD_Q) ||
      (tensor >= CASSPEC_T_WQKV_F8 && tensor <= CASSPEC_T_WD_F8))
    m->pack8_dirty = true;
  const auto& c = m->cfg;
  const size_t d = c.d_model, F = c.ffn, V = c.vocab;
  const bool state = tensor >= CASSPEC_T_RESIDUAL && tensor <= CASSPEC_T_ACT_S;  // step state, not weights
  const bool per_layer = tensor >= CASSPEC_T_ATTN_NORM && !state;
  if (per_layer && (layer < 0 || layer >= c.n_layers)) return CASSPEC_E_INVAL;
  if (tensor >= CASSPEC_T_WQKV_Q && !state && !c.with_int8) return CASSPEC_E_INVAL;
  void* p = nullptr;
  size_t nb = 0;
  const LayerPtrs* L = per_layer ? &m->layers[layer] : nullptr;
  switch (tensor) {
    case CASSPEC_T_EMBED: p = m->embed; nb = V * d * 2; break;
    case CASSPEC_T_LM_HEAD: p = m->lm_head; nb = V * d * 2; break;
    case CASSPEC_T_FINAL_NORM: p = m->final_norm; nb = d * 4; break;
    case CASSPEC_T_ATTN_NORM: p = L->attn_norm; nb = d * 4; break;
    case CASSPEC_T_FFN_NORM: p = L->ffn_norm; nb = d * 4; break;
    case CASSPEC_T_WQKV: p = L->wqkv; nb = 3 * d * d * 2; break;
    case CASSPEC_T_WO: p = L->wo; nb = d * d * 2; break;
    case CASSPEC_T_WG: p = L->wg; nb = F * d * 2; break;
    case CASSPEC_T_WU: p = L->wu; nb = F * d * 2; break;
    case CASSPEC_T_WD: p = L->wd; nb = d * F * 2; break;
    case CASSPEC_T_WQKV_Q: p = L->qkv_q; nb = 3 * d * d; break;
    case CASSPEC_T_WO_Q: p = L->wo_q; nb = d * d; break;
    case CASSPEC_T_WG_Q: p = L->wg_q; nb = F * d; break;
    case CASSPEC_T_WU_Q: p = L->wu_q; nb = F * d; break;
    case CASSPEC_T_WD_Q: p = L->wd_q; nb = d * F; break;
    case CASSPEC_T_WQKV_S: p = L->qkv_s; nb = 3 * d * 4; break;
    case CASSPEC_T_WO_S: p = L->wo_s; nb = d * 4; break;
    case CASSPEC_T_WG_S: p = L->wg_s; nb = F * 4; break;
    case CASSPEC_T_WU_S: p = L->wu_s; nb = F * 4; break;
    case CASSPEC_T_WD_S: p = L->wd_s; nb = d * 4; break;
    case CASSPEC_T_RESIDUAL: p = m->x; nb = (size_t)kMaxTree * d * 4; break;
    case CASSPEC_T_ACT_Q: p = m->xq; nb = (size_t)kMaxTree * std::max(d, F); break;
    case CASSPEC_T_ACT_S: p = m->xs; nb = (size_t)kMaxTree * 4; break;
    case CASSPEC_T_WQKV_Q4: p = L->qkv_q4; nb = 3 * d * d / 2; break;
    case CASSPEC_T_WO_Q4: p = L->wo_q4; nb = d * d / 2; break;
    case CASSPEC_T_WG_Q4: p = L->wg_q4; nb = F * d / 2; break;
    case CASSPEC_T_WU_Q4: p = L->wu_q4; nb = F * d / 2; break;
    case CASSPEC_T_WD_Q4: p = L->wd_q4; nb = d * F / 2; break;
    case CASSPEC_T_WQKV_S4: p = L->qkv_s4; nb = 3 * d * 4; break;
    case CASSPEC_T_WO_S4: p = L->wo_s4; nb = d * 4; break;
    case CASSPEC_T_WG_S4: p = L->wg_s4; nb = F * 4; break;
    case CASSPEC_T_WU_S4: p = L->wu_s4; nb = F * 4; break;
    case CASSPEC_T_WD_S4: p = L->wd_s4; nb = d * 4; break;
    case CASSPEC_T_WQKV_F8: p = L->qkv_f8; nb = 3 * d * d; break;
    case CASSPEC_T_WO_F8: p = L->wo_f8; nb = d * d; break;
    case CASSPEC_T_WG_F8: p = L->wg_f8; nb = F * d; break;
    case CASSPEC_T_WU_F8: p = L->wu_f8; nb = F * d; break;
    case CASSPEC_T_WD_F8: p = L->wd_f8; nb = d * F; break;
    default: return CASSPEC_E_INVAL;
  }
  *dev_ptr = p;
  if (bytes) *bytes = nb;
  return CASSPEC_OK;
}

int casspec_quantize_weights(casspec_model* m) {
  if (m == nullptr || !m->cfg.with_int8) return CASSPEC_E_INVAL;
  const auto& c = m->cfg;
  const int d = c.d_model, F = c.ffn;
  for (int l = 0; l < c.n_layers; ++l) {
    LayerPtrs& p = m->layers[l];
    CK(launch_quant_rows(p.wqkv, 3 * d, d, d, p.qkv_q, d, p.qkv_s, m->stream, false));
    CK(launch_quant_rows(p.wo, d, d, d, p.wo_q, d, p.wo_s, m->stream, false));
    CK(launch_quant_rows(p.wg, F, d, d, p.wg_q, d, p.wg_s, m->stream, false));
    CK(launch_quant_rows(p.wu, F, d, d, p.wu_q, d, p.wu_s, m->stream, false));
    CK(launch_quant_rows(p.wd, d, F, F, p.wd_q, F, p.wd_s, m->stream, false));
    // the W4A4 copies: codes in [-7, 7], two per byte (row stride K / 2 bytes)
    CK(launch_quant_rows(p.wqkv, 3 * d, d, d, p.qkv_q4, d / 2, p.qkv_s4, m->stream, false, 7, 1));
    CK(launch_quant_rows(p.wo, d, d, d, p.wo_q4, d / 2, p.wo_s4, m->stream, false, 7, 1));
    CK(launch_quant_rows(p.wg, F, d, d, p.wg_q4, d / 2, p.wg_s4, m->stream, false, 7, 1));
    CK(launch_quant_rows(p.wu, F, d, d, p.wu_q4, d / 2, p.wu_s4, m->stream, false, 7, 1));
    CK(launch_quant_rows(p.wd, d, F, F, p.wd_q4, F / 2, p.wd_s4, m->stream, false, 7, 1));
    // ... and as e4m3 bytes for the tensor-core path (same codes, same scales)
    CK(launch_quant_rows(p.wqkv, 3 * d, d, d, reinterpret_cast<int8_t*>(p.qkv_f8), d, p.qkv_s4, m->stream, false, 7, 2));
    CK(launch_quant_rows(p.wo, d, d, d, reinterpret_cast<int8_t*>(p.wo_f8), d, p.wo_s4, m->stream, false, 7, 2));
    CK(launch_quant_rows(p.wg, F, d, d, reinterpret_cast<int8_t*>(p.wg_f8), d, p.wg_s4, m->stream, false, 7, 2));
    CK(launch_quant_rows(p.wu, F, d, d, reinterpret_cast<int8_t*>(p.wu_f8), d, p.wu_s4, m->stream, false, 7, 2));
    CK(launch_quant_rows(p.wd, d, F, F, reinterpret_cast<int8_t*>(p.wd_f8), F, p.wd_s4, m->stream, false, 7, 2));
  }
  m->pack8_dirty = true;
  return CASSPEC_OK;
}

size_t casspec_kv_bytes(const casspec_model_config* cfg, int max_ctx) {
  if (!config_ok(cfg) || max_ctx < 1) return 0;
  return kv_region_bytes(*cfg, kv_ctx(max_ctx)) + kv_meta_bytes(*cfg, kv_ctx(max_ctx));
}

int casspec_kv_create(casspec_model* m, int max_ctx, void* dev_mem, size_t bytes, casspec_kv** out) {
  if (m == nullptr || dev_mem == nullptr || out == nullptr || max_ctx < 1) return CASSPEC_E_INVAL;
  if ((reinterpret_cast<uintptr_t>(dev_mem) & 255) != 0) return CASSPEC_E_INVAL;
  const int ctx = kv_ctx(max_ctx);
  const size_t region = kv_region_bytes(m->cfg, ctx);
  const size_t meta_bytes = kv_meta_bytes(m->cfg, ctx);
  if (bytes < region + meta_bytes) return CASSPEC_E_CAPACITY;
  casspec_kv* kv = new (std::nothrow) casspec_kv();
  if (kv == nullptr) return CASSPEC_E_CAPACITY;
  uint8_t* b = static_cast<uint8_t*>(dev_mem);
  kv->m = m;
  kv->base = reinterpret_cast<uint16_t*>(b);
  kv->ctx = ctx;
  uint8_t* meta = b + region;
  kv->dP = reinterpret_cast<int*>(meta);
  kv->compact_cnt = reinterpret_cast<unsigned*>(meta + 128);
  kv->tdepth = reinterpret_cast<int*>(meta + 256);
  kv->tanc = reinterpret_cast<unsigned long long*>(meta + 256 + kMaxTree * 4);
  kv->rope = reinterpret_cast<float2*>(meta + 1024);
  kv->layer_valid.assign(m->cfg.n_layers, 0);
  if (!encode_tmap_bf16(&kv->tm_kv, kv->base, (uint64_t)m->cfg.head_dim,
                        (uint64_t)m->cfg.n_layers * 2 * m->cfg.n_heads * ctx, (uint64_t)m->cfg.head_dim * 2, 64, 64)) {
    delete kv;
    return CASSPEC_E_CUDA;
  }
  // rotary table for every position of the cache, evaluated in fp64 on the host
  const int half = m->cfg.head_dim / 2;
  std::vector<float2> table((size_t)ctx * half);
  for (int p = 0; p < ctx; ++p)
    for (int j = 0; j < half; ++j) {
      const double ang = (double)p * std::pow((double)m->cfg.rope_base, -2.0 * j / (double)m->cfg.head_dim);
      table[(size_t)p * half + j] = make_float2((float)std::cos(ang), (float)std::sin(ang));
    }
  if (cudaMemsetAsync(b, 0, region + 1024, m->stream) != cudaSuccess ||
      cudaMemcpyAsync(kv->rope, table.data(), table.size() * sizeof(float2), cudaMemcpyHostToDevice, m->stream) !=
          cudaSuccess ||
      cudaStreamSynchronize(m->stream) != cudaSuccess) {
    delete kv;
    return CASSPEC_E_CUDA;
  }
  *out = kv;
  return CASSPEC_OK;
}

void casspec_kv_destroy(casspec_kv* kv) { delete kv; }

int casspec_kv_layer(casspec_kv* kv, int layer, void** k_dev, void** v_dev, int* ld_slots) {
  if (kv == nullptr || layer < 0 || layer >= kv->m->cfg.n_layers) return CASSPEC_E_INVAL;
  if (k_dev) *k_dev = kv_layer_k(kv, layer);
  if (v_dev) *v_dev = kv_layer_v(kv, layer);
  if (ld_slots) *ld_slots = kv->ctx;
  return CASSPEC_OK;
}

int casspec_kv_set_prefix(casspec_kv* kv, int P) {
  if (kv == nullptr || P < 0 || P > kv->ctx) return CASSPEC_E_INVAL;
  CK(launch_set_int(kv->dP, P, kv->m->stream));
  kv->m->launches++;
  kv->P_upper = P;
  kv->T = 0;
  std::fill(kv->layer_valid.begin(), kv->layer_valid.end(), 0);
  return CASSPEC_OK;
}

int casspec_kv_reset_tree(casspec_kv* kv) {
  if (kv == nullptr) return CASSPEC_E_INVAL;
  kv->T = 0;
  std::fill(kv->layer_valid.begin(), kv->layer_valid.end(), 0);
  return CASSPEC_OK;
}

int casspec_kv_length(casspec_kv* kv, int* P_out, int* T_out) {
  if (kv == nullptr) return CASSPEC_E_INVAL;
  CK(cudaStreamSynchronize(kv->m->stream));
  int P = 0;
  CK(cudaMemcpy(&P, kv->dP, 4, cudaMemcpyDeviceToHost));
  kv->P_upper = P;
  if (P_out) *P_out = P;
  if (T_out) *T_out = kv->T;
  return CASSPEC_OK;
}

int casspec_tree_step(casspec_model* m, casspec_kv* kv, const int32_t* tokens, const int32_t* parent_idx, int n,
                      const uint8_t* skip_mask, int quant_mode, float* logits_out) {
  if (m == nullptr || kv == nullptr || tokens == nullptr || parent_idx == nullptr || kv->m != m)
    return CASSPEC_E_INVAL;
  if (quant_mode < 0 || quant_mode > 2) return CASSPEC_E_INVAL;
  if (quant_mode != 0 && !m->cfg.with_int8) return CASSPEC_E_INVAL;
  if (n < 1 || n > kMaxTree) return CASSPEC_E_SHAPE;
  if (kv->T + n > kMaxTree || kv->P_upper + kv->T + n > kv->ctx) return CASSPEC_E_CAPACITY;
  const int NL = m->cfg.n_layers;
  std::vector<uint8_t> on(NL, kBlockAttn | kBlockFfn);
  if (skip_mask)
    for (int l = 0; l < NL; ++l) on[l] = layer_blocks(skip_mask[l]);
  for (int l = 0; l < NL; ++l)  // attention reads the K/V of the existing tree slots
    if ((on[l] & kBlockAttn) && kv->layer_valid[l] != kv->T) return CASSPEC_E_STATE;

  std::lock_guard<std::mutex> lock(m->mu);
  int rc = CASSPEC_OK;
  if (m->pack_dirty) {  // outside any capture: a graph never holds the packing
    int count = 0;
    if ((rc = pack_weights(m, count)) != CASSPEC_OK) return rc;
    m->launches += (uint64_t)count;
  }
  if (quant_mode != 0 && m->pack8_dirty) {
    int count = 0;
    if ((rc = pack_codes(m, count)) != CASSPEC_OK) return rc;
    m->launches += (uint64_t)count;
  }
  if ((m->flags & CASSPEC_OPT_GRAPHS) && !(m->flags & CASSPEC_OPT_TEST_STALL)) {
    GraphKey key{kv, tokens, parent_idx, logits_out, n, kv->T, quant_mode, on};
    auto it = m->graphs.find(key);
    if (it == m->graphs.end()) {
      if (cudaStreamBeginCapture(m->cap_stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
        return CASSPEC_E_CUDA;
      int count = 0;
      rc = enqueue_step(m, kv, tokens, parent_idx, n, on, quant_mode, logits_out, m->cap_stream, false, count);
      cudaGraph_t g = nullptr;
      const cudaError_t ec = cudaStreamEndCapture(m->cap_stream, &g);
      if (rc != CASSPEC_OK || ec != cudaSuccess || g == nullptr) {
        if (g) cudaGraphDestroy(g);
        cudaGetLastError();
        return rc != CASSPEC_OK ? rc : CASSPEC_E_CUDA;
      }
      cudaGraphExec_t ex = nullptr;
      const cudaError_t ei = cudaGraphInstantiate(&ex, g, 0);
      cudaGraphDestroy(g);
      if (ei != cudaSuccess) return CASSPEC_E_CUDA;
      it = m->graphs.emplace(key, std::make_pair(ex, count)).first;
    }
    if (cudaGraphLaunch(it->second.first, m->stream) != cudaSuccess) return CASSPEC_E_CUDA;
    m->launches += (uint64_t)it->second.second;
  } else {
    int count = 0;
    rc = enqueue_step(m, kv, tokens, parent_idx, n, on, quant_mode, logits_out, m->stream, m->prof_on, count);
    m->launches += (uint64_t)count;
    if (rc != CASSPEC_OK) return rc;
  }
  const int Tn = kv->T + n;
  for (int l = 0; l < NL; ++l)
    if (on[l] & kBlockAttn) kv->layer_valid[l] = Tn;
  kv->T = Tn;
  return CASSPEC_OK;
}

int casspec_argmax(casspec_model* m, const int32_t** argmax_dev, const float** margin_dev) {
  if (m == nullptr) return CASSPEC_E_INVAL;
  if (argmax_dev) *argmax_dev = m->am;
  if (margin_dev) *margin_dev = m->margin;
  return CASSPEC_OK;
}

int casspec_accept_greedy(casspec_model* m, const float* logits, const int32_t* tokens, const int32_t* parent_idx,
                          int n, int32_t* accepted_out) {
  if (m == nullptr || tokens == nullptr || parent_idx == nullptr || accepted_out == nullptr) return CASSPEC_E_INVAL;
  if (n < 1 || n > kMaxTree) return CASSPEC_E_SHAPE;
  const int* am = m->am;
  if (logits != nullptr) {
    CK(launch_row_argmax(logits, n, m->cfg.vocab, m->am2, m->stream));
    am = m->am2;
    m->launches++;
  }
  CK(launch_accept(am, tokens, parent_idx, n, accepted_out, m->status, m->stream));
  m->launches++;
  return CASSPEC_OK;
}

int casspec_kv_compact(casspec_kv* kv, const int32_t* accepted_out) {
  if (kv == nullptr || accepted_out == nullptr) return CASSPEC_E_INVAL;
  if (kv->T < 1) return CASSPEC_E_STATE;
  for (int v : kv->layer_valid)
    if (v != kv->T) return CASSPEC_E_STATE;
  casspec_model* m = kv->m;
  const auto& c = m->cfg;
  CK(launch_kv_compact(kv->base, c.n_layers, c.n_heads, kv->ctx, c.head_dim, accepted_out, kv->tanc, kv->T,
                       kv->dP, kv->compact_cnt, m->status, m->stream));
  m->launches++;
  kv->P_upper += kv->T;
  kv->T = 0;
  std::fill(kv->layer_valid.begin(), kv->layer_valid.end(), 0);
  return CASSPEC_OK;
}

int casspec_profile(casspec_model* m, int enable) {
  if (m == nullptr) return CASSPEC_E_INVAL;
  m->prof_on = enable != 0;
  if (m->prof_on)
    for (int k = 0; k < CASSPEC_K_COUNT; ++k) m->prof_used[k] = 0;
  return CASSPEC_OK;
}

int casspec_profile_read(casspec_model* m, int kind, double* total_ms, int* launches) {
  if (m == nullptr || kind < 0 || kind >= CASSPEC_K_COUNT) return CASSPEC_E_INVAL;
  CK(cudaStreamSynchronize(m->stream));
  double t = 0.0;
  for (int i = 0; i < m->prof_used[kind]; ++i) {
    float ms = 0.f;
    CK(cudaEventElapsedTime(&ms, m->prof_ev[kind][i].first, m->prof_ev[kind][i].second));
    t += ms;
  }
  if (total_ms) *total_ms = t;
  if (launches) *launches = m->prof_used[kind];
  return CASSPEC_OK;
}

int casspec_launch_count(casspec_model* m, uint64_t* count) {
  if (m == nullptr || count == nullptr) return CASSPEC_E_INVAL;
  *count = m->launches;
  return CASSPEC_OK;
}

int casspec_get_status(casspec_model* m, int* status_out) {
  if (m == nullptr) return CASSPEC_E_INVAL;
  CK(cudaStreamSynchronize(m->stream));
  int st = 0;
  CK(cudaMemcpy(&st, m->status, 4, cudaMemcpyDeviceToHost));
  if (st != 0) {
    // a kernel that gave up may have left fix-up counters behind: clear them all
    CK(cudaMemset(m->status, 0, 4));
    CK(cudaMemset(m->gemm_cnt, 0, (size_t)m->lay.max_tiles * 4));
    CK(cudaMemset(m->i8_cnt, 0, (size_t)m->lay.max_tiles * 4));
    CK(cudaMemset(m->chain_ready, 0, (size_t)kMaxPhases * kReadyPerPhase * 4));
    CK(cudaMemset(m->chain_done, 0, 256));
  }
  if (status_out) *status_out = st;
  return CASSPEC_OK;
}

const char* casspec_status_string(int s) {
  switch (s) {
    case CASSPEC_OK: return "ok";
    case CASSPEC_E_INVAL: return "invalid argument";
    case CASSPEC_E_SHAPE: return "unsupported size";
    case CASSPEC_E_CAPACITY: return "capacity exceeded";
    case CASSPEC_E_CUDA: return "CUDA error";
    case CASSPEC_E_TREE: return "invalid tree or accepted path";
    case CASSPEC_E_TIMEOUT: return "bounded device wait expired";
    case CASSPEC_E_STATE: return "call-order rule violated";
  }
  return "unknown status";
}

size_t casspec_linear_workspace_bytes(int N, int K, int n) {
  if (N < 1 || K < 8 || n < 1) return 0;
  const int tiles = cdiv(N, 128);
  return 4096 + gemm_partials_floats(tiles, kSmsBound) * 4;
}

int casspec_linear_bf16(const uint16_t* W, int N, int K, const uint16_t* X, int n, float* Y, int ldy, void* ws,
                        size_t ws_bytes, void* stream) {
  if (W == nullptr || X == nullptr || Y == nullptr || ws == nullptr) return CASSPEC_E_INVAL;
  if (n < 1 || n > kMaxTree || N < 1 || K < 8 || K % 8 != 0 || ldy < N) return CASSPEC_E_SHAPE;
  if (((uintptr_t)W & 15) || ((uintptr_t)X & 15) || ((uintptr_t)ws & 15)) return CASSPEC_E_INVAL;
  const int tiles = cdiv(N, 128);
  if (tiles > 1023) return CASSPEC_E_SHAPE;  // counters [0, tiles) and the status word at byte 4092
  if (ws_bytes < casspec_linear_workspace_bytes(N, K, n)) return CASSPEC_E_CAPACITY;
  const int sms = num_sms_of_current_device();
  if (sms <= 0) return CASSPEC_E_CUDA;
  const int BN = roundup16(n);
  CUtensorMap tw, tx;
  if (!encode_tmap_bf16(&tw, W, K, N, (uint64_t)K * 2, 64, 128) ||
      !encode_tmap_bf16(&tx, X, K, n, (uint64_t)K * 2, 64, BN))
    return CASSPEC_E_CUDA;
  const int kb = cdiv(K, 64);
  GemmArgs a = {};
  a.tiles = tiles;
  a.kblocks = kb;
  a.counters = static_cast<unsigned*>(ws);
  a.partials = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + 4096);
  a.status = reinterpret_cast<int*>(static_cast<uint8_t*>(ws) + 4092);
  a.ep.n = n;
  a.ep.N = N;
  a.ep.y = Y;
  a.ep.ldy = ldy;
  CK(launch_gemm_bf16(tw, tw, tx, BN, EPI_STORE, a, gemm_bf16_grid(tiles, kb, sms), static_cast<cudaStream_t>(stream),
                      false));
  return CASSPEC_OK;
}

int casspec_rmsnorm(const float* x, const float* g, int n, int d, float eps, uint16_t* y, int8_t* q, float* s,
                    void* stream) {
  if (x == nullptr || g == nullptr || (y == nullptr && q == nullptr) || ((q == nullptr) != (s == nullptr)))
    return CASSPEC_E_INVAL;
  if (n < 1 || d < 1) return CASSPEC_E_SHAPE;
  CK(launch_rmsnorm(x, g, n, d, eps, y, q, s, static_cast<cudaStream_t>(stream), false));
  return CASSPEC_OK;
}

int casspec_quantize_rows(const uint16_t* x, int n, int d, int8_t* q, float* s, void* stream) {
  if (x == nullptr || q == nullptr || s == nullptr) return CASSPEC_E_INVAL;
  if (n < 1 || d < 1) return CASSPEC_E_SHAPE;
  CK(launch_quant_rows(x, n, d, d, q, d, s, static_cast<cudaStream_t>(stream), false));
  return CASSPEC_OK;
}

int casspec_quantize_rows4(const uint16_t* x, int n, int d, uint8_t* q4, float* s, void* stream) {
  if (x == nullptr || q4 == nullptr || s == nullptr) return CASSPEC_E_INVAL;
  if (n < 1 || d < 8 || d % 8 != 0) return CASSPEC_E_SHAPE;
  CK(launch_quant_rows(x, n, d, d, reinterpret_cast<int8_t*>(q4), d / 2, s, static_cast<cudaStream_t>(stream), false,
                       7, 1));
  return CASSPEC_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------------------------
// One DyTC round (Sec. 4.2, Algorithm 1, then verification)
// ---------------------------------------------------------------------------------------------
namespace {
int read_dev_i32(casspec_model* m, const int32_t* dev, int count, int32_t* host) {
  CK(cudaMemcpyAsync(host, dev, (size_t)count * 4, cudaMemcpyDeviceToHost, m->stream));
  CK(cudaStreamSynchronize(m->stream));
  return CASSPEC_OK;
}
}  // namespace

extern "C" int casspec_dytc_round(casspec_dytc* s, casspec_model* m, casspec_kv* kv, const casspec_draft_cfg* cfgs,
                                  int32_t root_token, int32_t* history, int hist_len, int32_t* dev_work,
                                  float* dev_logits, int32_t* out_tokens, int* n_out, int* n_drafted_out) {
  if (s == nullptr || m == nullptr || kv == nullptr || cfgs == nullptr || dev_work == nullptr || out_tokens == nullptr ||
      n_out == nullptr || kv->m != m)
    return CASSPEC_E_INVAL;
  if (kv->T != 0) return CASSPEC_E_STATE;  // a round starts from a committed prefix
  casspec_dytc_params prm;
  if (casspec_dytc_get_params(s, &prm) != CASSPEC_OK) return CASSPEC_E_INVAL;
  const int K = prm.topk;
  if (K > 1 && dev_logits == nullptr) return CASSPEC_E_INVAL;
  const int V = m->cfg.vocab;
  int32_t* d_tok = dev_work;
  int32_t* d_par = dev_work + kMaxTree;
  int32_t* d_acc = dev_work + 2 * kMaxTree;
  int32_t* d_pld = dev_work + 3 * kMaxTree + 8;  // {match length, count, tokens...}
  int32_t* d_tki = dev_work + 5 * kMaxTree;      // top-K ids [64][8]
  float* d_tkp = reinterpret_cast<float*>(dev_work + 13 * kMaxTree);  // top-K probabilities [64][8]
  const int32_t* d_am = m->am;
  int rc;
  if ((rc = casspec_dytc_tree_reset(s)) != CASSPEC_OK) return rc;
  struct Expansion {
    int leaf, cfg, first;  // a branch node of an expansion and its top-1 child
  };
  std::vector<Expansion> exps;
  int32_t par[kMaxTree], tok[kMaxTree], ncfg[kMaxTree];
  int n = 1;
  tok[0] = root_token;
  par[0] = -1;
  while (true) {
    int leaf = -1, c = -1, k = 0;
    rc = casspec_dytc_tree_plan(s, &leaf, &c, &k);
    if (rc < 0) return rc;
    if (rc == 0) break;
    if ((rc = casspec_dytc_tree_get(s, &n, par, tok, ncfg, nullptr)) != CASSPEC_OK) return rc;
    tok[0] = root_token;
    // the chosen draft processes root .. leaf as one chain (valid for any layer mask), then each
    // drafted token in turn; the argmax of the last processed node is the next drafted token
    int32_t chain[kMaxTree];
    int len = 0;
    for (int v = leaf; v >= 0; v = par[v]) chain[len++] = v;
    int32_t ctok[kMaxTree], cpar[kMaxTree];
    for (int i = 0; i < len; ++i) {
      ctok[i] = tok[chain[len - 1 - i]];
      cpar[i] = i - 1;
    }
    if (cfgs[c].pld_n_max > 0 && cfgs[c].vc) {
      // the vertical cascade VC(model draft, prompt lookup), one holistic round: the lookup proposes
      // up to k tokens after history + path, the model draft runs once over root .. leaf plus the
      // proposals (a chain), and its greedy prefix match plus its own next token are appended
      if (history == nullptr || hist_len < 1) return CASSPEC_E_INVAL;
      const int kq = std::min(k, kMaxTree - len);
      int j = 0;
      int32_t pr[kMaxTree + 2];
      if (kq > 0) {
        if (len > 1)
          CK(cudaMemcpyAsync(history + hist_len, ctok + 1, (size_t)(len - 1) * 4, cudaMemcpyHostToDevice, m->stream));
        if ((rc = casspec_pld_draft(history, hist_len + len - 1, 1, cfgs[c].pld_n_max, kq, d_pld, m->stream)) !=
            CASSPEC_OK)
          return rc;
        if ((rc = read_dev_i32(m, d_pld, 2 + kq, pr)) != CASSPEC_OK) return rc;
        j = std::min(std::max(pr[1], 0), kq);
      }
      for (int i = 0; i < j; ++i) {
        ctok[len + i] = pr[2 + i];
        cpar[len + i] = len + i - 1;
      }
      casspec_kv_reset_tree(kv);
      CK(cudaMemcpyAsync(d_tok, ctok, (size_t)(len + j) * 4, cudaMemcpyHostToDevice, m->stream));
      CK(cudaMemcpyAsync(d_par, cpar, (size_t)(len + j) * 4, cudaMemcpyHostToDevice, m->stream));
      if ((rc = casspec_tree_step(m, kv, d_tok, d_par, len + j, cfgs[c].skip_mask, cfgs[c].quant_mode, nullptr)) !=
          CASSPEC_OK)
        return rc;
      int32_t am[kMaxTree + 1], drafted[kMaxTree + 1];
      if ((rc = read_dev_i32(m, d_am + (len - 1), j + 1, am)) != CASSPEC_OK) return rc;
      const int cnt = casspec_vc_accept(pr + 2, j, am, drafted);
      if (cnt < 0) return cnt;
      const int first = n;
      rc = casspec_dytc_tree_extend(s, leaf, c, cnt, drafted);
      if (rc < 0) return rc;
      if (rc > 0) exps.push_back({leaf, c, first});
      if (rc < cnt) break;  // the tree is full
      continue;
    }
    if (cfgs[c].pld_n_max > 0) {
      // the prompt-lookup bottom draft: the path below the root continues the committed history
      if (history == nullptr || hist_len < 1) return CASSPEC_E_INVAL;
      if (len > 1)
        CK(cudaMemcpyAsync(history + hist_len, ctok + 1, (size_t)(len - 1) * 4, cudaMemcpyHostToDevice, m->stream));
      if ((rc = casspec_pld_draft(history, hist_len + len - 1, 1, cfgs[c].pld_n_max, k, d_pld, m->stream)) != CASSPEC_OK)
        return rc;
      int32_t pr[kMaxTree + 2];
      if ((rc = read_dev_i32(m, d_pld, 2 + k, pr)) != CASSPEC_OK) return rc;
      if (pr[1] < 1) {  // no earlier occurrence: nothing drafted, a failure of this configuration
        casspec_dytc_record(s, c, 0);
        break;
      }
      const int first = n;
      rc = casspec_dytc_tree_extend(s, leaf, c, pr[1], pr + 2);
      if (rc < 0) return rc;
      if (rc > 0) exps.push_back({leaf, c, first});
      if (rc < pr[1]) break;  // the tree is full
      continue;
    }
    if (K > 1) {
      // the branches: the leaf and its active siblings; the draft runs over root .. leaf plus the
      // siblings (children of the leaf's parent, slot len - 2), so the branches' rows are contiguous
      int32_t br[kMaxTree];
      int nb = 0;
      if ((rc = casspec_dytc_tree_begin(s, leaf, 1, br, &nb)) != CASSPEC_OK) return rc;
      for (int b = 1; b < nb; ++b) {
        ctok[len + b - 1] = tok[br[b]];
        cpar[len + b - 1] = len - 2;
      }
      int n_dev = len + nb - 1;  // tree slots the draft holds (distinct nodes of the tree)
      casspec_kv_reset_tree(kv);
      CK(cudaMemcpyAsync(d_tok, ctok, (size_t)n_dev * 4, cudaMemcpyHostToDevice, m->stream));
      CK(cudaMemcpyAsync(d_par, cpar, (size_t)n_dev * 4, cudaMemcpyHostToDevice, m->stream));
      if ((rc = casspec_tree_step(m, kv, d_tok, d_par, n_dev, cfgs[c].skip_mask, cfgs[c].quant_mode, dev_logits)) !=
          CASSPEC_OK)
        return rc;
      int slot[kMaxTree], cur[kMaxTree];
      for (int b = 0; b < nb; ++b) {
        slot[b] = len - 1 + b;
        cur[b] = br[b];
      }
      const float* rows = dev_logits + (size_t)(len - 1) * V;
      bool full = false;
      for (int pos = 0; pos < k && !full; ++pos) {
        if ((rc = casspec_topk(rows, nb, V, K, d_tki, d_tkp, m->stream)) != CASSPEC_OK) return rc;
        int32_t ids[kMaxTree * CASSPEC_TOPK_MAX];
        float pr[kMaxTree * CASSPEC_TOPK_MAX];
        CK(cudaMemcpyAsync(pr, d_tkp, (size_t)nb * K * 4, cudaMemcpyDeviceToHost, m->stream));
        if ((rc = read_dev_i32(m, d_tki, nb * K, ids)) != CASSPEC_OK) return rc;
        int nxt = 0;
        for (int b = 0; b < nb; ++b) {
          const int child = casspec_dytc_tree_add(s, cur[b], c, ids + b * K, pr + b * K, K);
          if (child < 0) return child;
          if (child == 0) {  // the tree is full
            full = true;
            break;
          }
          if (pos == 0) exps.push_back({cur[b], c, child});
          cur[nxt] = child;
          slot[nxt] = slot[b];
          ctok[nxt] = ids[b * K];
          ++nxt;
        }
        if (full || pos + 1 == k) break;
        int tree_n = 0;
        if ((rc = casspec_dytc_tree_get(s, &tree_n, nullptr, nullptr, nullptr, nullptr)) != CASSPEC_OK) return rc;
        if (tree_n >= prm.m_max) break;
        // the next position: the branches' top-1 children, one tree step over all of them
        nb = nxt;
        for (int b = 0; b < nb; ++b) {
          cpar[n_dev + b] = slot[b];
          slot[b] = n_dev + b;
        }
        CK(cudaMemcpyAsync(d_tok + n_dev, ctok, (size_t)nb * 4, cudaMemcpyHostToDevice, m->stream));
        CK(cudaMemcpyAsync(d_par + n_dev, cpar + n_dev, (size_t)nb * 4, cudaMemcpyHostToDevice, m->stream));
        if ((rc = casspec_tree_step(m, kv, d_tok + n_dev, d_par + n_dev, nb, cfgs[c].skip_mask, cfgs[c].quant_mode,
                                    dev_logits)) != CASSPEC_OK)
          return rc;
        n_dev += nb;
        rows = dev_logits;
      }
      if (full) break;
      continue;
    }
    casspec_kv_reset_tree(kv);
    CK(cudaMemcpyAsync(d_tok, ctok, (size_t)len * 4, cudaMemcpyHostToDevice, m->stream));
    CK(cudaMemcpyAsync(d_par, cpar, (size_t)len * 4, cudaMemcpyHostToDevice, m->stream));
    if ((rc = casspec_tree_step(m, kv, d_tok, d_par, len, cfgs[c].skip_mask, cfgs[c].quant_mode, nullptr)) != CASSPEC_OK)
      return rc;
    int32_t drafted[kMaxTree];
    if ((rc = read_dev_i32(m, d_am + (len - 1), 1, &drafted[0])) != CASSPEC_OK) return rc;
    const int room = std::min(k, kMaxTree - len);  // physical tree slots of this expansion
    for (int i = 1; i < room; ++i) {
      ctok[len + i - 1] = drafted[i - 1];
      cpar[len + i - 1] = len + i - 2;
      CK(cudaMemcpyAsync(d_tok + len + i - 1, &ctok[len + i - 1], 4, cudaMemcpyHostToDevice, m->stream));
      CK(cudaMemcpyAsync(d_par + len + i - 1, &cpar[len + i - 1], 4, cudaMemcpyHostToDevice, m->stream));
      if ((rc = casspec_tree_step(m, kv, d_tok + len + i - 1, d_par + len + i - 1, 1, cfgs[c].skip_mask,
                                  cfgs[c].quant_mode, nullptr)) != CASSPEC_OK)
        return rc;
      if ((rc = read_dev_i32(m, d_am, 1, &drafted[i])) != CASSPEC_OK) return rc;
    }
    const int first = n;
    rc = casspec_dytc_tree_extend(s, leaf, c, room, drafted);
    if (rc < 0) return rc;
    if (rc > 0) exps.push_back({leaf, c, first});
    if (rc < room) break;  // the tree is full
  }
  if ((rc = casspec_dytc_tree_get(s, &n, par, tok, ncfg, nullptr)) != CASSPEC_OK) return rc;
  tok[0] = root_token;
  // verification by the target model over the whole tree, greedy acceptance
  casspec_kv_reset_tree(kv);
  CK(cudaMemcpyAsync(d_tok, tok, (size_t)n * 4, cudaMemcpyHostToDevice, m->stream));
  CK(cudaMemcpyAsync(d_par, par, (size_t)n * 4, cudaMemcpyHostToDevice, m->stream));
  if ((rc = casspec_tree_step(m, kv, d_tok, d_par, n, nullptr, 0, nullptr)) != CASSPEC_OK) return rc;
  if ((rc = casspec_accept_greedy(m, nullptr, d_tok, d_par, n, d_acc)) != CASSPEC_OK) return rc;
  int32_t acc[kMaxTree + 2];
  if ((rc = read_dev_i32(m, d_acc, n + 2, acc)) != CASSPEC_OK) return rc;
  const int L = acc[0];
  if (L < 1 || L > n) return CASSPEC_E_TREE;
  std::vector<uint8_t> on_path(n, 0);
  for (int i = 1; i <= L; ++i)
    if (acc[i] >= 0 && acc[i] < n) on_path[acc[i]] = 1;
  // first-draft-token outcomes of the expansion branches the target accepted (Sec. 4.2)
  for (const auto& e : exps)
    if (on_path[e.leaf]) casspec_dytc_record(s, e.cfg, on_path[e.first]);
  casspec_dytc_end_step(s);
  const long long p_upper = kv->P_upper;
  if ((rc = casspec_kv_compact(kv, d_acc)) != CASSPEC_OK) return rc;
  kv->P_upper = p_upper + L;  // the accepted length is known here: keep the capacity bound exact
  for (int i = 2; i <= L; ++i) out_tokens[i - 2] = tok[acc[i]];
  out_tokens[L - 1] = acc[L + 1];  // the bonus token: the next round's root
  *n_out = L;
  if (n_drafted_out) *n_drafted_out = n - 1;
  return CASSPEC_OK;
}
