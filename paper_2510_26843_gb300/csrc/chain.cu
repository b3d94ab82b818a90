// Persistent projection chain on the 5th-generation tensor cores (tcgen05 + TMEM, bulk copies + TMA).
//
// One launch runs a list of dependent projections of a tree step -- e.g. Wo (+residual), Wgate/Wup
// (+SwiGLU), Wdown (+residual) and the next layer's Wqkv (+rotary, K/V write) or the LM head
// (+argmax) -- with one CTA per SM.
//
// Work split: every projection Y[token][row] = sum_k X[token][k] W[row][k] is divided among the CTAs
// by OUTPUT ROWS.  CTA c owns a contiguous slice of 16-row groups (row_slice) and runs the whole K
// range for it.  The residual projections (Wo, Wdown: few rows per CTA) may instead give a slice to a
// cluster pair of CTAs, each running one half of K (S = 2); the pair adds its two partials through
// distributed shared memory as partial(rank 0) + partial(rank 1) on both CTAs.  Either way each output
// is reduced in one fixed order, so results do not depend on timing.
//
// MMA shape: the tokens are on M.  A = the split activation of one 64-column k-block, the hi plane in
// rows 0..63 and the lo plane in rows 64..127 (16 KB, 128-byte swizzle, TMA); B = the CTA's weight
// rows of that k-block (N = slice rows <= 256); D in TMEM, lane = plane row, column = output row.
// Two issuing threads take alternate k-blocks, each into its own accumulator.  The epilogue adds the
// accumulators, then the lo-plane lane to the hi-plane lane of each token, so 16 significant bits of
// the activation reach the fp32 accumulation.
//
// Weights are stored pre-packed per CTA (pack_rows_kernel) as the 128-byte-swizzled shared-memory
// image of the slice's k-blocks, in the order the CTA consumes them, so the weight producer streams
// them with plain bulk copies into a ring of 32 KB stages and never waits on activations: the weight
// stream runs on across phase boundaries.
//
// Phases are linked by per-k-block readiness counters instead of a grid barrier: a CTA counts the
// rows it finished into the counter of every 64-column block its slice touches, and a consumer loads
// k-block k once its counter holds all of the block's rows.  Each CTA walks its k-blocks starting
// from the block that its own slice of the producing projection feeds (rotated order, baked into the
// packed weights), so the first loads of a phase wait only on the CTA itself and its neighbours.
//
// Warps: 0 weight producer, 1 and 7 MMA issuers (warp 1 owns TMEM), 2-5 epilogue (warps 4, 5 hold
// the hi-plane lanes and run the per-token epilogue; warps 2, 3 hand over the lo-plane lanes through
// shared memory), 6 activation producer (the whole warp polls the readiness counters of 32 upcoming
// k-blocks at once).  Every wait is bounded (2 s) and reports CASSPEC_E_TIMEOUT instead of hanging.
#include "common.cuh"
#include "kernels.h"

namespace casspec {

constexpr int kChainThreads = 256;
constexpr uint32_t kWStage = 28672;  // weight ring stage: whole k-blocks of the CTA's slice
constexpr int kWStages = 4;
constexpr uint32_t kXStage = 16384;  // one k-block of the split activation: 128 rows x 128 B
constexpr int kXStages = 5;
constexpr int kRecvFloats = kPairMaxRows * 32;  // a pair partner's half-K partial of this CTA's 32 tokens
constexpr int kStgFloats = 2560;     // epilogue hand-over buffer: 32 rows x 64 tokens fp32 (two of them)
constexpr uint32_t kTmemCols = 512;  // one accumulator of up to 256 columns per MMA issuer

__host__ __device__ constexpr size_t chain_smem() {
  return 1024 + (size_t)kWStages * kWStage + (size_t)kXStages * kXStage + 2 * kStgFloats * 4 + kRecvFloats * 4 +
         128 * 4 + 512;
}
static_assert(chain_smem() <= 232448, "the chain's shared memory exceeds the 227 KB a CTA may use");
static_assert(kWStage % 1024 == 0 && kXStage % 1024 == 0, "ring stages keep the 1 KB alignment of the 128 B swizzle");
static_assert(kChainMaxSliceRows * 128 <= (int)kWStage && kChainMaxSliceRows <= 256, "a slice's k-block fits a weight stage");

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// generic-proxy global writes <-> async-proxy (TMA) reads of the split activations
__device__ __forceinline__ void fence_proxy_async_global() { asm volatile("fence.proxy.async.global;" ::: "memory"); }

// Wait until *p >= target (bounded; gives up on the CTA's abort flag).
__device__ __forceinline__ bool wait_count(const unsigned* p, unsigned target, volatile int* abort) {
  if (ld_acquire_u32(p) >= target) return true;
  const uint64_t t0 = globaltimer_ns();
  while (ld_acquire_u32(p) < target) {
    if (*abort) return false;
    if (globaltimer_ns() - t0 > kWaitLimitNs) return false;
  }
  return true;
}

// 8 fp32 -> 8 bf16 of the hi plane (bf16(x)) or of the lo plane (bf16(x - bf16(x)))
__device__ __forceinline__ uint4 split_pack8(const float* x, bool lo) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float a = x[2 * i], b = x[2 * i + 1];
    const uint16_t ha = f2bf(a), hb = f2bf(b);
    w[i] = lo ? pack_bf16x2(a - bf2f(ha), b - bf2f(hb)) : ((uint32_t)ha | ((uint32_t)hb << 16));
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

__global__ void __launch_bounds__(kChainThreads, 1)
    chain_kernel(const __grid_constant__ ChainMaps maps, const __grid_constant__ ChainArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* wring = smem;
  uint8_t* xring = wring + kWStages * kWStage;
  float* stg = reinterpret_cast<float*>(xring + kXStages * kXStage);  // [2][32][64]
  float* recv = stg + 2 * kStgFloats;                                 // [kPairMaxRows][32] from the partner
  float* rs = recv + kRecvFloats;                                     // [64] RMSNorm factors
  float* rs2 = rs + 64;                                               // [64] second half of the sums
  uint64_t* wfull = reinterpret_cast<uint64_t*>(rs2 + 64);
  uint64_t* wempty = wfull + kWStages;
  uint64_t* xfull = wempty + kWStages;
  uint64_t* xempty = xfull + kXStages;
  uint64_t* tfull = xempty + kXStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;  // [2]: one per MMA issuer
  uint64_t* pready = drain + 2;  // the partner CTA has written its half-K partial into `recv` (S = 2)
  uint64_t* pfree = pready + 1;  // the partner has consumed what this CTA wrote into its `recv`
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(pfree + 1);
  // [0] abort, [1] wait result, [2..5] accumulator-ready votes, [6] last CTA out
  volatile int* flags = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, cta = blockIdx.x;
  const int np = a.nphases;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kWStages; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], 2);  // released by both MMA issuers
    }
    for (int s = 0; s < kXStages; ++s) {
      mbar_init(&xfull[s], 1);
      mbar_init(&xempty[s], 1);  // released by the issuer that consumed the k-block
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 2);
      mbar_init(&tempty[b], 1);
    }
    mbar_init(&drain[0], 1);
    mbar_init(&drain[1], 1);
    mbar_init(pready, 1);
    mbar_init(pfree, 1);
    for (int f = 0; f < 8; ++f) flags[f] = 0;
    fence_mbar_init();
  }
  if (warp == 6 && lane == 0)
    for (int p = 0; p < np; ++p) tma_prefetch_desc(&maps.x[p]);
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (a.pairs) cluster_sync();  // the partner's barriers are initialised before any remote arrive
  const uint32_t tmem_base = *tmem_slot;
  pdl_trigger();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- weight producer (never waits on activations) ----------------
      const uint64_t pol = policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_parity = 0;
      for (int p = 0; p < np && !flags[0]; ++p) {
        const int mult = a.ph[p].epi == EPI_GLU ? 2 : 1;
        const int kb = a.ph[p].kb;
        const PhasePart s = phase_part(cta, G, a.ph[p].N / kRowGroup, kb, a.ph[p].S, a.ph[p].rot_groups);
        if (s.ng == 0) continue;
        const uint32_t chunk = (uint32_t)(s.ng * kRowGroup * mult) * 128u;  // one k-block of the slice
        const int kpb = (int)(kWStage / chunk);
        // the slice's packed stream; with S = 2 the second half of K follows the first
        const uint8_t* src = a.ph[p].wp + (size_t)s.g0 * kRowGroup * mult * kb * 128 + (size_t)s.klo * chunk;
        for (int j0 = 0; j0 < s.len; j0 += kpb) {
          const int nk = min(kpb, s.len - j0);
          if (!mbar_wait_bounded(&wempty[stage], phase ^ 1, flags)) {
            flags[0] = 1;
            set_status(a.status, CASSPEC_E_TIMEOUT);
            break;
          }
          const uint32_t bytes = (uint32_t)nk * chunk;
          mbar_expect_tx(&wfull[stage], bytes);
          armed |= 1u << stage;
          armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
          bulk_load_hint(wring + stage * kWStage, src + (size_t)j0 * chunk, bytes, &wfull[stage], pol);
          if (++stage == kWStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (flags[0]) {  // abort: let the copies already issued land before the CTA exits
        for (int s = 0; s < kWStages; ++s)
          if (armed & (1u << s)) mbar_wait_bounded(&wfull[s], (armed_parity >> s) & 1, nullptr);
      }
    }
  } else if (warp == 6) {
    // ---------------- activation producer (whole warp) ----------------
    // Inputs of a phase that reads an earlier kernel's output, and the readiness counters (reset by
    // the previous launch's last CTA), are valid only once the preceding kernels have completed.
    pdl_wait();
    const uint64_t pol = policy_evict_last();
    const uint32_t xbytes = 2u * (uint32_t)a.bn * 128u;
    int stage = 0;
    uint32_t phase = 0;
    uint32_t armed = 0, armed_parity = 0;
    bool ok = true;
    for (int p = 0; p < np && ok; ++p) {
      const int kb = a.ph[p].kb;
      const PhasePart s = phase_part(cta, G, a.ph[p].N / kRowGroup, kb, a.ph[p].S, a.ph[p].rot_groups);
      if (s.ng == 0) continue;
      const int in_phase = a.ph[p].in_phase, in_N = a.ph[p].in_N, in_S = a.ph[p].in_S;
      const int len = s.len;
      const unsigned* rdy = in_phase >= 0 ? a.ready + in_phase * kReadyPerPhase : nullptr;
      const unsigned extra = p == a.stall_phase ? 1u : 0u;  // test hook: a count that never completes
      int j = 0;
      while (j < len && ok) {
        int avail = len - j;
        if (rdy != nullptr) {
          // the lanes read the counters of the next 32 k-blocks at once (one round trip); the
          // consecutive ready ones from j on are loaded
          int jl = s.rot + j + lane;
          while (jl >= len) jl -= len;
          const int kl = s.klo + jl;
          const unsigned target = (unsigned)(min(64, in_N - 64 * kl) * in_S) + extra;
          const uint64_t t0 = globaltimer_ns();
          while (true) {
            const bool r = j + lane >= len || ld_acquire_u32(rdy + kl) >= target;
            const unsigned ball = __ballot_sync(0xffffffffu, r);
            avail = min(ball == 0xffffffffu ? 32 : __ffs(~ball) - 1, len - j);
            if (avail > 0) break;
            int give_up = (flags[0] || globaltimer_ns() - t0 > kWaitLimitNs) ? 1 : 0;
            give_up = __shfl_sync(0xffffffffu, give_up, 0);
            if (give_up) {
              ok = false;
              break;
            }
          }
          if (!ok) break;
          fence_proxy_async_global();
        }
        int issued_ok = 1;
        if (lane == 0) {
          for (int i = 0; i < avail; ++i) {
            int jk = s.rot + j + i;
            if (jk >= len) jk -= len;
            const int k = s.klo + jk;
            if (!mbar_wait_bounded(&xempty[stage], phase ^ 1, flags)) {
              issued_ok = 0;
              break;
            }
            mbar_expect_tx(&xfull[stage], xbytes);
            armed |= 1u << stage;
            armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
            uint8_t* sx = xring + stage * kXStage;
            if (a.bn == 64) {  // one 128-row box: hi plane rows 0..63, lo plane rows 64..127
              tma_load_2d(sx, &maps.x[p], &xfull[stage], k * 64, 0, pol);
            } else {
              tma_load_2d(sx, &maps.x[p], &xfull[stage], k * 64, 0, pol);          // hi plane -> rows 0..bn-1
              tma_load_2d(sx + 8192, &maps.x[p], &xfull[stage], k * 64, 64, pol);  // lo plane -> rows 64..
            }
            if (++stage == kXStages) {
              stage = 0;
              phase ^= 1;
            }
          }
        }
        ok = __shfl_sync(0xffffffffu, issued_ok, 0) != 0;
        j += avail;
      }
    }
    if (lane == 0) {
      if (!ok) {
        flags[0] = 1;
        set_status(a.status, CASSPEC_E_TIMEOUT);
      }
      if (flags[0]) {
        for (int s = 0; s < kXStages; ++s)
          if (armed & (1u << s)) mbar_wait_bounded(&xfull[s], (armed_parity >> s) & 1, nullptr);
      }
    }
  } else if (warp == 1 || warp == 7) {
    if (lane == 0) {
      // ---------------- MMA issuers ----------------
      // Two threads in two warps issue the MMAs, each into its own accumulator: the first takes the
      // even k-blocks of a phase, the second the odd ones (a single k-block: the first alone), four
      // k-steps per k-block.  A thread issues a tcgen05.mma only after its previous instructions, so
      // the loop between MMAs is kept to a few integer adds: descriptors are offsets from per-ring
      // bases, and one wait and one commit cover four MMAs.  The epilogue adds the accumulators.
      const int ib = warp == 1 ? 0 : 1;
      const uint64_t xd0 = sw128_kmajor_desc(smem_u32(xring));
      const uint64_t wd0 = sw128_kmajor_desc(smem_u32(wring));
      int ws = 0, xs = 0;
      uint32_t wph = 0, xph = 0;
      uint32_t used = 0;
      bool ok = true;
      for (int p = 0; p < np && ok; ++p) {
        const int mult = a.ph[p].epi == EPI_GLU ? 2 : 1;
        const int kb = a.ph[p].kb;
        const PhasePart s = phase_part(cta, G, a.ph[p].N / kRowGroup, kb, a.ph[p].S, a.ph[p].rot_groups);
        if (s.ng == 0) continue;
        const int ncols = s.ng * kRowGroup * mult;
        const uint32_t chunk = (uint32_t)ncols * 128u;
        const int kpb = (int)(kWStage / chunk);
        const uint32_t idesc = idesc_bf16_f32(128, ncols);
        // the accumulators are free once the previous phase's epilogue has read them
        if (!mbar_wait_bounded(tempty, (used & 1) ^ 1, flags)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(ib * ncols);
        uint32_t acc = 0;
        int j = 0;
        for (int j0 = 0; j0 < s.len && ok; j0 += kpb) {
          const int nk = min(kpb, s.len - j0);
          if (!mbar_wait_bounded(&wfull[ws], wph, flags)) {
            ok = false;
            break;
          }
          const uint64_t wd = wd0 + (uint64_t)((uint32_t)ws * (kWStage >> 4));
          for (int jj = 0; jj < nk; ++jj, ++j) {
            if ((j & 1) == ib) {
              if (!mbar_wait_bounded(&xfull[xs], xph, flags)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint64_t ad = xd0 + (uint64_t)((uint32_t)xs * (kXStage >> 4));
              const uint64_t bd = wd + (uint64_t)((uint32_t)jj * (chunk >> 4));
              tc_mma_bf16(d_tmem, ad, bd, idesc, acc);  // k-step 0: 32 B further along K per step
              tc_mma_bf16(d_tmem, ad + 2, bd + 2, idesc, 1u);
              tc_mma_bf16(d_tmem, ad + 4, bd + 4, idesc, 1u);
              tc_mma_bf16(d_tmem, ad + 6, bd + 6, idesc, 1u);
              acc = 1u;
              tc_commit(&xempty[xs]);
            }
            if (++xs == kXStages) {
              xs = 0;
              xph ^= 1;
            }
          }
          if (!ok) break;
          tc_commit(&wempty[ws]);
          if (++ws == kWStages) {
            ws = 0;
            wph ^= 1;
          }
        }
        if (!ok) break;
        tc_commit(tfull);
        ++used;
      }
      if (!ok) {
        flags[0] = 1;
        set_status(a.status, CASSPEC_E_TIMEOUT);
      }
      tc_commit(&drain[ib]);  // all MMAs complete before TMEM is released
      mbar_wait_bounded(&drain[ib], 0, nullptr);
    }
  } else {
    // ---------------- epilogue warps 2..5 ----------------
    // Control flow is identical in the four warps (every decision that follows a bounded wait is
    // voted through shared memory), so their named barriers always match, even after a timeout.
    const int q = warp & 3;             // TMEM lane quarter of this warp
    const bool hi = q < 2;              // lanes 0..63 hold the hi-plane rows, 64..127 the lo-plane rows
    const int t = (q & 1) * 32 + lane;  // token of this thread
    const int et = threadIdx.x - 64;    // 0..127
    auto bar = [] { named_bar_sync(1, 128); };
    pdl_wait();
    uint32_t used[2] = {0, 0};
    int pc = 0;
    uint32_t npair = 0;  // S = 2 phases done (parity of the pair barriers)
    for (int p = 0; p < np; ++p) {
      // The phase descriptor sits in parameter space behind a runtime index: copy what the loops use.
      const EpiParams ep = a.ph[p].ep;
      const int epi = a.ph[p].epi;
      const int mult = epi == EPI_GLU ? 2 : 1;
      const int S = a.ph[p].S;
      const PhasePart s = phase_part(cta, G, a.ph[p].N / kRowGroup, a.ph[p].kb, S, a.ph[p].rot_groups);
      if (s.ng == 0) continue;
      const int R = s.ng * kRowGroup;  // output rows (EPI_GLU: channels) of this CTA (S = 2: of the pair)
      const int r0 = s.g0 * kRowGroup;
      const int n = ep.n;
      const float* ss = a.ph[p].ss;
      const int buf = 0;  // one accumulator region (per issuer), reused phase after phase
      ++pc;

      // (1) the RMSNorm factor of this phase's tokens, once every producer has counted in (overlaps
      // this phase's MMAs): rs[t] = rsqrt(sum of the producers' partial sums of squares / K + eps)
      if (ss != nullptr) {
        const int in_phase = a.ph[p].in_phase;
        if (et == 0) {
          int ok = 1;
          if (in_phase >= 0) {
            const int Sin = a.ph[in_phase].S;
            const unsigned target = (unsigned)(min(a.ph[in_phase].N / kRowGroup, G / Sin) * Sin);
            ok = wait_count(a.done + in_phase, target, flags) ? 1 : 0;
            if (!ok) {
              flags[0] = 1;
              set_status(a.status, CASSPEC_E_TIMEOUT);
            }
          }
          flags[1] = ok;
        }
        bar();
        const bool ok = flags[1] != 0;
        if (ok) {
          const int parts = a.ph[p].ss_parts;
          const int tt = et & 63, half = et >> 6;
          const int c0 = half * (parts / 2), c1 = half ? parts : parts / 2;
          float acc = 0.f;
          for (int c = c0; c < c1; c += 16) {  // 16 loads in flight, summed in a fixed order
            float v16[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) v16[k] = c + k < c1 ? __ldcg(ss + (size_t)(c + k) * 64 + tt) : 0.f;
#pragma unroll
            for (int k = 0; k < 16; ++k) acc += v16[k];
          }
          (half ? rs2 : rs)[tt] = acc;
        }
        bar();
        if (ok && et < 64) rs[et] = rsqrtf((rs[et] + rs2[et]) / (float)a.ph[p].K + a.ph[p].eps);
        bar();
      }

      // residual epilogue: this CTA's slice of the residual rows (written by this CTA's own earlier
      // phases, same slicing, or by an earlier kernel) is loaded while the MMAs run
      // Everything the epilogue reads from memory that does not depend on this phase's result is
      // loaded while the MMAs run: the residual rows and the next norm's gains (S = 2), and the
      // rotary coefficients of the first 16-row group (QKV).
      float4 xo[5], gq[5], csn[4];  // (S = 2: up to kPairMaxRows / 4 = 20 rows per thread)
#pragma unroll
      for (int k = 0; k < 5; ++k) xo[k] = gq[k] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int k = 0; k < 4; ++k) csn[k] = make_float4(0.f, 0.f, 0.f, 0.f);
      // S = 2: rank r finishes tokens 32 r .. 32 r + 31, four threads per token, R / 4 rows each
      const int t2 = 32 * s.rank + (et >> 2), cq = et & 3, wq = R / 4, c0q = cq * wq;
      if (S == 2) {
        if (t2 < n) {
#pragma unroll
          for (int k = 0; k < 5; ++k)
            if (4 * k < wq) xo[k] = __ldcg(reinterpret_cast<const float4*>(ep.y + (size_t)t2 * ep.ldy + r0 + c0q) + k);
        }
        if (ep.xa_out != nullptr) {
#pragma unroll
          for (int k = 0; k < 5; ++k)
            if (4 * k < wq) gq[k] = __ldg(reinterpret_cast<const float4*>(ep.g_next + r0 + c0q) + k);
        }
      }
      int pos_t = 0, P = 0;
      if (epi == EPI_QKV) {
        P = __ldcg(ep.dP);
        pos_t = t < n ? __ldcg(ep.pos + t) : 0;
      }
      // rotary (cos, sin) of 16-row group `col` for this thread's token (zero for the v part)
      auto rope_load = [&](int col, float4* dst) {
        const int g = col / kRowGroup, gpp = ep.d / kRowGroup, part = g / gpp, gp = g - part * gpp;
        const int gph = ep.hd / kRowGroup, head = gp / gph, a0 = (gp - head * gph) * 8;
        if (part < 2) {
          const float4* cs = reinterpret_cast<const float4*>(ep.rope + (size_t)pos_t * (ep.hd >> 1) + a0);
#pragma unroll
          for (int k = 0; k < 4; ++k) dst[k] = __ldg(cs + k);
        }
      };
      if (epi == EPI_QKV && hi) rope_load(r0, csn);

      // (2) the accumulator of this phase
      const bool got = mbar_wait_bounded(&tfull[buf], used[buf] & 1, flags);
      if (lane == 0) flags[2 + q] = got ? 1 : 0;
      bar();
      const bool ready = flags[2] && flags[3] && flags[4] && flags[5];
      used[buf]++;
      bar();  // every warp has read the votes before they are rewritten
      if (!ready) {
        if (et == 0) {
          flags[0] = 1;
          set_status(a.status, CASSPEC_E_TIMEOUT);
        }
        continue;
      }
      tc_fence_after();
      const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16);
      const uint32_t acc2 = (uint32_t)(R * mult);  // the second issuer's accumulator
      const bool two = s.len > 1;                   // a single k-block leaves the second one unwritten

      if (S == 2) {
        // (3') the pair's residual projection: this CTA holds one half of K for the pair's rows.  Its
        // partial (hi + lo planes, both accumulators) goes to the staging area as [row][token]; the
        // partner reads it through distributed shared memory, and each CTA finishes 32 tokens of the
        // pair's rows as partial(rank 0) + partial(rank 1), in that order on both.
        float* Pp = stg;
        const int nch = R / 16;  // <= kPairMaxRows / 16 = 5: read in passes of up to 4 chunks
        for (int cb = 0; cb < nch; cb += 4) {
          float pv[4][16];  // both accumulators of the warp's lanes
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            if (cb + c < nch) {
              float w2[16];
              tmem_ld_x16(tbase + (uint32_t)((cb + c) * 16), pv[c]);
              if (two) tmem_ld_x16(tbase + acc2 + (uint32_t)((cb + c) * 16), w2);
              tmem_ld_wait();
              if (two) {
#pragma unroll
                for (int i = 0; i < 16; ++i) pv[c][i] += w2[i];
              }
            }
          }
          if (!hi) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
              if (cb + c < nch) {
#pragma unroll
                for (int i = 0; i < 16; ++i) Pp[((cb + c) * 16 + i) * 64 + t] = pv[c][i];
              }
          }
          tc_fence_before();
          bar();  // (the lo group's next pass writes other rows than the hi group adds here)
          if (hi) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
              if (cb + c < nch) {
#pragma unroll
                for (int i = 0; i < 16; ++i) Pp[((cb + c) * 16 + i) * 64 + t] += pv[c][i];
              }
          }
        }
        if (et == 0) mbar_arrive(&tempty[buf]);  // TMEM read: the next phase's MMAs may start
        // the partner's previous S = 2 phase has consumed what this CTA wrote into its `recv`
        if (et == 0) {
          int okf = 1;
          if (npair > 0 && !mbar_wait_cluster_bounded(pfree, (uint32_t)((npair - 1) & 1), flags)) {
            okf = 0;
            flags[0] = 1;
            set_status(a.status, CASSPEC_E_TIMEOUT);
          }
          flags[1] = okf;
        }
        bar();
        const int peer = s.rank ^ 1;
        if (flags[1]) {
          // push the partner's 32 tokens of this partial into its `recv` ([row][32], 16-byte stores)
          const uint32_t rv = map_to_rank(smem_u32(recv), (uint32_t)peer);
          for (int e = et; e < R * 8; e += 128) {
            const int row = e >> 3, tq = (e & 7) * 4;
            const float4 val = *reinterpret_cast<const float4*>(Pp + row * 64 + 32 * peer + tq);
            st_dsmem_f4(rv + (uint32_t)((row * 32 + tq) * 4), val);
          }
        }
        bar();
        if (et == 0) {
          int okp = flags[1];
          if (okp) {
            mbar_arrive_remote(map_to_rank(smem_u32(pready), (uint32_t)peer));
            okp = mbar_wait_cluster_bounded(pready, (uint32_t)(npair & 1), flags) ? 1 : 0;
            if (!okp) {
              flags[0] = 1;
              set_status(a.status, CASSPEC_E_TIMEOUT);
            }
          }
          flags[1] = okp;
        }
        bar();
        // this CTA's 32 tokens: partial(rank 0) + partial(rank 1), the same order on both CTAs
        float v[20];
        if (flags[1]) {
          const int tl = t2 - 32 * s.rank;  // token within this CTA's half
#pragma unroll
          for (int c = 0; c < 20; ++c)
            if (c < wq) {
              const float own = Pp[(c0q + c) * 64 + t2], got = recv[(c0q + c) * 32 + tl];
              v[c] = s.rank == 0 ? own + got : got + own;
            }
        }
        bar();
        // `recv` is read: the partner may fill it for the next pair phase (released before this CTA's
        // global stores below, which it does not depend on)
        if (et == 0 && flags[1]) mbar_arrive_remote(map_to_rank(smem_u32(pfree), (uint32_t)peer));
        if (flags[1]) {
          float ssq2 = 0.f;
          if (t2 < n) {
            float nv[20];
#pragma unroll
            for (int k = 0; k < 5; ++k) {
              nv[4 * k + 0] = xo[k].x + v[4 * k + 0];
              nv[4 * k + 1] = xo[k].y + v[4 * k + 1];
              nv[4 * k + 2] = xo[k].z + v[4 * k + 2];
              nv[4 * k + 3] = xo[k].w + v[4 * k + 3];
            }
            const int col = r0 + c0q;
            float4* dst = reinterpret_cast<float4*>(ep.y + (size_t)t2 * ep.ldy + col);
#pragma unroll
            for (int k = 0; k < 5; ++k)
              if (4 * k < wq) dst[k] = make_float4(nv[4 * k], nv[4 * k + 1], nv[4 * k + 2], nv[4 * k + 3]);
#pragma unroll
            for (int i = 0; i < 20; ++i)
              if (i < wq) ssq2 += nv[i] * nv[i];
            if (ep.xa_out != nullptr) {
#pragma unroll
              for (int k = 0; k < 5; ++k) {
                if (4 * k < wq) {
                  const float4 g4 = gq[k];
                  const float g[4] = {nv[4 * k] * g4.x, nv[4 * k + 1] * g4.y, nv[4 * k + 2] * g4.z, nv[4 * k + 3] * g4.w};
                  uint16_t h[4];
                  float l[4];
#pragma unroll
                  for (int e2 = 0; e2 < 4; ++e2) {
                    h[e2] = f2bf(g[e2]);
                    l[e2] = g[e2] - bf2f(h[e2]);
                  }
                  *reinterpret_cast<uint2*>(ep.xa_out + (size_t)t2 * ep.ldy + col + 4 * k) =
                      make_uint2((uint32_t)h[0] | ((uint32_t)h[1] << 16), (uint32_t)h[2] | ((uint32_t)h[3] << 16));
                  *reinterpret_cast<uint2*>(ep.xa_out + (size_t)(64 + t2) * ep.ldy + col + 4 * k) =
                      make_uint2(pack_bf16x2(l[0], l[1]), pack_bf16x2(l[2], l[3]));
                }
              }
            }
          }
          // the token's sum of squares over the pair's rows: its four threads, in a fixed order
          ssq2 += __shfl_xor_sync(0xffffffffu, ssq2, 1);
          ssq2 += __shfl_xor_sync(0xffffffffu, ssq2, 2);
          if (cq == 0 && ep.ss_out != nullptr) ep.ss_out[(size_t)s.slice * 64 + t2] = t2 < n ? ssq2 : 0.f;
        }
        ++npair;
      } else {
        // (3) 16 output rows (EPI_GLU: 16 channels, gate and up) at a time: the lo-plane warps hand
        // their lanes to the hi-plane warps through a double-buffered staging area
        float ssq = 0.f;                       // EPI_RESID: sum of squares of the updated rows
        float m1 = -INFINITY, m2 = -INFINITY;  // EPI_LMHEAD: max, second max
        int i1 = 0x7fffffff;                   //            argmax
        const float rsv = (ss != nullptr) ? rs[t] : 1.f;
        const int nchunks = R / 16;
        for (int c = 0; c < nchunks; ++c) {
          float* sb = stg + (c & 1) * kStgFloats;
          float v[32];
          // both lane groups read this chunk of both accumulators, then the lo-plane lanes hand over
          tmem_ld_x16(tbase + (uint32_t)(c * 16), v);
          if (mult == 2) tmem_ld_x16(tbase + (uint32_t)(R + c * 16), v + 16);
          if (two) {
            float w2[32];
            tmem_ld_x16(tbase + acc2 + (uint32_t)(c * 16), w2);
            if (mult == 2) tmem_ld_x16(tbase + acc2 + (uint32_t)(R + c * 16), w2 + 16);
            tmem_ld_wait();
  #pragma unroll
            for (int i = 0; i < 32; ++i) v[i] += w2[i];
          } else {
            tmem_ld_wait();
          }
          if (!hi) {
  #pragma unroll
            for (int i = 0; i < 16; ++i) sb[i * 64 + t] = v[i];
            if (mult == 2) {
  #pragma unroll
              for (int i = 0; i < 16; ++i) sb[(16 + i) * 64 + t] = v[16 + i];
            }
          }
          bar();
          if (hi) {
  #pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = (v[i] + sb[i * 64 + t]) * rsv;
            if (mult == 2) {
  #pragma unroll
              for (int i = 0; i < 16; ++i) v[16 + i] = (v[16 + i] + sb[(16 + i) * 64 + t]) * rsv;
            }
            const int col = r0 + c * 16;  // first output row (channel) of the chunk
            if (t < n) {
              if (epi == EPI_RESID) {
                float nv[16];
                float4 ox[4];
  #pragma unroll
                for (int k = 0; k < 4; ++k) ox[k] = __ldcg(reinterpret_cast<const float4*>(ep.y + (size_t)t * ep.ldy + col) + k);
  #pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const float4 o4 = ox[k];
                  nv[4 * k + 0] = o4.x + v[4 * k + 0];
                  nv[4 * k + 1] = o4.y + v[4 * k + 1];
                  nv[4 * k + 2] = o4.z + v[4 * k + 2];
                  nv[4 * k + 3] = o4.w + v[4 * k + 3];
                }
                float4* dst = reinterpret_cast<float4*>(ep.y + (size_t)t * ep.ldy + col);
  #pragma unroll
                for (int k = 0; k < 4; ++k) dst[k] = make_float4(nv[4 * k], nv[4 * k + 1], nv[4 * k + 2], nv[4 * k + 3]);
  #pragma unroll
                for (int i = 0; i < 16; ++i) ssq += nv[i] * nv[i];
                if (ep.xa_out != nullptr) {
                  float g[16];
  #pragma unroll
                  for (int k = 0; k < 4; ++k) {
                    const float4 g4 = __ldg(reinterpret_cast<const float4*>(ep.g_next + col) + k);
                    g[4 * k] = nv[4 * k] * g4.x;
                    g[4 * k + 1] = nv[4 * k + 1] * g4.y;
                    g[4 * k + 2] = nv[4 * k + 2] * g4.z;
                    g[4 * k + 3] = nv[4 * k + 3] * g4.w;
                  }
                  uint4* xh = reinterpret_cast<uint4*>(ep.xa_out + (size_t)t * ep.ldy + col);
                  uint4* xl = reinterpret_cast<uint4*>(ep.xa_out + (size_t)(64 + t) * ep.ldy + col);
                  xh[0] = split_pack8(g, false);
                  xh[1] = split_pack8(g + 8, false);
                  xl[0] = split_pack8(g, true);
                  xl[1] = split_pack8(g + 8, true);
                }
              } else if (epi == EPI_GLU) {
                float u[16];
  #pragma unroll
                for (int i = 0; i < 16; ++i) {
                  const float gt = v[i];
                  // fast exponential and division: ~1e-6 relative error, below the 16-bit split
                  u[i] = __fdividef(gt, 1.f + __expf(-gt)) * v[16 + i];
                }
                uint4* uh = reinterpret_cast<uint4*>(ep.u_out + (size_t)t * ep.N + col);
                uint4* ul = reinterpret_cast<uint4*>(ep.u_out + (size_t)(64 + t) * ep.N + col);
                uh[0] = split_pack8(u, false);
                uh[1] = split_pack8(u + 8, false);
                ul[0] = split_pack8(u, true);
                ul[1] = split_pack8(u + 8, true);
              } else if (epi == EPI_QKV) {
                // a 16-row group holds 8 rotary pairs: rows 0..7 are dims a0..a0+7 of one head of q, k
                // or v, rows 8..15 their partners a0+hd/2 .. (the packing order, qkv_src_row)
                const int g = col / kRowGroup;
                const int gpp = ep.d / kRowGroup;  // groups per part (q, k, v)
                const int part = g / gpp;
                const int gp = g - part * gpp;
                const int gph = ep.hd / kRowGroup;  // groups per head
                const int head = gp / gph;
                const int a0 = (gp - head * gph) * 8;
                const int half = ep.hd >> 1;
                float o[16];
                float4 cur[4];
  #pragma unroll
                for (int k = 0; k < 4; ++k) cur[k] = csn[k];
                if (c + 1 < nchunks) rope_load(col + 16, csn);  // the next group's, in flight meanwhile
                if (part < 2) {
                  float cv[8], sv[8];
  #pragma unroll
                  for (int k = 0; k < 4; ++k) {
                    const float4 c4 = cur[k];  // (cos, sin) of two frequencies
                    cv[2 * k] = c4.x;
                    sv[2 * k] = c4.y;
                    cv[2 * k + 1] = c4.z;
                    sv[2 * k + 1] = c4.w;
                  }
  #pragma unroll
                  for (int i = 0; i < 8; ++i) {
                    const float x = v[i], y = v[8 + i];
                    o[i] = x * cv[i] - y * sv[i];
                    o[8 + i] = y * cv[i] + x * sv[i];
                  }
                } else {
  #pragma unroll
                  for (int i = 0; i < 16; ++i) o[i] = v[i];
                }
                const uint4 first = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]),
                                               pack_bf16x2(o[4], o[5]), pack_bf16x2(o[6], o[7]));
                const uint4 second = make_uint4(pack_bf16x2(o[8], o[9]), pack_bf16x2(o[10], o[11]),
                                                pack_bf16x2(o[12], o[13]), pack_bf16x2(o[14], o[15]));
                uint16_t* base;
                if (part == 0)
                  base = ep.q_out + (size_t)t * ep.d + head * ep.hd;
                else
                  base = (part == 1 ? ep.kc : ep.vc) + ((size_t)head * ep.ctx + (P + ep.T + t)) * ep.hd;
                *reinterpret_cast<uint4*>(base + a0) = first;
                *reinterpret_cast<uint4*>(base + half + a0) = second;
              } else {  // EPI_LMHEAD
                // ep.N = vocabulary size (a multiple of 8); rows beyond it are zero padding of the last group
                if (ep.logits != nullptr) {
                  float4* dst = reinterpret_cast<float4*>(ep.logits + (size_t)t * ep.N + col);
  #pragma unroll
                  for (int k = 0; k < 4; ++k)
                    if (col + 4 * k < ep.N) dst[k] = make_float4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
                }
  #pragma unroll
                for (int i = 0; i < 16; ++i) {  // increasing vocabulary id: ties keep the lowest
                  if (col + i >= ep.N) break;
                  if (v[i] > m1) {
                    m2 = m1;
                    m1 = v[i];
                    i1 = col + i;
                  } else if (v[i] > m2) {
                    m2 = v[i];
                  }
                }
              }
            }
          }
        }
        // every TMEM read of this buffer is complete: hand it back to the MMA issuer
        tc_fence_before();
        bar();
        if (et == 0) mbar_arrive(&tempty[buf]);
        // per-slice partial results (slice index = CTA index)
        if (hi) {
          if (epi == EPI_RESID && ep.ss_out != nullptr) ep.ss_out[(size_t)s.slice * 64 + t] = t < n ? ssq : 0.f;
          if (epi == EPI_LMHEAD) {
            ep.am_v1[(size_t)s.slice * 64 + t] = m1;
            ep.am_i1[(size_t)s.slice * 64 + t] = i1 == 0x7fffffff ? r0 : i1;
            ep.am_v2[(size_t)s.slice * 64 + t] = m2;
          }
        }
      }
      // (4) publish: the slice's rows into the readiness counters of the 64-column blocks they
      // belong to, and the CTA into the phase's completion count
      fence_proxy_async_global();
      __threadfence();
      bar();
      if (et == 0) {
        __threadfence();
        if (a.ph[p].publish) {
          unsigned* rdy = a.ready + p * kReadyPerPhase;
          for (int k = r0 / 64; k * 64 < r0 + R; ++k) {
            const int lo = max(r0, 64 * k), hi_ = min(r0 + R, 64 * k + 64);
            atomicAdd(rdy + k, (unsigned)(hi_ - lo));
          }
        }
        atomicAdd(a.done + p, 1u);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (a.pairs) cluster_sync();  // no CTA leaves while its partner may still address its shared memory
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
  // The last CTA out returns the readiness and completion counters to zero for the next launch
  // (they belong to the previous launch until it completes, hence the dependency wait).
  if (threadIdx.x == 0) {
    pdl_wait();
    __threadfence();
    flags[6] = atomicAdd(a.done + kMaxPhases, 1u) == (unsigned)(G - 1) ? 1 : 0;
  }
  __syncthreads();
  if (flags[6]) {
    __threadfence();
    for (int i = threadIdx.x; i < np * kReadyPerPhase; i += blockDim.x) a.ready[i] = 0u;
    if (threadIdx.x <= kMaxPhases) a.done[threadIdx.x] = 0u;
  }
}

// ---------------------------------------------------------------------------------------------
// packing of a projection's weights into the per-CTA stream the chain consumes
// ---------------------------------------------------------------------------------------------
// Source row of packed row `row` of a QKV projection: each 16-row group holds dims a0..a0+7 and
// a0+hd/2 .. a0+hd/2+7 of one head of q, k or v (8 rotary pairs), a0 = 8 * (group within the head).
__host__ __device__ inline int qkv_src_row(int row, int d, int hd) {
  const int g = row / kRowGroup, i = row % kRowGroup;
  const int gpp = d / kRowGroup, part = g / gpp, gp = g - part * gpp;
  const int gph = hd / kRowGroup, head = gp / gph, a0 = (gp - head * gph) * 8;
  return part * d + head * hd + (i < 8 ? a0 + i : hd / 2 + a0 + (i - 8));
}

// One thread per 16-byte chunk of the packed image.  Logical rows `ch` (0 .. N-1; PACK_GLU: gate
// channels, each packed twice: gate row in the slice's first half, up row in its second half);
// source rows at or beyond `rows` (N rounded up to whole groups) are packed as zeros.
// CTA c's slice is packed contiguously: for its j-th consumed k-block (k = (k0 + j) mod kb) the
// slice's rows (128 bytes each, zero beyond K) in the 128-byte-swizzled image (16-byte chunk index
// XOR row % 8), so one bulk copy lands a k-block exactly as a swizzled TMA box would.
__global__ void pack_rows_kernel(const uint16_t* __restrict__ W, const uint16_t* __restrict__ W2, int N, int rows,
                                 int K, int kb, int G, int S, int kind, int d, int hd, int rot_groups, long long chunks,
                                 uint8_t* __restrict__ out) {
  const int mult = kind == PACK_GLU ? 2 : 1;
  const int Gs = G / S;  // row slices
  for (long long it = blockIdx.x * (long long)blockDim.x + threadIdx.x; it < chunks;
       it += (long long)gridDim.x * blockDim.x) {
    const int cch = (int)(it & 7);
    const long long rk = it >> 3;
    const int k = (int)(rk % kb);  // source k-block
    const long long lr = rk / kb;  // logical row x half
    const int h = (int)(lr % mult);
    const int ch = (int)(lr / mult);
    const int NG = N / kRowGroup;
    const int sl = row_slice_owner(ch / kRowGroup, NG, Gs);
    // the CTA that consumes k-block k of this slice, and where in its stream
    const int rank = (S == 2 && k >= kb / 2) ? 1 : 0;
    const PhasePart q = phase_part(sl * S + rank, G, NG, kb, S, rot_groups);
    const int R = q.ng * kRowGroup;
    const int r = h * R + (ch - q.g0 * kRowGroup);  // row within the slice's packed k-block
    const int j = (k - q.klo - q.rot + 2 * q.len) % q.len;  // consumption index within the CTA's k-range
    int src_row = ch;
    const uint16_t* src = W;
    if (kind == PACK_GLU) {
      src = h == 0 ? W : W2;
    } else if (kind == PACK_QKV) {
      src_row = qkv_src_row(ch, d, hd);
    }
    const int col = k * 64 + cch * 8;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (col < K && src_row < rows) v = *reinterpret_cast<const uint4*>(src + (size_t)src_row * K + col);
    // slice stream: [k-blocks of rank 0 in consumption order][k-blocks of rank 1 ...]
    const size_t slice_base = (size_t)q.g0 * kRowGroup * mult * kb * 128;
    const size_t off = slice_base + ((size_t)(q.klo + j) * R * mult + r) * 128 + (size_t)((cch ^ (r & 7)) << 4);
    *reinterpret_cast<uint4*>(out + off) = v;
  }
}

size_t pack_rows_bytes(int N, int K, int kind) {
  return (size_t)N * (kind == PACK_GLU ? 2 : 1) * (size_t)((K + 63) / 64) * 128;
}

cudaError_t launch_pack_rows(const uint16_t* W, const uint16_t* W2, int N, int rows, int K, int G, int S, int kind,
                             int d, int hd, int rot_groups, uint8_t* out, cudaStream_t s) {
  if (W == nullptr || out == nullptr || N < kRowGroup || N % kRowGroup != 0 || rows < 1 || rows > N || K < 8 ||
      K % 8 != 0 || G < 1 || (S != 1 && S != 2) || G % S != 0)
    return cudaErrorInvalidValue;
  if (kind == PACK_GLU && W2 == nullptr) return cudaErrorInvalidValue;
  if (kind == PACK_QKV && (N != 3 * d || hd % kRowGroup != 0 || d % hd != 0)) return cudaErrorInvalidValue;
  const int kb = (K + 63) / 64;
  if (S == 2 && kb < 2) return cudaErrorInvalidValue;
  const long long chunks = (long long)N * (kind == PACK_GLU ? 2 : 1) * kb * 8;
  const int threads = 256;
  long long blocks = (chunks + threads - 1) / threads;
  if (blocks > 65535LL * 16) blocks = 65535LL * 16;
  pack_rows_kernel<<<(unsigned)blocks, threads, 0, s>>>(W, W2, N, rows, K, kb, G, S, kind, d, hd, rot_groups, chunks,
                                                         out);
  return cudaGetLastError();
}

int chain_grid(int num_sms) { return num_sms; }

size_t chain_smem_bytes() { return chain_smem(); }

int chain_slice_rows(int N, int G, bool glu) {
  const int NG = N / kRowGroup;
  return (NG / G + (NG % G ? 1 : 0)) * kRowGroup * (glu ? 2 : 1);
}

cudaError_t launch_chain(const ChainMaps& maps, const ChainArgs& args, int grid, cudaStream_t stream, bool pdl) {
  if (args.nphases < 1 || args.nphases > kMaxPhases || args.bn < 16 || args.bn > 64 || args.bn % 16 != 0)
    return cudaErrorInvalidValue;
  for (int p = 0; p < args.nphases; ++p) {
    const ChainPhase& ph = args.ph[p];
    if (ph.wp == nullptr || (reinterpret_cast<uintptr_t>(ph.wp) & 15) != 0 || ph.N % kRowGroup != 0 || ph.kb < 1)
      return cudaErrorInvalidValue;
    if (chain_slice_rows(ph.N, grid, ph.epi == EPI_GLU) > kChainMaxSliceRows) return cudaErrorInvalidValue;
    if (ph.S != 1 && (ph.S != 2 || !args.pairs || ph.epi != EPI_RESID || ph.kb < 2 ||
                      chain_slice_rows(ph.N, grid / 2, false) > kPairMaxRows))
      return cudaErrorInvalidValue;
    if (ph.S == 1 && ph.epi == EPI_RESID && chain_slice_rows(ph.N, grid, false) > 64) return cudaErrorInvalidValue;
    if (ph.in_phase >= 0 && ph.in_S != args.ph[ph.in_phase].S) return cudaErrorInvalidValue;
    if (ph.in_phase >= p || (ph.in_phase >= 0 && (ph.in_N + 63) / 64 > kReadyPerPhase)) return cudaErrorInvalidValue;
    if (ph.publish && (ph.N + 63) / 64 > kReadyPerPhase) return cudaErrorInvalidValue;
  }
  auto kern = chain_kernel;
  constexpr size_t smem = chain_smem();
  static int configured = -1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured != dev) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kChainThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (args.pairs) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 2;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, kern, maps, args);
}

int chain_pairs_fit(int grid) {
  if (grid < 2 || grid % 2 != 0) return 0;
  auto kern = chain_kernel;
  constexpr size_t smem = chain_smem();
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kChainThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int nclusters = 0;
  if (cudaOccupancyMaxActiveClusters(&nclusters, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return nclusters * 2 >= grid ? 1 : 0;
}

}  // namespace casspec
