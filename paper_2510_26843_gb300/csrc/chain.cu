// Persistent projection chain on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// One launch runs a list of dependent projections of a tree step -- e.g. Wo (+residual), Wgate/Wup
// (+SwiGLU), Wdown (+residual), and the next layer's Wqkv (+rotary, K/V write) -- with a grid-wide
// barrier between phases.  Only the activations depend on the previous phase; the weights do not,
// so the weight stream runs on across phase boundaries and the HBM pipeline never drains between
// projections.  Per CTA (one per SM):
//   * warp 0 -- weight producer: streams the CTA's weight tiles (128 x 64 bf16, 128-byte swizzle,
//     L2 evict-first) of every phase through a deep mbarrier ring, never waiting on activations;
//   * warp 6 -- activation producer: after the phase barrier, streams the B operand tiles (BN x 64
//     of the hi plane and of the lo plane of the split activation, 128-byte swizzle) by TMA;
//   * warp 1 -- TMEM owner and single-thread MMA issuer: D += W hi^T + W lo^T (tcgen05.mma
//     kind::f16, M = 128 channels, N = BN tokens), double-buffered accumulators in TMEM;
//   * warps 2-5 -- epilogue: TMEM -> registers, stream-K fix-up (last CTA of a tile sums the partials
//     in CTA order), the per-token RMSNorm factor, fused epilogue; then the CTA's arrival at the
//     phase barrier.
// Work of each phase is split stream-K over (tile, k-block) units so all SMs stream equal bytes.
// Every wait is bounded (2 s) and reports CASSPEC_E_TIMEOUT instead of hanging.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace casspec {

constexpr int kChainThreads = 224;
constexpr uint32_t kWTile = 128 * 128;  // 128 rows x 64 bf16
constexpr int kXStages = 4;
constexpr uint32_t kChainSmemBudget = 232448u;  // 227 KB per CTA

__host__ __device__ constexpr uint32_t chain_x_stage(int BN) { return 2u * (uint32_t)BN * 128u; }
__host__ __device__ constexpr uint32_t chain_staging(int BN) { return (uint32_t)epi_staging_floats(BN) * 4u; }
__host__ __device__ constexpr uint32_t chain_fixed(int BN) {
  return 1024u + kXStages * chain_x_stage(BN) + chain_staging(BN) + 64u * 4u + 512u;
}
__host__ __device__ constexpr int chain_w_stages(int BN) {
  return (int)((kChainSmemBudget - chain_fixed(BN)) / kWTile) > 12 ? 12
                                                                   : (int)((kChainSmemBudget - chain_fixed(BN)) / kWTile);
}
__host__ __device__ constexpr size_t chain_smem(int BN) { return chain_fixed(BN) + (size_t)chain_w_stages(BN) * kWTile; }
// TMEM per accumulator buffer: one accumulator of 2*BN columns (the hi and lo planes stacked as
// one N = 2*BN operand); two buffers.
__host__ __device__ constexpr uint32_t chain_buf_cols(int BN) { return 2u * (uint32_t)BN; }
__host__ __device__ constexpr uint32_t chain_tmem_cols(int BN) {
  return 2 * chain_buf_cols(BN) <= 64 ? 64 : (2 * chain_buf_cols(BN) <= 128 ? 128 : 256);
}

__device__ __forceinline__ long long chain_u0(int c, long long U, int G) { return (long long)c * U / G; }
// CTA that owns unit x when U units are split into G contiguous ranges [c U / G, (c + 1) U / G)
__device__ __forceinline__ int chain_cta_of(long long x, long long U, int G) {
  return (int)(((x + 1) * (long long)G - 1) / U);
}
__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// generic-proxy global writes <-> async-proxy (TMA) reads of the split activations
__device__ __forceinline__ void fence_proxy_async_global() { asm volatile("fence.proxy.async.global;" ::: "memory"); }

template <int BN, typename Bar>
__device__ __forceinline__ void chain_epilogue(int epi, const EpiParams& e, int tile, int r, const float* v, float* stg,
                                               Bar bar, int i0, int i1) {
  switch (epi) {
    case EPI_RESID: run_epilogue<BN, EPI_RESID>(e, tile, r, v, stg, bar, i0, i1); break;
    case EPI_QKV: run_epilogue<BN, EPI_QKV>(e, tile, r, v, stg, bar, i0, i1); break;
    case EPI_GLU: run_epilogue<BN, EPI_GLU>(e, tile, r, v, stg, bar, i0, i1); break;
    case EPI_LMHEAD: run_epilogue<BN, EPI_LMHEAD>(e, tile, r, v, stg, bar, i0, i1); break;
    default: run_epilogue<BN, EPI_STORE>(e, tile, r, v, stg, bar, i0, i1); break;
  }
}

template <int BN>
__global__ void __launch_bounds__(kChainThreads, 1)
    chain_kernel(const __grid_constant__ ChainMaps maps, const __grid_constant__ ChainArgs a) {
  constexpr int SW = chain_w_stages(BN);
  constexpr int SX = kXStages;
  constexpr uint32_t XT = (uint32_t)BN * 128u;  // one hi or lo tile
  constexpr uint32_t XS = 2 * XT;
  constexpr uint32_t TMEM_COLS = chain_tmem_cols(BN);
  constexpr uint32_t IDESC = idesc_bf16_f32(128, 2 * BN);  // B = [hi; lo], N = 2 * BN

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* wring = smem;
  uint8_t* xring = smem + SW * kWTile;
  float* stg = reinterpret_cast<float*>(xring + SX * XS);
  float* rs = stg + epi_staging_floats(BN);
  uint64_t* wfull = reinterpret_cast<uint64_t*>(rs + 64);
  uint64_t* wempty = wfull + SW;
  uint64_t* xfull = wempty + SW;
  uint64_t* xempty = xfull + SX;
  uint64_t* tfull = xempty + SX;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  // [0] abort, [1] fix-up wait result, [2..9] per-warp accumulator-ready votes (two segments),
  // [2] after the main loops: this CTA is the last out
  volatile int* flags = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, cta = blockIdx.x;
  const int np = a.nphases;

  if (threadIdx.x == 0) {
    for (int s = 0; s < SW; ++s) {
      mbar_init(&wfull[s], 1);
      mbar_init(&wempty[s], 1);
    }
    for (int s = 0; s < SX; ++s) {
      mbar_init(&xfull[s], 1);
      mbar_init(&xempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);
    }
    mbar_init(drain, 1);
    for (int f = 0; f < 10; ++f) flags[f] = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    for (int p = 0; p < np; ++p) {
      tma_prefetch_desc(&maps.w[p]);
      if (a.ph[p].epi == EPI_GLU) tma_prefetch_desc(&maps.w2[p]);
      tma_prefetch_desc(&maps.x[p]);
    }
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
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
        const int kb = a.ph[p].kblocks;
        const bool glu = a.ph[p].epi == EPI_GLU;
        const long long U = (long long)a.ph[p].tiles * kb;
        const long long u1 = chain_u0(cta + 1, U, G);
        for (long long u = chain_u0(cta, U, G); u < u1; ++u) {
          if (!mbar_wait_bounded(&wempty[stage], phase ^ 1, flags)) {
            flags[0] = 1;
            set_status(a.status, CASSPEC_E_TIMEOUT);
            break;
          }
          const int t = (int)(u / kb), k = (int)(u % kb);
          mbar_expect_tx(&wfull[stage], kWTile);
          armed |= 1u << stage;
          armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
          uint8_t* sa = wring + stage * kWTile;
          if (glu) {
            tma_load_2d(sa, &maps.w[p], &wfull[stage], k * 64, t * 64, pol);
            tma_load_2d(sa + kWTile / 2, &maps.w2[p], &wfull[stage], k * 64, t * 64, pol);
          } else {
            tma_load_2d(sa, &maps.w[p], &wfull[stage], k * 64, t * 128, pol);
          }
          if (++stage == SW) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (flags[0]) {  // abort: let the copies already issued land before the CTA exits
        for (int s = 0; s < SW; ++s)
          if (armed & (1u << s)) mbar_wait_bounded(&wfull[s], (armed_parity >> s) & 1, nullptr);
      }
    }
  } else if (warp == 6) {
    if (lane == 0) {
      // ---------------- activation producer (waits for the phase barrier) ----------------
      const uint64_t pol = policy_evict_last();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_parity = 0;
      for (int p = 0; p < np && !flags[0]; ++p) {
        if (p == 0) {
          pdl_wait();  // inputs of the first phase come from the previous kernel
        } else {       // ... of the others from phase p - 1 of every CTA (one counter per phase:
                       // a CTA with no work may run ahead and arrive at later phases early)
          const uint64_t t0 = globaltimer_ns();
          while (ld_acquire_u32(a.bar + (p - 1)) < (unsigned)G) {
            if (flags[0]) break;
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
              flags[0] = 1;
              set_status(a.status, CASSPEC_E_TIMEOUT);
              break;
            }
          }
          if (flags[0]) break;
        }
        fence_proxy_async_global();
        const int kb = a.ph[p].kblocks;
        const long long U = (long long)a.ph[p].tiles * kb;
        const long long u1 = chain_u0(cta + 1, U, G);
        for (long long u = chain_u0(cta, U, G); u < u1; ++u) {
          if (!mbar_wait_bounded(&xempty[stage], phase ^ 1, flags)) {
            flags[0] = 1;
            set_status(a.status, CASSPEC_E_TIMEOUT);
            break;
          }
          const int k = (int)(u % kb);
          mbar_expect_tx(&xfull[stage], XS);
          armed |= 1u << stage;
          armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
          uint8_t* sx = xring + stage * XS;
          tma_load_2d(sx, &maps.x[p], &xfull[stage], k * 64, 0, pol);        // hi plane, tokens 0..BN-1
          tma_load_2d(sx + XT, &maps.x[p], &xfull[stage], k * 64, 64, pol);  // lo plane
          if (++stage == SX) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (flags[0]) {
        for (int s = 0; s < SX; ++s)
          if (armed & (1u << s)) mbar_wait_bounded(&xfull[s], (armed_parity >> s) & 1, nullptr);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int ws = 0, xs = 0;
      uint32_t wph = 0, xph = 0;
      uint32_t used[2] = {0, 0};
      int buf = 0;
      bool ok = true;
      for (int p = 0; p < np && ok; ++p) {
        const int kb = a.ph[p].kblocks;
        const long long U = (long long)a.ph[p].tiles * kb;
        const long long u1 = chain_u0(cta + 1, U, G);
        long long u = chain_u0(cta, U, G);
        while (u < u1 && ok) {
          const int t = (int)(u / kb);
          const long long seg_end = ((long long)(t + 1) * kb < u1) ? (long long)(t + 1) * kb : u1;
          if (!mbar_wait_bounded(&tempty[buf], (used[buf] & 1) ^ 1, flags)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + (uint32_t)buf * chain_buf_cols(BN);
          for (long long uu = u; uu < seg_end; ++uu) {
            if (!mbar_wait_bounded(&wfull[ws], wph, flags) || !mbar_wait_bounded(&xfull[xs], xph, flags)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(wring + ws * kWTile);
            const uint32_t sh = smem_u32(xring + xs * XS);
            // One MMA per 16-column k-step with the hi and lo planes stacked (N = 2 * BN, the X stage
            // holds them back to back), all into one accumulator: splitting even and odd k-steps
            // over two accumulators measured slower.
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_bf16(d_tmem, sw128_kmajor_desc(sa + kk * 32), sw128_kmajor_desc(sh + kk * 32), IDESC,
                          (uu > u || kk > 0) ? 1u : 0u);
            tc_commit(&wempty[ws]);
            tc_commit(&xempty[xs]);
            if (++ws == SW) {
              ws = 0;
              wph ^= 1;
            }
            if (++xs == SX) {
              xs = 0;
              xph ^= 1;
            }
          }
          if (!ok) break;
          tc_commit(&tfull[buf]);
          used[buf]++;
          buf ^= 1;
          u = seg_end;
        }
      }
      if (!ok) {
        flags[0] = 1;
        set_status(a.status, CASSPEC_E_TIMEOUT);
      }
      tc_commit(drain);  // all MMAs complete before TMEM is released
      mbar_wait_bounded(drain, 0, nullptr);
    }
  } else {
    // ---------------- epilogue warps 2..5 ----------------
    // Control flow is identical in the four warps (every decision that follows a bounded wait is
    // voted through shared memory), so their named barriers always match, even after a timeout.
    const int q = warp & 3;
    const int r = q * 32 + lane;
    auto bar = [] { named_bar_sync(1, 128); };
    // The phase-barrier counters belong to the previous launch until it has completed (its last
    // CTA resets them); a CTA without units could otherwise arrive before that reset.
    pdl_wait();
    uint32_t used[2] = {0, 0};
    int buf = 0, seg = 0;
    for (int p = 0; p < np; ++p) {
      // The phase descriptor sits in parameter space behind a runtime index: copy what the loops
      // use into registers once, so no load of it is ordered behind the epilogue's stores.
      const EpiParams ep = a.ph[p].ep;
      const int epi = a.ph[p].epi, kb = a.ph[p].kblocks, Kp = a.ph[p].K, n = ep.n;
      const float* ss = a.ph[p].ss;
      const int ss_tiles = a.ph[p].ss_tiles;
      const float eps = a.ph[p].eps;
      const long long U = (long long)a.ph[p].tiles * kb;
      const long long u1 = chain_u0(cta + 1, U, G);
      unsigned* counters = a.counters + p * 1024;
      bool have_rs = false;
      long long u = chain_u0(cta, U, G);
      while (u < u1) {
        const int t = (int)(u / kb);
        const long long seg_end = ((long long)(t + 1) * kb < u1) ? (long long)(t + 1) * kb : u1;
        const bool got = mbar_wait_bounded(&tfull[buf], used[buf] & 1, flags);
        if (lane == 0) flags[2 + (seg & 1) * 4 + q] = got ? 1 : 0;
        bar();
        const int vote = (seg & 1) * 4;
        const bool ready = flags[2 + vote] && flags[3 + vote] && flags[4 + vote] && flags[5 + vote];
        ++seg;
        used[buf]++;
        if (!ready) {  // the accumulator never arrived: give up on the rest (uniformly)
          flags[0] = 1;
          set_status(a.status, CASSPEC_E_TIMEOUT);
          u = seg_end;
          buf ^= 1;
          continue;
        }
        if (ss != nullptr && !have_rs) {
          // the phase's inputs are visible here: this accumulator was computed from them
          if (r < 64) {
            float ssum = 0.f;  // fixed summation order; loads issued 8 at a time
            for (int j0 = 0; j0 < ss_tiles; j0 += 8) {
              float t8[8];
#pragma unroll
              for (int k = 0; k < 8; ++k) t8[k] = j0 + k < ss_tiles ? __ldcg(ss + (j0 + k) * 64 + r) : 0.f;
#pragma unroll
              for (int k = 0; k < 8; ++k) ssum += t8[k];
            }
            rs[r] = rsqrtf(ssum / (float)Kp + eps);
          }
          bar();
          have_rs = true;
        }
        tc_fence_after();
        float v[BN];
        const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)buf * chain_buf_cols(BN);
#pragma unroll
        for (int c = 0; c < BN; c += 16) {  // hi-plane product + lo-plane product
          float t1[16];
          tmem_ld_x16(taddr + c, &v[c]);
          tmem_ld_x16(taddr + BN + c, t1);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 16; ++j) v[c + j] += t1[j];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[buf]);
        buf ^= 1;

        // Stream-K fix-up.  Every owner of a shared tile deposits its partial ([token][row] slot
        // t + cta) and counts itself in.  The owners for which the tile is their last segment of
        // the phase (all but possibly the one that holds the tile's tail at the start of its range)
        // reach it together at the end of the phase: each waits for every deposit, sums one slice
        // of the tokens over the owners in CTA order (deterministic) and runs the epilogue on it.
        // CTAs with no unit at all (phases with fewer units than CTAs) are not owners.
        const int c_first = chain_cta_of((long long)t * kb, U, G);
        const int c_last = chain_cta_of((long long)(t + 1) * kb - 1, U, G);
        int i0 = 0, i1 = n;
        bool finish = true;
        if (c_first != c_last) {
          const long long tile_end = (long long)(t + 1) * kb;
          int owners = 0, parts = 0, rank = 0;
          int own_list[6];  // the first 6 owners in CTA order
          for (int cc = c_first; cc <= c_last; ++cc) {
            const long long b0 = chain_u0(cc, U, G), b1 = chain_u0(cc + 1, U, G);
            if (b1 <= b0) continue;
#pragma unroll
            for (int o = 0; o < 6; ++o)
              if (o == owners) own_list[o] = cc;
            ++owners;
            if (b1 <= tile_end) {
              if (cc == cta) rank = parts;
              ++parts;
            }
          }
          // own partial token-major in shared memory ([token][row], the slot layout), then coalesced
          // 16-byte stores of the valid tokens into slot t + cta
#pragma unroll
          for (int i = 0; i < BN; ++i) stg[i * 128 + r] = v[i];
          bar();
          const int nf4 = n * 32;
          const float4* own4 = reinterpret_cast<const float4*>(stg);
          {
            float4* mine4 = reinterpret_cast<float4*>(a.partials + (size_t)(t + cta) * (64 * 128));
#pragma unroll
            for (int j = 0; j < BN / 4; ++j)
              if (r + 128 * j < nf4) __stcg(mine4 + r + 128 * j, own4[r + 128 * j]);
          }
          bar();  // then one gpu-scope fence (cumulative over the CTA's stores) before counting in
          if (threadIdx.x == 64) {
            __threadfence();
            atomicAdd(&counters[t], 1u);
          }
          finish = seg_end == u1;  // a participant: this is the CTA's last segment of the phase
          if (finish) {
            if (threadIdx.x == 64) {
              const uint64_t t0 = globaltimer_ns();
              int ok = 1;
              while (ld_acquire_u32(counters + t) < (unsigned)owners) {
                if (flags[0] || globaltimer_ns() - t0 > kWaitLimitNs) {
                  ok = 0;
                  flags[0] = 1;
                  set_status(a.status, CASSPEC_E_TIMEOUT);
                  break;
                }
              }
              flags[1] = ok;
            }
            bar();
            finish = flags[1] != 0;
            i0 = rank * n / parts;
            i1 = (rank + 1) * n / parts;
          }
          if (finish && i1 > i0) {
            __threadfence();
            const int f0 = i0 * 32, f1 = i1 * 32;  // float4s of the slice
            float4 acc[BN / 4];
#pragma unroll
            for (int j = 0; j < BN / 4; ++j) acc[j] = make_float4(0.f, 0.f, 0.f, 0.f);
            auto add4 = [](float4& x, const float4& y) {
              x.x += y.x;
              x.y += y.y;
              x.z += y.z;
              x.w += y.w;
            };
            if (owners <= 6 && f1 - f0 <= 4 * 128) {
              // a small slice (at most 4 float4s per thread) from at most 6 owners: every load in
              // flight together; sums in CTA order
              float4 t4[6][4];
#pragma unroll
              for (int o = 0; o < 6; ++o) {
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                  const int f = f0 + r + 128 * j;
                  float4 val = make_float4(0.f, 0.f, 0.f, 0.f);
                  if (o < owners && f < f1) {
                    const int cc = own_list[o];
                    val = cc == cta ? own4[f]
                                    : __ldcg(reinterpret_cast<const float4*>(a.partials + (size_t)(t + cc) * (64 * 128)) + f);
                  }
                  t4[o][j] = val;
                }
              }
#pragma unroll
              for (int o = 0; o < 6; ++o) {
#pragma unroll
                for (int j = 0; j < 4; ++j)
                  if (j < BN / 4) add4(acc[j], t4[o][j]);
              }
            } else {  // larger slices or many owners: one owner at a time, all its loads in flight
              for (int cc = c_first; cc <= c_last; ++cc) {
                if (cc != cta && chain_u0(cc + 1, U, G) <= chain_u0(cc, U, G)) continue;
                const float4* src = cc == cta ? own4
                                              : reinterpret_cast<const float4*>(a.partials + (size_t)(t + cc) * (64 * 128));
                float4 t4[BN / 4];
#pragma unroll
                for (int j = 0; j < BN / 4; ++j) {
                  const int f = f0 + r + 128 * j;
                  t4[j] = f < f1 ? (cc == cta ? src[f] : __ldcg(src + f)) : make_float4(0.f, 0.f, 0.f, 0.f);
                }
#pragma unroll
                for (int j = 0; j < BN / 4; ++j) add4(acc[j], t4[j]);
              }
            }
            bar();
            float4* st4 = reinterpret_cast<float4*>(stg);
#pragma unroll
            for (int j = 0; j < BN / 4; ++j) {
              const int f = f0 + r + 128 * j;
              if (f < f1) st4[f] = acc[j];
            }
            bar();
#pragma unroll
            for (int i = 0; i < BN; ++i) v[i] = stg[i * 128 + r];
          }
        }
        if (finish && i1 > i0) {
          if (ss != nullptr) {
#pragma unroll
            for (int i = 0; i < BN; ++i) v[i] *= rs[i];
          }
          chain_epilogue<BN>(epi, ep, t, r, v, stg, bar, i0, i1);
        }
        u = seg_end;
      }
      if (have_rs) bar();  // rs is rewritten by the next phase only after every thread used it
      if (p + 1 < np) {  // this CTA's writes of phase p are done: arrive at the phase barrier
        fence_proxy_async_global();
        __threadfence();
        bar();
        if (threadIdx.x == 64) {
          __threadfence();
          atomicAdd(&a.bar[p], 1u);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
  // The last CTA out returns the phase-barrier, exit and fix-up counters to zero for the next
  // launch (they belong to the previous launch until it completes, hence the dependency wait).
  if (threadIdx.x == 0) {
    pdl_wait();
    __threadfence();
    flags[2] = atomicAdd(&a.bar[kMaxPhases], 1u) == (unsigned)(G - 1) ? 1 : 0;
  }
  __syncthreads();
  if (flags[2]) {
    __threadfence();
    for (int p = threadIdx.x; p <= kMaxPhases; p += blockDim.x) a.bar[p] = 0u;
    for (int p = 0; p < np; ++p)
      for (int t = threadIdx.x; t < a.ph[p].tiles; t += blockDim.x) a.counters[p * 1024 + t] = 0u;
  }
}

int chain_grid(int num_sms) { return num_sms; }

size_t chain_smem_bytes(int BN) {
  switch (BN) {
    case 16: return chain_smem(16);
    case 32: return chain_smem(32);
    case 48: return chain_smem(48);
    default: return chain_smem(64);
  }
}

template <int BN>
static cudaError_t launch_bn(const ChainMaps& maps, const ChainArgs& args, int grid, cudaStream_t stream, bool pdl) {
  auto kern = chain_kernel<BN>;
  constexpr size_t smem = chain_smem(BN);
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
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, maps, args);
}

cudaError_t launch_chain(const ChainMaps& maps, const ChainArgs& args, int BN, int grid, cudaStream_t stream, bool pdl) {
  if (args.nphases < 1 || args.nphases > kMaxPhases) return cudaErrorInvalidValue;
  switch (BN) {
    case 16: return launch_bn<16>(maps, args, grid, stream, pdl);
    case 32: return launch_bn<32>(maps, args, grid, stream, pdl);
    case 48: return launch_bn<48>(maps, args, grid, stream, pdl);
    case 64: return launch_bn<64>(maps, args, grid, stream, pdl);
  }
  return cudaErrorInvalidValue;
}

}  // namespace casspec
