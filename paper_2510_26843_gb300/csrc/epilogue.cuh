// Epilogues of the projections.  A finished 128-row tile is held one row (output channel) per
// thread by 128 cooperating threads; thread r owns row r and the values v[0..BN) of tokens
// 0..BN-1 (only i < n are meaningful).  `stg` is a [128][BN+1] fp32 staging area in shared memory
// used where a row needs another row's values (rotary partner, gate/up pair, argmax over rows);
// `bar` synchronises the 128 threads (a named barrier).
#pragma once

#include "common.cuh"
#include "kernels.h"

namespace casspec {

template <int BN, typename Bar>
__device__ __forceinline__ void epi_qkv(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar) {
  const int o = tile * 128 + r;  // row of [Wq; Wk; Wv]
  const int part = o / e.d;      // 0: q, 1: k, 2: v
  const int within = o - part * e.d;
  const int head = within / e.hd;
  const int j = within - head * e.hd;
  const int half = e.hd >> 1;
#pragma unroll
  for (int i = 0; i < BN; ++i) stg[r * (BN + 1) + i] = v[i];
  bar();
  const int rp = r ^ half;  // heads are aligned to tiles (d % 128 == 0, hd | 128)
  const int P = __ldcg(e.dP);
  const int jj = j & (half - 1);
  if (part < 2) {
    const float sgn = (j < half) ? -1.f : 1.f;
#pragma unroll
    for (int i = 0; i < BN; ++i) {
      if (i < e.n) {
        const float2 cs = e.rope[(size_t)__ldcg(e.pos + i) * half + jj];
        const float out = v[i] * cs.x + sgn * stg[rp * (BN + 1) + i] * cs.y;
        if (part == 0)
          e.q_out[(size_t)i * e.d + within] = f2bf(out);
        else
          e.kc[((size_t)head * e.ctx + (P + e.T + i)) * e.hd + j] = f2bf(out);
      }
    }
  } else {
#pragma unroll
    for (int i = 0; i < BN; ++i)
      if (i < e.n) e.vc[((size_t)head * e.ctx + (P + e.T + i)) * e.hd + j] = f2bf(v[i]);
  }
  bar();
}

template <int BN, typename Bar>
__device__ __forceinline__ void epi_glu(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar) {
  if (r >= 64) {
#pragma unroll
    for (int i = 0; i < BN; ++i) stg[r * (BN + 1) + i] = v[i];
  }
  bar();
  const int ch = tile * 64 + r;
  if (r < 64 && ch < e.N) {
#pragma unroll
    for (int i = 0; i < BN; ++i) {
      if (i < e.n) {
        const float g = v[i];
        const float up = stg[(r + 64) * (BN + 1) + i];
        const float u = g / (1.f + expf(-g)) * up;
        const uint16_t hi = f2bf(u);
        e.u_out[(size_t)i * e.N + ch] = hi;
        e.u_out[(size_t)(64 + i) * e.N + ch] = f2bf(u - bf2f(hi));
      }
    }
  }
  bar();
}

template <int BN, typename Bar>
__device__ __forceinline__ void epi_lmhead(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar) {
  const int o = tile * 128 + r;
  const bool valid = o < e.N;
  if (e.logits != nullptr && valid) {
#pragma unroll
    for (int i = 0; i < BN; ++i)
      if (i < e.n) e.logits[(size_t)i * e.N + o] = v[i];
  }
#pragma unroll
  for (int i = 0; i < BN; ++i) stg[r * (BN + 1) + i] = valid ? v[i] : -INFINITY;
  bar();
  if (r < e.n) {
    float m1 = -INFINITY, m2 = -INFINITY;
    int i1 = 0;
    for (int row = 0; row < 128; ++row) {
      const float x = stg[row * (BN + 1) + r];
      if (x > m1) {
        m2 = m1;
        m1 = x;
        i1 = row;
      } else if (x > m2) {
        m2 = x;
      }
    }
    e.am_v1[tile * 64 + r] = m1;
    e.am_i1[tile * 64 + r] = tile * 128 + i1;
    e.am_v2[tile * 64 + r] = m2;
  }
  bar();
}

template <int BN>
__device__ __forceinline__ void epi_store(const EpiParams& e, int tile, int r, const float* v) {
  const int o = tile * 128 + r;
  if (o < e.N) {
#pragma unroll
    for (int i = 0; i < BN; ++i)
      if (i < e.n) e.y[(size_t)i * e.ldy + o] = v[i];
  }
}

// y += v (fp32 residual stream); optionally the tile's per-token sum of squares of the updated rows,
// the partial sums from which the next RMSNorm takes its scale (fixed order: deterministic), and
// split(y * g_next), the operand of the next projection.
template <int BN, typename Bar>
__device__ __forceinline__ void epi_resid(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar) {
  const int o = tile * 128 + r;
  const bool valid = o < e.N;
  const float gn = (e.xa_out != nullptr && valid) ? e.g_next[o] : 0.f;
#pragma unroll
  for (int i = 0; i < BN; ++i) {
    float nv = 0.f;
    if (i < e.n && valid) {
      float* p = e.y + (size_t)i * e.ldy + o;
      nv = __ldcg(p) + v[i];
      *p = nv;
      if (e.xa_out != nullptr) {
        const float a = nv * gn;
        const uint16_t hi = f2bf(a);
        e.xa_out[(size_t)i * e.ldy + o] = hi;
        e.xa_out[(size_t)(64 + i) * e.ldy + o] = f2bf(a - bf2f(hi));
      }
    }
    if (e.ss_out != nullptr) stg[r * (BN + 1) + i] = nv * nv;
  }
  if (e.ss_out == nullptr) return;
  bar();
  if (r < e.n) {
    float s = 0.f;
    for (int row = 0; row < 128; ++row) s += stg[row * (BN + 1) + r];
    e.ss_out[tile * 64 + r] = s;
  }
  bar();
}

template <int BN, int EPI, typename Bar>
__device__ __forceinline__ void run_epilogue(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar) {
  if constexpr (EPI == EPI_STORE) epi_store<BN>(e, tile, r, v);
  if constexpr (EPI == EPI_RESID) epi_resid<BN>(e, tile, r, v, stg, bar);
  if constexpr (EPI == EPI_QKV) epi_qkv<BN>(e, tile, r, v, stg, bar);
  if constexpr (EPI == EPI_GLU) epi_glu<BN>(e, tile, r, v, stg, bar);
  if constexpr (EPI == EPI_LMHEAD) epi_lmhead<BN>(e, tile, r, v, stg, bar);
}

}  // namespace casspec
