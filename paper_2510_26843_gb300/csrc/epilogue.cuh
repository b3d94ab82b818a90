// Epilogues of the projections.  A finished 128-row tile arrives one row (output channel) per
// thread from 128 cooperating threads: thread r owns row r and the values v[0..BN) of tokens
// 0..BN-1 (only i < n are meaningful).  The tile is first staged token-major in shared memory
// (`stg`, epi_staging_floats(BN) floats); then each warp takes whole tokens and each lane four
// consecutive channels, so every global access is a 16- or 8-byte vector and the per-token
// reductions (sum of squares, argmax) are warp shuffles in a fixed order (deterministic).
// `bar` synchronises the 128 threads (a named barrier).  Only tokens [i0, i1) (i1 <= n) are
// written: a tile may be finished in token slices by several CTAs.
#pragma once

#include "common.cuh"
#include "kernels.h"

namespace casspec {

constexpr int kEpiStride = 132;  // staging row of one token: 128 channels + 4 pad floats

__host__ __device__ constexpr int epi_staging_floats(int BN) {
  return 128 * (BN + 1) > BN * kEpiStride ? 128 * (BN + 1) : BN * kEpiStride;
}

template <int BN, typename Bar>
__device__ __forceinline__ void epi_stage(int r, const float* v, float* stg, Bar bar) {
  bar();  // the previous user of the staging area is done
#pragma unroll
  for (int i = 0; i < BN; ++i) stg[i * kEpiStride + r] = v[i];
  bar();
}

__device__ __forceinline__ float4 stg4(const float* stg, int i, int c) {
  return *reinterpret_cast<const float4*>(stg + i * kEpiStride + c);
}

__device__ __forceinline__ uint2 pack4_bf16(float a, float b, float c, float d) {
  return make_uint2(pack_bf16x2(a, b), pack_bf16x2(c, d));
}

// hi = bf16(x), lo = bf16(x - hi) of four values
__device__ __forceinline__ void split4(float4 x, uint2& hi, uint2& lo) {
  const uint16_t h0 = f2bf(x.x), h1 = f2bf(x.y), h2 = f2bf(x.z), h3 = f2bf(x.w);
  hi = make_uint2((uint32_t)h0 | ((uint32_t)h1 << 16), (uint32_t)h2 | ((uint32_t)h3 << 16));
  lo = pack4_bf16(x.x - bf2f(h0), x.y - bf2f(h1), x.z - bf2f(h2), x.w - bf2f(h3));
}

__device__ __forceinline__ float warp_sum(float s) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  return s;
}

// Q/K/V: rotary on q and k at the node's tree position; q -> q_out, k, v -> cache slot P + T + i.
template <int BN, typename Bar>
__device__ __forceinline__ void epi_qkv(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar,
                                         int i0, int i1) {
  epi_stage<BN>(r, v, stg, bar);
  const int w = r >> 5, l = r & 31;
  const int row = 4 * l;
  const int o = tile * 128 + row;  // first of this lane's 4 rows of [Wq; Wk; Wv]
  const int part = o / e.d;        // 0: q, 1: k, 2: v (a tile never straddles parts: d % 128 == 0)
  const int within = o - part * e.d;
  const int head = within / e.hd;
  const int j = within - head * e.hd;
  const int half = e.hd >> 1;
  const int prow = row ^ half;  // rotary partner rows (half is a multiple of 4)
  const int jj = j & (half - 1);
  const float sgn = (j < half) ? -1.f : 1.f;
  const int P = __ldcg(e.dP);
  constexpr int M = (BN + 3) / 4;  // tokens per warp: i = w + 4 m
  if (part < 2) {
    int pos[M];
#pragma unroll
    for (int m = 0; m < M; ++m) pos[m] = (w + 4 * m >= i0 && w + 4 * m < i1) ? __ldcg(e.pos + w + 4 * m) : 0;
#pragma unroll
    for (int m0 = 0; m0 < M; m0 += 8) {  // rotary tables of 8 tokens in flight at a time
      float4 c01[8], c23[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (m0 + k < M) {
          const float4* cs = reinterpret_cast<const float4*>(e.rope + (size_t)pos[m0 + k] * half + jj);
          c01[k] = cs[0];
          c23[k] = cs[1];
        }
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int i = w + 4 * (m0 + k);
        if (m0 + k < M && i >= i0 && i < i1) {
          const float4 x = stg4(stg, i, row), y = stg4(stg, i, prow);
          const uint2 out = pack4_bf16(x.x * c01[k].x + sgn * y.x * c01[k].y, x.y * c01[k].z + sgn * y.y * c01[k].w,
                                       x.z * c23[k].x + sgn * y.z * c23[k].y, x.w * c23[k].z + sgn * y.w * c23[k].w);
          if (part == 0)
            *reinterpret_cast<uint2*>(e.q_out + (size_t)i * e.d + within) = out;
          else
            *reinterpret_cast<uint2*>(e.kc + ((size_t)head * e.ctx + (P + e.T + i)) * e.hd + j) = out;
        }
      }
    }
  } else {
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const int i = w + 4 * m;
      if (i >= i0 && i < i1) {
        const float4 x = stg4(stg, i, row);
        *reinterpret_cast<uint2*>(e.vc + ((size_t)head * e.ctx + (P + e.T + i)) * e.hd + j) =
            pack4_bf16(x.x, x.y, x.z, x.w);
      }
    }
  }
  bar();
}

// gate/up tile (rows 0..63 gate, 64..127 up of channels tile*64..): u = silu(gate) * up, split.
template <int BN, typename Bar>
__device__ __forceinline__ void epi_glu(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar,
                                         int i0, int i1) {
  epi_stage<BN>(r, v, stg, bar);
  const int w = r >> 5, l = r & 31;
  const int c4 = (l & 15) * 4;  // 16 lanes per token, 4 channels each
  const int ch = tile * 64 + c4;
  if (ch < e.N) {  // N % 16 == 0: a 4-channel group is entirely valid or not
    constexpr int M = (BN + 7) / 8;  // token pairs per warp: i = 2 (w + 4 m) + (l >> 4)
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const int i = 2 * (w + 4 * m) + (l >> 4);
      if (i >= i0 && i < i1) {
        const float4 g = stg4(stg, i, c4), up = stg4(stg, i, 64 + c4);
        float4 u;
        // fast exponential and division: ~1e-6 relative error, below the 16-bit split
        u.x = __fdividef(g.x, 1.f + __expf(-g.x)) * up.x;
        u.y = __fdividef(g.y, 1.f + __expf(-g.y)) * up.y;
        u.z = __fdividef(g.z, 1.f + __expf(-g.z)) * up.z;
        u.w = __fdividef(g.w, 1.f + __expf(-g.w)) * up.w;
        uint2 hi, lo;
        split4(u, hi, lo);
        *reinterpret_cast<uint2*>(e.u_out + (size_t)i * e.N + ch) = hi;
        *reinterpret_cast<uint2*>(e.u_out + (size_t)(64 + i) * e.N + ch) = lo;
      }
    }
  }
  bar();
}

// LM head: logits (optional) and, per token, the tile's (max, argmax, second max) over its rows;
// ties go to the lowest vocabulary id.
template <int BN, typename Bar>
__device__ __forceinline__ void epi_lmhead(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar,
                                         int i0, int i1) {
  epi_stage<BN>(r, v, stg, bar);
  const int w = r >> 5, l = r & 31;
  const int o = tile * 128 + 4 * l;
  const bool valid = o < e.N;  // N % 8 == 0: a 4-row group is entirely valid or not
  constexpr int M = (BN + 3) / 4;
#pragma unroll
  for (int m = 0; m < M; ++m) {
    const int i = w + 4 * m;
    if (i < i0 || i >= i1) continue;  // warp-uniform
    const float4 x = stg4(stg, i, 4 * l);
    if (e.logits != nullptr && valid) *reinterpret_cast<float4*>(e.logits + (size_t)i * e.N + o) = x;
    float m1 = -INFINITY, m2 = -INFINITY;
    int i1 = 0x7fffffff;
    if (valid) {
      const float xs[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if (xs[k] > m1) {
          m2 = m1;
          m1 = xs[k];
          i1 = 4 * l + k;
        } else if (xs[k] > m2) {
          m2 = xs[k];
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float om1 = __shfl_xor_sync(0xffffffffu, m1, off);
      const float om2 = __shfl_xor_sync(0xffffffffu, m2, off);
      const int oi1 = __shfl_xor_sync(0xffffffffu, i1, off);
      if (om1 > m1 || (om1 == m1 && oi1 < i1)) {
        m2 = fmaxf(m1, om2);
        m1 = om1;
        i1 = oi1;
      } else {
        m2 = fmaxf(m2, om1);
      }
    }
    if (l == 0) {
      e.am_v1[tile * 64 + i] = m1;
      e.am_i1[tile * 64 + i] = tile * 128 + (i1 == 0x7fffffff ? 0 : i1);
      e.am_v2[tile * 64 + i] = m2;
    }
  }
  bar();
}

// y = v (stateless projection); any N and ldy.
template <int BN, typename Bar>
__device__ __forceinline__ void epi_store(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar,
                                         int i0, int i1) {
  epi_stage<BN>(r, v, stg, bar);
  const int w = r >> 5, l = r & 31;
  constexpr int M = (BN + 3) / 4;
#pragma unroll
  for (int m = 0; m < M; ++m) {
    const int i = w + 4 * m;
    if (i < i0 || i >= i1) continue;
#pragma unroll
    for (int k = 0; k < 4; ++k) {  // lane l: channels l, l + 32, l + 64, l + 96 (coalesced rows)
      const int c = l + 32 * k, o = tile * 128 + c;
      if (o < e.N) e.y[(size_t)i * e.ldy + o] = stg[i * kEpiStride + c];
    }
  }
  bar();
}

// y += v (fp32 residual stream); optionally the tile's per-token sum of squares of the updated rows
// (the partial sums from which the next RMSNorm takes its scale) and split(y * g_next), the operand
// of the next projection.  N = d (a multiple of 128).
template <int BN, typename Bar>
__device__ __forceinline__ void epi_resid(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar,
                                         int i0, int i1) {
  epi_stage<BN>(r, v, stg, bar);
  const int w = r >> 5, l = r & 31;
  const int o = tile * 128 + 4 * l;
  constexpr int M = (BN + 3) / 4;
  float4 old[M];  // every load first: one memory round trip
#pragma unroll
  for (int m = 0; m < M; ++m) {
    const int i = w + 4 * m;
    old[m] = (i >= i0 && i < i1) ? __ldcg(reinterpret_cast<const float4*>(e.y + (size_t)i * e.ldy + o))
                     : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  const float4 gn =
      e.xa_out != nullptr ? *reinterpret_cast<const float4*>(e.g_next + o) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int m = 0; m < M; ++m) {
    const int i = w + 4 * m;
    if (i < i0 || i >= i1) continue;  // warp-uniform
    const float4 x = stg4(stg, i, 4 * l);
    float4 nv;
    nv.x = old[m].x + x.x;
    nv.y = old[m].y + x.y;
    nv.z = old[m].z + x.z;
    nv.w = old[m].w + x.w;
    *reinterpret_cast<float4*>(e.y + (size_t)i * e.ldy + o) = nv;
    if (e.xa_out != nullptr) {
      uint2 hi, lo;
      split4(make_float4(nv.x * gn.x, nv.y * gn.y, nv.z * gn.z, nv.w * gn.w), hi, lo);
      *reinterpret_cast<uint2*>(e.xa_out + (size_t)i * e.ldy + o) = hi;
      *reinterpret_cast<uint2*>(e.xa_out + (size_t)(64 + i) * e.ldy + o) = lo;
    }
    if (e.ss_out != nullptr) {
      const float s = warp_sum(nv.x * nv.x + nv.y * nv.y + nv.z * nv.z + nv.w * nv.w);
      if (l == 0) e.ss_out[tile * 64 + i] = s;
    }
  }
  bar();
}

template <int BN, int EPI, typename Bar>
__device__ __forceinline__ void run_epilogue(const EpiParams& e, int tile, int r, const float* v, float* stg, Bar bar,
                                             int i0, int i1) {
  if constexpr (EPI == EPI_STORE) epi_store<BN>(e, tile, r, v, stg, bar, i0, i1);
  if constexpr (EPI == EPI_RESID) epi_resid<BN>(e, tile, r, v, stg, bar, i0, i1);
  if constexpr (EPI == EPI_QKV) epi_qkv<BN>(e, tile, r, v, stg, bar, i0, i1);
  if constexpr (EPI == EPI_GLU) epi_glu<BN>(e, tile, r, v, stg, bar, i0, i1);
  if constexpr (EPI == EPI_LMHEAD) epi_lmhead<BN>(e, tile, r, v, stg, bar, i0, i1);
}

}  // namespace casspec
