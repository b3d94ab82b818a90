// Tree attention (Sec. 4.2: parallel verification / drafting of a token tree).
//
// Node i of the tree attends to every committed prefix slot [0, P) and to the tree slots of its
// ancestors and itself (bit j of anc[i] <=> tree slot j, cache slot P + j).  One CTA handles one
// head and a contiguous range of 64-slot KV blocks (split-KV across SMs):
//   * K/V blocks are staged in shared memory with 16-byte cp.async, double buffered; the cache is
//     head-major ([H][ctx][hd]) so each block is one contiguous 64 * hd * 2-byte run;
//   * QK^T and PV run on tensor cores (mma.sync m16n8k16 bf16 -> fp32), one warp per 16 query
//     rows, with the ancestor mask applied to the scores and an online (running max) softmax whose
//     row reductions are quad shuffles;
//   * the CTA that finishes a head last (atomic counter) merges the per-split (max, sum, output)
//     partials in split order, so the result does not depend on CTA timing.
#include "common.cuh"
#include "kernels.h"

namespace casspec {

constexpr int kAttnThreads = 128;
constexpr int kAttnBlk = 64;

template <int HD>
__host__ __device__ constexpr size_t attn_smem_bytes() {
  return (size_t)(64 + 4 * kAttnBlk) * (HD + 8) * 2;
}

template <int HD>
__global__ void __launch_bounds__(kAttnThreads) tree_attn_kernel(const AttnArgs a) {
  constexpr int PITCH = HD + 8;  // bf16 per smem row: 16-byte skew keeps ldmatrix conflict-free
  constexpr int C8 = HD / 8;     // 16-byte chunks per row
  extern __shared__ __align__(16) uint16_t sm[];
  uint16_t* Qs = sm;
  uint16_t* Ks = Qs + 64 * PITCH;
  uint16_t* Vs = Ks + 2 * kAttnBlk * PITCH;
  __shared__ int s_last;

  const int head = blockIdx.x, split = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  pdl_trigger();
  pdl_wait();

  const int P = __ldcg(a.dP);
  const int total = P + a.T + a.n;
  const int nblk = (total + kAttnBlk - 1) / kAttnBlk;
  const int b0 = (int)((long long)split * nblk / a.splits);
  const int b1 = (int)((long long)(split + 1) * nblk / a.splits);
  const uint16_t* kbase = a.kc + (size_t)head * a.ctx * HD;
  const uint16_t* vbase = a.vc + (size_t)head * a.ctx * HD;

  for (int idx = tid; idx < 64 * C8; idx += kAttnThreads) {
    const int row = idx / C8, c8 = idx % C8;
    uint4 val = make_uint4(0, 0, 0, 0);
    if (row < a.n) val = __ldcg(reinterpret_cast<const uint4*>(a.q + (size_t)row * a.d + head * HD + c8 * 8));
    *reinterpret_cast<uint4*>(Qs + row * PITCH + c8 * 8) = val;
  }
  auto load_block = [&](int b, int buf) {
    const int s0 = b * kAttnBlk;
    for (int idx = tid; idx < kAttnBlk * C8; idx += kAttnThreads) {
      const int row = idx / C8, c8 = idx % C8;
      const int slot = s0 + row;
      uint16_t* dk = Ks + (buf * kAttnBlk + row) * PITCH + c8 * 8;
      uint16_t* dv = Vs + (buf * kAttnBlk + row) * PITCH + c8 * 8;
      if (slot < total) {
        cp_async16(dk, kbase + (size_t)slot * HD + c8 * 8);
        cp_async16(dv, vbase + (size_t)slot * HD + c8 * 8);
      } else {
        *reinterpret_cast<uint4*>(dk) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(dv) = make_uint4(0, 0, 0, 0);
      }
    }
    cp_async_commit();
  };
  if (b0 < b1) load_block(b0, 0);
  __syncthreads();  // Q staged

  const int row0 = warp * 16;
  const bool active = row0 < a.n;
  const int g = lane >> 2, t4 = lane & 3;
  const int rA = row0 + g, rB = rA + 8;
  const unsigned long long ancA = rA < a.n ? __ldcg(a.anc + rA) : 0ull;
  const unsigned long long ancB = rB < a.n ? __ldcg(a.anc + rB) : 0ull;

  uint32_t qf[HD / 16][4];
  if (active) {
#pragma unroll
    for (int kt = 0; kt < HD / 16; ++kt) {
      const int mi = lane >> 3;
      const uint16_t* p = Qs + (row0 + (lane & 7) + 8 * (mi & 1)) * PITCH + kt * 16 + 8 * (mi >> 1);
      ldmatrix_x4(qf[kt][0], qf[kt][1], qf[kt][2], qf[kt][3], p);
    }
  }
  float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;
  float oacc[HD / 8][4];
#pragma unroll
  for (int dt = 0; dt < HD / 8; ++dt) oacc[dt][0] = oacc[dt][1] = oacc[dt][2] = oacc[dt][3] = 0.f;

  for (int b = b0; b < b1; ++b) {
    const int buf = (b - b0) & 1;
    if (b + 1 < b1) {
      load_block(b + 1, buf ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (active) {
      const uint16_t* Kb = Ks + buf * kAttnBlk * PITCH;
      const uint16_t* Vb = Vs + buf * kAttnBlk * PITCH;
      float s[8][4];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
      for (int kt = 0; kt < HD / 16; ++kt) {
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          const int mi = lane >> 3;
          const uint16_t* p = Kb + (16 * np + 8 * (mi >> 1) + (lane & 7)) * PITCH + kt * 16 + 8 * (mi & 1);
          uint32_t k0, k1, k2, k3;
          ldmatrix_x4(k0, k1, k2, k3, p);
          mma_bf16_16816(s[2 * np], qf[kt][0], qf[kt][1], qf[kt][2], qf[kt][3], k0, k1);
          mma_bf16_16816(s[2 * np + 1], qf[kt][0], qf[kt][1], qf[kt][2], qf[kt][3], k2, k3);
        }
      }
      // mask + scale
      const int sbase = b * kAttnBlk;
      float mxA = -INFINITY, mxB = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int slot = sbase + nt * 8 + 2 * t4 + e;
          bool visA, visB;
          if (slot < P) {
            visA = visB = true;
          } else if (slot < total) {
            const int j = slot - P;
            visA = (ancA >> j) & 1ull;
            visB = (ancB >> j) & 1ull;
          } else {
            visA = visB = false;
          }
          s[nt][e] = visA ? s[nt][e] * a.scale_log2 : -INFINITY;
          s[nt][2 + e] = visB ? s[nt][2 + e] * a.scale_log2 : -INFINITY;
          mxA = fmaxf(mxA, s[nt][e]);
          mxB = fmaxf(mxB, s[nt][2 + e]);
        }
      }
      mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 1));
      mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 2));
      mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 1));
      mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 2));
      const float nA = fmaxf(mA, mxA), nB = fmaxf(mB, mxB);
      const float uA = (nA == -INFINITY) ? 0.f : nA, uB = (nB == -INFINITY) ? 0.f : nB;
      const float cA = exp2f(mA - uA), cB = exp2f(mB - uB);
      mA = nA;
      mB = nB;
      float sumA = 0.f, sumB = 0.f;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        s[nt][0] = exp2f(s[nt][0] - uA);
        s[nt][1] = exp2f(s[nt][1] - uA);
        s[nt][2] = exp2f(s[nt][2] - uB);
        s[nt][3] = exp2f(s[nt][3] - uB);
        sumA += s[nt][0] + s[nt][1];
        sumB += s[nt][2] + s[nt][3];
      }
      lA = lA * cA + sumA;
      lB = lB * cB + sumB;
#pragma unroll
      for (int dt = 0; dt < HD / 8; ++dt) {
        oacc[dt][0] *= cA;
        oacc[dt][1] *= cA;
        oacc[dt][2] *= cB;
        oacc[dt][3] *= cB;
      }
      // O += P V
#pragma unroll
      for (int kc = 0; kc < 4; ++kc) {
        const uint32_t a0 = pack_bf16x2(s[2 * kc][0], s[2 * kc][1]);
        const uint32_t a1 = pack_bf16x2(s[2 * kc][2], s[2 * kc][3]);
        const uint32_t a2 = pack_bf16x2(s[2 * kc + 1][0], s[2 * kc + 1][1]);
        const uint32_t a3 = pack_bf16x2(s[2 * kc + 1][2], s[2 * kc + 1][3]);
#pragma unroll
        for (int dp = 0; dp < HD / 16; ++dp) {
          const int mi = lane >> 3;
          const uint16_t* p = Vb + (16 * kc + (lane & 7) + 8 * (mi & 1)) * PITCH + 16 * dp + 8 * (mi >> 1);
          uint32_t v0, v1, v2, v3;
          ldmatrix_x4_trans(v0, v1, v2, v3, p);
          mma_bf16_16816(oacc[2 * dp], a0, a1, a2, a3, v0, v1);
          mma_bf16_16816(oacc[2 * dp + 1], a0, a1, a2, a3, v2, v3);
        }
      }
    }
    __syncthreads();  // this buffer is refilled two iterations later
  }
  lA += __shfl_xor_sync(0xffffffffu, lA, 1);
  lA += __shfl_xor_sync(0xffffffffu, lA, 2);
  lB += __shfl_xor_sync(0xffffffffu, lB, 1);
  lB += __shfl_xor_sync(0xffffffffu, lB, 2);

  if (a.splits == 1) {
    if (active) {
#pragma unroll
      for (int dt = 0; dt < HD / 8; ++dt) {
        const int col = head * HD + dt * 8 + 2 * t4;
        if (rA < a.n)
          *reinterpret_cast<uint32_t*>(a.o + (size_t)rA * a.d + col) = pack_bf16x2(oacc[dt][0] / lA, oacc[dt][1] / lA);
        if (rB < a.n)
          *reinterpret_cast<uint32_t*>(a.o + (size_t)rB * a.d + col) = pack_bf16x2(oacc[dt][2] / lB, oacc[dt][3] / lB);
      }
    }
    return;
  }

  // ---- partials of this split, then the last CTA of the head merges them in split order ----
  const size_t pbase = (size_t)head * a.splits + split;
  if (active) {
#pragma unroll
    for (int dt = 0; dt < HD / 8; ++dt) {
      const int col = dt * 8 + 2 * t4;
      if (rA < a.n) __stcg(reinterpret_cast<float2*>(a.part_o + (pbase * 64 + rA) * HD + col), make_float2(oacc[dt][0], oacc[dt][1]));
      if (rB < a.n) __stcg(reinterpret_cast<float2*>(a.part_o + (pbase * 64 + rB) * HD + col), make_float2(oacc[dt][2], oacc[dt][3]));
    }
    if (t4 == 0) {
      if (rA < a.n) __stcg(reinterpret_cast<float2*>(a.part_ml + (pbase * 64 + rA) * 2), make_float2(mA, lA));
      if (rB < a.n) __stcg(reinterpret_cast<float2*>(a.part_ml + (pbase * 64 + rB) * 2), make_float2(mB, lB));
    }
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const unsigned old = atomicAdd(&a.counters[head], 1u);
    s_last = (old == (unsigned)(a.splits - 1)) ? 1 : 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // merge: per-(row, split) weights 2^(m_s - M) / L staged in shared memory first (one pass of
  // independent loads), then every output is a weighted sum over splits with independent loads.
  float* w_s = reinterpret_cast<float*>(Ks);  // [64][splits] (K/V staging is free now)
  const int S = a.splits;
  for (int row = tid; row < a.n; row += kAttnThreads) {
    float M = -INFINITY;
    for (int sp = 0; sp < S; ++sp)
      M = fmaxf(M, __ldcg(a.part_ml + (((size_t)head * S + sp) * 64 + row) * 2));
    float L = 0.f;
    for (int sp = 0; sp < S; ++sp) {
      const float2 ml = __ldcg(reinterpret_cast<const float2*>(a.part_ml + (((size_t)head * S + sp) * 64 + row) * 2));
      const float w = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);
      w_s[row * S + sp] = w;
      L += ml.y * w;
    }
    const float invL = 1.f / L;
    for (int sp = 0; sp < S; ++sp) w_s[row * S + sp] *= invL;
  }
  __syncthreads();
  for (int idx = tid; idx < a.n * (HD / 4); idx += kAttnThreads) {
    const int row = idx / (HD / 4), c4 = (idx % (HD / 4)) * 4;
    float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int sp = 0; sp < S; ++sp) {
      const float w = w_s[row * S + sp];
      if (w == 0.f) continue;
      const float4 ov = __ldcg(reinterpret_cast<const float4*>(a.part_o + (((size_t)head * S + sp) * 64 + row) * HD + c4));
      o.x += ov.x * w;
      o.y += ov.y * w;
      o.z += ov.z * w;
      o.w += ov.w * w;
    }
    uint2 pk;
    pk.x = pack_bf16x2(o.x, o.y);
    pk.y = pack_bf16x2(o.z, o.w);
    *reinterpret_cast<uint2*>(a.o + (size_t)row * a.d + head * HD + c4) = pk;
  }
  if (tid == 0) a.counters[head] = 0u;
}

int attn_splits(int n_heads, int total_slots, int num_sms) {
  const int nblk = (total_slots + kAttnBlk - 1) / kAttnBlk;
  int s = (2 * num_sms) / n_heads;  // two CTAs per SM: the whole grid runs in one wave
  if (s > nblk) s = nblk;
  if (s > 64) s = 64;  // the merge stages 64 x splits weights in the K staging area
  if (s < 1) s = 1;
  return s;
}

template <int HD>
static cudaError_t launch_hd(const AttnArgs& a, int n_heads, cudaStream_t stream, bool pdl) {
  auto kern = tree_attn_kernel<HD>;
  constexpr size_t smem = attn_smem_bytes<HD>();
  static int configured = -1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured != dev) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_heads, a.splits);
  cfg.blockDim = dim3(kAttnThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

cudaError_t launch_tree_attention(const AttnArgs& a, int hd, int n_heads, cudaStream_t stream, bool pdl) {
  if (hd == 128) return launch_hd<128>(a, n_heads, stream, pdl);
  if (hd == 64) return launch_hd<64>(a, n_heads, stream, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace casspec
