// Tree attention (Sec. 4.2: parallel verification / drafting of a token tree).
//
// Node i of the tree attends to every committed prefix slot [0, P) and to the tree slots of its
// ancestors and itself (bit j of anc[i] <=> tree slot j, cache slot P + j).
//   * work split: the (head, 64-slot KV block) units of all heads are divided evenly over the grid
//     (contiguous ranges, stream-K style), so every SM streams the same number of K/V bytes; a CTA
//     whose range crosses a head boundary handles one segment per head;
//   * K/V blocks arrive by TMA (2-D tensor map over the whole cache, 128-byte swizzle, 64 slots x 64
//     dims per box) in an S-stage mbarrier ring fed by a dedicated producer warp;
//   * four compute warps, 16 query rows each, run QK^T and PV on tensor cores (mma.sync m16n8k16
//     bf16 -> fp32) with ldmatrix addresses XOR-swizzled to match the TMA layout, the ancestor mask
//     applied to the scores, and an online softmax whose row reductions are quad shuffles;
//   * a head split across CTAs is merged by the CTA that finishes it last (atomic counter), in
//     segment order, so the result does not depend on CTA timing.
#include "common.cuh"
#include "kernels.h"

namespace casspec {

constexpr int kAttnCompute = 128;                // 4 compute warps
constexpr int kAttnThreads = kAttnCompute + 32;  // + producer warp
constexpr int kAttnBlk = 64;
constexpr int kAttnStages = 3;

template <int HD>
__host__ __device__ constexpr uint32_t attn_tile_bytes() {
  return (uint32_t)kAttnBlk * HD * 2;
}
template <int HD>
__host__ __device__ constexpr size_t attn_smem_bytes() {
  return (size_t)kAttnStages * 2 * attn_tile_bytes<HD>() + (size_t)64 * HD * 2 + 128;
}

// Address of 16-byte chunk `c` (0 .. HD/8-1) of row `r` in a [64][HD] bf16 tile stored as HD/64
// sub-tiles of [64][128 B] with the 128-byte swizzle (TMA's layout; tile base 1024-byte aligned).
__device__ __forceinline__ uint32_t swz(uint32_t tile, int r, int c) {
  return tile + (uint32_t)(c >> 3) * 8192u + (uint32_t)r * 128u + ((uint32_t)((c & 7) ^ (r & 7)) << 4);
}

// CTA whose unit range [cU/G, (c+1)U/G) contains unit x.
__device__ __forceinline__ int cta_of(long long x, long long U, int G) { return (int)(((x + 1) * G - 1) / U); }

template <int HD>
__global__ void __launch_bounds__(kAttnThreads, 2) tree_attn_kernel(const __grid_constant__ CUtensorMap tmKV,
                                                                  const AttnArgs a) {
  constexpr uint32_t TILE = attn_tile_bytes<HD>();
  constexpr uint32_t STAGE = 2 * TILE;
  constexpr int S = kAttnStages;
  constexpr int NCH = HD / 8;  // 16-byte chunks per row
  extern __shared__ __align__(1024) uint8_t sm[];
  uint8_t* ring = sm;
  uint8_t* qs = sm + S * STAGE;
  uint64_t* full = reinterpret_cast<uint64_t*>(qs + 64 * HD * 2);
  uint64_t* empty = full + S;
  volatile int* flags = reinterpret_cast<volatile int*>(empty + S);  // [0] abort, [2..3] heads to merge

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = gridDim.x, cta = blockIdx.x;
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 4);
    }
    flags[0] = 0;
    flags[2] = -1;
    flags[3] = -1;
    fence_mbar_init();
  }
  if (tid == kAttnCompute) tma_prefetch_desc(&tmKV);
  __syncthreads();
  pdl_trigger();
  pdl_wait();
  if ((smem_u32(sm) & 1023u) != 0) {  // the swizzle addressing assumes 1024-byte aligned tiles
    if (tid == 0) set_status(a.status, CASSPEC_E_CUDA);
    return;
  }

  const int P = __ldcg(a.dP);
  const int total = P + a.T + a.n;
  const int nblk = (total + kAttnBlk - 1) / kAttnBlk;
  const long long U = (long long)a.n_heads * nblk;
  const long long u0 = (long long)cta * U / G, u1 = (long long)(cta + 1) * U / G;
  const int H = a.n_heads;

  if (warp == 4) {
    // ---------------- producer ----------------
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_parity = 0;
      for (long long u = u0; u < u1; ++u) {
        const int h = (int)(u / nblk), b = (int)(u % nblk);
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1, flags)) {
          flags[0] = 1;
          set_status(a.status, CASSPEC_E_TIMEOUT);
          break;
        }
        mbar_expect_tx(&full[stage], STAGE);
        armed |= 1u << stage;
        armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
        const int row_k = ((a.layer * 2 + 0) * H + h) * a.ctx + b * kAttnBlk;
        const int row_v = ((a.layer * 2 + 1) * H + h) * a.ctx + b * kAttnBlk;
        uint8_t* st = ring + stage * STAGE;
#pragma unroll
        for (int sub = 0; sub < HD / 64; ++sub) {
          tma_load_2d(st + sub * 8192, &tmKV, &full[stage], sub * 64, row_k, pol);
          tma_load_2d(st + TILE + sub * 8192, &tmKV, &full[stage], sub * 64, row_v, pol);
        }
        if (++stage == S) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (flags[0]) {  // abort: let the copies already issued land before the CTA exits
        for (int s = 0; s < S; ++s)
          if (armed & (1u << s)) mbar_wait_bounded(&full[s], (armed_parity >> s) & 1, nullptr);
      }
    }
    return;
  }

  // ---------------- compute warps ----------------
  const uint32_t qbase = smem_u32(qs);
  const int row0 = warp * 16;
  const bool active = row0 < a.n;
  const int g = lane >> 2, t4 = lane & 3;
  const int rA = row0 + g, rB = rA + 8;
  const unsigned long long ancA = rA < a.n ? __ldcg(a.anc + rA) : 0ull;
  const unsigned long long ancB = rB < a.n ? __ldcg(a.anc + rB) : 0ull;
  auto cbar = [] { named_bar_sync(1, kAttnCompute); };

  uint32_t qf[HD / 16][4];
  float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;
  float oacc[HD / 8][4];
  int stage = 0;
  uint32_t phase = 0;
  int h_cur = -1;
  bool ok = true;

  // End of this CTA's segment of head h: a head held by one CTA is written directly; otherwise the
  // partial (m, l, unnormalised O) goes to slot h + cta, and the head's last CTA is recorded.
  auto finish = [&](int h) {
    float LA = lA, LB = lB;  // complete the per-quad row sums
    LA += __shfl_xor_sync(0xffffffffu, LA, 1);
    LA += __shfl_xor_sync(0xffffffffu, LA, 2);
    LB += __shfl_xor_sync(0xffffffffu, LB, 1);
    LB += __shfl_xor_sync(0xffffffffu, LB, 2);
    const int c_first = cta_of((long long)h * nblk, U, G), c_last = cta_of((long long)(h + 1) * nblk - 1, U, G);
    if (c_first == c_last) {
      if (active) {
#pragma unroll
        for (int dt = 0; dt < HD / 8; ++dt) {
          const int col = h * HD + dt * 8 + 2 * t4;
          if (rA < a.n)
            *reinterpret_cast<uint32_t*>(a.o + (size_t)rA * a.d + col) = pack_bf16x2(oacc[dt][0] / LA, oacc[dt][1] / LA);
          if (rB < a.n)
            *reinterpret_cast<uint32_t*>(a.o + (size_t)rB * a.d + col) = pack_bf16x2(oacc[dt][2] / LB, oacc[dt][3] / LB);
        }
      }
      return;
    }
    const size_t slot = (size_t)h + cta;
    if (active) {
#pragma unroll
      for (int dt = 0; dt < HD / 8; ++dt) {
        const int col = dt * 8 + 2 * t4;
        if (rA < a.n)
          __stcg(reinterpret_cast<float2*>(a.part_o + (slot * 64 + rA) * HD + col), make_float2(oacc[dt][0], oacc[dt][1]));
        if (rB < a.n)
          __stcg(reinterpret_cast<float2*>(a.part_o + (slot * 64 + rB) * HD + col), make_float2(oacc[dt][2], oacc[dt][3]));
      }
      if (t4 == 0) {
        if (rA < a.n) __stcg(reinterpret_cast<float2*>(a.part_ml + (slot * 64 + rA) * 2), make_float2(mA, LA));
        if (rB < a.n) __stcg(reinterpret_cast<float2*>(a.part_ml + (slot * 64 + rB) * 2), make_float2(mB, LB));
      }
    }
    __threadfence();
    cbar();
    if (tid == 0) {
      const unsigned old = atomicAdd(&a.counters[h], 1u);
      if (old == (unsigned)(c_last - c_first)) {
        if (flags[2] < 0)
          flags[2] = h;
        else if (flags[3] < 0)
          flags[3] = h;
        else
          set_status(a.status, CASSPEC_E_CUDA);  // grid sizing keeps a CTA within two heads
      }
    }
    cbar();
  };

  for (long long u = u0; u < u1; ++u) {
    const int h = (int)(u / nblk), b = (int)(u % nblk);
    if (h != h_cur) {
      if (h_cur >= 0) finish(h_cur);
      cbar();  // nobody reads the previous head's Q any more
      for (int idx = tid; idx < 64 * NCH; idx += kAttnCompute) {
        const int row = idx / NCH, c = idx % NCH;
        uint4 val = make_uint4(0, 0, 0, 0);
        if (row < a.n) val = __ldcg(reinterpret_cast<const uint4*>(a.q + (size_t)row * a.d + h * HD + c * 8));
        asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(swz(qbase, row, c)), "r"(val.x), "r"(val.y),
                     "r"(val.z), "r"(val.w)
                     : "memory");
      }
      cbar();
      if (active) {
#pragma unroll
        for (int kt = 0; kt < HD / 16; ++kt) {
          const int mi = lane >> 3;
          ldmatrix_x4_a(qf[kt][0], qf[kt][1], qf[kt][2], qf[kt][3],
                        swz(qbase, row0 + (lane & 7) + 8 * (mi & 1), 2 * kt + (mi >> 1)));
        }
      }
      mA = mB = -INFINITY;
      lA = lB = 0.f;
#pragma unroll
      for (int dt = 0; dt < HD / 8; ++dt) oacc[dt][0] = oacc[dt][1] = oacc[dt][2] = oacc[dt][3] = 0.f;
      h_cur = h;
    }
    if (!mbar_wait_bounded(&full[stage], phase, flags)) {
      flags[0] = 1;
      set_status(a.status, CASSPEC_E_TIMEOUT);
      ok = false;
      break;
    }
    if (active) {
      const uint32_t kb = smem_u32(ring + stage * STAGE), vb = kb + TILE;
      float s[8][4];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
      for (int kt = 0; kt < HD / 16; ++kt) {
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          const int mi = lane >> 3;
          uint32_t k0, k1, k2, k3;
          ldmatrix_x4_a(k0, k1, k2, k3, swz(kb, 16 * np + 8 * (mi >> 1) + (lane & 7), 2 * kt + (mi & 1)));
          mma_bf16_16816(s[2 * np], qf[kt][0], qf[kt][1], qf[kt][2], qf[kt][3], k0, k1);
          mma_bf16_16816(s[2 * np + 1], qf[kt][0], qf[kt][1], qf[kt][2], qf[kt][3], k2, k3);
        }
      }
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
#pragma unroll
      for (int kc = 0; kc < 4; ++kc) {
        const uint32_t a0 = pack_bf16x2(s[2 * kc][0], s[2 * kc][1]);
        const uint32_t a1 = pack_bf16x2(s[2 * kc][2], s[2 * kc][3]);
        const uint32_t a2 = pack_bf16x2(s[2 * kc + 1][0], s[2 * kc + 1][1]);
        const uint32_t a3 = pack_bf16x2(s[2 * kc + 1][2], s[2 * kc + 1][3]);
#pragma unroll
        for (int dp = 0; dp < HD / 16; ++dp) {
          const int mi = lane >> 3;
          uint32_t v0, v1, v2, v3;
          ldmatrix_x4_trans_a(v0, v1, v2, v3, swz(vb, 16 * kc + (lane & 7) + 8 * (mi & 1), 2 * dp + (mi >> 1)));
          mma_bf16_16816(oacc[2 * dp], a0, a1, a2, a3, v0, v1);
          mma_bf16_16816(oacc[2 * dp + 1], a0, a1, a2, a3, v2, v3);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[stage]);
    if (++stage == S) {
      stage = 0;
      phase ^= 1;
    }
  }
  if (!ok) return;
  if (h_cur >= 0) finish(h_cur);

  // ---- merge the heads this CTA finished last (the K/V ring is idle now) ----
  float* w_s = reinterpret_cast<float*>(ring);  // [64][segments]
  constexpr int ITEMS = 64 * (HD / 4) / kAttnCompute;  // float4 outputs per thread
  for (int k = 2; k <= 3; ++k) {
    const int h = flags[k];
    if (h < 0) continue;
    const int c_first = cta_of((long long)h * nblk, U, G), c_last = cta_of((long long)(h + 1) * nblk - 1, U, G);
    const int nseg = c_last - c_first + 1;
    __threadfence();
    for (int row = tid; row < a.n; row += kAttnCompute) {
      float M = -INFINITY;
      for (int sg = 0; sg < nseg; ++sg) M = fmaxf(M, __ldcg(a.part_ml + (((size_t)h + c_first + sg) * 64 + row) * 2));
      float L = 0.f;
      for (int sg = 0; sg < nseg; ++sg) {
        const float2 ml =
            __ldcg(reinterpret_cast<const float2*>(a.part_ml + (((size_t)h + c_first + sg) * 64 + row) * 2));
        const float w = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);
        w_s[row * nseg + sg] = w;
        L += ml.y * w;
      }
      const float invL = 1.f / L;
      for (int sg = 0; sg < nseg; ++sg) w_s[row * nseg + sg] *= invL;
    }
    cbar();
    float4 o[ITEMS];
#pragma unroll
    for (int it = 0; it < ITEMS; ++it) o[it] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int sg = 0; sg < nseg; ++sg) {
      const size_t slot = (size_t)h + c_first + sg;
#pragma unroll
      for (int it = 0; it < ITEMS; ++it) {
        const int idx = tid + it * kAttnCompute;
        const int row = idx / (HD / 4), c4 = (idx % (HD / 4)) * 4;
        if (row < a.n) {
          const float w = w_s[row * nseg + sg];
          const float4 ov = __ldcg(reinterpret_cast<const float4*>(a.part_o + (slot * 64 + row) * HD + c4));
          o[it].x += ov.x * w;
          o[it].y += ov.y * w;
          o[it].z += ov.z * w;
          o[it].w += ov.w * w;
        }
      }
    }
#pragma unroll
    for (int it = 0; it < ITEMS; ++it) {
      const int idx = tid + it * kAttnCompute;
      const int row = idx / (HD / 4), c4 = (idx % (HD / 4)) * 4;
      if (row < a.n) {
        uint2 pk;
        pk.x = pack_bf16x2(o[it].x, o[it].y);
        pk.y = pack_bf16x2(o[it].z, o[it].w);
        *reinterpret_cast<uint2*>(a.o + (size_t)row * a.d + h * HD + c4) = pk;
      }
    }
    if (tid == 0) a.counters[h] = 0u;
    cbar();
  }
}

int attn_grid(int n_heads, int total_slots, int num_sms) {
  const long long U = (long long)n_heads * ((total_slots + kAttnBlk - 1) / kAttnBlk);
  const long long G = 2LL * num_sms;  // two CTAs per SM
  return (int)(U < G ? U : G);
}

template <int HD>
static cudaError_t launch_hd(const CUtensorMap& tm, const AttnArgs& a, int grid, cudaStream_t stream, bool pdl) {
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
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kAttnThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, tm, a);
}

cudaError_t launch_tree_attention(const CUtensorMap& tm, const AttnArgs& a, int hd, int grid, cudaStream_t stream,
                                  bool pdl) {
  if (hd == 128) return launch_hd<128>(tm, a, grid, stream, pdl);
  if (hd == 64) return launch_hd<64>(tm, a, grid, stream, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace casspec
