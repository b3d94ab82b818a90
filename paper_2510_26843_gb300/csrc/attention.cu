// Tree attention (Sec. 4.2: parallel verification / drafting of a token tree).
//
// Node i of the tree attends to every committed prefix slot [0, P) and to the tree slots of its
// ancestors and itself (bit j of anc[i] <=> tree slot j, cache slot P + j).
//   * S CTAs per head (split-KV, S * heads <= 2 per SM, so the whole grid is resident at once);
//     split s handles the s-th contiguous share of the head's 64-slot KV blocks;
//   * K/V blocks arrive by TMA (2-D tensor map over the whole cache, 128-byte swizzle, 64 slots x 64
//     dims per box) in an S-stage mbarrier ring fed by a dedicated producer warp;
//   * four compute warps, 16 query rows each, run QK^T and PV on tensor cores (mma.sync m16n8k16
//     bf16 -> fp32) with ldmatrix addresses XOR-swizzled to match the TMA layout, the ancestor mask
//     applied to the scores, and an online softmax whose row reductions are quad shuffles;
//   * each split writes its partial (running max, sum, unnormalised output) to global scratch and
//     counts itself in; once all S splits of the head have arrived, split s merges rows
//     s, s + S, ... over the S partials in split order (fixed, so results do not depend on timing)
//     and the last split out returns the head's counters to zero.
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

template <int HD>
__global__ void __launch_bounds__(kAttnThreads, 2) tree_attn_kernel(const __grid_constant__ CUtensorMap tmKV,
                                                                     const AttnArgs a) {
  constexpr uint32_t TILE = attn_tile_bytes<HD>();
  constexpr uint32_t STAGE = 2 * TILE;
  constexpr int S = kAttnStages;
  constexpr int NCH = HD / 8;  // 16-byte chunks per row
  static_assert(64 * kAttnMaxSplits * 12 + 64 * 4 <= S * STAGE, "merge weights must fit in the K/V ring");
  extern __shared__ __align__(1024) uint8_t sm[];
  uint8_t* ring = sm;
  uint8_t* qs = sm + S * STAGE;
  uint64_t* full = reinterpret_cast<uint64_t*>(qs + 64 * HD * 2);
  uint64_t* empty = full + S;
  volatile int* flags = reinterpret_cast<volatile int*>(empty + S);  // [0] abort, [1] merge go-ahead

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int C = a.splits;
  const int head = blockIdx.x / C;
  const int rank = blockIdx.x % C;
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 4);
    }
    flags[0] = 0;
    flags[1] = 0;
    fence_mbar_init();
  }
  // The committed length P is written only between steps (compaction, set_prefix), by kernels that
  // completed before this step's first kernel started, so it can be read before the dependency wait.
  // The blocks of this split that lie wholly inside the committed prefix do not depend on the
  // preceding kernels either: the producer loads the first of them into the ring before the wait,
  // and asks L2 for the rest, while the previous kernel finishes.
  const int Pp = *reinterpret_cast<const volatile int*>(a.dP);
  const bool aligned = (smem_u32(sm) & 1023u) == 0;  // the swizzle addressing needs 1024-byte tiles
  if (tid == kAttnCompute) {
    tma_prefetch_desc(&tmKV);
    if (Pp >= 0 && Pp <= a.ctx) {
      const int nb = min((Pp + a.T + a.n + kAttnBlk - 1) / kAttnBlk, a.ctx / kAttnBlk);
      const int row_k = ((a.layer * 2 + 0) * a.n_heads + head) * a.ctx;
      const int row_v = ((a.layer * 2 + 1) * a.n_heads + head) * a.ctx;
      for (int b = rank * nb / C + S; b < (rank + 1) * nb / C; ++b) {
#pragma unroll
        for (int sub = 0; sub < HD / 64; ++sub) {
          tma_prefetch_l2_2d(&tmKV, sub * 64, row_k + b * kAttnBlk);
          tma_prefetch_l2_2d(&tmKV, sub * 64, row_v + b * kAttnBlk);
        }
      }
    }
  }
  __syncthreads();
  pdl_trigger();
  if (warp != 4) pdl_wait();  // the producer waits after its prefix loads

  const int P = warp == 4 ? Pp : __ldcg(a.dP);
  const int total = P + a.T + a.n;
  const int nblk = (total + kAttnBlk - 1) / kAttnBlk;
  const int b0 = rank * nblk / C, b1 = (rank + 1) * nblk / C;
  if (!aligned && tid == 0) set_status(a.status, CASSPEC_E_CUDA);

  float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;
  float oacc[HD / 8][4];
#pragma unroll
  for (int dt = 0; dt < HD / 8; ++dt) oacc[dt][0] = oacc[dt][1] = oacc[dt][2] = oacc[dt][3] = 0.f;
  const int row0 = warp * 16;
  const bool active = warp < 4 && row0 < a.n;
  const int g = lane >> 2, t4 = lane & 3;
  const int rA = row0 + g, rB = rA + 8;
  auto cbar = [] { named_bar_sync(1, kAttnCompute); };

  if (warp == 4) {
    // ---------------- producer ----------------
    if (lane == 0 && aligned) {
      const uint64_t pol = policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_parity = 0;
      const int row_k = ((a.layer * 2 + 0) * a.n_heads + head) * a.ctx;
      const int row_v = ((a.layer * 2 + 1) * a.n_heads + head) * a.ctx;
      bool waited = false;
      for (int b = b0; b < b1; ++b) {
        if (!waited && (b - b0 >= S || (b + 1) * kAttnBlk > P || P < 0 || P > a.ctx)) {
          pdl_wait();  // from here on the blocks may hold this step's tree K/V
          waited = true;
          if (__ldcg(a.dP) != P) set_status(a.status, CASSPEC_E_STATE);  // P moved during a step
        }
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1, flags)) {
          flags[0] = 1;
          set_status(a.status, CASSPEC_E_TIMEOUT);
          break;
        }
        mbar_expect_tx(&full[stage], STAGE);
        armed |= 1u << stage;
        armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
        uint8_t* st = ring + stage * STAGE;
#pragma unroll
        for (int sub = 0; sub < HD / 64; ++sub) {
          tma_load_2d(st + sub * 8192, &tmKV, &full[stage], sub * 64, row_k + b * kAttnBlk, pol);
          tma_load_2d(st + TILE + sub * 8192, &tmKV, &full[stage], sub * 64, row_v + b * kAttnBlk, pol);
        }
        if (++stage == S) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (!waited) pdl_wait();
      if (flags[0]) {  // abort: let the copies already issued land before the ring is reused
        for (int s = 0; s < S; ++s)
          if (armed & (1u << s)) mbar_wait_bounded(&full[s], (armed_parity >> s) & 1, nullptr);
      }
    }
    __syncwarp();
  } else if (aligned) {
    // ---------------- compute warps ----------------
    const uint32_t qbase = smem_u32(qs);
    const unsigned long long ancA = rA < a.n ? __ldcg(a.anc + rA) : 0ull;
    const unsigned long long ancB = rB < a.n ? __ldcg(a.anc + rB) : 0ull;
    constexpr int QPT = 64 * NCH / kAttnCompute;  // 16-byte chunks of Q per thread
    uint4 qv[QPT];  // every load in flight before the first shared-memory store
#pragma unroll
    for (int k = 0; k < QPT; ++k) {
      const int idx = tid + k * kAttnCompute, row = idx / NCH, c = idx % NCH;
      qv[k] = row < a.n ? __ldcg(reinterpret_cast<const uint4*>(a.q + (size_t)row * a.d + head * HD + c * 8))
                        : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int k = 0; k < QPT; ++k) {
      const int idx = tid + k * kAttnCompute, row = idx / NCH, c = idx % NCH;
      asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(swz(qbase, row, c)), "r"(qv[k].x), "r"(qv[k].y),
                   "r"(qv[k].z), "r"(qv[k].w)
                   : "memory");
    }
    cbar();
    uint32_t qf[HD / 16][4];
    if (active) {
#pragma unroll
      for (int kt = 0; kt < HD / 16; ++kt) {
        const int mi = lane >> 3;
        ldmatrix_x4_a(qf[kt][0], qf[kt][1], qf[kt][2], qf[kt][3],
                      swz(qbase, row0 + (lane & 7) + 8 * (mi & 1), 2 * kt + (mi >> 1)));
      }
    }
    int stage = 0;
    uint32_t phase = 0;
    for (int b = b0; b < b1; ++b) {
      if (!mbar_wait_bounded(&full[stage], phase, flags)) {
        flags[0] = 1;
        set_status(a.status, CASSPEC_E_TIMEOUT);
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
        if (sbase + kAttnBlk <= P) {  // a block of the committed prefix: visible to every node
#pragma unroll
          for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              s[nt][e] *= a.scale_log2;
              s[nt][2 + e] *= a.scale_log2;
              mxA = fmaxf(mxA, s[nt][e]);
              mxB = fmaxf(mxB, s[nt][2 + e]);
            }
          }
        } else {
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
  }

  // ---- this split's partial to global scratch, then count in ----
  const int n = a.n;
  const size_t pslot = (size_t)head * C + rank;
  if (warp < 4) {
    lA += __shfl_xor_sync(0xffffffffu, lA, 1);
    lA += __shfl_xor_sync(0xffffffffu, lA, 2);
    lB += __shfl_xor_sync(0xffffffffu, lB, 1);
    lB += __shfl_xor_sync(0xffffffffu, lB, 2);
    float* po = a.part_o + pslot * 64 * HD;
#pragma unroll
    for (int dt = 0; dt < HD / 8; ++dt) {
      const int col = dt * 8 + 2 * t4;
      if (rA < n) __stcg(reinterpret_cast<float2*>(po + rA * HD + col), make_float2(oacc[dt][0], oacc[dt][1]));
      if (rB < n) __stcg(reinterpret_cast<float2*>(po + rB * HD + col), make_float2(oacc[dt][2], oacc[dt][3]));
    }
    if (t4 == 0) {
      if (rA < n) __stcg(a.part_ml + pslot * 64 + rA, make_float2(mA, lA));
      if (rB < n) __stcg(a.part_ml + pslot * 64 + rB, make_float2(mB, lB));
    }
  }
  __syncthreads();
  if (tid == 0) {
    // every split of this head is resident (the grid fits the GPU at two CTAs per SM), so this
    // wait ends as soon as the slowest split has written its partial
    __threadfence();
    atomicAdd(a.cnt + head, 1u);
    const uint64_t t0 = globaltimer_ns();
    int ok = 1;
    while (ld_acquire_gpu(a.cnt + head) < (unsigned)C) {
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        ok = 0;
        set_status(a.status, CASSPEC_E_TIMEOUT);
        break;
      }
    }
    flags[1] = ok;
  }
  __syncthreads();

  // ---- merge: this split finishes rows rank, rank + C, ... over all C partials, in split order ----
  // (the K/V ring is drained: its shared memory holds the merge weights)
  if (flags[1]) {
    __threadfence();
    constexpr int V4 = HD / 4;
    const float* pob = a.part_o + (size_t)head * C * 64 * HD;
    const float2* pml = a.part_ml + (size_t)head * C * 64;
    const int nr = rank < n ? (n - rank + C - 1) / C : 0;  // rows of this split
    float2* ml_s = reinterpret_cast<float2*>(ring);          // [nr][C] (max, sum)
    float* w_s = reinterpret_cast<float*>(ring + 64 * kAttnMaxSplits * 8);  // [nr][C] weights
    float* inv_s = w_s + 64 * kAttnMaxSplits;                                // [nr] 1 / sum
    if (tid < nr * C) ml_s[tid] = __ldcg(pml + (tid % C) * 64 + rank + (tid / C) * C);
    __syncthreads();
    if (tid < nr) {
      float M = -INFINITY;
      for (int k = 0; k < C; ++k) M = fmaxf(M, ml_s[tid * C + k].x);
      float L = 0.f;
      for (int k = 0; k < C; ++k) {
        const float2 ml = ml_s[tid * C + k];
        const float w = ml.x == -INFINITY ? 0.f : exp2f(ml.x - M);  // an empty split weighs 0
        w_s[tid * C + k] = w;
        L += ml.y * w;
      }
      inv_s[tid] = 1.f / L;
    }
    __syncthreads();
    for (int idx = tid; idx < nr * V4; idx += kAttnThreads) {
      const int j = idx / V4, c4 = (idx % V4) * 4, row = rank + j * C;
      float4 ov[kAttnMaxSplits];  // every partial of this element in flight at once
#pragma unroll
      for (int k = 0; k < kAttnMaxSplits; ++k)
        if (k < C) ov[k] = __ldcg(reinterpret_cast<const float4*>(pob + ((size_t)k * 64 + row) * HD + c4));
      float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int k = 0; k < kAttnMaxSplits; ++k) {
        if (k < C) {
          const float w = w_s[j * C + k];
          o.x += ov[k].x * w;
          o.y += ov[k].y * w;
          o.z += ov[k].z * w;
          o.w += ov[k].w * w;
        }
      }
      const float inv = inv_s[j];
      const float r0 = o.x * inv, r1 = o.y * inv, r2 = o.z * inv, r3 = o.w * inv;
      const uint16_t h0 = f2bf(r0), h1 = f2bf(r1), h2 = f2bf(r2), h3 = f2bf(r3);
      uint2 hi, lo;  // split output: hi = bf16(o) in rows 0..63, lo = bf16(o - hi) in rows 64..127
      hi.x = (uint32_t)h0 | ((uint32_t)h1 << 16);
      hi.y = (uint32_t)h2 | ((uint32_t)h3 << 16);
      lo.x = pack_bf16x2(r0 - bf2f(h0), r1 - bf2f(h1));
      lo.y = pack_bf16x2(r2 - bf2f(h2), r3 - bf2f(h3));
      *reinterpret_cast<uint2*>(a.o + (size_t)row * a.d + head * HD + c4) = hi;
      *reinterpret_cast<uint2*>(a.o + (size_t)(64 + row) * a.d + head * HD + c4) = lo;
    }
  }
  __syncthreads();
  if (tid == 0) {  // the last split out (every split has stopped reading the arrival counter)
    __threadfence();
    if (atomicAdd(a.cnt + a.n_heads + head, 1u) == (unsigned)(C - 1)) {
      a.cnt[head] = 0u;
      a.cnt[a.n_heads + head] = 0u;
    }
  }
}

int attn_splits(int n_heads, int num_sms) {
  int c = (2 * num_sms) / n_heads;  // two CTAs per SM: the whole grid is resident at once
  if (c > kAttnMaxSplits) c = kAttnMaxSplits;
  if (c < 1) c = 1;
  return c;
}

template <int HD>
static cudaError_t launch_hd(const CUtensorMap& tm, const AttnArgs& a, cudaStream_t stream, bool pdl) {
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
  cfg.gridDim = dim3(a.n_heads * a.splits);
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

cudaError_t launch_tree_attention(const CUtensorMap& tm, const AttnArgs& a, int hd, cudaStream_t stream, bool pdl) {
  if (a.splits < 1 || a.splits > kAttnMaxSplits) return cudaErrorInvalidValue;
  if (hd == 128) return launch_hd<128>(tm, a, stream, pdl);
  if (hd == 64) return launch_hd<64>(tm, a, stream, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace casspec
