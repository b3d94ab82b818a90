// Tree attention (Sec. 4.2: parallel verification / drafting of a token tree) on the 5th-generation
// tensor cores.
//
// Node i of the tree attends to every committed prefix slot [0, P) and to the tree slots of its
// ancestors and itself (bit j of anc[i] <=> tree slot j, cache slot P + j).
//   * C CTAs per head (split-KV) form one thread-block cluster; heads * C <= 2 per SM, so the whole
//     grid is resident at once.  Split s handles the s-th contiguous share of the head's 64-slot KV
//     blocks;
//   * K and V blocks arrive by TMA (2-D tensor map over the whole cache, 128-byte swizzle, 64 slots x
//     64 dims per box) in two mbarrier rings (K: 3 stages, released once the block's scores are
//     computed; V: 2 stages, released after P V), each fed by one producer thread, which loads the
//     blocks that lie wholly in the committed prefix before waiting on the preceding kernel;
//   * one thread issues tcgen05.mma: S = Q K^T per block (M = 64 query rows, N = 64 slots, both
//     operands K-major) into one of two TMEM score buffers, and O += P V (N = head dim, V read
//     MN-major straight from its cache layout) into a TMEM accumulator.  S of block i is issued
//     before P V of block i - 1, so the scores of the next block are computed while the softmax
//     warps work on the current one;
//   * four softmax warps read S from TMEM (M = 64 puts query rows 16 q .. 16 q + 15 in lanes 0..15 of
//     lane quarter q; the 16x256b load shape spreads each 16-row group over all 32 threads, two rows
//     per quad), apply the ancestor mask, keep the online softmax state in registers against a
//     reference max that moves only when a score exceeds it by 2^8 (then the O rows are rescaled in
//     TMEM), and write P as bf16 into one of two 128-byte-swizzled tiles, the A operand of P V;
//   * each split leaves its partial (running max, sum, unnormalised output) in its own shared memory;
//     after a cluster barrier, split s merges rows s, s + C, ... over the C partials, read through
//     distributed shared memory in split order (fixed, so results do not depend on timing).
#include "common.cuh"
#include "kernels.h"

namespace casspec {

constexpr int kAttnThreads = 192;  // warp 0 producers (lane 0: K, lane 1: V), warp 1 MMA, warps 2..5 softmax
constexpr int kAttnBlk = 64;
constexpr int kAttnKStages = 3;
constexpr int kAttnVStages = 2;
constexpr uint32_t kAttnTmemCols = 256;  // two 64-column score buffers + the output (<= 128 columns)
constexpr uint32_t kAttnO = 128;         // TMEM column of the output accumulator
constexpr float kRescaleLog2 = 8.f;      // the reference max moves when a score exceeds it by 2^8

template <int HD>
__host__ __device__ constexpr uint32_t attn_tile_bytes() {  // a [64][HD] bf16 tile
  return (uint32_t)kAttnBlk * HD * 2;
}
template <int HD>
__host__ __device__ constexpr size_t attn_smem_bytes() {
  // Q, the K and V rings, two P tiles, barriers (two CTAs per SM: <= 113 KB each)
  return attn_tile_bytes<HD>() * (1 + kAttnKStages + kAttnVStages) + 2 * 8192 + 256;
}

// Byte offset of 16-byte chunk `c` (0 .. HD/8-1) of row `r` in a [64][HD] bf16 tile stored as HD/64
// sub-tiles of [64][128 B] with the 128-byte swizzle (TMA's layout; tile base 1024-byte aligned).
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return (uint32_t)(c >> 3) * 8192u + (uint32_t)r * 128u + ((uint32_t)((c & 7) ^ (r & 7)) << 4);
}

__device__ __forceinline__ float fast_exp2(float x) {  // 2^x, ~2 ulp; 2^-inf = 0
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int HD>
__global__ void __launch_bounds__(kAttnThreads, 2) tree_attn_kernel(const __grid_constant__ CUtensorMap tmKV,
                                                                     const AttnArgs a) {
  constexpr uint32_t TILE = attn_tile_bytes<HD>();
  constexpr int NK = kAttnKStages, NV = kAttnVStages;
  constexpr int NCH = HD / 8;  // 16-byte chunks per row
  // the partial (O rows fp32 + (max, sum)) reuses the drained K/V rings
  static_assert(64 * HD * 4 + 64 * 8 <= (NK + NV) * TILE, "the partial must fit in the K/V rings");
  // The kernel has no static shared memory, so the dynamic block starts the CTA's shared window; the
  // swizzled tiles need it 1 KB aligned (checked: results are flagged invalid otherwise).
  extern __shared__ __align__(1024) uint8_t sm[];
  uint8_t* qs = sm;                // Q: [64][HD]
  uint8_t* kring = qs + TILE;      // NK x K
  uint8_t* vring = kring + NK * TILE;  // NV x V
  uint8_t* ps = vring + NV * TILE;     // two P tiles [64][64]
  uint64_t* k_full = reinterpret_cast<uint64_t*>(ps + 2 * 8192);
  uint64_t* k_empty = k_full + NK;
  uint64_t* v_full = k_empty + NK;
  uint64_t* v_empty = v_full + NV;
  uint64_t* s_full = v_empty + NV;  // [2]
  uint64_t* s_free = s_full + 2;    // [2]
  uint64_t* p_full = s_free + 2;    // [2]
  uint64_t* pv_done = p_full + 2;   // [2]: P V of block j completes phase j / 2 of pv_done[j % 2]
  uint64_t* q_full = pv_done + 2;
  uint64_t* drain = q_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* flags = reinterpret_cast<volatile int*>(tmem_slot + 1);  // [0] abort
  float* part_o = reinterpret_cast<float*>(kring);                        // [64][HD] after the blocks
  float2* part_ml = reinterpret_cast<float2*>(kring + 64 * HD * 4);       // [64]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int C = a.splits;
  const int head = blockIdx.x / C;
  const int rank = (int)cluster_ctarank();  // == blockIdx.x % C: the head's splits are one cluster
  if (tid == 0) {
    for (int s = 0; s < NK; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < NV; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_free[b], 4);  // one arrival per softmax warp
    }
    mbar_init(&p_full[0], 4);
    mbar_init(&p_full[1], 4);
    mbar_init(&pv_done[0], 1);
    mbar_init(&pv_done[1], 1);
    mbar_init(q_full, 4);
    mbar_init(drain, 1);
    flags[0] = 0;
    if ((smem_u32(sm) & 1023u) != 0) set_status(a.status, CASSPEC_E_CUDA);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kAttnTmemCols);
    tmem_relinquish();
  }
  // The committed length P is written only between steps (compaction, set_prefix), by kernels that
  // completed before this step's first kernel started, so it can be read before the dependency wait.
  const int Pp = *reinterpret_cast<const volatile int*>(a.dP);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();
  if (warp != 0) pdl_wait();  // the producers wait after their prefix loads

  const int P = warp == 0 ? Pp : __ldcg(a.dP);
  const int total = P + a.T + a.n;
  const int nblk = (total + kAttnBlk - 1) / kAttnBlk;
  const int b0 = rank * nblk / C, b1 = (rank + 1) * nblk / C;
  const int nb = b1 - b0;

  if (warp == 0) {
    // ---------------- producers: lane 0 loads K blocks, lane 1 V blocks ----------------
    if (lane < 2) {
      if (lane == 0) tma_prefetch_desc(&tmKV);
      const bool isk = lane == 0;
      const int ns = isk ? NK : NV;
      uint8_t* ring = isk ? kring : vring;
      uint64_t* full = isk ? k_full : v_full;
      uint64_t* empty = isk ? k_empty : v_empty;
      const uint64_t pol = policy_evict_first();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_parity = 0;
      const int row0 = ((a.layer * 2 + (isk ? 0 : 1)) * a.n_heads + head) * a.ctx;
      bool waited = false;
      for (int b = b0; b < b1; ++b) {
        if (!waited && (b - b0 >= ns || (b + 1) * kAttnBlk > P || P < 0 || P > a.ctx)) {
          pdl_wait();  // from here on the blocks may hold this step's tree K/V
          waited = true;
          if (__ldcg(a.dP) != P) set_status(a.status, CASSPEC_E_STATE);  // P moved during a step
        }
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1, flags)) {
          flags[0] = 1;
          set_status(a.status, CASSPEC_E_TIMEOUT);
          break;
        }
        mbar_expect_tx(&full[stage], TILE);
        armed |= 1u << stage;
        armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
        uint8_t* st = ring + stage * TILE;
#pragma unroll
        for (int sub = 0; sub < HD / 64; ++sub)
          tma_load_2d(st + sub * 8192, &tmKV, &full[stage], sub * 64, row0 + b * kAttnBlk, pol);
        if (++stage == ns) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (!waited) pdl_wait();
      if (flags[0]) {  // abort: let the copies already issued land before the shared memory is reused
        for (int s = 0; s < ns; ++s)
          if (armed & (1u << s)) mbar_wait_bounded(&full[s], (armed_parity >> s) & 1, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16_f32(64, 64);
      const uint32_t id_o = idesc_bf16_f32(64, HD) | kIdescBMnMajor;
      const uint64_t qd = sw128_kmajor_desc(smem_u32(qs));
      bool ok = nb == 0 || mbar_wait_bounded(q_full, 0, flags);
      // P V of block j: A = P tile j & 1, 4 k-steps of 16 slots; B = V of its stage, MN-major
      // (64-dim groups 8 KB apart, 8-slot groups 1 KB apart, 2 KB per k-step)
      auto issue_pv = [&](int j) -> bool {
        const int vs = j % NV;
        const uint64_t pd = sw128_kmajor_desc(smem_u32(ps + (j & 1) * 8192));
        if (!mbar_wait_bounded(&p_full[j & 1], (uint32_t)(j >> 1) & 1, flags)) return false;
        if (!mbar_wait_bounded(&v_full[vs], (uint32_t)(j / NV) & 1, flags)) return false;
        tc_fence_after();
        const uint32_t vb = smem_u32(vring + vs * TILE);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          tc_mma_bf16(tmem + kAttnO, pd + (uint64_t)(2 * kk), sw128_mnmajor_desc(vb + 2048u * kk, 8192u, 1024u), id_o,
                      (j > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&v_empty[vs]);
        tc_commit(&pv_done[j & 1]);
        return true;
      };
      if (ok) {
        tc_fence_after();
        for (int i = 0; i < nb && ok; ++i) {
          const int sb = i & 1, ks = i % NK;
          if (i >= 2 && !mbar_wait_bounded(&s_free[sb], (uint32_t)((i - 2) >> 1) & 1, flags)) {
            ok = false;
            break;
          }
          if (!mbar_wait_bounded(&k_full[ks], (uint32_t)(i / NK) & 1, flags)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t kd = sw128_kmajor_desc(smem_u32(kring + ks * TILE));
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint64_t off = (uint64_t)((kk >> 2) * 512 + (kk & 3) * 2);  // 8 KB per 64 dims, 32 B per step
            tc_mma_bf16(tmem + (uint32_t)(sb * 64), qd + off, kd + off, id_s, kk > 0 ? 1u : 0u);
          }
          tc_commit(&s_full[sb]);
          tc_commit(&k_empty[ks]);  // the K block is consumed once its scores are complete
          if (i >= 1 && !issue_pv(i - 1)) ok = false;
        }
        if (ok && nb > 0 && !issue_pv(nb - 1)) ok = false;
      }
      if (!ok) {
        flags[0] = 1;
        set_status(a.status, CASSPEC_E_TIMEOUT);
      }
      tc_commit(drain);  // every MMA complete before TMEM is released
      mbar_wait_bounded(drain, 0, nullptr);
    }
    __syncwarp();
  } else {
    // ---------------- softmax warps 2..5 ----------------
    // TMEM lane quarter qq holds query rows 16 qq .. 16 qq + 15 (M = 64).  Read with the 16x256b
    // shape, thread t of the warp holds rows rA = 16 qq + t/4 and rB = rA + 8 at columns
    // 8 j + 2 (t % 4) + {0, 1}: the four threads of a quad share a row pair, so row reductions are two
    // quad shuffles.
    const int qq = warp & 3;
    const int g = lane >> 2, t4 = lane & 3;
    const int rA = 16 * qq + g, rB = rA + 8;
    const uint32_t tl = tmem + ((uint32_t)(qq * 32) << 16);
    // Q of this head: rows >= n are zero
    {
      const int et = tid - 64;  // 0..127
      constexpr int QPT = 64 * NCH / 128;
      uint4 qv[QPT];
#pragma unroll
      for (int k = 0; k < QPT; ++k) {
        const int idx = et + k * 128, r = idx / NCH, c = idx % NCH;
        qv[k] = r < a.n ? __ldcg(reinterpret_cast<const uint4*>(a.q + (size_t)r * a.d + head * HD + c * 8))
                        : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int k = 0; k < QPT; ++k) {
        const int idx = et + k * 128, r = idx / NCH, c = idx % NCH;
        *reinterpret_cast<uint4*>(qs + swz(r, c)) = qv[k];
      }
      fence_proxy_async_smem();  // generic-proxy writes -> the tensor cores' operand reads
      __syncwarp();
      if (lane == 0) mbar_arrive(q_full);
    }
    const unsigned long long ancA = rA < a.n ? __ldcg(a.anc + rA) : 0ull;
    const unsigned long long ancB = rB < a.n ? __ldcg(a.anc + rB) : 0ull;
    float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;  // lA, lB: this thread's columns only
    bool ok = true;
    for (int i = 0; i < nb; ++i) {
      const int sb = i & 1;
      if (!mbar_wait_bounded(&s_full[sb], (uint32_t)(i >> 1) & 1, flags)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[32];
      tmem_ld_16x256b_x8(tl + (uint32_t)(sb * 64), s);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[sb]);  // the score buffer may take block i + 2
      const int sbase = (b0 + i) * kAttnBlk;
      float mxA = -INFINITY, mxB = -INFINITY;
      if (sbase + kAttnBlk <= P) {  // a block of the committed prefix: visible to every node
#pragma unroll
        for (int j = 0; j < 8; ++j) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            s[4 * j + e] *= a.scale_log2;
            s[4 * j + 2 + e] *= a.scale_log2;
            mxA = fmaxf(mxA, s[4 * j + e]);
            mxB = fmaxf(mxB, s[4 * j + 2 + e]);
          }
        }
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int slot = sbase + 8 * j + 2 * t4 + e;
            bool visA, visB;
            if (slot < P) {
              visA = visB = true;
            } else if (slot < total) {
              visA = (ancA >> (slot - P)) & 1ull;
              visB = (ancB >> (slot - P)) & 1ull;
            } else {
              visA = visB = false;
            }
            s[4 * j + e] = visA ? s[4 * j + e] * a.scale_log2 : -INFINITY;
            s[4 * j + 2 + e] = visB ? s[4 * j + 2 + e] * a.scale_log2 : -INFINITY;
            mxA = fmaxf(mxA, s[4 * j + e]);
            mxB = fmaxf(mxB, s[4 * j + 2 + e]);
          }
        }
      }
      mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 1));
      mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 2));
      mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 1));
      mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 2));
      // Reference max per row: P = 2^(s - m) with m raised only when a score exceeds it by more than
      // kRescaleLog2 (P <= 2^kRescaleLog2 otherwise).  Moving m rescales l and the O row by
      // 2^(m_old - m_new), which needs the previous block's P V complete; most blocks skip that.
      const bool upA = mxA > mA + kRescaleLog2, upB = mxB > mB + kRescaleLog2;
      const float nA = upA ? mxA : mA, nB = upB ? mxB : mB;
      const float uA = nA == -INFINITY ? 0.f : nA, uB = nB == -INFINITY ? 0.f : nB;
      const float cA = upA ? fast_exp2(mA - uA) : 1.f, cB = upB ? fast_exp2(mB - uB) : 1.f;  // 0 from -inf
      mA = nA;
      mB = nB;
      float sumA = 0.f, sumB = 0.f;
      uint32_t pk[16];  // [2 j]: row A, [2 j + 1]: row B
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float a0 = fast_exp2(s[4 * j] - uA), a1 = fast_exp2(s[4 * j + 1] - uA);
        const float b0v = fast_exp2(s[4 * j + 2] - uB), b1v = fast_exp2(s[4 * j + 3] - uB);
        sumA += a0 + a1;
        sumB += b0v + b1v;
        pk[2 * j] = pack_bf16x2(a0, a1);
        pk[2 * j + 1] = pack_bf16x2(b0v, b1v);
      }
      lA = lA * cA + sumA;
      lB = lB * cB + sumB;
      // The O rows of this warp move with m: P V of block i - 1 must have completed.  P tile i & 1
      // was last read by P V of block i - 2.
      const bool resc = i >= 1 && __any_sync(0xffffffffu, upA || upB);
      if (resc || i >= 2) {
        // (waits stay within one phase of each barrier: P V of block i + 1 or later needs this
        // warp's P of block i first)
        const int w = resc ? i - 1 : i - 2;
        if (!mbar_wait_bounded(&pv_done[w & 1], (uint32_t)(w >> 1) & 1, flags)) {
          ok = false;
          break;
        }
        tc_fence_after();
      }
      if (resc) {
#pragma unroll
        for (int h = 0; h < HD / 64; ++h) {
          float o[32];
          tmem_ld_16x256b_x8(tl + kAttnO + (uint32_t)(64 * h), o);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            o[4 * j] *= cA;
            o[4 * j + 1] *= cA;
            o[4 * j + 2] *= cB;
            o[4 * j + 3] *= cB;
          }
          tmem_st_16x256b_x8(tl + kAttnO + (uint32_t)(64 * h), o);
        }
        tmem_st_wait();
      }
      {
        uint8_t* pt = ps + sb * 8192;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          *reinterpret_cast<uint32_t*>(pt + (uint32_t)rA * 128u + ((uint32_t)(j ^ (rA & 7)) << 4) + 4u * t4) = pk[2 * j];
          *reinterpret_cast<uint32_t*>(pt + (uint32_t)rB * 128u + ((uint32_t)(j ^ (rB & 7)) << 4) + 4u * t4) = pk[2 * j + 1];
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[sb]);
    }
    // this split's partial into its own shared memory (the rings are drained once the last P V
    // completed): unnormalised O rows, (max, sum)
    if (ok && nb > 0 && !mbar_wait_bounded(&pv_done[(nb - 1) & 1], (uint32_t)((nb - 1) >> 1) & 1, flags)) ok = false;
    if (!ok) {
      flags[0] = 1;
      set_status(a.status, CASSPEC_E_TIMEOUT);
    }
    lA += __shfl_xor_sync(0xffffffffu, lA, 1);
    lA += __shfl_xor_sync(0xffffffffu, lA, 2);
    lB += __shfl_xor_sync(0xffffffffu, lB, 1);
    lB += __shfl_xor_sync(0xffffffffu, lB, 2);
    if (ok) tc_fence_after();
#pragma unroll
    for (int h = 0; h < HD / 64; ++h) {
      float o[32];
      if (ok && nb > 0) {
        tmem_ld_16x256b_x8(tl + kAttnO + (uint32_t)(64 * h), o);
        tmem_ld_wait();
      } else {
#pragma unroll
        for (int e = 0; e < 32; ++e) o[e] = 0.f;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int col = 64 * h + 8 * j + 2 * t4;
        *reinterpret_cast<float2*>(part_o + rA * HD + col) = make_float2(o[4 * j], o[4 * j + 1]);
        *reinterpret_cast<float2*>(part_o + rB * HD + col) = make_float2(o[4 * j + 2], o[4 * j + 3]);
      }
    }
    if (t4 == 0) {
      part_ml[rA] = make_float2(ok && nb > 0 ? mA : -INFINITY, lA);
      part_ml[rB] = make_float2(ok && nb > 0 ? mB : -INFINITY, lB);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kAttnTmemCols);
  }
  cluster_sync();  // every split's partial is in its shared memory

  // ---- merge: this split finishes rows rank, rank + C, ... over the C partials, in split order ----
  // A thread takes two (row, 4-column) items per batch and issues every load of both, the (max, sum)
  // and the four output columns of all C partials, before using any: one round trip through
  // distributed shared memory per batch.  The weights are formed per item.
  const int n = a.n;
  const int nr = rank < n ? (n - rank + C - 1) / C : 0;  // rows of this split
  constexpr int V4 = HD / 4;
  for (int base = 0; base < nr * V4; base += 2 * kAttnThreads) {  // 8 rows (C = 8): one batch
    float4 ov[2][kAttnMaxSplits];
    float2 ml[2][kAttnMaxSplits];
#pragma unroll
    for (int it = 0; it < 2; ++it) {
      const int idx = base + tid + it * kAttnThreads;
      if (idx < nr * V4) {
        const int j = idx / V4, c4 = (idx % V4) * 4, r = rank + j * C;
        const uint32_t src = smem_u32(part_o + r * HD + c4), srm = smem_u32(part_ml + r);
#pragma unroll
        for (int k = 0; k < kAttnMaxSplits; ++k)
          if (k < C) {
            ov[it][k] = ld_dsmem_f4(map_to_rank(src, (uint32_t)k));
            ml[it][k] = ld_dsmem_f2(map_to_rank(srm, (uint32_t)k));
          }
      }
    }
#pragma unroll
    for (int it = 0; it < 2; ++it) {
      const int idx = base + tid + it * kAttnThreads;
      if (idx < nr * V4) {
        const int j = idx / V4, c4 = (idx % V4) * 4, r = rank + j * C;
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < kAttnMaxSplits; ++k)
          if (k < C) M = fmaxf(M, ml[it][k].x);
        float L = 0.f;
        float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int k = 0; k < kAttnMaxSplits; ++k) {
          if (k < C) {
            const float w = ml[it][k].x == -INFINITY ? 0.f : exp2f(ml[it][k].x - M);  // an empty split weighs 0
            L += ml[it][k].y * w;
            o.x += ov[it][k].x * w;
            o.y += ov[it][k].y * w;
            o.z += ov[it][k].z * w;
            o.w += ov[it][k].w * w;
          }
        }
        const float inv = 1.f / L;
        const float r0 = o.x * inv, r1 = o.y * inv, r2 = o.z * inv, r3 = o.w * inv;
        const uint16_t h0 = f2bf(r0), h1 = f2bf(r1), h2 = f2bf(r2), h3 = f2bf(r3);
        uint2 hi, lo;  // split output: hi = bf16(o) in rows 0..63, lo = bf16(o - hi) in rows 64..127
        hi.x = (uint32_t)h0 | ((uint32_t)h1 << 16);
        hi.y = (uint32_t)h2 | ((uint32_t)h3 << 16);
        lo.x = pack_bf16x2(r0 - bf2f(h0), r1 - bf2f(h1));
        lo.y = pack_bf16x2(r2 - bf2f(h2), r3 - bf2f(h3));
        *reinterpret_cast<uint2*>(a.o + (size_t)r * a.d + head * HD + c4) = hi;
        *reinterpret_cast<uint2*>(a.o + (size_t)(64 + r) * a.d + head * HD + c4) = lo;
      }
    }
  }
  cluster_sync();  // no split leaves while another still reads its partial
}

int attn_splits(int n_heads, int num_sms) {
  int c = (2 * num_sms) / n_heads;  // two CTAs per SM: the whole grid is resident at once
  if (c > kAttnMaxSplits) c = kAttnMaxSplits;
  if (c < 1) c = 1;
  return c;
}

static_assert(attn_smem_bytes<128>() + 1024 <= 232448 / 2, "two attention CTAs per SM");

template <int HD>
static cudaError_t launch_hd(const CUtensorMap& tm, const AttnArgs& a, cudaStream_t stream, bool pdl) {
  auto kern = tree_attn_kernel<HD>;
  constexpr size_t smem = attn_smem_bytes<HD>();
  static int configured = -1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured != dev) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    // the whole shared memory as carveout: two CTAs per SM
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_heads * a.splits);
  cfg.blockDim = dim3(kAttnThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)a.splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kern, tm, a);
}

cudaError_t launch_tree_attention(const CUtensorMap& tm, const AttnArgs& a, int hd, cudaStream_t stream, bool pdl) {
  if (a.splits < 1 || a.splits > kAttnMaxSplits || a.n < 1 || a.n > 64 || a.T < 0 || a.T + a.n > 64)
    return cudaErrorInvalidValue;
  if (hd == 128) return launch_hd<128>(tm, a, stream, pdl);
  if (hd == 64) return launch_hd<64>(tm, a, stream, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace casspec
