// Exact quantised projections on the 5th-generation tensor cores (App. C's W4A4 and W8A8 drafts).
//
// Two operand kinds share one weight-streaming kernel:
//   * kOpE4M3 (W4A4): codes in [-7, 7] are exact FP8 e4m3 values, a product of two codes is at
//     most 49, and every partial sum over K <= 65536 is an integer below 2^22, so
//     tcgen05.mma.kind::f8f6f4 with e4m3 operands and fp32 accumulation returns the exact integer
//     sum in any summation order.
//   * kOpS8 (W8A8): codes in [-127, 127] as int8 bytes.  Four converter warps widen each stage's
//     weight and activation codes to fp16 in shared memory (every integer of magnitude <= 2048 is
//     exact in fp16) and tcgen05.mma.kind::f16 sums them in fp32.  One accumulator covers at most
//     8 k-blocks (1024 columns), so every partial sum is an integer of magnitude
//     <= 1024 * 127^2 < 2^24 and exact; the epilogue converts each accumulator to int32 and adds
//     them, so the result is the exact int32 sum of the integer mma.sync path.
// Common structure:
//   * swap-AB: 128 output channels on M, the n <= 64 tokens (padded to BN) on N;
//   * a stage holds a 128 x 128-code weight tile (16 KB, one 2-D TMA box of bytes with the 128-byte
//     swizzle; gate/up: 64 rows of each) and the BN x 128 activation codes;
//   * stream-K over (tile, 128-column k-block) units with the last-arriver fix-up (exact integer
//     partials), double-buffered TMEM accumulators, warp roles as in the bf16 projection;
//   * the epilogue dequantises y = acc * s_x[token] * s_w[row] in fp32 (the order of the int8
//     projection) and runs the fused epilogue.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

#include <cudaTypedefs.h>

namespace casspec {

constexpr int kOpE4M3 = 0, kOpS8 = 1;
constexpr uint32_t kF8ATile = 128 * 128;  // 128 rows x 128 codes
constexpr int kS8Region = 8;              // k-blocks per fp32 accumulator in kOpS8 (1024 columns)
constexpr int kF8MaxContrib = 8;          // stream-K contributors per tile whose partials are read together
constexpr size_t kF8SmemMax = 232448;     // dynamic shared memory limit per CTA

// kOpS8: converter warps (8 for the small token counts of drafts, 4 where the epilogue needs the
// registers of BN = 48 or 64 tokens)
__host__ __device__ constexpr int f8_conv_warps(int OP, int BN) { return OP == kOpS8 ? (BN <= 32 ? 8 : 4) : 0; }
__host__ __device__ constexpr int f8_threads(int OP, int BN) { return 192 + 32 * f8_conv_warps(OP, BN); }
__host__ __device__ constexpr uint32_t f8_stage_bytes(int BN) { return kF8ATile + (uint32_t)BN * 128u; }
// kOpS8: a 16-bit stage, the widened weight tile (two 64-column swizzle atoms of 16 KB) and the widened
// activation codes (two atoms of BN x 128 B)
__host__ __device__ constexpr uint32_t f8_cstage_bytes(int OP, int BN) {
  return OP == kOpS8 ? 2u * kF8ATile + (uint32_t)BN * 256u : 0u;
}
__host__ __device__ constexpr int f8_cstages(int OP, int BN) { return OP == kOpS8 ? (BN <= 16 ? 3 : 2) : 0; }
__host__ __device__ constexpr uint32_t f8_staging_bytes(int BN) { return (uint32_t)epi_staging_floats(BN) * 4u; }
__host__ __device__ constexpr int f8_stages(int OP, int BN) {
  return OP == kOpS8
             ? ((int)((kF8SmemMax - 1280 - f8_staging_bytes(BN) - (size_t)f8_cstages(OP, BN) * f8_cstage_bytes(OP, BN)) /
                      f8_stage_bytes(BN)) > 8
                    ? 8
                    : (int)((kF8SmemMax - 1280 - f8_staging_bytes(BN) -
                             (size_t)f8_cstages(OP, BN) * f8_cstage_bytes(OP, BN)) /
                            f8_stage_bytes(BN)))
             : ((int)((200u * 1024u - f8_staging_bytes(BN) - 1024u) / f8_stage_bytes(BN)) > 8
                    ? 8
                    : (int)((200u * 1024u - f8_staging_bytes(BN) - 1024u) / f8_stage_bytes(BN)));
}
__host__ __device__ constexpr size_t f8_smem_bytes(int OP, int BN) {
  return 1024 + (size_t)f8_stages(OP, BN) * f8_stage_bytes(BN) + (size_t)f8_cstages(OP, BN) * f8_cstage_bytes(OP, BN) +
         f8_staging_bytes(BN) + 256;
}
__host__ __device__ constexpr uint32_t f8_tmem_cols(int BN) { return 2 * BN <= 32 ? 32 : (2 * BN <= 64 ? 64 : 128); }
static_assert(f8_smem_bytes(kOpS8, 64) <= kF8SmemMax && f8_smem_bytes(kOpS8, 16) <= kF8SmemMax &&
                  f8_stages(kOpS8, 64) >= 3,
              "W8A8 stages fit the shared memory");
static_assert(f8_stage_bytes(16) % 1024 == 0 && f8_stage_bytes(48) % 1024 == 0 &&
                  f8_cstage_bytes(kOpS8, 16) % 1024 == 0 && f8_cstage_bytes(kOpS8, 48) % 1024 == 0,
              "stages keep the 1 KB alignment of the 128 B swizzle");
static_assert(kS8Region * 128 * 127 * 127 < (1 << 24), "one W8A8 accumulator holds exact integer sums");

// Instruction descriptor of tcgen05.mma.kind::f8f6f4 with e4m3 A/B, fp32 D, both operands K-major.
__host__ __device__ constexpr uint32_t idesc_e4m3_f32(int M, int N) {
  return (1u << 4)                       // D format: f32
         | (0u << 7)                     // A format: e4m3
         | (0u << 10)                    // B format: e4m3
         | ((uint32_t)(N >> 3) << 17)    // N / 8
         | ((uint32_t)(M >> 4) << 24);   // M / 16
}

__device__ __forceinline__ void tc_mma_e4m3(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ int f8_cta_of_unit(long long x, long long U, int G) {
  return (int)(((x + 1) * (long long)G - 1) / U);
}

// Instruction descriptor of tcgen05.mma.kind::f16 with fp16 A/B, fp32 D, both operands K-major.
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N) {
  return (1u << 4)                     // D format: f32
         | (0u << 7)                   // A format: f16
         | (0u << 10)                  // B format: f16
         | ((uint32_t)(N >> 3) << 17)  // N / 8
         | ((uint32_t)(M >> 4) << 24); // M / 16
}

// 16 int8 codes -> 16 fp16 values, exactly: a code q, biased to u = q + 128 by flipping its top bit,
// is placed as the low mantissa byte under the exponent of 1024 (the fp16 1024 + u, exact with 10
// mantissa bits); one fp16x2 subtraction of 1152 = 1024 + 128 leaves q for two codes at once.
__device__ __forceinline__ uint32_t s8pair_to_f16x2(uint32_t biased, uint32_t sel) {
  const uint32_t h = __byte_perm(biased, 0x64646464u, sel);
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(h), "r"(0x64806480u));
  return r;
}
__device__ __forceinline__ void s8x16_to_f16(const uint4 w, uint4& lo, uint4& hi) {
  const uint32_t b0 = w.x ^ 0x80808080u, b1 = w.y ^ 0x80808080u, b2 = w.z ^ 0x80808080u, b3 = w.w ^ 0x80808080u;
  lo = make_uint4(s8pair_to_f16x2(b0, 0x5140), s8pair_to_f16x2(b0, 0x7362), s8pair_to_f16x2(b1, 0x5140),
                  s8pair_to_f16x2(b1, 0x7362));
  hi = make_uint4(s8pair_to_f16x2(b2, 0x5140), s8pair_to_f16x2(b2, 0x7362), s8pair_to_f16x2(b3, 0x5140),
                  s8pair_to_f16x2(b3, 0x7362));
}

// Widen one 16-code chunk of a 128-byte-swizzled byte tile (row r, logical chunk c) into the
// fp16 tile of two 64-column swizzle atoms `atom` bytes apart (row r, logical chunks 2c, 2c + 1).
__device__ __forceinline__ void s8_widen_chunk(const uint8_t* raw, uint8_t* cv, uint32_t atom, int r, int c) {
  const int sw = r & 7;
  const uint4 w = *reinterpret_cast<const uint4*>(raw + r * 128 + ((c ^ sw) << 4));
  uint4 lo, hi;
  s8x16_to_f16(w, lo, hi);
  uint8_t* dst = cv + (c >> 2) * atom + r * 128;
  const int j0 = (c & 3) * 2;
  *reinterpret_cast<uint4*>(dst + ((j0 ^ sw) << 4)) = lo;
  *reinterpret_cast<uint4*>(dst + (((j0 + 1) ^ sw) << 4)) = hi;
}

// BATCH (kOpS8, BN <= 32, chosen for n >= 4): the stream-K fix-up reads every contributor's partial in
// one batch; a separate instantiation, so the one-token drafts run the smaller code without it.
template <int BN, int EPI, int OP, bool BATCH>
__global__ void __launch_bounds__(f8_threads(OP, BN), 1)
    gemm_f8_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmW2,
                   const __grid_constant__ CUtensorMap tmX, const GemmF8Args a) {
  constexpr int S = f8_stages(OP, BN);
  constexpr int C = f8_cstages(OP, BN);
  constexpr int NCONV = f8_conv_warps(OP, BN);
  constexpr uint32_t STAGE = f8_stage_bytes(BN);
  constexpr uint32_t CSTAGE = f8_cstage_bytes(OP, BN);
  constexpr uint32_t TMEM_COLS = f8_tmem_cols(BN);
  constexpr uint32_t IDESC = OP == kOpS8 ? idesc_f16_f32(128, BN) : idesc_e4m3_f32(128, BN);
  // k-blocks one fp32 accumulator may sum (kOpE4M3: a whole tile segment)
  constexpr int REGION = OP == kOpS8 ? kS8Region : (1 << 30);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* cring = smem + S * STAGE;  // kOpS8: the widened fp16 stages
  float* stg = reinterpret_cast<float*>(cring + C * CSTAGE);
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(stg) + f8_staging_bytes(BN));
  uint64_t* empty = full + S;
  uint64_t* tfull = empty + S;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* cfull = drain + 1;
  uint64_t* cempty = cfull + C;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(cempty + C);
  volatile int* flags = reinterpret_cast<volatile int*>(tmem_slot + 1);  // [0] abort, [1] last-arriver

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, cta = blockIdx.x;
  const int kb = a.kblocks;
  const long long U = (long long)a.tiles * kb;
  const long long u0 = (long long)cta * U / G, u1 = (long long)(cta + 1) * U / G;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], OP == kOpS8 ? NCONV : 1);  // kOpS8: released by the converter warps
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);
    }
    mbar_init(drain, 1);
    for (int c = 0; c < C; ++c) {
      mbar_init(&cfull[c], NCONV);
      mbar_init(&cempty[c], 1);
    }
    flags[0] = 0;
    flags[1] = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmW);
    if (EPI == EPI_GLU) tma_prefetch_desc(&tmW2);
    tma_prefetch_desc(&tmX);
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
      // ---------------- TMA producer ----------------
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_x = policy_evict_last();
      auto load_w = [&](int stage, long long u) {
        const int t = (int)(u / kb), k = (int)(u % kb);
        uint8_t* sa = smem + stage * STAGE;
        if (a.wpk != nullptr) {  // the tile's 16 KB swizzled image, contiguous (pack_tiles8_kernel)
          bulk_load_hint(sa, a.wpk + ((size_t)t * kb + k) * kF8ATile, kF8ATile, &full[stage], pol_w);
        } else if (EPI == EPI_GLU) {
          tma_load_2d(sa, &tmW, &full[stage], k * 128, t * 64, pol_w);                  // gate rows
          tma_load_2d(sa + kF8ATile / 2, &tmW2, &full[stage], k * 128, t * 64, pol_w);  // up rows
        } else {
          tma_load_2d(sa, &tmW, &full[stage], k * 128, t * 128, pol_w);
        }
      };
      auto load_x = [&](int stage, long long u) {
        const int k = (int)(u % kb);
        tma_load_2d(smem + stage * STAGE + kF8ATile, &tmX, &full[stage], k * 128, 0, pol_x);
      };
      const long long total = u1 - u0;
      const int pre = (int)(total < S ? total : S);
      uint32_t armed = 0, armed_parity = 0;
      for (int j = 0; j < pre; ++j) {  // weights first: they do not depend on the previous kernel
        mbar_expect_tx(&full[j], STAGE);
        armed |= 1u << j;
        load_w(j, u0 + j);
      }
      pdl_wait();
      for (int j = 0; j < pre; ++j) load_x(j, u0 + j);
      int stage = pre % S;
      uint32_t phase = (uint32_t)((pre / S) & 1);
      for (long long u = u0 + pre; u < u1; ++u) {
        if (!mbar_wait_bounded(&empty[stage], phase ^ 1, flags)) {
          flags[0] = 1;
          set_status(a.status, CASSPEC_E_TIMEOUT);
          break;
        }
        mbar_expect_tx(&full[stage], STAGE);
        armed |= 1u << stage;
        armed_parity = (armed_parity & ~(1u << stage)) | (phase << stage);
        load_w(stage, u);
        load_x(stage, u);
        if (++stage == S) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (flags[0]) {
        for (int s = 0; s < S; ++s)
          if (armed & (1u << s)) mbar_wait_bounded(&full[s], (armed_parity >> s) & 1, nullptr);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer (one thread) ----------------
      int stage = 0;  // kOpE4M3: the byte stages; kOpS8: the widened stages
      uint32_t phase = 0;
      uint32_t used[2] = {0, 0};
      int buf = 0;
      long long u = u0;
      bool ok = true;
      while (u < u1 && ok) {
        const int t = (int)(u / kb);
        const long long seg_end = ((long long)(t + 1) * kb < u1) ? (long long)(t + 1) * kb : u1;
        // one accumulator per REGION k-blocks of the tile segment
        for (long long r0 = u; r0 < seg_end && ok; r0 += REGION) {
          const long long r1 = (r0 + REGION < seg_end) ? r0 + REGION : seg_end;
          if (!mbar_wait_bounded(&tempty[buf], (used[buf] & 1) ^ 1, flags)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
          for (long long uu = r0; uu < r1; ++uu) {
            if (OP == kOpS8) {
              if (!mbar_wait_bounded(&cfull[stage], phase, flags)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t sa = smem_u32(cring + stage * CSTAGE);
              const uint32_t sb = sa + 2 * kF8ATile;
#pragma unroll
              for (int kk = 0; kk < 8; ++kk)  // kind::f16 (fp16 operands per IDESC): 16 columns per MMA
                tc_mma_bf16(d_tmem, sw128_kmajor_desc(sa + (kk >> 2) * kF8ATile + (kk & 3) * 32),
                            sw128_kmajor_desc(sb + (kk >> 2) * (BN * 128) + (kk & 3) * 32), IDESC,
                            (uu > r0 || kk > 0) ? 1u : 0u);
              tc_commit(&cempty[stage]);
              if (++stage == C) {
                stage = 0;
                phase ^= 1;
              }
            } else {
              if (!mbar_wait_bounded(&full[stage], phase, flags)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t sa = smem_u32(smem + stage * STAGE);
              const uint32_t sb = sa + kF8ATile;
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)  // 32 codes (32 bytes) per MMA
                tc_mma_e4m3(d_tmem, sw128_kmajor_desc(sa + kk * 32), sw128_kmajor_desc(sb + kk * 32), IDESC,
                            (uu > r0 || kk > 0) ? 1u : 0u);
              tc_commit(&empty[stage]);
              if (++stage == S) {
                stage = 0;
                phase ^= 1;
              }
            }
          }
          if (!ok) break;
          tc_commit(&tfull[buf]);
          used[buf]++;
          buf ^= 1;
        }
        u = seg_end;
      }
      if (!ok) {
        flags[0] = 1;
        set_status(a.status, CASSPEC_E_TIMEOUT);
      }
      tc_commit(drain);
      mbar_wait_bounded(drain, 0, nullptr);
    }
  } else if (OP == kOpS8 && warp >= 6) {
    // ---------------- converter warps 6.. (kOpS8) ----------------
    // Each byte stage is widened into the next fp16 stage: 128 weight rows and BN activation rows of
    // 8 chunks of 16 codes.  A quarter-warp takes one chunk of 8 consecutive rows, so both the reads
    // and the writes of the 128-byte-swizzled tiles fall in 8 distinct 16-byte bank groups.
    constexpr int CT = 32 * NCONV;
    const int ct = threadIdx.x - 192;  // 0 .. CT - 1
    int stage = 0, cst = 0;
    uint32_t phase = 0, cph = 0;
    bool ok = true;
    for (long long u = u0; u < u1; ++u) {
      if (!mbar_wait_bounded(&full[stage], phase, flags) || !mbar_wait_bounded(&cempty[cst], cph ^ 1, flags)) {
        ok = false;
        break;
      }
      const uint8_t* raw = smem + stage * STAGE;
      uint8_t* cv = cring + cst * CSTAGE;
#pragma unroll
      for (int task = ct; task < 1024; task += CT) s8_widen_chunk(raw, cv, kF8ATile, task & 127, task >> 7);
      for (int task = ct; task < BN * 8; task += CT)
        s8_widen_chunk(raw + kF8ATile, cv + 2 * kF8ATile, (uint32_t)BN * 128u, task % BN, task / BN);
      fence_proxy_async_smem();  // the MMAs read these tiles through the async proxy
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&cfull[cst]);
        mbar_arrive(&empty[stage]);
      }
      if (++stage == S) {
        stage = 0;
        phase ^= 1;
      }
      if (++cst == C) {
        cst = 0;
        cph ^= 1;
      }
    }
    if (!ok) {
      flags[0] = 1;
      set_status(a.status, CASSPEC_E_TIMEOUT);
    }
  } else if (warp >= 2 && warp <= 5) {
    // ---------------- epilogue warps 2..5 ----------------
    const int q = warp & 3;
    const int r = q * 32 + lane;
    auto bar = [] { named_bar_sync(1, 128); };
    // the weight scale of this thread's output row
    float sw_r = 0.f;
    uint32_t used[2] = {0, 0};
    int buf = 0;
    long long u = u0;
    bool ok = true;
    while (u < u1 && ok) {
      const int t = (int)(u / kb);
      const long long seg_end = ((long long)(t + 1) * kb < u1) ? (long long)(t + 1) * kb : u1;
      float v[BN];
      int iv[OP == kOpS8 ? BN : 1];  // kOpS8: the exact int32 sum of the segment's accumulators
      if constexpr (OP == kOpS8) {
#pragma unroll
        for (int i = 0; i < BN; ++i) iv[i] = 0;
      }
      for (long long r0 = u; r0 < seg_end; r0 += REGION) {
        if (!mbar_wait_bounded(&tfull[buf], used[buf] & 1, flags)) {
          flags[0] = 1;
          set_status(a.status, CASSPEC_E_TIMEOUT);
          ok = false;
          break;
        }
        used[buf]++;
        tc_fence_after();
        const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN);
#pragma unroll
        for (int c = 0; c < BN; c += 16) tmem_ld_x16(taddr + c, &v[c]);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[buf]);
        buf ^= 1;
        if constexpr (OP == kOpS8) {
#pragma unroll
          for (int i = 0; i < BN; ++i) iv[i] += __float2int_rn(v[i]);  // an integer below 2^24: exact
        }
      }
      if (!ok) break;

      // stream-K fix-up: the last CTA to finish a shared tile adds the others' (exact integer)
      // partials to its own; integer sums, so the order does not matter
      const int c_first = f8_cta_of_unit((long long)t * kb, U, G);
      const int c_last = f8_cta_of_unit((long long)(t + 1) * kb - 1, U, G);
      bool finish = true;
      if (c_first != c_last) {
        float* mine = a.partials + (size_t)(t + cta) * (64 * 128);
#pragma unroll
        for (int i = 0; i < BN; ++i) {
          if (i < a.ep.n) {
            if constexpr (OP == kOpS8)
              __stcg(mine + i * 128 + r, __int_as_float(iv[i]));
            else
              __stcg(mine + i * 128 + r, v[i]);
          }
        }
        __threadfence();
        bar();
        if (threadIdx.x == 64) {
          const unsigned old = atomicAdd(&a.counters[t], 1u);
          flags[1] = (old == (unsigned)(c_last - c_first)) ? 1 : 0;
        }
        bar();
        finish = flags[1] != 0;
        if (finish) {
          __threadfence();
          auto add_partial = [&](int cc) {
            const float* pp = a.partials + (size_t)(t + cc) * (64 * 128);
#pragma unroll
            for (int i = 0; i < BN; ++i)
              if (i < a.ep.n) {
                const float pv = __ldcg(pp + i * 128 + r);
                if constexpr (OP == kOpS8)
                  iv[i] += __float_as_int(pv);
                else
                  v[i] += pv;
              }
          };
          if (BATCH && c_last - c_first < kF8MaxContrib) {
            // the loads of every contributor's partial are issued together: one memory round trip
            // instead of one per contributor
#pragma unroll
            for (int k = 0; k < kF8MaxContrib; ++k)
              if (k <= c_last - c_first && c_first + k != cta) add_partial(c_first + k);
          } else {
            for (int cc = c_first; cc <= c_last; ++cc)
              if (cc != cta) add_partial(cc);
          }
          if (threadIdx.x == 64) a.counters[t] = 0u;
        }
      }
      if (finish) {
        if (EPI == EPI_GLU) {
          const int ch = t * 64 + (r & 63);
          sw_r = ch < a.N ? (r < 64 ? a.sw[ch] : a.sw2[ch]) : 0.f;
        } else {
          const int o = t * 128 + r;
          sw_r = o < a.N ? a.sw[o] : 0.f;
        }
        // the activation scales come from the previous kernel; its codes were loaded after the
        // dependency wait and have been consumed, so they are visible here
#pragma unroll
        for (int i = 0; i < BN; ++i) {
          const float sxi = i < a.ep.n ? __ldcg(a.sx + i) : 0.f;
          float acc;
          if constexpr (OP == kOpS8)
            acc = (float)iv[i];
          else
            acc = v[i];
          v[i] = acc * sxi * sw_r;
        }
        run_epilogue<BN, EPI>(a.ep, t, r, v, stg, bar, 0, a.ep.n);
      }
      u = seg_end;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------------------------
// Weight codes packed for the projection: one 16 KB image per (128-row tile, 128-column k-block),
// tiles in order and k-blocks in order within a tile, each image exactly what a 2-D TMA box with the
// 128-byte swizzle would leave in shared memory (row r at 128 r, its 16-byte chunk c at c ^ (r % 8));
// rows past N and columns past K are zero.  EPI_GLU tiles hold 64 gate rows, then the same 64 up
// rows.  The stream is then read with plain bulk copies of whole contiguous images.
// ---------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) pack_tiles8_kernel(const uint8_t* __restrict__ src,
                                                          const uint8_t* __restrict__ src2, int N, int K, int glu,
                                                          int kb, uint8_t* __restrict__ dst) {
  const int t = blockIdx.x / kb, k = blockIdx.x % kb;
  uint8_t* img = dst + (size_t)blockIdx.x * kF8ATile;
  for (int idx = threadIdx.x; idx < 1024; idx += 256) {
    const int r = idx >> 3, c = idx & 7;
    const uint8_t* base = src;
    int row = t * 128 + r;
    if (glu) {
      row = t * 64 + (r & 63);
      base = r < 64 ? src : src2;
    }
    const int col = k * 128 + c * 16;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (row < N && col < K) v = *reinterpret_cast<const uint4*>(base + (size_t)row * K + col);
    *reinterpret_cast<uint4*>(img + r * 128 + ((c ^ (r & 7)) << 4)) = v;
  }
}

size_t pack_tiles8_bytes(int N, int K, int glu) {
  const size_t tiles = glu ? (size_t)((N + 63) / 64) : (size_t)((N + 127) / 128);
  return tiles * (size_t)((K + 127) / 128) * kF8ATile;
}

cudaError_t launch_pack_tiles8(const uint8_t* src, const uint8_t* src2, int N, int K, int glu, uint8_t* dst,
                               cudaStream_t stream) {
  if (src == nullptr || dst == nullptr || N < 1 || K < 16 || K % 16 != 0 || (glu && src2 == nullptr))
    return cudaErrorInvalidValue;
  const int kb = (K + 127) / 128;
  const int tiles = glu ? (N + 63) / 64 : (N + 127) / 128;
  pack_tiles8_kernel<<<tiles * kb, 256, 0, stream>>>(src, src2, N, K, glu, kb, dst);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------------------------
bool encode_tmap_u8(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t rows, uint64_t row_stride_bytes,
                    uint32_t box_inner, uint32_t box_rows) {
  void* p = nullptr;
  cudaDriverEntryPointQueryResult qr;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &qr) != cudaSuccess ||
      qr != cudaDriverEntryPointSuccess)
    return false;
  auto fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int EPI, int OP, bool BATCH>
static cudaError_t launch_f8_t(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX,
                               const GemmF8Args& args, int grid, cudaStream_t stream, bool pdl) {
  auto kern = gemm_f8_kernel<BN, EPI, OP, BATCH>;
  constexpr size_t smem = f8_smem_bytes(OP, BN);
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
  cfg.blockDim = dim3(f8_threads(OP, BN));
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, tmW, tmW2, tmX, args);
}

template <int BN, int OP, bool BATCH>
static cudaError_t launch_f8_epi(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int epi,
                                 const GemmF8Args& args, int grid, cudaStream_t s, bool pdl) {
  switch (epi) {
    case EPI_STORE: return launch_f8_t<BN, EPI_STORE, OP, BATCH>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_RESID: return launch_f8_t<BN, EPI_RESID, OP, BATCH>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_QKV: return launch_f8_t<BN, EPI_QKV, OP, BATCH>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_GLU: return launch_f8_t<BN, EPI_GLU, OP, BATCH>(tmW, tmW2, tmX, args, grid, s, pdl);
  }
  return cudaErrorInvalidValue;
}

template <int BN, int OP>
static cudaError_t launch_f8_bn(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int epi,
                                const GemmF8Args& args, int grid, cudaStream_t s, bool pdl) {
  if constexpr (OP == kOpS8 && BN <= 32) {
    if (args.ep.n >= 4) return launch_f8_epi<BN, OP, true>(tmW, tmW2, tmX, epi, args, grid, s, pdl);
  }
  return launch_f8_epi<BN, OP, false>(tmW, tmW2, tmX, epi, args, grid, s, pdl);
}

template <int OP>
static cudaError_t launch_f8_op(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int BN,
                                int epi, const GemmF8Args& args, int grid, cudaStream_t stream, bool pdl) {
  if (args.tiles < 1 || args.kblocks < 1 || args.sx == nullptr || args.sw == nullptr ||
      (epi == EPI_GLU && args.sw2 == nullptr))
    return cudaErrorInvalidValue;
  switch (BN) {
    case 16: return launch_f8_bn<16, OP>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 32: return launch_f8_bn<32, OP>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 48: return launch_f8_bn<48, OP>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 64: return launch_f8_bn<64, OP>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_f8(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int BN, int epi,
                           const GemmF8Args& args, int grid, cudaStream_t stream, bool pdl) {
  return launch_f8_op<kOpE4M3>(tmW, tmW2, tmX, BN, epi, args, grid, stream, pdl);
}

cudaError_t launch_gemm_s8tc(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int BN,
                             int epi, const GemmF8Args& args, int grid, cudaStream_t stream, bool pdl) {
  return launch_f8_op<kOpS8>(tmW, tmW2, tmX, BN, epi, args, grid, stream, pdl);
}

}  // namespace casspec
