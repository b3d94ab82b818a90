// Exact W4A4 projection on the 5th-generation tensor cores (App. C's W4A4 drafts).
//
// Codes in [-7, 7] are exact FP8 e4m3 values, a product of two codes is at most 49, and every
// partial sum over K <= 65536 is an integer below 2^22, so tcgen05.mma.kind::f8f6f4 with e4m3
// operands and fp32 accumulation returns the exact integer sum in any summation order.  The kernel
// is the bf16 weight-streaming projection with 8-bit operands:
//   * swap-AB: 128 output channels on M, the n <= 64 tokens (padded to BN) on N;
//   * a stage holds a 128 x 128-code weight tile (16 KB, one 2-D TMA box of bytes with the 128-byte
//     swizzle; gate/up: 64 rows of each) and the BN x 128 activation codes; four MMAs of K = 32;
//   * stream-K over (tile, 128-column k-block) units with the last-arriver fix-up (exact integer
//     partials), double-buffered TMEM accumulators, warp roles as in the bf16 projection;
//   * the epilogue dequantises y = acc * s_x[token] * s_w[row] in fp32 (the order of the int8
//     projection) and runs the fused epilogue.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

#include <cudaTypedefs.h>

namespace casspec {

constexpr int kF8Threads = 192;
constexpr uint32_t kF8ATile = 128 * 128;  // 128 rows x 128 e4m3 codes

__host__ __device__ constexpr uint32_t f8_stage_bytes(int BN) { return kF8ATile + (uint32_t)BN * 128u; }
__host__ __device__ constexpr uint32_t f8_staging_bytes(int BN) { return (uint32_t)epi_staging_floats(BN) * 4u; }
__host__ __device__ constexpr int f8_stages(int BN) {
  return (int)((200u * 1024u - f8_staging_bytes(BN) - 1024u) / f8_stage_bytes(BN)) > 8
             ? 8
             : (int)((200u * 1024u - f8_staging_bytes(BN) - 1024u) / f8_stage_bytes(BN));
}
__host__ __device__ constexpr size_t f8_smem_bytes(int BN) {
  return 1024 + (size_t)f8_stages(BN) * f8_stage_bytes(BN) + f8_staging_bytes(BN) + 256;
}
__host__ __device__ constexpr uint32_t f8_tmem_cols(int BN) { return 2 * BN <= 32 ? 32 : (2 * BN <= 64 ? 64 : 128); }

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

template <int BN, int EPI>
__global__ void __launch_bounds__(kF8Threads, 1)
    gemm_f8_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmW2,
                   const __grid_constant__ CUtensorMap tmX, const GemmF8Args a) {
  constexpr int S = f8_stages(BN);
  constexpr uint32_t STAGE = f8_stage_bytes(BN);
  constexpr uint32_t TMEM_COLS = f8_tmem_cols(BN);
  constexpr uint32_t IDESC = idesc_e4m3_f32(128, BN);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* stg = reinterpret_cast<float*>(smem + S * STAGE);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * STAGE + f8_staging_bytes(BN));
  uint64_t* empty = full + S;
  uint64_t* tfull = empty + S;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* flags = reinterpret_cast<volatile int*>(tmem_slot + 1);  // [0] abort, [1] last-arriver

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, cta = blockIdx.x;
  const int kb = a.kblocks;
  const long long U = (long long)a.tiles * kb;
  const long long u0 = (long long)cta * U / G, u1 = (long long)(cta + 1) * U / G;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);
    }
    mbar_init(drain, 1);
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
        if (EPI == EPI_GLU) {
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
      int stage = 0;
      uint32_t phase = 0;
      uint32_t used[2] = {0, 0};
      int buf = 0;
      long long u = u0;
      bool ok = true;
      while (u < u1 && ok) {
        const int t = (int)(u / kb);
        const long long seg_end = ((long long)(t + 1) * kb < u1) ? (long long)(t + 1) * kb : u1;
        if (!mbar_wait_bounded(&tempty[buf], (used[buf] & 1) ^ 1, flags)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
        for (long long uu = u; uu < seg_end; ++uu) {
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
                        (uu > u || kk > 0) ? 1u : 0u);
          tc_commit(&empty[stage]);
          if (++stage == S) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc_commit(&tfull[buf]);
        used[buf]++;
        buf ^= 1;
        u = seg_end;
      }
      if (!ok) {
        flags[0] = 1;
        set_status(a.status, CASSPEC_E_TIMEOUT);
      }
      tc_commit(drain);
      mbar_wait_bounded(drain, 0, nullptr);
    }
  } else {
    // ---------------- epilogue warps 2..5 ----------------
    const int q = warp & 3;
    const int r = q * 32 + lane;
    auto bar = [] { named_bar_sync(1, 128); };
    // the weight scale of this thread's output row
    float sw_r = 0.f;
    uint32_t used[2] = {0, 0};
    int buf = 0;
    long long u = u0;
    bool have_sx = false;
    float sx[BN];
    while (u < u1) {
      const int t = (int)(u / kb);
      const long long seg_end = ((long long)(t + 1) * kb < u1) ? (long long)(t + 1) * kb : u1;
      if (!mbar_wait_bounded(&tfull[buf], used[buf] & 1, flags)) {
        flags[0] = 1;
        set_status(a.status, CASSPEC_E_TIMEOUT);
        break;
      }
      used[buf]++;
      tc_fence_after();
      float v[BN];
      const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN);
#pragma unroll
      for (int c = 0; c < BN; c += 16) tmem_ld_x16(taddr + c, &v[c]);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[buf]);
      buf ^= 1;
      if (!have_sx) {  // the activation scales come from the previous kernel: read after its codes landed
#pragma unroll
        for (int i = 0; i < BN; ++i) sx[i] = i < a.ep.n ? __ldcg(a.sx + i) : 0.f;
        have_sx = true;
      }

      // stream-K fix-up: the last CTA to finish a shared tile sums the (exact integer) partials
      const int c_first = f8_cta_of_unit((long long)t * kb, U, G);
      const int c_last = f8_cta_of_unit((long long)(t + 1) * kb - 1, U, G);
      bool finish = true;
      if (c_first != c_last) {
        float* mine = a.partials + (size_t)(t + cta) * (64 * 128);
#pragma unroll
        for (int i = 0; i < BN; ++i)
          if (i < a.ep.n) __stcg(mine + i * 128 + r, v[i]);
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
          float acc[BN];
#pragma unroll
          for (int i = 0; i < BN; ++i) acc[i] = 0.f;
          for (int cc = c_first; cc <= c_last; ++cc) {
            if (cc == cta) {
#pragma unroll
              for (int i = 0; i < BN; ++i) acc[i] += v[i];
            } else {
              const float* pp = a.partials + (size_t)(t + cc) * (64 * 128);
#pragma unroll
              for (int i = 0; i < BN; ++i)
                if (i < a.ep.n) acc[i] += __ldcg(pp + i * 128 + r);
            }
          }
#pragma unroll
          for (int i = 0; i < BN; ++i) v[i] = acc[i];
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
#pragma unroll
        for (int i = 0; i < BN; ++i) v[i] = v[i] * sx[i] * sw_r;
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

template <int BN, int EPI>
static cudaError_t launch_f8_t(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX,
                               const GemmF8Args& args, int grid, cudaStream_t stream, bool pdl) {
  auto kern = gemm_f8_kernel<BN, EPI>;
  constexpr size_t smem = f8_smem_bytes(BN);
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
  cfg.blockDim = dim3(kF8Threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, tmW, tmW2, tmX, args);
}

template <int BN>
static cudaError_t launch_f8_bn(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int epi,
                                const GemmF8Args& args, int grid, cudaStream_t s, bool pdl) {
  switch (epi) {
    case EPI_STORE: return launch_f8_t<BN, EPI_STORE>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_RESID: return launch_f8_t<BN, EPI_RESID>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_QKV: return launch_f8_t<BN, EPI_QKV>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_GLU: return launch_f8_t<BN, EPI_GLU>(tmW, tmW2, tmX, args, grid, s, pdl);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_f8(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int BN, int epi,
                           const GemmF8Args& args, int grid, cudaStream_t stream, bool pdl) {
  if (args.tiles < 1 || args.kblocks < 1 || args.sx == nullptr || args.sw == nullptr ||
      (epi == EPI_GLU && args.sw2 == nullptr))
    return cudaErrorInvalidValue;
  switch (BN) {
    case 16: return launch_f8_bn<16>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 32: return launch_f8_bn<32>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 48: return launch_f8_bn<48>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 64: return launch_f8_bn<64>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
  }
  return cudaErrorInvalidValue;
}

}  // namespace casspec
