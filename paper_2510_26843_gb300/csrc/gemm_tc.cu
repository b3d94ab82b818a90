// Weight-streaming projection on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// Y[i][o] = sum_k X[i][k] W[o][k] for the n <= 64 tokens of a tree step.  At this batch the
// projection is bound by reading W once from HBM, so the kernel is built around the weight stream:
//   * swap-AB: the 128 output channels of a tile are the MMA's M side, the tokens (n padded to BN,
//     a multiple of 16) its N side, so one tcgen05.mma.kind::f16 (M=128, N=BN, K=16) covers all
//     tokens and the accumulator is a 128-lane x BN-column block of tensor memory;
//   * every CTA streams its own weight tiles with 2-D TMA (128 x 64 bf16 = 16 KB per stage, 128-byte
//     swizzle, L2 evict-first) through an S-stage mbarrier ring; the activation tile (BN x 64, reused
//     by all CTAs from L2, evict-last) rides in the same stage;
//   * stream-K over (tile, k-block) units: CTA c of G takes units [cU/G, (c+1)U/G), so all SMs
//     stream the same number of weight bytes.  A tile split across CTAs is finished by the CTA that
//     arrives last on the tile's counter; it sums the partial tiles in CTA order (deterministic) and
//     runs the epilogue.  No CTA ever waits for another;
//   * warp roles: warp 0 = TMA producer, warp 1 = TMEM owner + single-thread MMA issuer, warps 2-5 =
//     epilogue (TMEM -> registers -> fix-up -> fused epilogue).  The accumulator is double buffered in
//     TMEM so the epilogue of one tile overlaps the MMAs of the next;
//   * programmatic dependent launch: the producer issues the first S weight tiles before
//     griddepcontrol.wait, so the weight stream of this projection overlaps the tail of the kernel
//     that produces its activations.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

#include <cudaTypedefs.h>

namespace casspec {

constexpr int kGemmThreads = 192;
constexpr uint32_t kATileBytes = 128 * 128;  // 128 rows x 64 bf16

__host__ __device__ constexpr uint32_t gemm_stage_bytes(int BN) { return kATileBytes + (uint32_t)BN * 128u; }
__host__ __device__ constexpr uint32_t gemm_staging_bytes(int BN) { return (uint32_t)epi_staging_floats(BN) * 4u; }
#ifndef CASSPEC_GEMM_SMEM_BUDGET
#define CASSPEC_GEMM_SMEM_BUDGET (200u * 1024u)
#endif
#ifndef CASSPEC_GEMM_MAX_STAGES
#define CASSPEC_GEMM_MAX_STAGES 8
#endif
__host__ __device__ constexpr int gemm_stages(int BN) {
  return (int)((CASSPEC_GEMM_SMEM_BUDGET - gemm_staging_bytes(BN) - 1024u) / gemm_stage_bytes(BN)) >
                 CASSPEC_GEMM_MAX_STAGES
             ? CASSPEC_GEMM_MAX_STAGES
             : (int)((CASSPEC_GEMM_SMEM_BUDGET - gemm_staging_bytes(BN) - 1024u) / gemm_stage_bytes(BN));
}
__host__ __device__ constexpr size_t gemm_smem_bytes(int BN) {
  return 1024 + (size_t)gemm_stages(BN) * gemm_stage_bytes(BN) + gemm_staging_bytes(BN) + 256;
}
__host__ __device__ constexpr uint32_t gemm_tmem_cols(int BN) { return 2 * BN <= 32 ? 32 : (2 * BN <= 64 ? 64 : 128); }

// CTA that owns stream-K unit x when U units are split evenly over G CTAs.
__device__ __forceinline__ int cta_of_unit(long long x, long long U, int G) {
  return (int)(((x + 1) * (long long)G - 1) / U);
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_bf16_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmW2,
                        const __grid_constant__ CUtensorMap tmX, const GemmArgs a) {
  constexpr int S = gemm_stages(BN);
  constexpr uint32_t STAGE = gemm_stage_bytes(BN);
  constexpr uint32_t TMEM_COLS = gemm_tmem_cols(BN);
  constexpr uint32_t IDESC = idesc_bf16_f32(128, BN);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* stg = reinterpret_cast<float*>(smem + S * STAGE);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * STAGE + gemm_staging_bytes(BN));
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
          const int x = a.w_blocked ? 0 : k * 64, y = a.w_blocked ? (int)u * 64 : t * 64;
          tma_load_2d(sa, &tmW, &full[stage], x, y, pol_w);                    // gate rows
          tma_load_2d(sa + kATileBytes / 2, &tmW2, &full[stage], x, y, pol_w);  // up rows
        } else {
          const int x = a.w_blocked ? 0 : k * 64, y = a.w_blocked ? (int)u * 128 : t * 128;
          tma_load_2d(sa, &tmW, &full[stage], x, y, pol_w);
        }
      };
      auto load_x = [&](int stage, long long u) {
        const int k = (int)(u % kb);
        tma_load_2d(smem + stage * STAGE + kATileBytes, &tmX, &full[stage], k * 64, 0, pol_x);
      };
      const long long total = u1 - u0;
      const int pre = (int)(total < S ? total : S);
      uint32_t armed = 0, armed_parity = 0;  // per stage: armed at least once / parity of the last arm
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
      if (flags[0]) {  // abort: let the copies already issued land before the CTA exits
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
          const uint32_t sb = sa + kATileBytes;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            tc_mma_bf16(d_tmem, sw128_kmajor_desc(sa + kk * 32), sw128_kmajor_desc(sb + kk * 32), IDESC,
                        (uu > u || kk > 0) ? 1u : 0u);
          }
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
      // all MMAs issued by this thread complete before TMEM is released
      tc_commit(drain);
      mbar_wait_bounded(drain, 0, nullptr);
    }
  } else {
    // ---------------- epilogue warps 2..5 ----------------
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int r = q * 32 + lane;
    auto bar = [] { named_bar_sync(1, 128); };
    uint32_t used[2] = {0, 0};
    int buf = 0;
    long long u = u0;
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

      // stream-K fix-up: the last CTA to finish a shared tile sums the partials in CTA order
      const int c_first = cta_of_unit((long long)t * kb, U, G);
      const int c_last = cta_of_unit((long long)(t + 1) * kb - 1, U, G);
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
          if (threadIdx.x == 64) a.counters[t] = 0u;  // ready for the next launch
        }
      }
      if (finish) run_epilogue<BN, EPI>(a.ep, t, r, v, stg, bar, 0, a.ep.n);
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
static PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

bool encode_tmap_bf16(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t rows, uint64_t row_stride_bytes,
                      uint32_t box_inner, uint32_t box_rows) {
  auto fn = get_encode_fn();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int gemm_bf16_grid(int tiles, int kblocks, int num_sms) {
  const long long U = (long long)tiles * kblocks;
  return (int)(U < num_sms ? U : num_sms);
}

size_t gemm_partials_floats(int tiles, int grid) { return (size_t)(tiles + grid) * 64 * 128; }

template <int BN, int EPI>
static cudaError_t launch_t(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX,
                            const GemmArgs& args, int grid, cudaStream_t stream, bool pdl) {
  auto kern = gemm_bf16_tc_kernel<BN, EPI>;
  constexpr size_t smem = gemm_smem_bytes(BN);
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
  cfg.blockDim = dim3(kGemmThreads);
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
static cudaError_t launch_bn(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int epi,
                             const GemmArgs& args, int grid, cudaStream_t s, bool pdl) {
  switch (epi) {
    case EPI_STORE: return launch_t<BN, EPI_STORE>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_RESID: return launch_t<BN, EPI_RESID>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_QKV: return launch_t<BN, EPI_QKV>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_GLU: return launch_t<BN, EPI_GLU>(tmW, tmW2, tmX, args, grid, s, pdl);
    case EPI_LMHEAD: return launch_t<BN, EPI_LMHEAD>(tmW, tmW2, tmX, args, grid, s, pdl);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_bf16(const CUtensorMap& tmW, const CUtensorMap& tmW2, const CUtensorMap& tmX, int BN, int epi,
                             const GemmArgs& args, int grid, cudaStream_t stream, bool pdl) {
  switch (BN) {
    case 16: return launch_bn<16>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 32: return launch_bn<32>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 48: return launch_bn<48>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
    case 64: return launch_bn<64>(tmW, tmW2, tmX, epi, args, grid, stream, pdl);
  }
  return cudaErrorInvalidValue;
}

}  // namespace casspec
