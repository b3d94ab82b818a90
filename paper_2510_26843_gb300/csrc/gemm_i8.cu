// W8A8 / W4A4 projection for the activation-quantisation drafts (App. C, QSpec-style DSIA).
//
// y[i][o] = (sum_k qx[i][k] * qw[o][k]) * sx[i] * sw[o], with the integer sum exact in int32
// (|sum| <= K * 127^2 < 2^31 for K < 133,000).  tcgen05.mma has no integer kind on sm_103a, so the
// contraction uses the warp-level mma.sync.m16n8k32 s8 x s8 -> s32 path; at draft batch sizes the
// projection is bound by streaming the int8 weights, half the bytes of the bf16 weights.
//   * one CTA = 8 warps = one 128-row output tile (warp w: rows 16w..16w+15) x at most 4 blocks of
//     128 columns; `ksplit` CTAs share a tile along K;
//   * weights go straight from HBM into mma fragments with 16-byte loads (no shared memory), all
//     of the CTA's loads issued before the first MMA, so each CTA pays one memory latency.  The
//     activation slice of the k-range is staged once in shared memory.  Both operands use the same
//     permutation of the 128 columns of a block inside the fragments, which leaves the dot product
//     unchanged: thread (group g, lane t) takes bytes [16t, 16t+16) and [64+16t, 64+16t+16);
//   * W4A4: the weights are packed 4-bit codes (half the bytes again), loaded 8 bytes per fragment
//     piece and widened to int8 in registers just before their MMA; the activations are int8 codes
//     in [-7, 7], so the same s8 MMA gives the exact integer sum;
//   * the CTA that finishes a tile last (atomic counter) sums the int32 partials, dequantises
//     once, and runs the same fused epilogue as the bf16 projection.
#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace casspec {

constexpr int kI8Threads = 256;

__device__ __forceinline__ uint4 ldg_nc16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ uint2 ldg_nc8(const void* p) {
  uint2 v;
  asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
  return v;
}

// 16 signed 4-bit codes (8 bytes, column 2j in the low nibble of byte j) -> 16 int8 in column order:
// each nibble is sign-extended per byte as (v ^ 8) - 8, then low and high nibbles are interleaved.
__device__ __forceinline__ uint4 unpack_s4x16(uint2 w) {
  uint32_t out[4];
  const uint32_t in[2] = {w.x, w.y};
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint32_t lo = __vsub4((in[h] & 0x0F0F0F0Fu) ^ 0x08080808u, 0x08080808u);
    const uint32_t hi = __vsub4(((in[h] >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u, 0x08080808u);
    out[2 * h] = __byte_perm(lo, hi, 0x5140);
    out[2 * h + 1] = __byte_perm(lo, hi, 0x7362);
  }
  return make_uint4(out[0], out[1], out[2], out[3]);
}

constexpr int kI8MaxKb = 4;  // k-blocks of 128 per CTA (all of its weight loads in flight at once)

template <int BN, int EPI, bool W4>
__global__ void __launch_bounds__(kI8Threads) gemm_i8_kernel(const GemmI8Args a) {
  extern __shared__ float stg[];  // the CTA's X slice, then the dequantised tile, then the epilogue staging
  __shared__ int s_last;
  const int tile = blockIdx.x, ks = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t4 = lane & 3;
  pdl_trigger();

  const int KB = (a.K + 127) / 128;
  const int kb0 = (int)((long long)ks * KB / a.ksplit), kb1 = (int)((long long)(ks + 1) * KB / a.ksplit);
  const int nkb = kb1 - kb0;  // <= kI8MaxKb: ksplit >= ceil(KB / kI8MaxKb)
  const int n = a.ep.n;

  // weight rows of this thread's fragments: tile rows lr and lr + 8
  const size_t wld = W4 ? (size_t)a.K / 2 : (size_t)a.K;  // bytes per weight row
  const int8_t* wrow[2];
  bool wok[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int lr = warp * 16 + g + 8 * h;
    if (EPI == EPI_GLU) {
      const int ch = tile * 64 + (lr & 63);
      wok[h] = ch < a.N;
      wrow[h] = (lr < 64 ? a.W : a.W2) + (size_t)(wok[h] ? ch : 0) * wld;
    } else {
      const int o = tile * 128 + lr;
      wok[h] = o < a.N;
      wrow[h] = a.W + (size_t)(wok[h] ? o : 0) * wld;
    }
  }
  // every weight load of the CTA's k-range first (the weights do not depend on the previous kernel);
  // 4-bit codes stay packed in registers until their MMA
  uint4 A[kI8MaxKb][W4 ? 1 : 4];
  uint2 A4[kI8MaxKb][W4 ? 4 : 1];
#pragma unroll
  for (int j = 0; j < kI8MaxKb; ++j) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int col = (kb0 + j) * 128 + c * 64 + 16 * t4;
        const bool ok = j < nkb && wok[h] && col < a.K;
        if (W4)
          A4[j][2 * h + c] = ok ? ldg_nc8(wrow[h] + col / 2) : make_uint2(0u, 0u);
        else
          A[j][2 * h + c] = ok ? ldg_nc16(wrow[h] + col) : make_uint4(0, 0, 0, 0);
      }
    }
  }
  pdl_wait();
  // the activations of the k-range, [BN][nkb * 128] int8 in shared memory (zero beyond n and K)
  int8_t* xs = reinterpret_cast<int8_t*>(stg);
  const int xrow = nkb * 128;
  {
    constexpr int kPieces = (BN * kI8MaxKb * 8 + kI8Threads - 1) / kI8Threads;  // 16-byte pieces per thread
    const int per_tok = nkb * 8;
    const int pieces = BN * per_tok;
    uint4 xv[kPieces];
#pragma unroll
    for (int k = 0; k < kPieces; ++k) {
      const int idx = tid + k * kI8Threads;
      const int tok = idx / per_tok, c = (idx % per_tok) * 16;
      const int col = kb0 * 128 + c;
      xv[k] = (idx < pieces && tok < n && col < a.K)
                  ? __ldcg(reinterpret_cast<const uint4*>(a.X + (size_t)tok * a.K + col))
                  : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int k = 0; k < kPieces; ++k) {
      const int idx = tid + k * kI8Threads;
      if (idx < pieces) *reinterpret_cast<uint4*>(xs + (idx / per_tok) * xrow + (idx % per_tok) * 16) = xv[k];
    }
  }
  __syncthreads();

  int acc[BN / 8][4];
#pragma unroll
  for (int j = 0; j < BN / 8; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0;
#pragma unroll
  for (int kbl = 0; kbl < kI8MaxKb; ++kbl) {
    if (kbl < nkb) {
      uint4 Aw[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) Aw[e] = W4 ? unpack_s4x16(A4[kbl][e]) : A[kbl][W4 ? 0 : e];
#pragma unroll
      for (int j = 0; j < BN / 8; ++j) {
        const int tok = 8 * j + g;
        uint4 B[2];
#pragma unroll
        for (int c = 0; c < 2; ++c)
          B[c] = *reinterpret_cast<const uint4*>(xs + tok * xrow + kbl * 128 + c * 64 + 16 * t4);
#pragma unroll
        for (int s2 = 0; s2 < 4; ++s2) {
          const uint4 lo = Aw[s2 >> 1], hi = Aw[2 + (s2 >> 1)], b = B[s2 >> 1];
          const bool odd = s2 & 1;
          mma_s8_16832(acc[j], odd ? lo.z : lo.x, odd ? hi.z : hi.x, odd ? lo.w : lo.y, odd ? hi.w : hi.y,
                       odd ? b.z : b.x, odd ? b.w : b.y);
        }
      }
    }
  }
  __syncthreads();  // the X slice is dead: the shared memory now takes the dequantised tile

  auto scale_w = [&](int row) -> float {
    if (EPI == EPI_GLU) {
      const int ch = tile * 64 + (row & 63);
      if (ch >= a.N) return 0.f;
      return row < 64 ? a.sw[ch] : a.sw2[ch];
    }
    const int o = tile * 128 + row;
    return o < a.N ? a.sw[o] : 0.f;
  };

  if (a.ksplit > 1) {
    int* part = a.partials + ((size_t)tile * a.ksplit + ks) * (64 * 128);
#pragma unroll
    for (int j = 0; j < BN / 8; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int tok = 8 * j + 2 * t4 + (e & 1), row = warp * 16 + g + 8 * (e >> 1);
        if (tok < n) __stcg(part + tok * 128 + row, acc[j][e]);
      }
    __syncthreads();
    if (tid == 0) {
      __threadfence();
      s_last = (atomicAdd(&a.counters[tile], 1u) == (unsigned)(a.ksplit - 1)) ? 1 : 0;
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    for (int idx = tid; idx < n * 128; idx += kI8Threads) {
      const int tok = idx >> 7, row = idx & 127;
      int sum = 0;
      for (int k = 0; k < a.ksplit; ++k)
        sum += __ldcg(a.partials + ((size_t)tile * a.ksplit + k) * (64 * 128) + tok * 128 + row);
      stg[row * (BN + 1) + tok] = (float)sum * __ldcg(a.sx + tok) * scale_w(row);
    }
    if (tid == 0) a.counters[tile] = 0u;
  } else {
#pragma unroll
    for (int j = 0; j < BN / 8; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int tok = 8 * j + 2 * t4 + (e & 1), row = warp * 16 + g + 8 * (e >> 1);
        if (tok < n) stg[row * (BN + 1) + tok] = (float)acc[j][e] * __ldcg(a.sx + tok) * scale_w(row);
      }
  }
  __syncthreads();
  float v[BN];
  if (tid < 128) {
#pragma unroll
    for (int i = 0; i < BN; ++i) v[i] = stg[tid * (BN + 1) + i];
  }
  __syncthreads();
  if (tid < 128) run_epilogue<BN, EPI>(a.ep, tile, tid, v, stg, [] { named_bar_sync(1, 128); }, 0, a.ep.n);
}

int gemm_i8_ksplit(int tiles, int K, int num_sms) {
  (void)tiles;
  (void)num_sms;
  return ((K + 127) / 128 + kI8MaxKb - 1) / kI8MaxKb;
}

template <int BN, int EPI>
static cudaError_t launch_t(const GemmI8Args& a, cudaStream_t s, bool pdl) {
  if (a.w4 && a.K % 16 != 0) return cudaErrorInvalidValue;  // whole 8-byte groups of codes per fragment
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.tiles, a.ksplit);
  cfg.blockDim = dim3(kI8Threads);
  cfg.dynamicSmemBytes = (size_t)epi_staging_floats(BN) * 4;  // >= BN * 4 * 128 bytes of X slice
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return a.w4 ? cudaLaunchKernelEx(&cfg, gemm_i8_kernel<BN, EPI, true>, a)
              : cudaLaunchKernelEx(&cfg, gemm_i8_kernel<BN, EPI, false>, a);
}

template <int BN>
static cudaError_t launch_bn(const GemmI8Args& a, int epi, cudaStream_t s, bool pdl) {
  switch (epi) {
    case EPI_STORE: return launch_t<BN, EPI_STORE>(a, s, pdl);
    case EPI_RESID: return launch_t<BN, EPI_RESID>(a, s, pdl);
    case EPI_QKV: return launch_t<BN, EPI_QKV>(a, s, pdl);
    case EPI_GLU: return launch_t<BN, EPI_GLU>(a, s, pdl);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_i8(const GemmI8Args& a, int BN, int epi, cudaStream_t stream, bool pdl) {
  switch (BN) {
    case 16: return launch_bn<16>(a, epi, stream, pdl);
    case 32: return launch_bn<32>(a, epi, stream, pdl);
    case 48: return launch_bn<48>(a, epi, stream, pdl);
    case 64: return launch_bn<64>(a, epi, stream, pdl);
  }
  return cudaErrorInvalidValue;
}

}  // namespace casspec
