// The small kernels of the tree step: tree preparation, embedding gather, RMSNorm (+ per-token
// int8 quantisation), LM-head argmax reduction, greedy acceptance and KV compaction.
#include "common.cuh"
#include "kernels.h"

namespace casspec {

static cudaLaunchConfig_t make_cfg(dim3 grid, dim3 block, size_t smem, cudaStream_t s, bool pdl,
                                   cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cfg;
}

// Note on loads: a kernel launched with programmatic dependent launch may start before its
// predecessor finishes; everything a predecessor kernel wrote is therefore read with L1-bypassing
// loads (__ldcg / ld.global.cg), never through L1 or the read-only path, which could hold lines
// cached before griddepcontrol.wait returned.

// ---------------------------------------------------------------------------------------------
// Tree preparation (Alg. 1 tree T_r; Sec. 4.2 tree attention).  New node i occupies tree slot
// T + i; its depth is 0 for parent -1 (child of the last committed token) else depth(parent) + 1;
// its position is P + depth; its ancestor mask is anc(parent) | bit(T + i).
// ---------------------------------------------------------------------------------------------
__global__ void tree_prep_kernel(const int* __restrict__ parent, int n, int T, const int* dP, int* tdepth,
                                 unsigned long long* tanc, int* pos, unsigned long long* anc_new, int* status) {
  __shared__ int s_depth[kMaxTree];
  __shared__ unsigned long long s_anc[kMaxTree];
  __shared__ int s_par[kMaxTree];
  pdl_trigger();
  pdl_wait();
  const int P = __ldcg(dP);
  if (threadIdx.x < T) {
    s_depth[threadIdx.x] = __ldcg(tdepth + threadIdx.x);
    s_anc[threadIdx.x] = __ldcg(tanc + threadIdx.x);
  }
  if (threadIdx.x < n) s_par[threadIdx.x] = __ldcg(parent + threadIdx.x);
  __syncthreads();
  if (threadIdx.x == 0) {
    bool bad = false;
    for (int i = 0; i < n; ++i) {
      const int j = T + i;
      const int p = s_par[i];
      int dep;
      unsigned long long an;
      if (p == -1) {
        dep = 0;
        an = 1ull << j;
      } else if (p >= 0 && p < j) {
        dep = s_depth[p] + 1;
        an = s_anc[p] | (1ull << j);
      } else {
        bad = true;  // reported; the node is treated as a depth-0 node so the step stays well defined
        dep = 0;
        an = 1ull << j;
      }
      s_depth[j] = dep;
      s_anc[j] = an;
    }
    if (bad) set_status(status, CASSPEC_E_TREE);
  }
  __syncthreads();
  if (threadIdx.x < n) {
    const int j = T + threadIdx.x;
    tdepth[j] = s_depth[j];
    tanc[j] = s_anc[j];
    pos[threadIdx.x] = P + s_depth[j];
    anc_new[threadIdx.x] = s_anc[j];
  }
}

cudaError_t launch_tree_prep(const int* parent, int n, int T, const int* dP, int* tdepth, unsigned long long* tanc,
                             int* pos, unsigned long long* anc_new, int* status, cudaStream_t s, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(1), dim3(64), 0, s, pdl, attr);
  return cudaLaunchKernelEx(&cfg, tree_prep_kernel, parent, n, T, dP, tdepth, tanc, pos, anc_new, status);
}

// ---------------------------------------------------------------------------------------------
// Block reductions (256 threads)
// ---------------------------------------------------------------------------------------------
__device__ __forceinline__ float block_sum(float v, float* red) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = 0.f;
  for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += red[k];  // fixed order: deterministic
  return t;
}
__device__ __forceinline__ float block_max(float v, float* red) {
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = red[0];
  for (int k = 1; k < (int)(blockDim.x >> 5); ++k) t = fmaxf(t, red[k]);
  return t;
}

// Per-row symmetric int8 quantisation rule (App. C activation-quantisation DSIA, W8A8 reading):
// inv = 127 / amax (IEEE division), q = rint(x * inv) (IEEE multiply, ties to even), clamp +-127,
// scale = amax / 127; amax = 0 gives q = 0, scale 0.
// e4m3 byte of an integer code in [-7, 7] (exact: e4m3 holds every integer up to 16); byte a of the
// constant is the code of +a
__device__ __forceinline__ uint8_t e4m3_of_code(int q) {
  const uint32_t a = (uint32_t)(q < 0 ? -q : q);
  const uint8_t m = (uint8_t)((0x4E4C4A4844403800ull >> (8 * a)) & 0xFFu);
  return q < 0 ? (uint8_t)(m | 0x80u) : m;
}

__device__ __forceinline__ int8_t quant_one(float x, float inv, int qmax) {
  int q = __float2int_rn(__fmul_rn(x, inv));
  q = q > qmax ? qmax : (q < -qmax ? -qmax : q);
  return (int8_t)q;
}

// ---------------------------------------------------------------------------------------------
// Embedding gather: x[i][:] = E[tokens[i]][:] widened to the fp32 residual stream, plus the row's
// sum of squares (the first RMSNorm's scale), ss[i].
// ---------------------------------------------------------------------------------------------
__global__ void embed_kernel(const uint16_t* __restrict__ E, const int* tokens, int d, int vocab,
                             const float* __restrict__ g, float* __restrict__ x, float* __restrict__ ss,
                             uint16_t* __restrict__ xa) {
  __shared__ float red[32];
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x;
  int tok = __ldcg(tokens + i);
  tok = tok < 0 ? 0 : (tok >= vocab ? vocab - 1 : tok);
  const uint16_t* row = E + (size_t)tok * d;
  float acc = 0.f;
  for (int c = threadIdx.x * 2; c < d; c += blockDim.x * 2) {
    const uint32_t two = *reinterpret_cast<const uint32_t*>(row + c);
    const float f0 = bf2f(two & 0xFFFF), f1 = bf2f(two >> 16);
    *reinterpret_cast<float2*>(x + (size_t)i * d + c) = make_float2(f0, f1);
    acc += f0 * f0 + f1 * f1;
    if (xa != nullptr) {  // split(x * g) for the first projection that normalises x
      const float a0 = f0 * g[c], a1 = f1 * g[c + 1];
      const uint16_t h0 = f2bf(a0), h1 = f2bf(a1);
      *reinterpret_cast<uint32_t*>(xa + (size_t)i * d + c) = (uint32_t)h0 | ((uint32_t)h1 << 16);
      *reinterpret_cast<uint32_t*>(xa + (size_t)(64 + i) * d + c) = pack_bf16x2(a0 - bf2f(h0), a1 - bf2f(h1));
    }
  }
  acc = block_sum(acc, red);
  if (threadIdx.x == 0) ss[i] = acc;
}

cudaError_t launch_embed(const uint16_t* E, const int* tokens, int n, int d, int vocab, const float* g, float* x,
                         float* ss, uint16_t* xa, cudaStream_t s, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n), dim3(256), 0, s, pdl, attr);
  return cudaLaunchKernelEx(&cfg, embed_kernel, E, tokens, d, vocab, g, x, ss, g != nullptr ? xa : nullptr);
}

// ---------------------------------------------------------------------------------------------
// RMSNorm (pre-norm): y = bf16(x * rsqrt(mean(x^2) + eps) * g), fp32 arithmetic; optionally the
// per-token int8 quantisation of the bf16 row.  One CTA per row; the row stays in registers
// (16-byte loads, all issued before the first reduction), so the kernel is one memory round trip.
// ---------------------------------------------------------------------------------------------
constexpr int kRowThreads = 512;
constexpr int kRowVec = 8;  // float4 per thread: rows up to 16384 fp32 values

__global__ void __launch_bounds__(kRowThreads) rmsnorm_kernel(const float* __restrict__ x, const float* __restrict__ g,
                                                              int d, float eps, uint16_t* __restrict__ y,
                                                              int8_t* __restrict__ q, float* __restrict__ sq,
                                                              int qmax, int e4m3) {
  __shared__ float red[32];
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x;
  const int nv = d / 4;
  float4 gv[kRowVec];
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) {
    const int c = threadIdx.x + k * kRowThreads;
    gv[k] = c < nv ? reinterpret_cast<const float4*>(g)[c] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)i * d);
  float4 xv[kRowVec];
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) {
    const int c = threadIdx.x + k * kRowThreads;
    xv[k] = c < nv ? __ldcg(xr + c) : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  float ss = 0.f;
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) ss += xv[k].x * xv[k].x + xv[k].y * xv[k].y + xv[k].z * xv[k].z + xv[k].w * xv[k].w;
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / (float)d + eps);
  uint16_t b[kRowVec][4];
  float amax = 0.f;
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) {
    b[k][0] = f2bf(xv[k].x * r * gv[k].x);
    b[k][1] = f2bf(xv[k].y * r * gv[k].y);
    b[k][2] = f2bf(xv[k].z * r * gv[k].z);
    b[k][3] = f2bf(xv[k].w * r * gv[k].w);
    const int c = threadIdx.x + k * kRowThreads;
    if (c < nv) {
      if (y) {
        uint2 pk;
        pk.x = (uint32_t)b[k][0] | ((uint32_t)b[k][1] << 16);
        pk.y = (uint32_t)b[k][2] | ((uint32_t)b[k][3] << 16);
        reinterpret_cast<uint2*>(y + (size_t)i * d)[c] = pk;
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) amax = fmaxf(amax, fabsf(bf2f(b[k][e])));
    }
  }
  if (q == nullptr) return;
  amax = block_max(amax, red);
  const float inv = amax > 0.f ? __fdiv_rn((float)qmax, amax) : 0.f;
#pragma unroll
  for (int k = 0; k < kRowVec; ++k) {
    const int c = threadIdx.x + k * kRowThreads;
    if (c < nv) {
      char4 o;
      o.x = amax > 0.f ? quant_one(bf2f(b[k][0]), inv, qmax) : 0;
      o.y = amax > 0.f ? quant_one(bf2f(b[k][1]), inv, qmax) : 0;
      o.z = amax > 0.f ? quant_one(bf2f(b[k][2]), inv, qmax) : 0;
      o.w = amax > 0.f ? quant_one(bf2f(b[k][3]), inv, qmax) : 0;
      if (e4m3) {
        o.x = (int8_t)e4m3_of_code(o.x);
        o.y = (int8_t)e4m3_of_code(o.y);
        o.z = (int8_t)e4m3_of_code(o.z);
        o.w = (int8_t)e4m3_of_code(o.w);
      }
      reinterpret_cast<char4*>(q + (size_t)i * d)[c] = o;
    }
  }
  if (threadIdx.x == 0) sq[i] = amax > 0.f ? __fdiv_rn(amax, (float)qmax) : 0.f;
}

cudaError_t launch_rmsnorm(const float* x, const float* g, int n, int d, float eps, uint16_t* y, int8_t* q, float* sq,
                           cudaStream_t s, bool pdl, int qmax, int fmt) {
  if (d % 4 != 0 || d > 4 * kRowVec * kRowThreads || qmax < 1 || qmax > 127 || (fmt != 0 && fmt != 2) ||
      (fmt == 2 && qmax > 7))
    return cudaErrorInvalidValue;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n), dim3(kRowThreads), 0, s, pdl, attr);
  return cudaLaunchKernelEx(&cfg, rmsnorm_kernel, x, g, d, eps, y, q, sq, qmax, fmt == 2 ? 1 : 0);
}

// Per-row symmetric quantisation of bf16 rows to codes in [-qmax, qmax] (16-byte loads kept in
// registers; rows up to 16384).  fmt 0: int8 codes; 1: two 4-bit codes per byte (column 2j in the
// low nibble of byte j, 2j + 1 in the high one, two's complement), ldq then counted in bytes; 2: one
// e4m3 byte per code (codes in [-7, 7]).
constexpr int kQVec = 4;  // uint4 (8 bf16) per thread
__global__ void __launch_bounds__(kRowThreads) quant_rows_kernel(const uint16_t* __restrict__ x, int d, int ldx,
                                                                 int8_t* __restrict__ q, int ldq,
                                                                 float* __restrict__ sq, int qmax, int fmt) {
  __shared__ float red[32];
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x;
  const int nv = d / 8;
  const uint16_t* xr = x + (size_t)i * ldx;
  uint4 xv[kQVec];
#pragma unroll
  for (int k = 0; k < kQVec; ++k) {
    const int c = threadIdx.x + k * kRowThreads;
    xv[k] = c < nv ? __ldcg(reinterpret_cast<const uint4*>(xr) + c) : make_uint4(0, 0, 0, 0);
  }
  float amax = 0.f;
#pragma unroll
  for (int k = 0; k < kQVec; ++k) {
    const uint32_t w[4] = {xv[k].x, xv[k].y, xv[k].z, xv[k].w};
#pragma unroll
    for (int e = 0; e < 4; ++e) amax = fmaxf(amax, fmaxf(fabsf(bf2f(w[e] & 0xFFFF)), fabsf(bf2f(w[e] >> 16))));
  }
  amax = block_max(amax, red);
  const float inv = amax > 0.f ? __fdiv_rn((float)qmax, amax) : 0.f;
#pragma unroll
  for (int k = 0; k < kQVec; ++k) {
    const int c = threadIdx.x + k * kRowThreads;
    if (c < nv) {
      const uint32_t w[4] = {xv[k].x, xv[k].y, xv[k].z, xv[k].w};
      uint32_t o[2] = {0u, 0u}, p4 = 0u;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float v = bf2f(e & 1 ? (w[e >> 1] >> 16) : (w[e >> 1] & 0xFFFF));
        const int8_t qq = amax > 0.f ? quant_one(v, inv, qmax) : (int8_t)0;
        o[e >> 2] |= ((uint32_t)(fmt == 2 ? e4m3_of_code(qq) : (uint8_t)qq)) << (8 * (e & 3));
        p4 |= ((uint32_t)qq & 0xFu) << (4 * e);
      }
      if (fmt == 1)
        reinterpret_cast<uint32_t*>(reinterpret_cast<uint8_t*>(q) + (size_t)i * ldq)[c] = p4;
      else
        reinterpret_cast<uint2*>(q + (size_t)i * ldq)[c] = make_uint2(o[0], o[1]);
    }
  }
  if (threadIdx.x == 0) sq[i] = amax > 0.f ? __fdiv_rn(amax, (float)qmax) : 0.f;
}

cudaError_t launch_quant_rows(const uint16_t* x, int n, int d, int ldx, int8_t* q, int ldq, float* sq, cudaStream_t s,
                              bool pdl, int qmax, int fmt) {
  if (d % 8 != 0 || ldx % 8 != 0 || ldq % (fmt == 1 ? 4 : 8) != 0 || d > 8 * kQVec * kRowThreads || qmax < 1 ||
      qmax > 127 || fmt < 0 || fmt > 2 || (fmt != 0 && qmax > 7))
    return cudaErrorInvalidValue;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n), dim3(kRowThreads), 0, s, pdl, attr);
  return cudaLaunchKernelEx(&cfg, quant_rows_kernel, x, d, ldx, q, ldq, sq, qmax, fmt);
}

// ---------------------------------------------------------------------------------------------
// Activation sparsity (App. C, TEAL's magnitude rule): in every token row t of a split activation
// (hi plane row t, lo plane row 64 + t), the z = floor(s K) entries of smallest |hi + lo| become 0 in
// both planes; among equal magnitudes the higher index goes first (the lower is kept).  With
// planes = 1 only the hi plane is read and zeroed (the bf16 activation a quantised draft stores and
// quantises; its lo plane is not used).  One CTA per
// row: a radix select over the magnitude's fp32 bits (4 passes of 8 bits) finds the z-th smallest
// magnitude T and how many entries equal to T are to go; the entries below T and the highest-index
// entries equal to T are zeroed.
// ---------------------------------------------------------------------------------------------
constexpr int kSpThreads = 256;
__global__ void __launch_bounds__(kSpThreads) sparsify_kernel(uint16_t* __restrict__ x, int ld, int K, int z, int planes) {
  extern __shared__ uint32_t sp_key[];  // [K] magnitude bits
  __shared__ unsigned hist[256], part[kSpThreads];
  __shared__ unsigned s_prefix, s_rem;
  pdl_trigger();
  pdl_wait();
  const int t = blockIdx.x, tid = threadIdx.x;
  uint16_t* hi = x + (size_t)t * ld;
  uint16_t* lo = x + (size_t)(64 + t) * ld;
  for (int c = tid; c < K; c += kSpThreads)
    sp_key[c] = __float_as_uint(fabsf(planes == 2 ? bf2f(hi[c]) + bf2f(lo[c]) : bf2f(hi[c])));
  if (tid == 0) {
    s_prefix = 0u;
    s_rem = (unsigned)z;
  }
  unsigned mask = 0u;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int b = tid; b < 256; b += kSpThreads) hist[b] = 0u;
    __syncthreads();
    const unsigned prefix = s_prefix;
    for (int c = tid; c < K; c += kSpThreads) {
      const unsigned k = sp_key[c];
      if ((k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (tid == 0) {  // the bucket that holds the rem-th smallest candidate
      unsigned rem = s_rem, b = 0u;
      for (; b < 255u && hist[b] < rem; ++b) rem -= hist[b];
      s_rem = rem;
      s_prefix = prefix | (b << shift);
    }
    mask |= 255u << shift;
    __syncthreads();
  }
  const unsigned T = s_prefix, rem = s_rem;  // z-th smallest magnitude; entries equal to it to zero
  const int per = (K + kSpThreads - 1) / kSpThreads;
  const int c0 = min(K, tid * per), c1 = min(K, c0 + per);
  unsigned eq = 0u;
  for (int c = c0; c < c1; ++c) eq += sp_key[c] == T ? 1u : 0u;
  part[tid] = eq;
  __syncthreads();
  unsigned after = 0u;  // entries equal to T at higher indices than the one in hand
  for (int k = tid + 1; k < kSpThreads; ++k) after += part[k];
  for (int c = c1 - 1; c >= c0; --c) {
    const unsigned k = sp_key[c];
    bool drop = k < T;
    if (k == T) drop = after++ < rem;
    if (drop) {
      hi[c] = 0;
      if (planes == 2) lo[c] = 0;
    }
  }
}

cudaError_t launch_sparsify(uint16_t* x, int ld, int n, int K, float s, cudaStream_t st, bool pdl, int planes) {
  if (n < 1 || n > 64 || K < 1 || ld < K || !(s >= 0.f && s < 1.f) || (planes != 1 && planes != 2))
    return cudaErrorInvalidValue;
  const int z = (int)floor((double)s * K + 1e-9);
  if (z <= 0) return cudaSuccess;
  const size_t smem = (size_t)K * 4;
  static int configured = -1;
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured != dev) {
    const cudaError_t e = cudaFuncSetAttribute(sparsify_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 65536);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  if (smem > 65536) return cudaErrorInvalidValue;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n), dim3(kSpThreads), smem, st, pdl, attr);
  return cudaLaunchKernelEx(&cfg, sparsify_kernel, x, ld, K, z, planes);
}

// ---------------------------------------------------------------------------------------------
// Argmax over the vocabulary: (max, lowest index of the max, second max) partials per LM-head
// tile are merged; the merge is a total order (ties -> lower id), so lane order does not matter.
// ---------------------------------------------------------------------------------------------
struct Top2 {
  float v1;
  int i1;
  float v2;
};
__device__ __forceinline__ Top2 merge_top2(Top2 a, Top2 b) {
  Top2 r;
  const bool b_wins = (b.v1 > a.v1) || (b.v1 == a.v1 && b.i1 < a.i1);
  r.v1 = b_wins ? b.v1 : a.v1;
  r.i1 = b_wins ? b.i1 : a.i1;
  r.v2 = fmaxf(fmaxf(a.v2, b.v2), fminf(a.v1, b.v1));
  return r;
}

__global__ void argmax_reduce_kernel(const float* __restrict__ v1, const int* __restrict__ i1,
                                     const float* __restrict__ v2, int tiles, int* am, float* margin) {
  pdl_trigger();
  pdl_wait();
  const int row = blockIdx.x, lane = threadIdx.x;
  Top2 acc = {-INFINITY, 0x7fffffff, -INFINITY};
  for (int t = lane; t < tiles; t += 32)
    acc = merge_top2(acc, Top2{__ldcg(v1 + t * 64 + row), __ldcg(i1 + t * 64 + row), __ldcg(v2 + t * 64 + row)});
  for (int o = 16; o > 0; o >>= 1) {
    Top2 other{__shfl_xor_sync(0xffffffffu, acc.v1, o), __shfl_xor_sync(0xffffffffu, acc.i1, o),
               __shfl_xor_sync(0xffffffffu, acc.v2, o)};
    acc = merge_top2(acc, other);
  }
  if (lane == 0) {
    am[row] = acc.i1;
    margin[row] = acc.v1 - acc.v2;
  }
}

cudaError_t launch_argmax_reduce(const float* v1, const int* i1, const float* v2, int tiles, int n, int* am,
                                 float* margin, cudaStream_t s, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n), dim3(32), 0, s, pdl, attr);
  return cudaLaunchKernelEx(&cfg, argmax_reduce_kernel, v1, i1, v2, tiles, am, margin);
}

__global__ void row_argmax_kernel(const float* __restrict__ logits, int V, int* am) {
  __shared__ float sv[8];
  __shared__ int si[8];
  const int row = blockIdx.x;
  const float* lr = logits + (size_t)row * V;
  float best = -INFINITY;
  int bi = 0x7fffffff;
  for (int c = threadIdx.x; c < V; c += blockDim.x) {
    const float x = __ldcg(lr + c);
    if (x > best || (x == best && c < bi)) {
      best = x;
      bi = c;
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (ov > best || (ov == best && oi < bi)) {
      best = ov;
      bi = oi;
    }
  }
  if ((threadIdx.x & 31) == 0) {
    sv[threadIdx.x >> 5] = best;
    si[threadIdx.x >> 5] = bi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
      if (sv[w] > best || (sv[w] == best && si[w] < bi)) {
        best = sv[w];
        bi = si[w];
      }
    am[row] = bi;
  }
}

cudaError_t launch_row_argmax(const float* logits, int n, int V, int* am, cudaStream_t s) {
  row_argmax_kernel<<<n, 256, 0, s>>>(logits, V, am);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// Greedy acceptance (Sec. 5.1 lossless verification): a node matches when its parent matches and
// its token equals the parent's argmax; the deepest match (lowest index among equals) is accepted
// with its root path; the bonus token is the argmax there.
// ---------------------------------------------------------------------------------------------
__global__ void accept_kernel(const int* __restrict__ am, const int* __restrict__ tokens,
                              const int* __restrict__ parent, int n, int* acc, int* status) {
  // Warp-parallel: thread c owns node c.  Pointer jumping (6 rounds for up to 64 nodes) gives every
  // node its depth, whether every edge on its root path matches (child token == parent's argmax),
  // and its ancestor set; a max-reduction picks the deepest matching node (lowest index on ties), and
  // the nodes of its ancestor set write themselves into the path at their depth.
  __shared__ int s_ptr[2][kMaxTree], s_depth[2][kMaxTree], s_match[2][kMaxTree], s_am[kMaxTree];
  __shared__ unsigned long long s_anc[2][kMaxTree];
  __shared__ int s_best, s_bad;
  const int c = threadIdx.x;
  const bool live = c < n;
  int par = -1, tok = 0;
  if (live) {
    par = __ldcg(parent + c);
    tok = __ldcg(tokens + c);
    s_am[c] = __ldcg(am + c);
  }
  if (c == 0) s_bad = 0;
  __syncthreads();
  if (live && (c == 0 ? par != -1 : (par < 0 || par >= c))) atomicOr(&s_bad, 1);
  __syncthreads();
  if (s_bad) {
    if (c == 0) {
      set_status(status, CASSPEC_E_TREE);
      acc[0] = 0;
    }
    return;
  }
  int b = 0;
  if (live) {
    s_ptr[0][c] = par;
    s_depth[0][c] = c == 0 ? 0 : 1;
    s_match[0][c] = c == 0 ? 1 : (tok == s_am[par] ? 1 : 0);
    s_anc[0][c] = 1ull << c;
  }
  __syncthreads();
  for (int r = 0; r < 6; ++r, b ^= 1) {  // 2^6 = 64 >= the deepest path
    if (live) {
      const int q = s_ptr[b][c];
      if (q >= 0) {
        s_ptr[b ^ 1][c] = s_ptr[b][q];
        s_depth[b ^ 1][c] = s_depth[b][c] + s_depth[b][q];
        s_match[b ^ 1][c] = s_match[b][c] & s_match[b][q];
        s_anc[b ^ 1][c] = s_anc[b][c] | s_anc[b][q];
      } else {
        s_ptr[b ^ 1][c] = q;
        s_depth[b ^ 1][c] = s_depth[b][c];
        s_match[b ^ 1][c] = s_match[b][c];
        s_anc[b ^ 1][c] = s_anc[b][c];
      }
    }
    __syncthreads();
  }
  // deepest matching node, lowest index on ties: key = depth * 128 + (127 - c)
  int key = (live && s_match[b][c]) ? s_depth[b][c] * 128 + (127 - c) : -1;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) key = max(key, __shfl_xor_sync(0xffffffffu, key, o));
  if ((c & 31) == 0) s_ptr[b ^ 1][c >> 5] = key;  // (the other buffer is free now)
  __syncthreads();
  if (c == 0) {
    int k = s_ptr[b ^ 1][0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) k = max(k, s_ptr[b ^ 1][w]);
    s_best = 127 - (k & 127);
  }
  __syncthreads();
  const int best = s_best;
  const int L = s_depth[b][best] + 1;
  if (live && ((s_anc[b][best] >> c) & 1ull)) acc[s_depth[b][c] + 1] = c;
  if (c == 0) {
    acc[0] = L;
    acc[L + 1] = s_am[best];
  }
}

cudaError_t launch_accept(const int* am, const int* tokens, const int* parent, int n, int* acc, int* status,
                          cudaStream_t s) {
  accept_kernel<<<1, 64, 0, s>>>(am, tokens, parent, n, acc, status);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// KV compaction: K/V of accepted tree slot path[k] -> committed slot P + k in every layer.  One
// thread owns one 16-byte chunk of one (layer, K|V, head) row and walks k upwards; since
// path[k] >= k, a source slot is never overwritten before it is read.  The CTA that finishes last
// advances P (all CTAs read P before any of them can finish).
// ---------------------------------------------------------------------------------------------
__global__ void kv_compact_kernel(uint16_t* kv, int n_layers, int n_heads, int ctx, int hd, const int* __restrict__ acc,
                                  const unsigned long long* __restrict__ tanc, int T, int* dP, unsigned* counter,
                                  int* status) {
  __shared__ int s_path[kMaxTree];
  __shared__ int s_ok, s_last;
  const int P = __ldcg(dP);
  if (threadIdx.x == 0) {
    const int L = __ldcg(acc);
    // a root-first chain of the current tree: the root (slot 0), then each node a child of the one
    // before it (ancestor sets include the node itself, so anc(j) == anc(prev) | {j} <=> parent(j) == prev)
    bool ok = L >= 1 && L <= T;
    unsigned long long prev_anc = 0ull;
    for (int k = 0; ok && k < L; ++k) {
      const int j = __ldcg(acc + 1 + k);
      ok = j >= 0 && j < T && (k == 0 ? j == 0 : j > s_path[k - 1]);
      if (ok) {
        const unsigned long long an = __ldcg(tanc + j);
        ok = an == (prev_anc | (1ull << j));
        prev_anc = an;
      }
      s_path[k] = j;
    }
    s_ok = ok ? L : 0;
    if (!ok && blockIdx.x == 0) set_status(status, CASSPEC_E_TREE);
  }
  __syncthreads();
  const int L = s_ok;
  const int chunks = hd / 8;
  const long long items = (long long)n_layers * 2 * n_heads * chunks;
  for (long long it = (long long)blockIdx.x * blockDim.x + threadIdx.x; L > 0 && it < items;
       it += (long long)gridDim.x * blockDim.x) {
    const int c = (int)(it % chunks);
    const long long row = it / chunks;  // (layer, kv, head) rows of [ctx][hd]
    uint16_t* base = kv + (size_t)row * ctx * hd + c * 8;
    for (int k = 0; k < L; ++k) {
      const int src = P + s_path[k], dst = P + k;
      if (src != dst)
        *reinterpret_cast<uint4*>(base + (size_t)dst * hd) = *reinterpret_cast<const uint4*>(base + (size_t)src * hd);
    }
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const unsigned old = atomicAdd(counter, 1u);
    s_last = (old == gridDim.x - 1) ? 1 : 0;
  }
  __syncthreads();
  if (s_last && threadIdx.x == 0) {
    if (L > 0) *dP = P + L;
    *counter = 0u;
  }
}

cudaError_t launch_kv_compact(uint16_t* kv, int n_layers, int n_heads, int ctx, int hd, const int* acc,
                              const unsigned long long* tanc, int T, int* dP, unsigned* counter, int* status,
                              cudaStream_t s) {
  const long long items = (long long)n_layers * 2 * n_heads * (hd / 8);
  long long blocks = (items + 255) / 256;
  if (blocks > 1024) blocks = 1024;
  kv_compact_kernel<<<(int)blocks, 256, 0, s>>>(kv, n_layers, n_heads, ctx, hd, acc, tanc, T, dP, counter, status);
  return cudaGetLastError();
}

__global__ void set_int_kernel(int* p, int v) { *p = v; }
cudaError_t launch_set_int(int* p, int v, cudaStream_t s) {
  set_int_kernel<<<1, 1, 0, s>>>(p, v);
  return cudaGetLastError();
}

}  // namespace casspec
