// Prompt-lookup bottom draft (PLD; the default bottom draft M_dn of Sec. 4.1, whose match length is
// its confidence, Sec. 4.2): the tokens that followed the latest earlier occurrence of the history's
// longest matching final n-gram (n in [n_min, n_max]).
//   One CTA: every thread takes candidate end positions p (strided), measures the common suffix of
//   x[..p] and x (the suffix staged in shared memory, coalesced reads of x), and keeps the key
//   (length << 32 | p + 1); a max-reduction over the CTA picks the longest match, then the most
//   recent one.  Integer work, latency-bound for histories of a few thousand tokens.
#include "common.cuh"

namespace casspec {

constexpr int kPldThreads = 1024;
constexpr int kPldMaxN = 64;

__global__ void __launch_bounds__(kPldThreads) pld_kernel(const int32_t* __restrict__ x, int L, int n_min, int n_max,
                                                          int k, int32_t* __restrict__ out) {
  __shared__ int32_t suf[kPldMaxN];  // suf[s] = x[L - 1 - s]
  __shared__ unsigned long long wbest[kPldThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid < n_max && tid < L) suf[tid] = x[L - 1 - tid];
  __syncthreads();
  unsigned long long best = 0ull;
  for (int p = tid; p < L - 1; p += kPldThreads) {
    int s = 0;
    while (s < n_max && s <= p && x[p - s] == suf[s]) ++s;
    if (s >= n_min) {
      const unsigned long long key = ((unsigned long long)s << 32) | (unsigned)(p + 1);
      best = key > best ? key : best;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const unsigned long long o = __shfl_xor_sync(0xffffffffu, best, off);
    best = o > best ? o : best;
  }
  if (lane == 0) wbest[warp] = best;
  __syncthreads();
  if (warp == 0) {
    best = wbest[lane];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const unsigned long long o = __shfl_xor_sync(0xffffffffu, best, off);
      best = o > best ? o : best;
    }
    if (lane == 0) wbest[0] = best;
  }
  __syncthreads();
  best = wbest[0];
  const int n = (int)(best >> 32);
  const int p = (int)(best & 0xffffffffull) - 1;
  const int cnt = n == 0 ? 0 : min(k, L - 1 - p);
  if (tid == 0) {
    out[0] = n;
    out[1] = cnt;
  }
  for (int i = tid; i < cnt; i += kPldThreads) out[2 + i] = x[p + 1 + i];
}

}  // namespace casspec

extern "C" CASSPEC_API int casspec_pld_draft(const int32_t* tokens, int L, int n_min, int n_max, int k, int32_t* out,
                                             void* cuda_stream) {
  if (out == nullptr || (L > 0 && tokens == nullptr) || L < 0 || n_min < 1 || n_max < n_min ||
      n_max > casspec::kPldMaxN || k < 0 || k > CASSPEC_MAX_TREE)
    return CASSPEC_E_INVAL;
  casspec::pld_kernel<<<1, casspec::kPldThreads, 0, static_cast<cudaStream_t>(cuda_stream)>>>(tokens, L, n_min, n_max, k,
                                                                                             out);
  return cudaGetLastError() == cudaSuccess ? CASSPEC_OK : CASSPEC_E_CUDA;
}
