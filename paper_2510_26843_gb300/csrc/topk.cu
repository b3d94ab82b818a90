// K-best candidates per logit row (Sec. 4.2, Algorithm 1: the top-K tokens of each drafted position,
// whose normalised probabilities rank the sibling candidates of the draft tree).
//   One CTA per row: each thread keeps a sorted list of its K best (value descending, token id
//   ascending on ties) and the row maximum; a second pass sums exp(x - max) in a fixed order; K
//   rounds of a block-wide (value, id) maximum then pick the winners, each winner's thread advancing
//   in its list.  Outputs the token ids and their softmax probabilities over the whole row.
#include <climits>

#include "common.cuh"

namespace casspec {

constexpr int kTopkThreads = 256;
constexpr int kTopkMax = 8;

__device__ __forceinline__ bool topk_better(float v, int i, float w, int j) { return v > w || (v == w && i < j); }

__global__ void __launch_bounds__(kTopkThreads) topk_kernel(const float* __restrict__ logits, int V, int K,
                                                            int32_t* __restrict__ idx_out, float* __restrict__ prob_out) {
  __shared__ float s_v[kTopkThreads / 32];
  __shared__ int s_i[kTopkThreads / 32];
  __shared__ float s_red[kTopkThreads / 32];
  const int row = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* x = logits + (size_t)row * V;
  float lv[kTopkMax];
  int li[kTopkMax];
#pragma unroll
  for (int j = 0; j < kTopkMax; ++j) {
    lv[j] = -INFINITY;
    li[j] = INT_MAX;
  }
  float mx = -INFINITY;
  for (int i = tid; i < V; i += kTopkThreads) {
    const float v = x[i];
    mx = fmaxf(mx, v);
    if (topk_better(v, i, lv[kTopkMax - 1], li[kTopkMax - 1])) {  // insertion into the sorted list
#pragma unroll
      for (int pos = kTopkMax - 1; pos >= 0; --pos) {
        const bool shift = pos > 0 && topk_better(v, i, lv[pos - 1], li[pos - 1]);
        const bool here = !shift && topk_better(v, i, lv[pos], li[pos]);
        if (shift) {
          lv[pos] = lv[pos - 1];
          li[pos] = li[pos - 1];
        } else if (here) {
          lv[pos] = v;
          li[pos] = i;
        }
        if (!shift) break;
      }
    }
  }
  // row maximum
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  if (lane == 0) s_red[warp] = mx;
  __syncthreads();
  float M = s_red[0];
#pragma unroll
  for (int w = 1; w < kTopkThreads / 32; ++w) M = fmaxf(M, s_red[w]);
  __syncthreads();
  // sum of exp(x - M), fixed order
  float z = 0.f;
  for (int i = tid; i < V; i += kTopkThreads) z += expf(x[i] - M);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(0xffffffffu, z, off);
  if (lane == 0) s_red[warp] = z;
  __syncthreads();
  float Z = 0.f;
#pragma unroll
  for (int w = 0; w < kTopkThreads / 32; ++w) Z += s_red[w];
  // K rounds of a block-wide maximum over the lists' heads
  int head = 0;
  for (int r = 0; r < K; ++r) {
    float v = -INFINITY;
    int i = INT_MAX;
#pragma unroll
    for (int j = 0; j < kTopkMax; ++j)
      if (j == head) {
        v = lv[j];
        i = li[j];
      }
    const int own_i = i;  // this thread's head (token ids are unique within the row)
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, v, off);
      const int oi = __shfl_xor_sync(0xffffffffu, i, off);
      if (topk_better(ov, oi, v, i)) {
        v = ov;
        i = oi;
      }
    }
    __syncthreads();  // the previous round's winner has been read
    if (lane == 0) {
      s_v[warp] = v;
      s_i[warp] = i;
    }
    __syncthreads();
    float bv = s_v[0];
    int bi = s_i[0];
#pragma unroll
    for (int w = 1; w < kTopkThreads / 32; ++w)
      if (topk_better(s_v[w], s_i[w], bv, bi)) {
        bv = s_v[w];
        bi = s_i[w];
      }
    if (own_i == bi && bi != INT_MAX) ++head;  // the winner's owner moves to its next candidate
    if (tid == 0) {
      const bool valid = bi != INT_MAX;
      idx_out[(size_t)row * K + r] = valid ? bi : -1;
      prob_out[(size_t)row * K + r] = valid ? expf(bv - M) / Z : 0.f;
    }
  }
}

}  // namespace casspec

extern "C" CASSPEC_API int casspec_topk(const float* logits, int n, int V, int K, int32_t* idx_out, float* prob_out,
                                        void* cuda_stream) {
  if (logits == nullptr || idx_out == nullptr || prob_out == nullptr || n < 1 || V < 1 || K < 1 ||
      K > casspec::kTopkMax)
    return CASSPEC_E_INVAL;
  casspec::topk_kernel<<<n, casspec::kTopkThreads, 0, static_cast<cudaStream_t>(cuda_stream)>>>(logits, V, K, idx_out,
                                                                                                 prob_out);
  return cudaGetLastError() == cudaSuccess ? CASSPEC_OK : CASSPEC_E_CUDA;
}
