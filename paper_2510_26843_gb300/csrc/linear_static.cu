// casspec_linear_bf16_static: the stream-K tcgen05 projection of casspec_linear_bf16 with its
// scratch (fix-up counters + partial tiles) in a file-scope static device array instead of a
// caller workspace, so the call allocates nothing.
//
// It serves callers that cannot hand over a workspace: plain C callers without an allocator for
// device memory, and code that must not call one on the hot path (a device allocation, or a
// caching allocator growing its pool, can synchronise the device).  The price is one fixed
// scratch per device, shared by every call: calls that overlap in time on one device (different
// streams or threads) race on it and must be serialised by the caller.
#include <mutex>

#include "../../include/casspec.h"
#include "kernels.h"

namespace casspec {
namespace {

// Counters (first 4 KB; the last int of it is the call's status word) + partial slots of 64 x 128
// fp32 (32 KB each).  A call needs ceil(N/128) + grid slots, grid <= number of SMs (152 on GB300).
constexpr size_t kStaticCounterBytes = 4096;
constexpr size_t kStaticStatusOffset = kStaticCounterBytes - 4;
constexpr size_t kStaticSlots = 256;
constexpr size_t kStaticScratchBytes = kStaticCounterBytes + kStaticSlots * 64 * 128 * 4;  // 8 MB + 4 KB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_linear_scratch[kStaticScratchBytes];

struct DeviceScratch {
  void* ptr = nullptr;
  int sms = 0;
};
std::mutex g_scratch_mu;
DeviceScratch g_scratch[kMaxDevices];

// Device address of the scratch array and the SM count of the current device (looked up once per
// device, with that device current).
int scratch_of_current_device(DeviceScratch* out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return CASSPEC_E_CUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  DeviceScratch& s = g_scratch[dev];
  if (s.ptr == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_linear_scratch) != cudaSuccess || p == nullptr) return CASSPEC_E_CUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
      return CASSPEC_E_CUDA;
    s.ptr = p;
    s.sms = sms;
  }
  *out = s;
  return CASSPEC_OK;
}

}  // namespace
}  // namespace casspec

using namespace casspec;

extern "C" int casspec_linear_bf16_static(const uint16_t* W, int N, int K, const uint16_t* X, int n, float* Y,
                                          int ldy, void* cuda_stream) {
  if (W == nullptr || X == nullptr || Y == nullptr) return CASSPEC_E_INVAL;
  if (n < 1 || n > CASSPEC_MAX_TREE || N < 1 || K < 8 || K % 8 != 0 || ldy < N) return CASSPEC_E_SHAPE;
  if (((uintptr_t)W & 15) || ((uintptr_t)X & 15)) return CASSPEC_E_INVAL;
  DeviceScratch s;
  const int rc = scratch_of_current_device(&s);
  if (rc != CASSPEC_OK) return rc;
  const int tiles = (N + 127) / 128;
  const int kb = (K + 63) / 64;
  const int grid = gemm_bf16_grid(tiles, kb, s.sms);
  if ((size_t)(tiles + grid) > kStaticSlots) return CASSPEC_E_CAPACITY;  // N beyond the static scratch
  const int BN = (n + 15) / 16 * 16;
  CUtensorMap tw, tx;
  if (!encode_tmap_bf16(&tw, W, K, N, (uint64_t)K * 2, 64, 128) ||
      !encode_tmap_bf16(&tx, X, K, n, (uint64_t)K * 2, 64, BN))
    return CASSPEC_E_CUDA;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  // The counters must be zero when the kernel starts; clearing them per call also recovers from a
  // call that ended early.
  if (cudaMemsetAsync(s.ptr, 0, kStaticCounterBytes, stream) != cudaSuccess) return CASSPEC_E_CUDA;
  GemmArgs a = {};
  a.tiles = tiles;
  a.kblocks = kb;
  a.counters = static_cast<unsigned*>(s.ptr);
  a.partials = reinterpret_cast<float*>(static_cast<unsigned char*>(s.ptr) + kStaticCounterBytes);
  a.status = reinterpret_cast<int*>(static_cast<unsigned char*>(s.ptr) + kStaticStatusOffset);
  a.ep.n = n;
  a.ep.N = N;
  a.ep.y = Y;
  a.ep.ldy = ldy;
  if (launch_gemm_bf16(tw, tw, tx, BN, EPI_STORE, a, grid, stream, false) != cudaSuccess) return CASSPEC_E_CUDA;
  return CASSPEC_OK;
}

extern "C" int casspec_linear_bf16_static_status(void* cuda_stream, int* status_out) {
  if (status_out == nullptr) return CASSPEC_E_INVAL;
  DeviceScratch s;
  const int rc = scratch_of_current_device(&s);
  if (rc != CASSPEC_OK) return rc;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  int st = 0;
  if (cudaMemcpyAsync(&st, static_cast<unsigned char*>(s.ptr) + kStaticStatusOffset, 4, cudaMemcpyDeviceToHost,
                      stream) != cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess)
    return CASSPEC_E_CUDA;
  *status_out = st;
  return CASSPEC_OK;
}
