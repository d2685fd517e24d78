// Allocation-free variant of the vote + top-k step (see
// mmshift_scores_topk_noalloc in include/mmshift.h): its scratch lives in a
// file-scope device array instead of a caller workspace.
#include <mutex>
#include <string>

#include "common.cuh"

namespace mmshift {
mmshift_status noalloc_prepare(const mmshift_shape* s, const mmshift_params* p, Problem* P);
mmshift_status noalloc_cuda_fail(cudaError_t e);
}  // namespace mmshift

using namespace mmshift;

namespace {

// Shared by every call on a device; holds coverage bitmaps and, when the
// caller passes no scores buffer, the scores.
__device__ __align__(256) unsigned char g_noalloc_scratch[MMSHIFT_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_addr[kMaxDevices] = {};

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

// Device address of the scratch array on the current device. In host code the
// symbol only names a host-side stand-in, so the address is looked up once per
// device with that device current and kept for the life of the process (a
// later cudaDeviceReset would invalidate it; the header says so).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_addr[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_addr[dev] = ptr;
  }
  *out = g_addr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" mmshift_status mmshift_scores_topk_noalloc(const mmshift_shape* s,
                                                      const mmshift_params* p,
                                                      const float* group_mass,
                                                      const float* anchor, float* scores,
                                                      int32_t* out_idx,
                                                      mmshift_stream_t stream) {
  Problem P;
  mmshift_status st = noalloc_prepare(s, p, &P);
  if (st != MMSHIFT_OK) return st;
  if (!p || !out_idx || (P.G && !group_mass)) return MMSHIFT_ERR_INVALID_ARG;
  if (P.mode == MMSHIFT_SCORE_VOTE && !anchor) return MMSHIFT_ERR_INVALID_ARG;
  const size_t bits_bytes = round256((size_t)P.L * P.Hkv * P.G * P.total_words * sizeof(uint32_t));
  const size_t score_bytes = scores ? 0 : round256((size_t)P.L * P.Hkv * P.total_T * sizeof(float));
  if (bits_bytes + score_bytes > MMSHIFT_NOALLOC_SCRATCH_BYTES) return MMSHIFT_ERR_WORKSPACE;
  void* base = nullptr;
  const cudaError_t ea = scratch_address(&base);
  if (ea != cudaSuccess) return noalloc_cuda_fail(ea);
  Buffers bf;
  memset(&bf, 0, sizeof(bf));
  bf.gmass = const_cast<float*>(group_mass);
  bf.anchor = const_cast<float*>(anchor);
  bf.bits = static_cast<uint32_t*>(base);
  bf.scores = scores ? scores : reinterpret_cast<float*>(static_cast<char*>(base) + bits_bytes);
  bf.scores_out = scores ? 1 : 0;
  const cudaStream_t cs = (cudaStream_t)stream;
  cudaError_t e = cudaSuccess;
  if (P.mode == MMSHIFT_SCORE_VOTE) e = launch_cover(P, bf, cs);
  if (e == cudaSuccess) e = launch_topk(P, bf, cs, out_idx, false);
  return e == cudaSuccess ? MMSHIFT_OK : noalloc_cuda_fail(e);
}
