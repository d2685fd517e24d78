// Steps 2-4 on the 5th-generation tensor cores (tcgen05 + TMA + TMEM).
#include "common.cuh"

namespace mmshift {

bool umma_supported(const Problem& P) { (void)P; return false; }

cudaError_t launch_score_umma(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* K) {
  (void)P; (void)bf; (void)st; (void)K;
  return cudaErrorNotSupported;
}

}  // namespace mmshift
