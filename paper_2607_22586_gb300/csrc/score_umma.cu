// Steps 2-4 on the 5th-generation tensor cores (tcgen05 + TMA + TMEM).
#include "common.cuh"

namespace mmshift {

bool umma_supported(const Problem& P) { (void)P; return false; }
int umma_launches(const Problem& P) { (void)P; return 3; }

cudaError_t launch_score_umma(const Problem& P, const Buffers& bf, cudaStream_t st,
                              const void* K, cudaEvent_t* ev) {
  (void)P; (void)bf; (void)st; (void)K; (void)ev;
  return cudaErrorNotSupported;
}

}  // namespace mmshift
