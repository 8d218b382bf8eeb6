// Scoring kernel, mean form of Eq. 6 (the kernel template is in k_score.cuh).
#include "k_score.cuh"

namespace bkv {

cudaError_t launch_score_mean(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32,
                              const CUtensorMap& qmap, const ScoreArgs& a, cudaStream_t st) {
  return launch_score_agg<true, false>(s, kmap, kmap32, qmap, a, st);
}

}  // namespace bkv
