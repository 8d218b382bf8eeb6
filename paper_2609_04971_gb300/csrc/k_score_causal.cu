// Scoring kernel, max form of Eq. 6 with the causal mask inside the recent
// window (the kernel template is in k_score.cuh).
#include "k_score.cuh"

namespace bkv {

cudaError_t launch_score_causal(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32,
                                const CUtensorMap& qmap, const ScoreArgs& a, cudaStream_t st) {
  return launch_score_agg<false, true>(s, kmap, kmap32, qmap, a, st);
}

}  // namespace bkv
