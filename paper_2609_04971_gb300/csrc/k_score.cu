// Scoring kernel, max form of Eq. 6 (the kernel template is in k_score.cuh).
#include "k_score.cuh"

namespace bkv {

cudaError_t launch_score(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32, const CUtensorMap& qmap,
                         const ScoreArgs& a, cudaStream_t st) {
  if (a.causal) return a.mean ? launch_score_causal_mean(s, kmap, kmap32, qmap, a, st)
                              : launch_score_causal(s, kmap, kmap32, qmap, a, st);
  if (a.mean) return launch_score_mean(s, kmap, kmap32, qmap, a, st);
  return launch_score_agg<false, false>(s, kmap, kmap32, qmap, a, st);
}

}  // namespace bkv
