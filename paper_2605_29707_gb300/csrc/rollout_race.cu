// rollout_race.cu -- the sequential draft loop's kernels instantiated for the seeded exponential
// race (Gumbel-max sampling, kRace), compiled apart from rollout.cu's greedy and inverse-CDF ones.
#include "rollout_kernels.cuh"

namespace dm {

cudaError_t launch_rollout_race(const RolloutParams& p, int grid, size_t smem, cudaStream_t stream,
                                const CUtensorMap& tm) {
  return launch_rollout_b<true>(p, grid, smem, stream, tm);
}

}  // namespace dm
