// tc_softmax_k8.cu -- the fused vocabulary GEMM + online softmax / top-k with 8-entry lists
// (draft branching k <= 8), compiled apart from the 16 / 32-entry variants.
#include "tc_pair.cuh"

namespace dm {

cudaError_t launch_tc_vocab_pair_k8(const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t s) {
  return launch_tc_vocab_pair_instance<8>(maps, p, grid, s);
}

cudaError_t launch_tc_softmax_k8(int bn, bool swap, const CUtensorMap* maps, const TcParams& p, int grid,
                                 cudaStream_t s) {
#define DM_SM(BN, SW) \
  if (bn == BN && swap == SW) return launch_tc_instance<BN, SW, kModeSoftmax, 8>(maps, p, grid, s);
  DM_SM(16, true) DM_SM(32, true) DM_SM(64, true) DM_SM(128, true) DM_SM(256, false)
#undef DM_SM
  return cudaErrorInvalidValue;
}

cudaError_t launch_tc_softmax_deferred_k8(int bn, const CUtensorMap* maps, const TcParams& p, int grid,
                                          cudaStream_t s) {
  if (bn == 16) return launch_tc_instance<16, true, kModeSoftmax, 8, 6>(maps, p, grid, s, true);
  if (bn == 32) return launch_tc_instance<32, true, kModeSoftmax, 8, 5>(maps, p, grid, s, true);
  return cudaErrorInvalidValue;
}

int tc_softmax_deferred_smem_k8(int bn) {
  if (bn == 16) return TcCfg<16, true, kModeSoftmax, 8, 6>::kSmemBytes;
  if (bn == 32) return TcCfg<32, true, kModeSoftmax, 8, 5>::kSmemBytes;
  return 0;
}

}  // namespace dm
