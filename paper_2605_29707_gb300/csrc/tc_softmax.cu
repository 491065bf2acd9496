// tc_softmax.cu -- instantiations of the fused vocabulary GEMM + online softmax / top-k
// epilogue (section 4.1.1 base logits and the section 4.1.2 W2 term in one accumulator).
#include "tc_gemm.cuh"

namespace dm {

cudaError_t launch_tc_softmax(int bn, bool swap, int kmax, const CUtensorMap* maps, const TcParams& p,
                              int grid, cudaStream_t s) {
#define DM_SM(BN, SW, KM)                                                              \
  if (bn == BN && swap == SW && kmax == KM)                                            \
    return launch_tc_instance<BN, SW, kModeSoftmax, KM>(maps, p, grid, s);
  DM_SM(16, true, 16) DM_SM(32, true, 16) DM_SM(64, true, 16) DM_SM(128, true, 16) DM_SM(256, false, 16)
  DM_SM(16, true, 32) DM_SM(32, true, 32) DM_SM(64, true, 32) DM_SM(128, true, 32) DM_SM(256, false, 32)
#undef DM_SM
  return cudaErrorInvalidValue;
}

}  // namespace dm
