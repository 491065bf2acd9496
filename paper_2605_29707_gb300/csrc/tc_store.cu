// tc_store.cu -- instantiations of the split-K projection GEMM with an fp32 partial-sum
// epilogue (GRU input projection E . W_ih^T and the hidden half of W1 [H_i; S_{i-1}]).
#include "tc_gemm.cuh"

namespace dm {

cudaError_t launch_tc_softmax(int bn, bool swap, int kmax, const CUtensorMap* maps, const TcParams& p,
                              int grid, cudaStream_t s);

static cudaError_t launch_tc_store(int bn, bool swap, const CUtensorMap* maps, const TcParams& p, int grid,
                                   cudaStream_t s) {
#define DM_ST(BN, SW)                 \
  if (bn == BN && swap == SW) return launch_tc_instance<BN, SW, kModeStore, 16>(maps, p, grid, s);
  DM_ST(16, true) DM_ST(32, true) DM_ST(64, true) DM_ST(128, true) DM_ST(256, false)
#undef DM_ST
  return cudaErrorInvalidValue;
}

cudaError_t launch_tc_gemm(int mode, int bn, bool swap, int kmax, const CUtensorMap* maps, const TcParams& p,
                           int grid, cudaStream_t stream) {
  if (mode == kModeSoftmax) return launch_tc_softmax(bn, swap, kmax, maps, p, grid, stream);
  return launch_tc_store(bn, swap, maps, p, grid, stream);
}

}  // namespace dm
