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

cudaError_t launch_tc_store_chained(int bn, const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t s) {
#define DM_STC(BN) \
  if (bn == BN) return launch_tc_instance<BN, true, kModeStore, 16, 4>(maps, p, grid, s, true);
  DM_STC(16) DM_STC(32) DM_STC(64) DM_STC(128)
#undef DM_STC
  return cudaErrorInvalidValue;
}

int tc_store_chained_smem(int bn) {
  switch (bn) {
    case 16: return TcCfg<16, true, kModeStore, 16, 4>::kSmemBytes;
    case 32: return TcCfg<32, true, kModeStore, 16, 4>::kSmemBytes;
    case 64: return TcCfg<64, true, kModeStore, 16, 4>::kSmemBytes;
    case 128: return TcCfg<128, true, kModeStore, 16, 4>::kSmemBytes;
    default: return 0;
  }
}

cudaError_t launch_tc_store_dependent(const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t s) {
  return launch_tc_instance<256, false, kModeStore, 16>(maps, p, grid, s, true);
}

cudaError_t launch_tc_gemm(int mode, int bn, bool swap, int kmax, const CUtensorMap* maps, const TcParams& p,
                           int grid, cudaStream_t stream) {
  if (mode == kModeSoftmax) return launch_tc_softmax(bn, swap, kmax, maps, p, grid, stream);
  return launch_tc_store(bn, swap, maps, p, grid, stream);
}

}  // namespace dm
