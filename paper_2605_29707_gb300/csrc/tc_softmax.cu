// tc_softmax.cu -- instantiations of the fused vocabulary GEMM + online softmax / top-k
// epilogue (section 4.1.1 base logits and the section 4.1.2 W2 term in one accumulator).
#include "tc_pair.cuh"

namespace dm {

cudaError_t launch_tc_vocab_pair(int kmax, const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t s) {
  if (kmax == 8) return launch_tc_vocab_pair_k8(maps, p, grid, s);
  if (kmax == 16) return launch_tc_vocab_pair_instance<16>(maps, p, grid, s);
  if (kmax == 32) return launch_tc_vocab_pair_instance<32>(maps, p, grid, s);
  return cudaErrorInvalidValue;
}

cudaError_t launch_tc_softmax(int bn, bool swap, int kmax, const CUtensorMap* maps, const TcParams& p,
                              int grid, cudaStream_t s) {
  // tokens on M in CTA pairs: the 2-SM MMA kernel (tc_pair.cuh)
  if (!swap && bn == 256 && p.mcast == 2) return launch_tc_vocab_pair(kmax, maps, p, grid, s);
  if (kmax == 8) return launch_tc_softmax_k8(bn, swap, maps, p, grid, s);
#define DM_SM(BN, SW, KM)                                                              \
  if (bn == BN && swap == SW && kmax == KM)                                            \
    return launch_tc_instance<BN, SW, kModeSoftmax, KM>(maps, p, grid, s);
  DM_SM(16, true, 16) DM_SM(32, true, 16) DM_SM(64, true, 16) DM_SM(128, true, 16) DM_SM(256, false, 16)
  DM_SM(16, true, 32) DM_SM(32, true, 32) DM_SM(64, true, 32) DM_SM(128, true, 32) DM_SM(256, false, 32)
#undef DM_SM
  return cudaErrorInvalidValue;
}

// Deferred variants: 6 stages (BN 16) / 5 stages (BN 32) keep a CTA near 118 KB of shared
// memory so that it fits on an SM next to a GRU CTA.
cudaError_t launch_tc_softmax_deferred(int bn, int kmax, const CUtensorMap* maps, const TcParams& p, int grid,
                                       cudaStream_t s) {
  if (p.defer < 1 || p.defer > kMaxDefer) return cudaErrorInvalidValue;
  if (kmax == 8) return launch_tc_softmax_deferred_k8(bn, maps, p, grid, s);
  if (bn == 16 && kmax == 16) return launch_tc_instance<16, true, kModeSoftmax, 16, 6>(maps, p, grid, s, true);
  if (bn == 16 && kmax == 32) return launch_tc_instance<16, true, kModeSoftmax, 32, 6>(maps, p, grid, s, true);
  if (bn == 32 && kmax == 16) return launch_tc_instance<32, true, kModeSoftmax, 16, 5>(maps, p, grid, s, true);
  if (bn == 32 && kmax == 32) return launch_tc_instance<32, true, kModeSoftmax, 32, 5>(maps, p, grid, s, true);
  return cudaErrorInvalidValue;
}

int tc_softmax_deferred_smem(int bn, int kmax) {
  if (kmax == 8) return tc_softmax_deferred_smem_k8(bn);
  if (bn == 16) return kmax <= 16 ? TcCfg<16, true, kModeSoftmax, 16, 6>::kSmemBytes
                                  : TcCfg<16, true, kModeSoftmax, 32, 6>::kSmemBytes;
  if (bn == 32) return kmax <= 16 ? TcCfg<32, true, kModeSoftmax, 16, 5>::kSmemBytes
                                  : TcCfg<32, true, kModeSoftmax, 32, 5>::kSmemBytes;
  return 0;
}

}  // namespace dm
