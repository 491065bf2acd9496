// tc_pair.cuh -- the fused vocabulary GEMM + online softmax / top-k for many tokens (tokens on the
// MMA's M side) on CTA pairs with the 2-SM tensor-core MMA (tcgen05 cta_group::2).
//
// The two CTAs of a cluster hold consecutive 128-token tiles of one vocabulary chunk.  Each
// 256 x 256 tile of logits is one MMA per K step: rows 0..127 (the even CTA's tokens) accumulate
// in the even CTA's TMEM and rows 128..255 in the odd CTA's, and each CTA stages only its own
// 128 token rows and its own half (128 rows) of the 256 weight rows of every K block: 32 KB per
// stage instead of the 48 KB a one-CTA 128 x 256 tile needs, so six stages fit where four did, and
// every weight byte reaches one SM's shared memory once.
//
// Roles (192 threads per CTA):
//   warp 0 lane 0   both CTAs: TMA loads of the CTA's token rows and weight half into its ring,
//                   each load signalling the even CTA's stage barrier, which expects the bytes
//                   of both CTAs;
//   warp 1          both CTAs: the pair's TMEM (two 256-column accumulators); then even CTA
//                   lane 0 issues the MMAs once a stage of both CTAs has landed, releases the
//                   stage and publishes finished accumulators in both CTAs (multicast commits);
//   warps 2..5      both CTAs: the softmax / top-k epilogue of the CTA's 128 tokens, as in the
//                   one-CTA kernel; the odd CTA's epilogue reports a drained accumulator to the
//                   even CTA with one remote arrival.
// The logits of the section 4.1.1 LM head and the section 4.1.2 W2 term share the accumulator,
// and no logit leaves the chip.
#pragma once

#include "tc_gemm.cuh"

namespace dm {

template <int KMAX>
struct PairCfg {
  static constexpr int kABytes = 128 * 128;  // 128 token rows x 64 bf16
  static constexpr int kBBytes = 128 * 128;  // this CTA's 128 of the tile's 256 weight rows x 64 bf16
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = 6;
  static constexpr int kListBytes = 128 * 32 * 4;  // per-thread scratch of one 32-value chunk (rare path)
  static constexpr int kBarBytes = 512;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kListBytes + kBarBytes;
  static constexpr int kRec = 2 + 2 * KMAX;
  static_assert(kSmemBytes <= 227 * 1024, "one CTA's dynamic shared memory limit");
};

template <int KMAX>
__global__ void __launch_bounds__(192, 1)
    tc_vocab_pair_kernel(const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
                         const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmB2,
                         const TcParams p) {
  using C = PairCfg<KMAX>;
  constexpr int BN = 256;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::kStages * C::kABytes;
  float* scratch = reinterpret_cast<float*>(sB + C::kStages * C::kBBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(scratch) + C::kListBytes);
  uint64_t* full = bars;                    // even CTA: the stage of both CTAs landed
  uint64_t* empty = full + C::kStages;      // stage consumed by the pair's MMAs
  uint64_t* tfull = empty + C::kStages;     // accumulator finished
  uint64_t* tempty = tfull + 2;             // even CTA: accumulator drained by both epilogues
  uint64_t* drain = tempty + 2;             // every MMA of the pair done
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);  // [2]
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool lead = rank == 0;
  constexpr uint16_t kPairMask = 0x3;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);   // the even CTA's producer, expecting both CTAs' bytes
      mbar_init(&empty[s], 1);  // one multicast commit of the even CTA releases it in both
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 128 + 1);  // the even CTA's 128 epilogue threads + the odd CTA's report
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (threadIdx.x == 32) {
    tma_prefetch_desc(&tmA1);
    tma_prefetch_desc(&tmB1);
    if (p.nkb2 > 0) {
      tma_prefetch_desc(&tmA2);
      tma_prefetch_desc(&tmB2);
    }
  }
  // ---- the pair's tensor memory: two 256-column accumulators, allocated by one warp of each CTA
  //      in two steps; both CTAs must see the same column addresses before any MMA is issued
  //      (otherwise the device status reports DOMINO_ERR_UNSUPPORTED and the pair frees what it
  //      holds and leaves)
  if (warp == 1) tmem_alloc_pair(&tmem_slot[0], 256);
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers initialised, both first allocations written
  tc_fence_after();
  const uint32_t acc0 = tmem_slot[0];
  bool same = acc0 == ld_cluster_u32(cluster_addr(&tmem_slot[0], rank ^ 1u));
  uint32_t acc1 = 0;
  if (same) {
    if (warp == 1) tmem_alloc_pair(&tmem_slot[1], 256);
    tc_fence_before();
    __syncthreads();
    cluster_sync();
    tc_fence_after();
    acc1 = tmem_slot[1];
    same = acc1 == ld_cluster_u32(cluster_addr(&tmem_slot[1], rank ^ 1u));
    if (!same && warp == 1) tmem_dealloc_pair(acc1, 256);
  }
  if (!same) {
    if (threadIdx.x == 0) set_status(p.status, kStatusUnsupported);
    if (warp == 1) tmem_dealloc_pair(acc0, 256);
    cluster_sync();  // no CTA leaves while its peer may still read its slots
    return;
  }
  const uint32_t acc[2] = {acc0, acc1};
  // the merge kernel launched as this grid's programmatic dependent may start; it waits for this
  // grid before it reads the records
  if (DOMINO_VOCAB_TRIGGER) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (both CTAs)
    if (lane == 0) {
      const uint64_t pol_w = p.w_evict_first ? l2_policy_evict_first() : l2_policy_evict_normal();
      const uint64_t pol_t = l2_policy_evict_last();
      const uint32_t lead_full = cluster_addr(full, 0);
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      bool ok = true;
      bool waited = p.pdl_wait != 3;
      TcItem it;
      for (int i = 0; ok && tc_get_item<kModeSoftmax>(p, i, it); ++i) {
        for (int kb = 0; kb < it.kb1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, p.status)) { ok = false; break; }
          const bool seg2 = kb >= p.nkb1;
          if (seg2 && !waited) {
            // launched as a programmatic dependent of the kernel that writes u: the W_lm segment
            // streamed meanwhile; this thread alone reads u (through TMA)
            asm volatile("griddepcontrol.wait;" ::: "memory");
            waited = true;
          }
          if (lead) mbar_arrive_expect_tx(&full[stage], 2 * C::kStageBytes);
          const int kx = (seg2 ? kb - p.nkb1 : kb) * 64;
          const uint32_t bar = lead_full + static_cast<uint32_t>(stage * sizeof(uint64_t));
          tma_load_2d_pair(sA + stage * C::kABytes, seg2 ? &tmA2 : &tmA1, bar, kx, it.tok * 128, pol_t);
          tma_load_2d_pair(sB + stage * C::kBBytes, seg2 ? &tmB2 : &tmB1, bar, kx,
                           it.w * BN + static_cast<int>(rank) * 128, pol_w);
          ++issued;
          if (++stage == C::kStages) { stage = 0; phase ^= 1u; }
        }
      }
      // every load of the pair lands before either CTA can exit: the even CTA waits for its
      // stages' last phases (both CTAs' bytes), and the teardown's cluster barrier holds the odd one
      if (lead) {
        const int outstanding = issued < C::kStages ? issued : C::kStages;
        for (int j = 1; j <= outstanding; ++j) {
          int s = stage - j;
          uint32_t ph = phase;
          if (s < 0) { s += C::kStages; ph ^= 1u; }
          const long long t0 = clock64();
          while (!mbar_try_wait_cluster(&full[s], ph)) {
            if (clock64() - t0 > kWaitCycles) { set_status(p.status, kStatusTimeout); break; }
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && lead) {
      // ---------------------------------------------------------- MMA issuer (even CTA)
      constexpr uint32_t kIdesc = idesc_bf16_f32(256, BN);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      TcItem it;
      for (int i = 0; ok && tc_get_item<kModeSoftmax>(p, i, it); ++i) {
        const int ab = i & 1;
        const uint32_t aph = (i >> 1) & 1;
        if (!mbar_wait_cluster(&tempty[ab], aph ^ 1u, abort_flag, p.status)) break;
        tc_fence_after();
        for (int kb = 0; kb < it.kb1; ++kb) {
          if (!mbar_wait_cluster(&full[stage], phase, abort_flag, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t da = smem_desc_sw128(smem_u32(sA + stage * C::kABytes));
          const uint64_t db = smem_desc_sw128(smem_u32(sB + stage * C::kBBytes));
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16_pair(acc[ab], da + static_cast<uint64_t>(2 * kk), db + static_cast<uint64_t>(2 * kk), kIdesc,
                             (kb > 0 || kk > 0) ? 1u : 0u);
          tc_commit_pair_multicast(&empty[stage], kPairMask);  // release it in both CTAs
          if (++stage == C::kStages) { stage = 0; phase ^= 1u; }
        }
        if (ok) tc_commit_pair_multicast(&tfull[ab], kPairMask);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (128 threads each)
    const int q = warp & 3;  // TMEM lanes 32q .. 32q+31 belong to this warp
    const int ep = threadIdx.x - 64;
    const uint32_t lane_off = static_cast<uint32_t>(32 * q) << 16;
    const uint32_t lead_tempty = cluster_addr(tempty, 0);
    OnlineTopK<KMAX> st;
    st.init();
    float* my_scratch = scratch + ep;
    bool aborted = false;
    TcItem it;
    it.tok = 0;
    for (int i = 0; tc_get_item<kModeSoftmax>(p, i, it); ++i) {
      const int ab = i & 1;
      const uint32_t aph = (i >> 1) & 1;
      const bool ok = mbar_wait_cluster(&tfull[ab], aph, abort_flag, p.status);
      if (epi_any(!ok)) { aborted = true; break; }
      tc_fence_after();
      const uint32_t tcol = acc[ab] + lane_off;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        float r[32];
        tc_ld_x32(tcol + c0, r);
        tc_wait_ld();
        const int v0 = it.w * BN + c0;
        const int nvalid = p.rows_w - v0;
        if (p.bias != nullptr) {
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (j < nvalid) r[j] += __bfloat162float(p.bias[v0 + j]);
        }
        {
          // the rare path re-reads the chunk from this thread's shared-memory scratch
          float cm = -INFINITY;
#pragma unroll
          for (int j = 0; j < 32; ++j) cm = fmaxf(cm, j < nvalid ? r[j] : -INFINITY);
          if (cm > st.tv[KMAX - 1]) {
#pragma unroll
            for (int j = 0; j < 32; ++j) my_scratch[j * 128] = r[j];
          }
        }
        stream_chunk<32, KMAX>(r, my_scratch, 128, v0, 1, nvalid, st.mx, st.se, st.tv, st.ti);
      }
      tc_fence_before();
      if (lead) {
        mbar_arrive(&tempty[ab]);
      } else {
        named_bar_sync(1, 128);  // every thread of this epilogue has read the accumulator
        if (ep == 0) mbar_arrive_cluster(lead_tempty + static_cast<uint32_t>(ab * sizeof(uint64_t)));
      }
    }
    if (!aborted) {
      const int tok = (blockIdx.x % p.tok_tiles) * 128 + 32 * q + lane;
      const int chunk = blockIdx.x / p.tok_tiles;
      if (tok < p.rows_tok) st.store(p.out + static_cast<size_t>(tok) * C::kRec * p.nchunks + chunk, p.nchunks);
    }
  }

  // ------------------------------------------------------------ teardown
  tc_fence_before();
  __syncthreads();
  if (warp == 1 && lane == 0) {
    // every MMA of the pair (issued by the even CTA) has completed in both CTAs' TMEM
    if (lead) tc_commit_pair_multicast(drain, kPairMask);
    const long long t0 = clock64();
    while (!mbar_try_wait_cluster(drain, 0)) {
      if (clock64() - t0 > kWaitCycles) { set_status(p.status, kStatusTimeout); break; }
    }
  }
  cluster_sync();  // neither CTA frees its TMEM or shared memory while the pair still uses them
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(acc[0], 256);
    tmem_dealloc_pair(acc[1], 256);
  }
}

template <int KMAX>
cudaError_t launch_tc_vocab_pair_instance(const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t stream) {
  using C = PairCfg<KMAX>;
  auto kern = tc_vocab_pair_kernel<KMAX>;
  if (p.mcast != 2 || p.tok_tiles % 2 != 0 || grid % 2 != 0 || p.defer != 0) return cudaErrorInvalidValue;
  {
    const cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), C::kSmemBytes, true);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attrs[2];
  attrs[0].id = cudaLaunchAttributeClusterDimension;
  attrs[0].val.clusterDim.x = 2;
  attrs[0].val.clusterDim.y = 1;
  attrs[0].val.clusterDim.z = 1;
  attrs[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attrs[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attrs;
  cfg.numAttrs = p.pdl_wait == 3 ? 2 : 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, maps[0], maps[1], maps[2], maps[3], p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dm
