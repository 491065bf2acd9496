// tc_gemm.cuh -- persistent tcgen05 GEMM for sm_103a with two K segments and two epilogues.
//
// Warp roles (192 threads):
//   warp 0      one thread issues TMA tile loads into a STAGES-deep shared-memory ring;
//   warp 1      allocates TMEM; one thread issues tcgen05.mma (M = 128, N = BN, K = 16 per
//               instruction) into one of two TMEM accumulators and commits to mbarriers;
//   warps 2..5  epilogue: tcgen05.ld the finished accumulator and either
//               - softmax mode: fold every logit into a per-(token, CTA) running max, running
//                 sum of exp and a top-KMAX list (value desc, id asc), so that the logits never
//                 leave the chip (the vocabulary projection of section 4.1.1 plus the W2 term
//                 of section 4.1.2 in one accumulator), or
//               - store mode: write fp32 partial sums (split-K) of a plain projection.
// The two accumulators let the epilogue of tile i overlap the main loop of tile i+1.
#pragma once

#include <math.h>

#include "kernels.h"
#include "ptx.cuh"
#include "topk.cuh"

#ifndef DOMINO_VOCAB_TRIGGER
#define DOMINO_VOCAB_TRIGGER 1  // let the merge kernel launch while this grid runs
#endif

namespace dm {

template <int BN, bool SWAP, int MODE, int KMAX, int ST = 0>
struct TcCfg {
  static constexpr int kABytes = 128 * 128;  // 128 rows x 64 bf16
  static constexpr int kBBytes = BN * 128;   // BN rows x 64 bf16
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kTPT = SWAP ? 128 / BN : 1;  // epilogue threads per token (swap)
  static constexpr int kTrStride = 128 + kTPT;      // conflict-free transpose pitch (floats)
  static constexpr int kTrBytes = (SWAP && MODE == kModeSoftmax) ? BN * kTrStride * 4 : 0;
  static constexpr int kBudget = 200 * 1024;
  static constexpr int kSt0 = (kBudget - kTrBytes) / kStageBytes;
  static constexpr int kStages = ST > 0 ? ST : (kSt0 > 8 ? 8 : kSt0);
  static constexpr int kTmemCols =
      (2 * BN <= 32) ? 32 : (2 * BN <= 64) ? 64 : (2 * BN <= 128) ? 128 : (2 * BN <= 256) ? 256 : 512;
  static constexpr int kBarBytes = 512;  // ring, accumulator and per-deferred-tile barriers
  // per-thread scratch of one 32-value chunk (rare path of the normal orientation)
  static constexpr int kListBytes = (MODE == kModeSoftmax && !SWAP) ? 128 * 32 * 4 : 0;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kTrBytes + kListBytes + kBarBytes;
  static constexpr int kRec = 2 + 2 * KMAX;
  static_assert(kStages >= 2, "pipeline needs at least two stages");
  static_assert(kSmemBytes <= 227 * 1024, "one CTA's dynamic shared memory limit");
  // CTAs of this kernel that fit on one 228 KB SM (1 KB of shared memory reserved per CTA)
  // never hold more than the SM's 512 TMEM columns between them.  (Across kernels, see the
  // trigger after the allocation in the kernel body.)
  static constexpr int kPerSm = (228 * 1024) / (kSmemBytes + 1024);
  static_assert(kPerSm <= 1 || kPerSm * kTmemCols <= 512, "co-resident CTAs fit in TMEM");
  static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "UMMA N for M = 128");
};

struct TcItem {
  int tok, w, kb0, kb1, split;
};

template <int MODE>
__device__ __forceinline__ bool tc_get_item(const TcParams& p, int i, TcItem& it) {
  const int nkb = p.nkb1 + p.nkb2;
  if (MODE == kModeSoftmax) {
    const int tok = blockIdx.x % p.tok_tiles;
    const int chunk = blockIdx.x / p.tok_tiles;
    const int w = chunk * p.w_per_chunk + i;
    if (chunk >= p.nchunks || i >= p.w_per_chunk || w >= p.w_tiles) return false;
    it.tok = tok; it.w = w; it.kb0 = 0; it.kb1 = nkb; it.split = 0;
    return true;
  } else {
    const int idx = blockIdx.x + i * gridDim.x;
    if (idx >= p.total_items) return false;
    const int split = idx % p.splits;
    const int rest = idx / p.splits;
    it.w = rest % p.w_tiles;
    it.tok = rest / p.w_tiles;
    it.split = split;
    it.kb0 = split * p.kb_per_split;
    it.kb1 = min(nkb, it.kb0 + p.kb_per_split);
    return true;
  }
}

// TMEM column of item i's accumulator: two alternating buffers; in deferred mode the first
// p.defer tiles each keep their own column block (holding the first segment until the second
// is added) and later tiles alternate between the two blocks after them.
template <int BN>
__device__ __forceinline__ uint32_t tc_acc_col(const TcParams& p, int i) {
  if (!p.defer) return static_cast<uint32_t>((i & 1) * BN);
  if (i < p.defer) return static_cast<uint32_t>(i * BN);
  return static_cast<uint32_t>((p.defer + ((i - p.defer) & 1)) * BN);
}

// Running log-sum-exp state and top-KMAX list of one token over a stream of logits.
template <int KM>
struct OnlineTopK {
  float mx, se;
  float tv[KM];
  int ti[KM];

  __device__ __forceinline__ void init() {
    mx = -INFINITY;
    se = 0.f;
#pragma unroll
    for (int q = 0; q < KM; ++q) { tv[q] = -INFINITY; ti[q] = -1; }
  }

  // Stream insert: ids arrive in increasing order, so an equal value never displaces an
  // earlier (lower) id.
  __device__ __forceinline__ void push(float x, int id) {
    if (x > mx) {
      se = se * __expf(mx - x) + 1.f;
      mx = x;
    } else {
      se += __expf(x - mx);
    }
    if (x > tv[KM - 1]) {
#pragma unroll
      for (int q = 0; q < KM; ++q) {
        const bool sw = x > tv[q];
        const float a = tv[q];
        const int b = ti[q];
        tv[q] = sw ? x : a;
        ti[q] = sw ? id : b;
        x = sw ? a : x;
        id = sw ? b : id;
      }
    }
  }

  __device__ __forceinline__ void merge_lse(float omx, float ose) {
    const float m = fmaxf(mx, omx);
    if (m == -INFINITY) return;
    const float a = (mx == -INFINITY) ? 0.f : se * __expf(mx - m);
    const float b = (omx == -INFINITY) ? 0.f : ose * __expf(omx - m);
    mx = m;
    se = a + b;
  }

  // Merge with the state held by lane (laneid ^ offset): both lanes end with the same state
  // (the best KM of the two lists by a bitonic merge).
  __device__ __forceinline__ void merge_shfl_xor(int offset) {
    const float omx = __shfl_xor_sync(0xffffffffu, mx, offset);
    const float ose = __shfl_xor_sync(0xffffffffu, se, offset);
    float ov[KM];
    int oi[KM];
#pragma unroll
    for (int q = 0; q < KM; ++q) {
      ov[q] = __shfl_xor_sync(0xffffffffu, tv[q], offset);
      oi[q] = __shfl_xor_sync(0xffffffffu, ti[q], offset);
    }
    merge_lse(omx, ose);
    merge_lists<KM>(tv, ti, ov, oi);
  }

  // Partial records are stored field-major: field f of chunk c at base[f * stride + c], so a
  // merge kernel reading one field of consecutive chunks issues coalesced loads.
  __device__ __forceinline__ void store(float* base, int stride) const {
    base[0] = mx;
    base[stride] = se;
#pragma unroll
    for (int q = 0; q < KM; ++q) {
      base[(2 + q) * stride] = tv[q];
      reinterpret_cast<int*>(base)[(2 + KM + q) * stride] = ti[q];
    }
  }
};

// ---- streaming softmax/top-k of one epilogue thread ---------------------------------------
// Running max, sum of exp and the top-KMAX list (value desc, id asc) live in registers.  The hot
// path per chunk of values is branch-free: one chunk max, one rescale, one exp per value, and a
// single compare of the chunk max with the list's last value.  Only when that compare passes
// (rare once the list has filled) does the chunk join the list.  A 16-value chunk and a list of
// at most 16 entries (the small-batch swap orientation) are merged by a bitonic sort of the chunk
// and a bitonic merge, a short dependency chain; wider chunks or lists walk the chunk's values, read
// back from shared memory, through the register insertion network, which is emitted once (the
// unrolled networks cost more than they save there).  Values of one thread arrive in increasing
// id order, so an equal value never displaces an earlier entry.
template <int N, int KM>
__device__ __forceinline__ void stream_chunk(const float (&r)[N], const float* sx, int sstride, int v0, int vstride,
                                             int nvalid, float& mx, float& se, float (&tv)[KM], int (&ti)[KM]) {
  float cm = -INFINITY;
#pragma unroll
  for (int j = 0; j < N; ++j) cm = fmaxf(cm, j < nvalid ? r[j] : -INFINITY);
  if (cm > mx) {
    se = (mx == -INFINITY) ? 0.f : se * __expf(mx - cm);
    mx = cm;
  }
  if (mx == -INFINITY) return;
  float sum = 0.f;
#pragma unroll
  for (int j = 0; j < N; ++j) sum += (j < nvalid) ? __expf(r[j] - mx) : 0.f;
  se += sum;
  if (cm > tv[KM - 1]) {
    if constexpr (N == 16 && KM <= 16) {
      float c[16];
      int ci[16];
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        const bool in = q < nvalid;
        c[q] = in ? r[q] : -INFINITY;
        ci[q] = in ? v0 + q * vstride : -1;
      }
      bitonic_sort<16>(c, ci);
      float h[KM];
      int hi[KM];
#pragma unroll
      for (int q = 0; q < KM; ++q) { h[q] = c[q]; hi[q] = ci[q]; }
      merge_lists<KM>(tv, ti, h, hi);
      return;
    }
    const int n = nvalid < N ? nvalid : N;
#pragma unroll 1
    for (int j = 0; j < n; ++j) {
      float x = sx[j * sstride];
      if (!(x > tv[KM - 1])) continue;
      int id = v0 + j * vstride;
#pragma unroll
      for (int q = 0; q < KM; ++q) {
        const bool sw = x > tv[q];
        const float a = tv[q];
        const int b = ti[q];
        tv[q] = sw ? x : a;
        ti[q] = sw ? id : b;
        x = sw ? a : x;
        id = sw ? b : id;
      }
    }
  }
}

// Returns the OR of `pred` over the 128 epilogue threads (named barrier 1).
__device__ __forceinline__ bool epi_any(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, 1, 128, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)pred)
      : "memory");
  return r != 0;
}

// Deferred variants (ST > 0) must fit their registers beside a GRU CTA on one SM: the bound of
// two CTAs per SM caps them at 168 registers per thread.
template <int BN, bool SWAP, int MODE, int KMAX, int ST>
__global__ void __launch_bounds__(192, ST > 0 ? 2 : 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
                   const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmB2,
                   const TcParams p) {
  using C = TcCfg<BN, SWAP, MODE, KMAX, ST>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::kStages * C::kABytes;
  float* tr = reinterpret_cast<float*>(sB + C::kStages * C::kBBytes);
  float* scratch = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(tr) + C::kTrBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(scratch) + C::kListBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + C::kStages;
  uint64_t* tfull = bars + 2 * C::kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* tdone = tempty + 2;  // deferred tile i < p.defer: its accumulator is complete
  uint64_t* drain = tdone + kMaxDefer;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], p.mcast > 1 ? p.mcast : 1);  // every CTA of a multicast cluster releases it
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 128);
    }
    for (int d = 0; d < kMaxDefer; ++d) mbar_init(&tdone[d], 1);
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
  if (warp == 1) {
    tmem_alloc(tmem_slot, static_cast<uint32_t>(p.tmem_cols));
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // Weight multicast (p.mcast > 1, tokens-on-M orientation): the CTAs of a cluster hold
  // consecutive token tiles of one vocabulary chunk and stream the same weight tiles; each loads
  // 1/mcast of every weight box into all of them.  No CTA may multicast before every CTA of the
  // cluster has initialised its barriers.
  const uint16_t mc_mask = static_cast<uint16_t>((1u << (p.mcast > 1 ? p.mcast : 1)) - 1u);
  if (p.mcast > 1) cluster_sync();
  // A kernel launched as this grid's programmatic dependent may start now: it waits for this
  // grid to complete before it reads anything this kernel writes.  The trigger comes after the
  // TMEM allocation, so a dependent that allocates TMEM on this SM can only wait for columns
  // this CTA frees when it ends, never the other way round.
  if (DOMINO_VOCAB_TRIGGER) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const uint64_t pol_w = p.w_evict_first ? l2_policy_evict_first() : l2_policy_evict_normal();
      const uint64_t pol_t = l2_policy_evict_last();
      const uint64_t polA = SWAP ? pol_w : pol_t;
      const uint64_t polB = SWAP ? pol_t : pol_w;
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      bool ok = true;
      TcItem it;
      // Deferred mode (p.defer = D > 0 tiles): pass 0 streams only the first K segment of tiles
      // 0..D-1; the second segment's activations (u) come from the preceding kernel, so pass 1
      // loads them only after griddepcontrol.wait (the hardware's wait for the preceding grid
      // to complete) and adds the second segment to tiles 0..D-1; pass 2 runs tiles D.. whole.
      // Chained launch: the preceding grid wrote this kernel's token operand (pdl_wait = 1), or
      // wrote nothing it reads but must complete before this grid does (pdl_wait = 2).
      if (p.pdl_wait == 1) asm volatile("griddepcontrol.wait;" ::: "memory");
      const int passes = p.defer ? 3 : 1;
      for (int pass = 0; pass < passes && ok; ++pass) {
      if (pass == 1) asm volatile("griddepcontrol.wait;" ::: "memory");
      for (int i = (pass == 2 ? p.defer : 0); ok && tc_get_item<MODE>(p, i, it); ++i) {
        if (pass < 2 && p.defer && i >= p.defer) break;
        const int kb_lo = (p.defer && pass == 1) ? p.nkb1 : it.kb0;
        const int kb_hi = (p.defer && pass == 0) ? p.nkb1 : it.kb1;
        for (int kb = kb_lo; kb < kb_hi; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, p.status)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[stage], C::kStageBytes);
          const bool seg2 = kb >= p.nkb1;
          const int kx = (seg2 ? kb - p.nkb1 : kb) * 64;
          const int ay = SWAP ? it.w * 128 : it.tok * 128;
          const int by = SWAP ? it.tok * BN : it.w * BN;
          tma_load_2d(sA + stage * C::kABytes, seg2 ? &tmA2 : &tmA1, &full[stage], kx, ay, polA);
          if (!SWAP && p.mcast > 1) {
            // this CTA's BN / mcast rows of the weight box (the map's box is that high)
            const int part = static_cast<int>(cluster_ctarank());
            const int rows = BN / p.mcast;
            tma_load_2d_multicast(sB + stage * C::kBBytes + part * rows * 128, seg2 ? &tmB2 : &tmB1, &full[stage],
                                  kx, by + part * rows, mc_mask, polB);
          } else {
            tma_load_2d(sB + stage * C::kBBytes, seg2 ? &tmB2 : &tmB1, &full[stage], kx, by, polB);
          }
          ++issued;
          if (++stage == C::kStages) { stage = 0; phase ^= 1u; }
        }
      }
      }
      if (p.pdl_wait == 2) asm volatile("griddepcontrol.wait;" ::: "memory");
      // Let every load this thread issued land before the CTA can exit (each is the last
      // one on its stage; a completed phase of that parity returns at once).  With multicast,
      // wait until every CTA of the cluster has consumed them (the stage's release).
      const int outstanding = issued < C::kStages ? issued : C::kStages;
      for (int j = 1; j <= outstanding; ++j) {
        int s = stage - j;
        uint32_t ph = phase;
        if (s < 0) { s += C::kStages; ph ^= 1u; }
        uint64_t* last = p.mcast > 1 ? &empty[s] : &full[s];
        const long long t0 = clock64();
        while (!mbar_try_wait(last, ph)) {
          if (clock64() - t0 > kWaitCycles) { set_status(p.status, kStatusTimeout); break; }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t kIdesc = idesc_bf16_f32(128, BN);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      TcItem it;
      const int passes = p.defer ? 3 : 1;
      for (int pass = 0; pass < passes && ok; ++pass) {
      for (int i = (pass == 2 ? p.defer : 0); ok && tc_get_item<MODE>(p, i, it); ++i) {
        if (pass < 2 && p.defer && i >= p.defer) break;
        // A deferred tile (i < p.defer) keeps its own TMEM block and signals its own barrier,
        // so it never waits for the epilogue; later tiles take turns on two blocks.
        const bool own = p.defer && i < p.defer;
        const int jd = own ? 0 : i - p.defer;
        const int ab = jd & 1;
        const uint32_t aph = (jd >> 1) & 1;
        const bool last_pass = !p.defer || pass >= 1;  // passes that finish a tile
        const uint32_t d_tmem = tmem_base + tc_acc_col<BN>(p, i);
        if (last_pass && !own) {
          if (!mbar_wait(&tempty[ab], aph ^ 1u, abort_flag, p.status)) break;
          tc_fence_after();
        }
        const int kb_lo = (p.defer && pass == 1) ? p.nkb1 : it.kb0;
        const int kb_hi = (p.defer && pass == 0) ? p.nkb1 : it.kb1;
        for (int kb = kb_lo; kb < kb_hi; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, p.status)) { ok = false; break; }
          tc_fence_after();
          const uint64_t da = smem_desc_sw128(smem_u32(sA + stage * C::kABytes));
          const uint64_t db = smem_desc_sw128(smem_u32(sB + stage * C::kBBytes));
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            tc_mma_bf16(d_tmem, da + static_cast<uint64_t>(2 * kk), db + static_cast<uint64_t>(2 * kk),
                        kIdesc, (kb > it.kb0 || kk > 0) ? 1u : 0u);
          }
          if (p.mcast > 1) tc_commit_multicast(&empty[stage], mc_mask);  // release it in every CTA
          else tc_commit(&empty[stage]);
          if (++stage == C::kStages) { stage = 0; phase ^= 1u; }
        }
        if (ok && last_pass) tc_commit(own ? &tdone[i] : &tfull[ab]);
      }
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (128 threads)
    const int q = warp & 3;  // TMEM lanes 32q .. 32q+31 belong to this warp
    const int ep = threadIdx.x - 64;
    const uint32_t lane_off = static_cast<uint32_t>(32 * q) << 16;
    OnlineTopK<KMAX> st;
    if (MODE == kModeSoftmax) st.init();
    float* my_scratch = scratch + ep;
    bool aborted = false;
    TcItem it;
    it.tok = 0;
    for (int i = 0; tc_get_item<MODE>(p, i, it); ++i) {
      const bool own = p.defer && i < p.defer;
      const int jd = own ? 0 : i - p.defer;
      const int ab = jd & 1;
      const uint32_t aph = (jd >> 1) & 1;
      const bool ok = own ? mbar_wait(&tdone[i], 0u, abort_flag, p.status)
                          : mbar_wait(&tfull[ab], aph, abort_flag, p.status);
      if (epi_any(!ok)) { aborted = true; break; }
      tc_fence_after();
      const uint32_t tcol = tmem_base + lane_off + tc_acc_col<BN>(p, i);

      if constexpr (MODE == kModeStore) {
        if constexpr (SWAP) {
          const int n = it.w * 128 + 32 * q + lane;
          float* out = p.out + static_cast<size_t>(it.split) * p.rows_tok * p.ld_out;
#pragma unroll
          for (int c0 = 0; c0 < BN; c0 += (BN < 32 ? BN : 32)) {
            float r[BN < 32 ? 16 : 32];
            if constexpr (BN < 32) tc_ld_x16(tcol + c0, r); else tc_ld_x32(tcol + c0, r);
            tc_wait_ld();
#pragma unroll
            for (int j = 0; j < (BN < 32 ? 16 : 32); ++j) {
              const int tok = it.tok * BN + c0 + j;
              if (tok < p.rows_tok && n < p.rows_w) out[static_cast<size_t>(tok) * p.ld_out + n] = r[j];
            }
          }
        } else {
          const int tok = it.tok * 128 + 32 * q + lane;
          float* orow = p.out + (static_cast<size_t>(it.split) * p.rows_tok + tok) * p.ld_out;
#pragma unroll 1
          for (int c0 = 0; c0 < BN; c0 += 32) {
            float r[32];
            tc_ld_x32(tcol + c0, r);
            tc_wait_ld();
            const int n0 = it.w * BN + c0;
            if (tok < p.rows_tok) {
              if (n0 + 32 <= p.rows_w) {
#pragma unroll
                for (int j = 0; j < 32; j += 4)
                  *reinterpret_cast<float4*>(orow + n0 + j) = make_float4(r[j], r[j + 1], r[j + 2], r[j + 3]);
              } else {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  if (n0 + j < p.rows_w) orow[n0 + j] = r[j];
              }
            }
          }
        }
        tc_fence_before();
        mbar_arrive(&tempty[ab]);
      } else if constexpr (SWAP) {
        // vocabulary rows on TMEM lanes, tokens on columns: stage through shared memory so
        // that each thread owns one token and a strided slice of the tile's vocabulary
        const int vrow = 32 * q + lane;
        const int v = it.w * 128 + vrow;
        const bool vvalid = v < p.rows_w;
        const float bv = (p.bias != nullptr && vvalid) ? __bfloat162float(p.bias[v]) : 0.f;
#pragma unroll
        for (int c0 = 0; c0 < BN; c0 += (BN < 32 ? BN : 32)) {
          float r[BN < 32 ? 16 : 32];
          if constexpr (BN < 32) tc_ld_x16(tcol + c0, r); else tc_ld_x32(tcol + c0, r);
          tc_wait_ld();
#pragma unroll
          for (int j = 0; j < (BN < 32 ? 16 : 32); ++j) tr[(c0 + j) * C::kTrStride + vrow] = r[j] + bv;
        }
        tc_fence_before();
        if (!own) mbar_arrive(&tempty[ab]);  // a deferred tile's block is never reused
        named_bar_sync(1, 128);
        const int tt = ep / C::kTPT;
        const int sub = ep % C::kTPT;
        const int vbase = it.w * 128;
        const float* trow = tr + tt * C::kTrStride;
        const int left = p.rows_w - vbase - sub;  // valid entries: sub + TPT * jj < rows_w - vbase
        const int nvalid_all = left <= 0 ? 0 : (left + C::kTPT - 1) / C::kTPT;
        constexpr int kSub = BN < 32 ? BN : 32;
#pragma unroll 1
        for (int j0 = 0; j0 < BN; j0 += kSub) {
          float r[kSub];
          const float* sx = trow + sub + C::kTPT * j0;
#pragma unroll
          for (int j = 0; j < kSub; ++j) r[j] = sx[C::kTPT * j];
          stream_chunk<kSub, KMAX>(r, sx, C::kTPT, vbase + sub + C::kTPT * j0, C::kTPT, nvalid_all - j0, st.mx, st.se,
                                   st.tv, st.ti);
        }
        named_bar_sync(1, 128);
      } else {
        // tokens on TMEM lanes: each thread streams its own row across the vocabulary tile
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
        mbar_arrive(&tempty[ab]);
      }
    }

    if (MODE == kModeSoftmax && !aborted) {
      const int tok_tile = blockIdx.x % p.tok_tiles;
      const int chunk = blockIdx.x / p.tok_tiles;

      if constexpr (SWAP) {
#pragma unroll
        for (int off = C::kTPT / 2; off >= 1; off >>= 1) st.merge_shfl_xor(off);
        const int tt = ep / C::kTPT;
        const int tok = tok_tile * BN + tt;
        if (ep % C::kTPT == 0 && tok < p.rows_tok)
          st.store(p.out + static_cast<size_t>(tok) * C::kRec * p.nchunks + chunk, p.nchunks);
      } else {
        const int tok = tok_tile * 128 + 32 * q + lane;
        if (tok < p.rows_tok) st.store(p.out + static_cast<size_t>(tok) * C::kRec * p.nchunks + chunk, p.nchunks);
      }
    }
  }

  // ------------------------------------------------------------ teardown
  tc_fence_before();
  __syncthreads();
  if (p.mcast > 1) cluster_sync();  // no CTA leaves while a peer may still write into it
  if (warp == 1) {
    if (lane == 0) {
      // every MMA this thread issued must be finished before the TMEM is released
      tc_commit(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(drain, 0)) {
        if (clock64() - t0 > kWaitCycles) { set_status(p.status, kStatusTimeout); break; }
      }
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, static_cast<uint32_t>(p.tmem_cols));
  }
}

template <int BN, bool SWAP, int MODE, int KMAX, int ST = 0>
cudaError_t launch_tc_instance(const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t stream,
                               bool pdl = false) {
  using C = TcCfg<BN, SWAP, MODE, KMAX, ST>;
  auto kern = tc_gemm_kernel<BN, SWAP, MODE, KMAX, ST>;
  {
    const cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), C::kSmemBytes, true);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchAttribute attrs[2];
  int na = 0;
  if (pdl) attrs[na++] = attr[0];
  if (p.mcast > 1) {
    if (SWAP || MODE != kModeSoftmax || p.mcast > 8 || p.tok_tiles % p.mcast != 0 || grid % p.mcast != 0 ||
        BN % (8 * p.mcast) != 0)
      return cudaErrorInvalidValue;
    attrs[na].id = cudaLaunchAttributeClusterDimension;
    attrs[na].val.clusterDim.x = p.mcast;
    attrs[na].val.clusterDim.y = 1;
    attrs[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attrs;
  cfg.numAttrs = na;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, maps[0], maps[1], maps[2], maps[3], p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dm
