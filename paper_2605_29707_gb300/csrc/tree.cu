// tree.cu -- merge of the per-CTA softmax partials into log-probabilities and top-k lists,
// then the best-first draft tree (the "Tree" cost of the paper's Fig. 1), one CTA per sequence.
//
// Merge: one warp per draft position combines the (max, sum-exp, top-KMAX) records of every
// vocabulary chunk into lse = max + log(sum) and the k best (value desc, id asc) tokens, with
// logp = logit - lse.
// Tree: warp 0 selects N nodes best-first.  The frontier is every child of an already selected
// node (or of the anchor) not yet selected; the next node is the frontier entry with the greatest
// (score, lower token id, lower parent index).  For each expanded node ("slot") the warp caches
// its best remaining child, so a step is one argmax over the slots plus two child refreshes.
#include <math.h>

#include "kernels.h"
#include "ptx.cuh"

namespace dm {

constexpr int kTreeThreads = 512;
constexpr int kMaxK = 64;
constexpr int kMaxTopk = 32;
constexpr int kMaxN = 256;

template <int KM>
__device__ __forceinline__ void lane_insert(float (&tv)[KM], int (&ti)[KM], float x, int id) {
#pragma unroll
  for (int q = 0; q < KM; ++q) {
    const bool sw = x > tv[q] || (x == tv[q] && (unsigned)id < (unsigned)ti[q]);
    const float a = tv[q];
    const int b = ti[q];
    tv[q] = sw ? x : a;
    ti[q] = sw ? id : b;
    x = sw ? a : x;
    id = sw ? b : id;
  }
}

__device__ __forceinline__ void warp_argmax2(uint32_t hi, uint32_t lo, uint32_t& mhi, uint32_t& mlo,
                                             int& src) {
  mhi = __reduce_max_sync(0xffffffffu, hi);
  mlo = __reduce_max_sync(0xffffffffu, hi == mhi ? lo : 0u);
  const unsigned ball = __ballot_sync(0xffffffffu, hi == mhi && lo == mlo);
  src = __ffs(ball) - 1;
}

template <int KM>
__global__ void __launch_bounds__(kTreeThreads) merge_tree_kernel(const TreeParams p) {
  __shared__ float s_lp[kMaxK * kMaxTopk];
  __shared__ int s_id[kMaxK * kMaxTopk];
  __shared__ float sl_score[kMaxN + 1];
  __shared__ int sl_depth[kMaxN + 1];
  __shared__ unsigned sl_popped[kMaxN + 1];
  __shared__ unsigned sl_hi[kMaxN + 1];
  __shared__ unsigned sl_lo[kMaxN + 1];
  __shared__ int sl_j[kMaxN + 1];

  const int b = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int kWarps = kTreeThreads / 32;
  constexpr int kRec = 2 + 2 * KM;
  const int K = p.K, k = p.k, N = p.N;

  // ---------------------------------------------------------------- merge
  for (int j = warp; j < K; j += kWarps) {
    const int m = b * K + j;
    float mx = -INFINITY, se = 0.f;
    float tv[KM];
    int ti[KM];
#pragma unroll
    for (int q = 0; q < KM; ++q) { tv[q] = -INFINITY; ti[q] = -1; }
    for (int c = lane; c < p.nchunks; c += 32) {
      const float* r = p.partials + (static_cast<size_t>(m) * p.nchunks + c) * kRec;
      const float cm = r[0], cs = r[1];
      const float nm = fmaxf(mx, cm);
      if (nm != -INFINITY) {
        se = (mx == -INFINITY ? 0.f : se * __expf(mx - nm)) + (cm == -INFINITY ? 0.f : cs * __expf(cm - nm));
        mx = nm;
      }
      for (int q = 0; q < KM; ++q) {  // the chunk's list is sorted: stop at the first loser
        const float x = r[2 + q];
        const int id = reinterpret_cast<const int*>(r)[2 + KM + q];
        if (!(x > tv[KM - 1] || (x == tv[KM - 1] && (unsigned)id < (unsigned)ti[KM - 1]))) break;
        lane_insert<KM>(tv, ti, x, id);
      }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      const float om = __shfl_xor_sync(0xffffffffu, mx, o);
      const float os = __shfl_xor_sync(0xffffffffu, se, o);
      const float nm = fmaxf(mx, om);
      if (nm != -INFINITY) {
        se = (mx == -INFINITY ? 0.f : se * __expf(mx - nm)) + (om == -INFINITY ? 0.f : os * __expf(om - nm));
        mx = nm;
      }
    }
    const float lse = mx + logf(se);
    for (int q = 0; q < k; ++q) {
      uint32_t mhi, mlo;
      int src;
      warp_argmax2(f32_ord(tv[0]), ~static_cast<uint32_t>(ti[0]), mhi, mlo, src);
      const float val = __shfl_sync(0xffffffffu, tv[0], src);
      const int id = __shfl_sync(0xffffffffu, ti[0], src);
      if (lane == src) {
#pragma unroll
        for (int i = 0; i + 1 < KM; ++i) { tv[i] = tv[i + 1]; ti[i] = ti[i + 1]; }
        tv[KM - 1] = -INFINITY;
        ti[KM - 1] = -1;
      }
      if (lane == 0) {
        const float lp = val - lse;
        p.topk_ids[static_cast<size_t>(m) * k + q] = id;
        p.topk_logp[static_cast<size_t>(m) * k + q] = lp;
        s_id[j * k + q] = id;
        s_lp[j * k + q] = lp;
      }
    }
  }
  __syncthreads();
  if (warp != 0) return;

  // ---------------------------------------------------------------- tree (warp 0)
  // slot 0 is the anchor; slot i+1 is node i.  Child key: hi = ordered score, lo = token
  // (lower wins) then parent (lower wins); hi == 0 marks "no child left".
  auto refresh = [&](int s) {
    const int d = sl_depth[s];
    uint32_t hi = 0, lo = 0;
    if (lane < k && !((sl_popped[s] >> lane) & 1u)) {
      const float sc = sl_score[s] + s_lp[d * k + lane];
      hi = f32_ord(sc);
      lo = ((0x3FFFFFu - static_cast<uint32_t>(s_id[d * k + lane])) << 10) | (0x3FFu - static_cast<uint32_t>(s));
    }
    uint32_t mhi, mlo;
    int src;
    warp_argmax2(hi, lo, mhi, mlo, src);
    if (lane == 0) {
      sl_hi[s] = mhi;
      sl_lo[s] = mlo;
      sl_j[s] = src;
    }
    __syncwarp();
  };

  if (lane == 0) {
    sl_score[0] = 0.f;
    sl_depth[0] = 0;
    sl_popped[0] = 0u;
  }
  __syncwarp();
  refresh(0);
  const size_t ob = static_cast<size_t>(b) * N;
  for (int i = 0; i < N; ++i) {
    uint32_t hi = 0, lo = 0;
    int sb = -1;
    for (int s = lane; s <= i; s += 32) {
      const uint32_t h = sl_hi[s], l = sl_lo[s];
      if (h > hi || (h == hi && h != 0 && l > lo)) { hi = h; lo = l; sb = s; }
    }
    uint32_t mhi, mlo;
    int src;
    warp_argmax2(hi, lo, mhi, mlo, src);
    const int s = __shfl_sync(0xffffffffu, sb, src);
    const int jj = sl_j[s];
    const int d = sl_depth[s];
    const int tok = s_id[d * k + jj];
    const float sc = sl_score[s] + s_lp[d * k + jj];
    __syncwarp();
    if (lane == 0) {
      p.tree_parent[ob + i] = s - 1;
      p.tree_token[ob + i] = tok;
      p.tree_depth[ob + i] = d + 1;
      if (p.tree_score) p.tree_score[ob + i] = sc;
      sl_score[i + 1] = sc;
      sl_depth[i + 1] = d + 1;
      sl_popped[i + 1] = 0u;
      sl_popped[s] |= 1u << jj;
    }
    __syncwarp();
    refresh(s);
    if (d + 1 < K) {
      refresh(i + 1);
    } else {
      if (lane == 0) sl_hi[i + 1] = 0u;
      __syncwarp();
    }
  }
}

cudaError_t launch_merge_tree(const TreeParams& p, cudaStream_t stream) {
  if (p.K > kMaxK || p.k > kMaxTopk || p.N > kMaxN) return cudaErrorInvalidValue;
  if (p.kmax == 16) merge_tree_kernel<16><<<p.B, kTreeThreads, 0, stream>>>(p);
  else if (p.kmax == 32) merge_tree_kernel<32><<<p.B, kTreeThreads, 0, stream>>>(p);
  else return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace dm
