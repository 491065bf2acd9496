// tree.cu -- merge of the per-CTA softmax partials into log-probabilities and top-k lists,
// then the best-first draft tree (the "Tree" cost of the paper's Fig. 1).
//
// Merge: one CTA per draft row (sequence b, position j).  Thread c reads chunk c's record
// (running max, sum of exp, top-KMAX list; field-major, so the loads are coalesced), the CTA
// reduces lse = max + log(sum) and extracts the k best (value desc, id asc) tokens; logp =
// logit - lse.
// Tree: the CTA that merges the last row of a sequence (atomic counter) selects N nodes
// best-first with one warp.  The frontier is every child (from its position's top-k list) of
// the anchor or of an already selected node that is not selected yet; the next node is the
// frontier entry with the greatest (score, lower token id, lower parent index).  Each expanded
// node ("slot") caches its best remaining child.  Children of a slot have non-increasing scores
// (sorted log-probs plus the same parent score), so the best remaining child is the first
// unselected one, or a lower-token child of exactly the same score; one lane refreshes a slot
// by that short scan.
#include <math.h>

#include "kernels.h"
#include "ptx.cuh"

#ifndef DOMINO_TREE_PDL
#define DOMINO_TREE_PDL 1  // launch the merge kernel as a programmatic dependent of the vocab GEMM
#endif

namespace dm {

constexpr int kMergeThreads = 256;
constexpr int kMaxK = 64;
constexpr int kMaxTopk = 32;
constexpr int kMaxN = 256;

__device__ __forceinline__ void warp_argmax2(uint32_t hi, uint32_t lo, uint32_t& mhi, uint32_t& mlo, int& src) {
  mhi = __reduce_max_sync(0xffffffffu, hi);
  mlo = __reduce_max_sync(0xffffffffu, hi == mhi ? lo : 0u);
  const unsigned ball = __ballot_sync(0xffffffffu, hi == mhi && lo == mlo);
  src = __ffs(ball) - 1;
}

template <int KM>
__device__ __forceinline__ void insert_keyed(float (&tv)[KM], int (&ti)[KM], float x, int id) {
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

__device__ __forceinline__ void lse_merge(float& mx, float& se, float om, float os) {
  const float nm = fmaxf(mx, om);
  if (nm == -INFINITY) return;
  se = (mx == -INFINITY ? 0.f : se * __expf(mx - nm)) + (om == -INFINITY ? 0.f : os * __expf(om - nm));
  mx = nm;
}

struct TreeSlots {
  float score[kMaxN + 1];
  int depth[kMaxN + 1];
  unsigned mask[kMaxN + 1];
  unsigned hi[kMaxN + 1];
  unsigned lo[kMaxN + 1];
  int j[kMaxN + 1];
};

// Best remaining child of slot s (one thread).  The caller passes the slot's depth d, score
// and popped mask in registers; children of a slot have non-increasing scores, so the best
// remaining one is the first unpopped child, or an unpopped child of exactly the same score
// with a lower token id.
__device__ __forceinline__ void refresh_slot(TreeSlots& S, int s, int d, float base, unsigned mask, const float* lp,
                                             const int* ids, int K, int k) {
  if (d >= K) { S.hi[s] = 0u; return; }
  const unsigned all = (k == 32) ? 0xffffffffu : ((1u << k) - 1u);
  const unsigned avail = ~mask & all;
  if (avail == 0u) { S.hi[s] = 0u; return; }
  const int j0 = __ffs(avail) - 1;
  const float* row_lp = lp + d * k;
  const int* row_id = ids + d * k;
  const float best_sc = base + row_lp[j0];
  int best_j = j0, best_tok = row_id[j0];
  for (int j = j0 + 1; j < k; ++j) {
    const float sc = base + row_lp[j];
    if (sc < best_sc) break;
    if (!((mask >> j) & 1u) && row_id[j] < best_tok) { best_j = j; best_tok = row_id[j]; }
  }
  S.hi[s] = f32_ord(best_sc);
  S.lo[s] = ((0x3FFFFFu - static_cast<unsigned>(best_tok)) << 10) | (0x3FFu - static_cast<unsigned>(s));
  S.j[s] = best_j;
}

template <int KM>
__global__ void __launch_bounds__(kMergeThreads) merge_tree_kernel(const TreeParams p) {
  constexpr int F = 2 + 2 * KM;
  constexpr int kWarps = kMergeThreads / 32;
  __shared__ float s_mx[kWarps], s_se[kWarps];
  __shared__ int s_last;
  __shared__ float s_cv[kWarps * kMaxTopk];
  __shared__ int s_ci[kWarps * kMaxTopk];
  __shared__ float s_lp[kMaxK * kMaxTopk];
  __shared__ int s_id[kMaxK * kMaxTopk];
  __shared__ TreeSlots S;

  const int m = blockIdx.x;
  const int K = p.K, k = p.k, N = p.N, nch = p.nchunks;
  const int b = m / K;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // launched as a programmatic dependent of the vocabulary GEMM: wait for its partials
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const float* base = p.partials + static_cast<size_t>(m) * F * nch;
  const int* ibase = reinterpret_cast<const int*>(base);

  // ------------------------------------------------------------ this thread's chunks
  float mx = -INFINITY, se = 0.f;
  float tv[KM];
  int ti[KM];
#pragma unroll
  for (int q = 0; q < KM; ++q) { tv[q] = -INFINITY; ti[q] = -1; }
  for (int c = tid; c < nch; c += kMergeThreads) {
    const float cm = __ldg(base + c), cs = __ldg(base + nch + c);
    float v[KM];
    int id[KM];
#pragma unroll
    for (int q = 0; q < KM; ++q) {
      v[q] = __ldg(base + (2 + q) * nch + c);
      id[q] = __ldg(ibase + (2 + KM + q) * nch + c);
    }
    lse_merge(mx, se, cm, cs);
    if (c == tid) {
#pragma unroll
      for (int q = 0; q < KM; ++q) { tv[q] = v[q]; ti[q] = id[q]; }
    } else {
#pragma unroll
      for (int q = 0; q < KM; ++q) insert_keyed<KM>(tv, ti, v[q], id[q]);
    }
  }

  // ------------------------------------------------------------ lse over the CTA
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, mx, o);
    const float os = __shfl_xor_sync(0xffffffffu, se, o);
    lse_merge(mx, se, om, os);
  }
  if (lane == 0) { s_mx[warp] = mx; s_se[warp] = se; }
  __syncthreads();
  mx = -INFINITY;
  se = 0.f;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) lse_merge(mx, se, s_mx[w], s_se[w]);
  const float lse = mx + logf(se);

  // ------------------------------------------------------------ k best: per warp, then across warps
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
    if (lane == 0) { s_cv[warp * kMaxTopk + q] = val; s_ci[warp * kMaxTopk + q] = id; }
  }
  __syncthreads();
  if (warp == 0) {
    int ptr = 0;  // lane w < kWarps walks warp w's sorted candidate list
    for (int q = 0; q < k; ++q) {
      uint32_t hi = 0u, lo = 0u;
      if (lane < kWarps && ptr < k) {
        hi = f32_ord(s_cv[lane * kMaxTopk + ptr]);
        lo = ~static_cast<uint32_t>(s_ci[lane * kMaxTopk + ptr]);
      }
      uint32_t mhi, mlo;
      int src;
      warp_argmax2(hi, lo, mhi, mlo, src);
      if (lane == src) {
        p.topk_ids[static_cast<size_t>(m) * k + q] = s_ci[lane * kMaxTopk + ptr];
        p.topk_logp[static_cast<size_t>(m) * k + q] = s_cv[lane * kMaxTopk + ptr] - lse;
        ++ptr;
      }
    }
  }

  // ------------------------------------------------------------ last row of the sequence?
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(p.seq_done + b, 1u) == static_cast<unsigned>(K - 1));
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const size_t rows = static_cast<size_t>(b) * K * k;
  for (int e = tid; e < K * k; e += kMergeThreads) {
    s_id[e] = __ldcg(p.topk_ids + rows + e);
    s_lp[e] = __ldcg(p.topk_logp + rows + e);
  }
  __syncthreads();
  if (warp != 0) return;

  // ------------------------------------------------------------ tree (warp 0)
  const size_t ob = static_cast<size_t>(b) * N;
  if (lane == 0) {
    S.score[0] = 0.f;
    S.depth[0] = 0;
    S.mask[0] = 0u;
    refresh_slot(S, 0, 0, 0.f, 0u, s_lp, s_id, K, k);
  }
  __syncwarp();
  for (int i = 0; i < N; ++i) {
    uint32_t hi = 0u, lo = 0u;
    int sb = -1;
    for (int s2 = lane; s2 <= i; s2 += 32) {
      const uint32_t h = S.hi[s2], l = S.lo[s2];
      if (h > hi || (h == hi && h != 0u && l > lo)) { hi = h; lo = l; sb = s2; }
    }
    uint32_t mhi, mlo;
    int src;
    warp_argmax2(hi, lo, mhi, mlo, src);
    const int s = __shfl_sync(0xffffffffu, sb, src);
    if (lane == 0) {
      const int jj = S.j[s];
      const int d = S.depth[s];
      const float base_s = S.score[s];
      const unsigned mask_s = S.mask[s] | (1u << jj);
      const int tok = s_id[d * k + jj];
      const float sc = base_s + s_lp[d * k + jj];
      p.tree_parent[ob + i] = s - 1;
      p.tree_token[ob + i] = tok;
      p.tree_depth[ob + i] = d + 1;
      if (p.tree_score) p.tree_score[ob + i] = sc;
      S.mask[s] = mask_s;
      S.score[i + 1] = sc;
      S.depth[i + 1] = d + 1;
      S.mask[i + 1] = 0u;
      refresh_slot(S, s, d, base_s, mask_s, s_lp, s_id, K, k);
      refresh_slot(S, i + 1, d + 1, sc, 0u, s_lp, s_id, K, k);
    }
    __syncwarp();
  }
}

cudaError_t launch_merge_tree(const TreeParams& p, cudaStream_t stream) {
  if (p.K > kMaxK || p.k > kMaxTopk || p.N > kMaxN) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.B * p.K);
  cfg.blockDim = dim3(kMergeThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = DOMINO_TREE_PDL ? 1 : 0;
  cudaError_t e;
  if (p.kmax == 16) e = cudaLaunchKernelEx(&cfg, merge_tree_kernel<16>, p);
  else if (p.kmax == 32) e = cudaLaunchKernelEx(&cfg, merge_tree_kernel<32>, p);
  else return cudaErrorInvalidValue;
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dm
