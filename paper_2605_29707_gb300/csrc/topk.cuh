// topk.cuh -- merging of best-first (value desc, id asc) candidate lists held in registers.
#pragma once

namespace dm {

// Total order of (logit, token) candidates: greater logit first, then lower token id.  Padding
// entries carry (-inf, -1), which sorts after every real entry.
__device__ __forceinline__ bool better(float a, int ia, float b, int ib) {
  return a > b || (a == b && static_cast<unsigned>(ia) < static_cast<unsigned>(ib));
}

// Sort a bitonic sequence best-first (half-cleaners of decreasing span).
template <int KK>
__device__ __forceinline__ void bitonic_clean(float (&v)[KK], int (&id)[KK]) {
#pragma unroll
  for (int h = KK / 2; h > 0; h >>= 1) {
#pragma unroll
    for (int q = 0; q < KK; ++q) {
      if ((q & h) == 0) {
        const int r = q + h;
        const bool keep = better(v[q], id[q], v[r], id[r]);
        const float a = v[q], b = v[r];
        const int ia = id[q], ib = id[r];
        v[q] = keep ? a : b;
        id[q] = keep ? ia : ib;
        v[r] = keep ? b : a;
        id[r] = keep ? ib : ia;
      }
    }
  }
}

// (v, id) <- best KK of the union of two best-first lists: the half-cleaner of a ++ reverse(b)
// keeps the KK best as a bitonic sequence, which bitonic_clean sorts.  Depth 1 + log2(KK)
// compare-exchange stages, each of independent pairs.
template <int KK>
__device__ __forceinline__ void merge_lists(float (&v)[KK], int (&id)[KK], const float (&w)[KK], const int (&iw)[KK]) {
#pragma unroll
  for (int q = 0; q < KK; ++q) {
    const float b = w[KK - 1 - q];
    const int ib = iw[KK - 1 - q];
    const bool keep = better(v[q], id[q], b, ib);
    v[q] = keep ? v[q] : b;
    id[q] = keep ? id[q] : ib;
  }
  bitonic_clean<KK>(v, id);
}

// Sort KK candidates best-first (bitonic sorting network, depth log2(KK)(log2(KK)+1)/2).
template <int KK>
__device__ __forceinline__ void bitonic_sort(float (&v)[KK], int (&id)[KK]) {
#pragma unroll
  for (int size = 2; size <= KK; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
#pragma unroll
      for (int q = 0; q < KK; ++q) {
        const int r = q ^ stride;
        if (r > q) {
          // blocks with (q & size) == 0 end best-first, the others worst-first; the last
          // pass (size == KK) leaves the whole array best-first
          const bool q_better = better(v[q], id[q], v[r], id[r]);
          const bool sw = ((q & size) == 0) ? !q_better : q_better;
          const float a = v[q], b = v[r];
          const int ia = id[q], ib = id[r];
          v[q] = sw ? b : a;
          id[q] = sw ? ib : ia;
          v[r] = sw ? a : b;
          id[r] = sw ? ia : ib;
        }
      }
    }
  }
}

}  // namespace dm
