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

}  // namespace dm
